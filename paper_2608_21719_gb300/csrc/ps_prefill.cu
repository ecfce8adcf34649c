// ps_prefill.cu -- chunked-prefill attention over the paged KV cache on the
// 5th-generation tensor cores (tcgen05 + TMEM), sm_103a.
//
// The prefill phase (PowerSlider Sec. 2.2) attends every new prompt token
// causally over its sequence's cache; unlike decode it is a dense
// contraction with high arithmetic intensity (Sec. 3 Obs. 2, App. B: the
// intensity grows with the number of tokens processed together).  Sequence s
// has L_s cached tokens whose last Q_s are the new (query) tokens; query i sits
// at position p = L_s - Q_s + i and sees keys 0 .. p.
//
// Tiling.  One CTA per (query tile, KV head j, sequence s).  A query tile is
// 128 MMA rows: 128 / g consecutive query tokens times the g query heads of
// group j (row = token * g + head), so every K/V tile staged in shared memory
// serves the whole group.  Keys stream in tiles of 128 through shared-memory
// rings; every 16-key chunk of a tile comes from one (block, kv-head) page of
// the cache, addressed through the block table: for K as two TMA boxes (its
// 64-column halves, stored [half][key][64], the K-major layout Q K^T needs),
// for V as one box holding both halves ([chunk][half][16][64]; V is the
// MN-major operand of P V, whose 64-column groups may sit 2 KiB apart), which
// halves V's copies per tile.
//
// Per key tile n (warp roles, 7 warps):
//   warps 0, 6 TMA producers: Q once and K_n into a three-stage ring (warp 0),
//              V_n into a three-stage ring (warp 6).  A K stage is released
//              as soon as its Q K^T has run, a V stage once its P V has run.
//   warp 1     MMA issuer (one thread): S_n = Q K_n^T into one of two TMEM
//              score buffers (M = 128, N = 128, K = 128), then, once the
//              softmax has written P_{n-1}, O += P_{n-1} V_{n-1} with P read
//              from TMEM and V (MN-major) from shared memory, into the TMEM
//              output accumulator.  Completion is signalled with
//              tcgen05.commit on mbarriers.
//   warps 2-5  softmax, one TMEM lane (= one row) per thread: load the score
//              row, mask it causally, update the running max m and sum l in
//              fp32 (base 2, log2 e folded into the scale), write the bf16
//              probabilities into TMEM P buffer n & 1 (the A operand of the
//              P V MMA), and rescale the output row in TMEM when the max has
//              grown.  Only that rescale waits for the previous P V, so the
//              exponentials of tile n+1 overlap the P V of tile n.
// The rescale is lazy: the reference max m only moves when the tile max
// exceeds it by more than 2^8, so P <= 256 and no value leaves fp32/bf16
// range; the final O / l is the same quotient whichever reference max was
// used.  The QK^T of tile n+1 runs on the tensor cores while the softmax works
// on tile n.
//
// Every mbarrier wait gives up after ~2 s of globaltimer, or at once when
// another role has given up, and raises PS_DEVICE_TIMEOUT in the optional
// device status word; the producer then waits for its own copies, the MMA
// issuer for its own MMAs, and TMEM is freed on every path.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <mutex>

#include "ps_decode.h"
#include "ps_internal.h"

namespace {

constexpr int kD = 128;            // head_dim
constexpr int kRows = 128;         // MMA M: query rows per tile
constexpr int kKeys = 128;         // MMA N of S, K of P.V: keys per tile
constexpr int kChunk = 16;         // keys per TMA box (one page slice)
#ifndef PS_PREFILL_KSTAGES
#define PS_PREFILL_KSTAGES 3
#endif
#ifndef PS_PREFILL_VSTAGES
#define PS_PREFILL_VSTAGES 3
#endif
constexpr int kKStages = PS_PREFILL_KSTAGES;  // K ring: a stage is free once its Q K^T is done
constexpr int kVStages = PS_PREFILL_VSTAGES;  // V ring: a stage is free once its P V is done
constexpr int kThreads = 224;
constexpr int kHalf = kRows * 64 * 2;   // one 64-column half of a 128-row tile: 16 KiB
constexpr int kTile = 2 * kHalf;        // 32 KiB
constexpr int kOffQ = 0;
constexpr int kOffK = kOffQ + kTile;
constexpr int kOffV = kOffK + kKStages * kTile;
constexpr int kOffBar = kOffV + kVStages * kTile;
constexpr int kSmemBytes = 1024 + kOffBar + 256;  // 1 KiB of alignment slack
static_assert(kSmemBytes <= 227 * 1024, "shared memory");
constexpr uint32_t kTmemCols = 512;
// TMEM columns: S buffers at 0 and 128, O at 256, two P buffers (bf16 pairs
// packed in 32-bit columns, 64 columns each) at 384 and 448.
constexpr uint32_t kColO = 256, kColP = 384;
constexpr float kRescaleLog2 = 8.0f;
constexpr unsigned long long kWaitLimitNs = 2000000000ull;

struct PrefillParams {
    const int *block_table, *seq_lens, *q_start;
    uint16_t *out;
    unsigned *status;
    int num_seqs, total_q, num_q_heads, num_kv_heads, group, tokens_per_tile, num_qtiles;
    int block_size, max_blocks_per_seq;
    long long num_blocks;
    float scale_log2;
};

// ------------------------------------------------------------ PTX wrappers --

__device__ __forceinline__ uint32_t saddr(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *tm, int c0, int c1, int c2,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(c2), "r"(bar)
        : "memory");
}
// The same with an L2 cache-policy hint (from createpolicy).
__device__ __forceinline__ void tma_load_4d_hint(uint32_t dst, const CUtensorMap *tm, int c0, int c1, int c2, int c3,
                                                 uint32_t bar, uint64_t policy) {
    asm volatile("cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%2, %3, %4, %5}], [%6], %7;" ::"r"(dst), "l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1),
        "r"(c2), "r"(c3), "r"(bar), "l"(policy) : "memory");
}

__device__ __forceinline__ void tma_load_3d_hint(uint32_t dst, const CUtensorMap *tm, int c0, int c1, int c2,
                                                 uint32_t bar, uint64_t policy) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.L2::cache_hint"
        " [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(c2), "r"(bar), "l"(policy)
        : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
// Shared-memory matrix descriptor, 128-byte swizzle (sm_100 family format):
// start address, leading and stride byte offsets in 16-byte units, version 1.
__device__ __forceinline__ uint64_t smem_desc(uint32_t addr, uint32_t lbo, uint32_t sbo) {
    return (uint64_t)((addr >> 4) & 0x3FFF) | ((uint64_t)((lbo >> 4) & 0x3FFF) << 16) |
           ((uint64_t)((sbo >> 4) & 0x3FFF) << 32) | (1ull << 46) | (2ull << 61);
}
// Instruction descriptor of kind::f16: f32 accumulator, bf16 A and B, A
// K-major, B K-major (b_mn = 0) or MN-major (b_mn = 1), shape M x N.
__host__ __device__ constexpr uint32_t instr_desc(int m, int n, int b_mn) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)b_mn << 16) | ((uint32_t)(n >> 3) << 17) |
           ((uint32_t)(m >> 4) << 24);
}
__device__ __forceinline__ void umma(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}
// The same with A read from tensor memory (row = TMEM lane, K packed in bf16
// pairs along the columns: a K step of 16 is 8 columns).
__device__ __forceinline__ void umma_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}
__device__ __forceinline__ void umma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float *v) {
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_st16u(uint32_t taddr, const uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]), "r"(v[8]), "r"(v[9]),
        "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15])
        : "memory");
}
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const float (&v)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
        "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
        "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
        "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
        "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
        "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
        "r"(__float_as_uint(v[15])), "r"(__float_as_uint(v[16])), "r"(__float_as_uint(v[17])),
        "r"(__float_as_uint(v[18])), "r"(__float_as_uint(v[19])), "r"(__float_as_uint(v[20])),
        "r"(__float_as_uint(v[21])), "r"(__float_as_uint(v[22])), "r"(__float_as_uint(v[23])),
        "r"(__float_as_uint(v[24])), "r"(__float_as_uint(v[25])), "r"(__float_as_uint(v[26])),
        "r"(__float_as_uint(v[27])), "r"(__float_as_uint(v[28])), "r"(__float_as_uint(v[29])),
        "r"(__float_as_uint(v[30])), "r"(__float_as_uint(v[31]))
        : "memory");
}
__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
// Registers written by tcgen05.ld are only valid after tcgen05.wait::ld.  The
// loads and the wait are volatile asm, which the compiler keeps in order;
// passing every loaded value through an empty volatile asm after the wait
// keeps their first uses behind it too.
template <int N>
__device__ __forceinline__ void tmem_loaded(float *v) {
#pragma unroll
    for (int i = 0; i < N; ++i) asm volatile("" : "+f"(v[i]));
}
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Bounded wait; also returns false as soon as another role raised `abort`.
__device__ __forceinline__ bool wait_phase(uint32_t bar, uint32_t parity, volatile int *abort, unsigned *status) {
    for (int i = 0; i < 64; ++i)
        if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (*abort) return false;
        if (global_ns() - t0 > kWaitLimitNs) {
            *abort = 1;
            if (status) atomicOr(status, (unsigned)PS_DEVICE_TIMEOUT);
            return false;
        }
    }
    return true;
}
// The same, taken by a whole warp: every lane waits and the warp agrees on
// the outcome, so the warp stays converged for .sync.aligned instructions.
__device__ __forceinline__ bool warp_wait(uint32_t bar, uint32_t parity, volatile int *abort, unsigned *status) {
    return __all_sync(0xffffffffu, wait_phase(bar, parity, abort, status));
}
// Bounded wait without the abort shortcut: used to drain this thread's own
// copies and MMAs, which complete whatever the other roles did.
__device__ __forceinline__ void drain_phase(uint32_t bar, uint32_t parity) {
    const unsigned long long t0 = global_ns();
    while (!mbar_try_wait(bar, parity))
        if (global_ns() - t0 > kWaitLimitNs) return;
}


__global__ void __launch_bounds__(kThreads, 1)
    ps_prefill_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV, const PrefillParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    // Consecutive CTAs share a (sequence, KV head), heaviest (last) query
    // tile first: the few K/V streams in flight at a time stay in L2.
    const int qt = p.num_qtiles - 1 - (int)blockIdx.x;
    const int j = blockIdx.y, s = blockIdx.z;
    const int g = p.group, tpt = p.tokens_per_tile;

    // Sequence geometry (uniform over the CTA).
    const int qs0 = __ldg(p.q_start + s), qs1 = __ldg(p.q_start + s + 1);
    const int Q = qs1 - qs0;
    const int L = __ldg(p.seq_lens + s);
    const int tok0 = qt * tpt;
    // max_q_len below a chunk leaves that chunk's later rows uncovered.
    if (qt == p.num_qtiles - 1 && j == 0 && tid == 0 && Q > p.num_qtiles * tpt && p.status)
        atomicOr(p.status, (unsigned)PS_DEVICE_LEN_CLAMPED);
    if (tok0 >= Q) return;
    const long long cap = (long long)p.max_blocks_per_seq * p.block_size;
    if (Q < 0 || L < Q || (long long)L > cap || qs0 < 0 || qs1 > p.total_q) {
        if (tid == 0 && j == 0 && p.status) atomicOr(p.status, (unsigned)PS_DEVICE_LEN_CLAMPED);
        return;
    }
    const int tok_end = min(Q, tok0 + tpt);
    const int kv_limit = L - Q + tok_end;  // keys this tile needs: [0, kv_limit)
    const int ntiles = (kv_limit + kKeys - 1) / kKeys;

    uint64_t *bars = reinterpret_cast<uint64_t *>(sm + kOffBar);
    const uint32_t bar_q = saddr(bars + 0);
    auto bar_kfull = [&](int st) { return saddr(bars + 1 + st); };                        // [kKStages]
    auto bar_kfree = [&](int st) { return saddr(bars + 1 + kKStages + st); };             // [kKStages]
    auto bar_vfull = [&](int st) { return saddr(bars + 1 + 2 * kKStages + st); };         // [kVStages]
    auto bar_vfree = [&](int st) { return saddr(bars + 1 + 2 * kKStages + kVStages + st); };
    constexpr int kB = 1 + 2 * kKStages + 2 * kVStages;
    auto bar_sfull = [&](int b) { return saddr(bars + kB + b); };
    auto bar_sfree = [&](int b) { return saddr(bars + kB + 2 + b); };
    auto bar_pfull = [&](int b) { return saddr(bars + kB + 4 + b); };
    auto bar_pfree = [&](int b) { return saddr(bars + kB + 6 + b); };
    const uint32_t bar_mma_end = saddr(bars + kB + 8);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + kB + 9);
    volatile int *abort = reinterpret_cast<volatile int *>(bars + kB + 10);
    static_assert((1 + 2 * kKStages + 2 * kVStages + 11) * 8 <= 256, "barrier area");

    if (tid == 0) {
        mbar_init(bar_q, 1);
        for (int i = 0; i < kKStages; ++i) {
            mbar_init(bar_kfull(i), 1);
            mbar_init(bar_kfree(i), 1);
        }
        for (int i = 0; i < kVStages; ++i) {
            mbar_init(bar_vfull(i), 1);
            mbar_init(bar_vfree(i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar_sfull(i), 1);
            mbar_init(bar_sfree(i), 4);
            mbar_init(bar_pfull(i), 128);
            mbar_init(bar_pfree(i), 1);
        }
        mbar_init(bar_mma_end, 1);
        *abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(saddr(tmem_slot)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    const uint32_t sQ = saddr(sm + kOffQ), sK = saddr(sm + kOffK), sV = saddr(sm + kOffV);

    if (warp == 0 || warp == 6) {
        // ----------------------------------------------------- producers --
        const bool is_k = warp == 0;
        if (is_k && lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmQ)) : "memory");
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
            mbar_expect_tx(bar_q, (uint32_t)(2 * 128 * g * tpt));
            tma_load_3d(sQ, &tmQ, 0, j * g, qs0 + tok0, bar_q);
            tma_load_3d(sQ + kHalf, &tmQ, 64, j * g, qs0 + tok0, bar_q);
        }
        if (!is_k && lane == 0)
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
        const int stages = is_k ? kKStages : kVStages;
        const uint32_t ring = is_k ? sK : sV;
        const CUtensorMap *tm = is_k ? &tmK : &tmV;
        const int *bt_row = p.block_table + (size_t)s * p.max_blocks_per_seq;
        const int half = (lane >> 3) & 1, c = lane & 7;  // K: lanes 0-15, 8 chunks x 2 halves; V: lanes 0-7
        // Every K/V page is read by all query tiles of its (sequence, head):
        // ask L2 to keep it (evict last).
        uint64_t keep;
        asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(keep));
        int issued = 0;
        for (int n = 0; n < ntiles; ++n) {
            const int st = n % stages, use = n / stages;
            if (n >= stages &&
                !warp_wait(is_k ? bar_kfree(st) : bar_vfree(st), (use - 1) & 1, abort, p.status))
                break;
            const int base = n * kKeys;
            const int nc = (min(kKeys, kv_limit - base) + kChunk - 1) / kChunk;
            const uint32_t full = is_k ? bar_kfull(st) : bar_vfull(st);
            if (lane == 0) mbar_expect_tx(full, (uint32_t)(nc * 2 * kChunk * 128));
            __syncwarp();
            if (is_k ? (lane < 16 && c < nc) : (lane < nc)) {
                const int cc = is_k ? c : lane;
                const int t0 = base + cc * kChunk;
                const int lb = t0 / p.block_size;
                const int b = __ldg(bt_row + lb);
                int page = -1;  // out of range: TMA fills zeros
                if (b >= 0 && (long long)b < p.num_blocks) page = b * p.num_kv_heads + j;
                else if (p.status && is_k) atomicOr(p.status, (unsigned)PS_DEVICE_BAD_BLOCK);
                if (is_k)
                    tma_load_3d_hint(ring + st * kTile + half * kHalf + cc * (kChunk * 128), tm, half * 64,
                                     t0 - lb * p.block_size, page, full, keep);
                else  // both 64-column halves of the chunk in one box: [half][16][64]
                    tma_load_4d_hint(ring + st * kTile + cc * (2 * kChunk * 128), tm, 0, t0 - lb * p.block_size, 0,
                                     page, full, keep);
            }
            issued = n + 1;
        }
        // Drain: the last copies of each stage must land before the CTA exits.
        for (int n = max(0, issued - stages); n < issued; ++n)
            drain_phase(is_k ? bar_kfull(n % stages) : bar_vfull(n % stages), (n / stages) & 1);
        if (is_k) drain_phase(bar_q, 0);
    } else if (warp == 1) {
        // ---------------------------------------------------- MMA issuer --
        constexpr uint32_t idS = instr_desc(kRows, kKeys, 0);
        constexpr uint32_t idO = instr_desc(kRows, kD, 1);
        bool ok = warp_wait(bar_q, 0, abort, p.status);
        for (int n = 0; ok && n <= ntiles; ++n) {
            if (n < ntiles) {
                const int st = n % kKStages, b = n & 1;
                if (!warp_wait(bar_kfull(st), (n / kKStages) & 1, abort, p.status)) { ok = false; break; }
                if (n >= 2 && !warp_wait(bar_sfree(b), ((n >> 1) - 1) & 1, abort, p.status)) { ok = false; break; }
                tc_fence_after();
                if (lane == 0) {
                    const uint32_t kb = sK + st * kTile;
#pragma unroll
                    for (int kk = 0; kk < kD / 16; ++kk) {
                        const uint32_t off = (kk >> 2) * kHalf + (kk & 3) * 32;
                        umma(tmem + b * kKeys, smem_desc(sQ + off, 16, 1024), smem_desc(kb + off, 16, 1024), idS,
                             kk > 0);
                    }
                    umma_commit(bar_sfull(b));
                    umma_commit(bar_kfree(st));
                }
                __syncwarp();
            }
            if (n >= 1) {
                const int m = n - 1, st = m % kVStages;
                if (!warp_wait(bar_vfull(st), (m / kVStages) & 1, abort, p.status)) { ok = false; break; }
                const uint32_t vb = sV + st * kTile;
                const int valid = kv_limit - m * kKeys;
                if (valid < kKeys) {
                    // Rows past the last needed key hold other tokens' data
                    // or stale bytes; P is zero there, so make V zero too.
                    uint8_t *v = sm + kOffV + st * kTile;
                    const int nvec = (kKeys - valid) * 8;
                    for (int e = lane; e < 2 * nvec; e += 32) {
                        const int h = e / nvec, r = e - h * nvec;
                        const int key = valid + (r >> 3);
                        *reinterpret_cast<uint4 *>(v + (key >> 4) * (2 * kChunk * 128) + h * (kChunk * 128) +
                                                   (key & 15) * 128 + (r & 7) * 16) = make_uint4(0, 0, 0, 0);
                    }
                    fence_proxy_async_smem();
                    __syncwarp();
                }
                if (!warp_wait(bar_pfull(m & 1), (m >> 1) & 1, abort, p.status)) { ok = false; break; }
                tc_fence_after();
                if (lane == 0) {
                    const uint32_t pt = tmem + kColP + (m & 1) * (kKeys / 2);
#pragma unroll
                    for (int kk = 0; kk < kKeys / 16; ++kk)
                        umma_ts(tmem + kColO, pt + kk * 8, smem_desc(vb + kk * 4096, 2048, 1024), idO,
                                (m > 0 || kk > 0) ? 1u : 0u);
                    umma_commit(bar_pfree(m & 1));
                    umma_commit(bar_vfree(st));
                }
                __syncwarp();
            }
        }
        // Every MMA issued above has finished before TMEM and smem go away.
        if (lane == 0) umma_commit(bar_mma_end);
        __syncwarp();
        drain_phase(bar_mma_end, 0);
    } else {
        // ------------------------------------------------------- softmax --
        const int quarter = warp & 3;  // TMEM lanes 32 * quarter .. + 31
        const int r = quarter * 32 + lane;
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
        const int tl = r / g, hl = r - tl * g;
        const bool row_valid = (tl < tpt) && (tok0 + tl < Q);
        const int limit = row_valid ? (L - Q + tok0 + tl + 1) : kv_limit;
        const float sl2 = p.scale_log2;
        float m_ref = -INFINITY, l = 0.f;
        bool ok = true;
        for (int n = 0; n < ntiles; ++n) {
            const int b = n & 1;
            if (!warp_wait(bar_sfull(b), (n >> 1) & 1, abort, p.status)) { ok = false; break; }
            tc_fence_after();
            float sv[kKeys];
#pragma unroll
            for (int c = 0; c < 4; ++c) tmem_ld32(trow + b * kKeys + c * 32, sv + c * 32);
            tmem_wait_ld();
            tmem_loaded<kKeys>(sv);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_sfree(b));
            const int base = n * kKeys;
            if (base + kKeys > limit) {
#pragma unroll
                for (int i = 0; i < kKeys; ++i)
                    if (base + i >= limit) sv[i] = -INFINITY;
            }
            float mx = sv[0];
#pragma unroll
            for (int i = 1; i < kKeys; ++i) mx = fmaxf(mx, sv[i]);
            const float m_tile = mx * sl2;
            const bool grow = m_tile > m_ref + kRescaleLog2;  // always true on the first tile
            const float alpha = grow ? ex2(m_ref - m_tile) : 1.f;
            if (n >= 1 && __any_sync(0xffffffffu, grow)) {
                // O must hold key tiles 0 .. n-1 before it is rescaled.
                if (!warp_wait(bar_pfree((n - 1) & 1), ((n - 1) >> 1) & 1, abort, p.status)) { ok = false; break; }
                tc_fence_after();
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    float ov[32];
                    tmem_ld32(trow + kColO + c * 32, ov);
                    tmem_wait_ld();
                    tmem_loaded<32>(ov);
#pragma unroll
                    for (int i = 0; i < 32; ++i) ov[i] *= alpha;
                    tmem_st32(trow + kColO + c * 32, ov);
                }
                tmem_wait_st();
            }
            if (grow) {
                l *= alpha;
                m_ref = m_tile;
            }
            // P buffer b was last read by the P V of tile n - 2.
            if (n >= 2) {
                if (!warp_wait(bar_pfree(b), ((n >> 1) - 1) & 1, abort, p.status)) { ok = false; break; }
                tc_fence_after();
            }
            // P row (bf16 pairs) into TMEM buffer b, row = this thread's lane:
            // the A operand of the P V MMA.
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                uint32_t w[16];
#pragma unroll
                for (int e = 0; e < 16; ++e) {
                    const int i = c * 32 + 2 * e;
                    const __nv_bfloat162 pr =
                        __floats2bfloat162_rn(ex2(fmaf(sv[i], sl2, -m_ref)), ex2(fmaf(sv[i + 1], sl2, -m_ref)));
                    const float2 back = __bfloat1622float2(pr);
                    l += back.x + back.y;
                    w[e] = *reinterpret_cast<const uint32_t *>(&pr);
                }
                tmem_st16u(trow + kColP + b * (kKeys / 2) + c * 16, w);
            }
            tmem_wait_st();
            tc_fence_before();
            mbar_arrive(bar_pfull(b));
        }
        if (ok && warp_wait(bar_pfree((ntiles - 1) & 1), ((ntiles - 1) >> 1) & 1, abort, p.status)) {
            tc_fence_after();
            const float inv = 1.f / l;
            uint16_t *orow = p.out + ((size_t)(qs0 + tok0 + tl) * p.num_q_heads + (size_t)j * g + hl) * kD;
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                float ov[32];
                tmem_ld32(trow + kColO + c * 32, ov);
                tmem_wait_ld();
                tmem_loaded<32>(ov);
                if (row_valid) {
#pragma unroll
                    for (int v = 0; v < 4; ++v) {
                        uint32_t w[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const __nv_bfloat162 pr = __floats2bfloat162_rn(ov[v * 8 + 2 * e] * inv, ov[v * 8 + 2 * e + 1] * inv);
                            w[e] = *reinterpret_cast<const uint32_t *>(&pr);
                        }
                        *reinterpret_cast<uint4 *>(orow + c * 32 + v * 8) = make_uint4(w[0], w[1], w[2], w[3]);
                    }
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
    }
}

// ------------------------------------------------------------------ host --

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encoder() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *f = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(f);
    });
    return fn;
}

bool encode3d(CUtensorMap *tm, const void *base, cuuint64_t d1, cuuint64_t d2, cuuint32_t b1, cuuint32_t b2) {
    EncodeTiledFn fn = encoder();
    if (!fn) return false;
    cuuint64_t dims[3] = {(cuuint64_t)kD, d1, d2};
    cuuint64_t strides[2] = {(cuuint64_t)kD * 2, d1 * kD * 2};
    cuuint32_t box[3] = {64, b1, b2};
    cuuint32_t estr[3] = {1, 1, 1};
    return fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// V as [page][slot][half][64]: dims (64, slot, half, page) with the half
// stride (128 B) inside the slot stride (256 B), so that one box {64, 16, 2}
// lands as [half][16][64] (both halves of a 16-key chunk in one copy).
bool encode_v4d(CUtensorMap *tm, const void *base, cuuint64_t bs, cuuint64_t pages) {
    EncodeTiledFn fn = encoder();
    if (!fn) return false;
    cuuint64_t dims[4] = {64, bs, 2, pages};
    cuuint64_t strides[3] = {(cuuint64_t)kD * 2, 64 * 2, bs * kD * 2};
    cuuint32_t box[4] = {64, kChunk, 2, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    return fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15) == 0; }

}  // namespace

extern "C" ps_status_t ps_prefill_attention(const void *q, const void *k_cache, const void *v_cache,
                                            const int *block_table, const int *seq_lens, const int *q_start,
                                            void *out, int num_seqs, int total_q_tokens, int max_q_len,
                                            int num_q_heads, int num_kv_heads, int head_dim, int block_size,
                                            int max_blocks_per_seq, long long num_blocks, float scale,
                                            unsigned int *device_status, void *stream) {
    if (!q || !k_cache || !v_cache || !block_table || !seq_lens || !q_start || !out) return PS_ERR_INVALID_ARG;
    if (!aligned16(q) || !aligned16(k_cache) || !aligned16(v_cache) || !aligned16(out)) return PS_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(block_table) & 3) || (reinterpret_cast<uintptr_t>(seq_lens) & 3) ||
        (reinterpret_cast<uintptr_t>(q_start) & 3) || (reinterpret_cast<uintptr_t>(device_status) & 3))
        return PS_ERR_INVALID_ARG;
    if (num_seqs < 0 || total_q_tokens < 0 || max_q_len < 0 || max_q_len > total_q_tokens ||
        num_q_heads <= 0 || num_kv_heads <= 0 || head_dim <= 0 || block_size <= 0 || max_blocks_per_seq <= 0 ||
        num_blocks <= 0 || num_q_heads % num_kv_heads != 0 || !std::isfinite(scale))
        return PS_ERR_INVALID_ARG;
    const int g = num_q_heads / num_kv_heads;
    if (head_dim != kD || g > 16 || block_size % kChunk != 0) return PS_ERR_UNSUPPORTED;
    if ((long long)max_blocks_per_seq * block_size > INT32_MAX || num_blocks * num_kv_heads > INT32_MAX ||
        num_seqs > 65535)
        return PS_ERR_UNSUPPORTED;
    if (num_seqs == 0 || total_q_tokens == 0 || max_q_len == 0) return PS_OK;
    const int tpt = kRows / g;
    const long long nqt = (max_q_len + tpt - 1) / tpt;
    if (nqt > 65535) return PS_ERR_UNSUPPORTED;

    CUtensorMap tmQ, tmK, tmV;
    if (!encode3d(&tmQ, q, (cuuint64_t)num_q_heads, (cuuint64_t)total_q_tokens, (cuuint32_t)g, (cuuint32_t)tpt) ||
        !encode3d(&tmK, k_cache, (cuuint64_t)block_size, (cuuint64_t)(num_blocks * num_kv_heads), kChunk, 1) ||
        !encode_v4d(&tmV, v_cache, (cuuint64_t)block_size, (cuuint64_t)(num_blocks * num_kv_heads)))
        return PS_ERR_CUDA;
    // The shared-memory limit is a per-device function attribute: set it for
    // the current device on every call (cheap), so that a process driving
    // several GPUs works on each of them.
    if (cudaFuncSetAttribute(ps_prefill_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) !=
        cudaSuccess)
        return PS_ERR_CUDA;

    PrefillParams pp;
    pp.block_table = block_table;
    pp.seq_lens = seq_lens;
    pp.q_start = q_start;
    pp.out = static_cast<uint16_t *>(out);
    pp.status = device_status;
    pp.num_seqs = num_seqs;
    pp.total_q = total_q_tokens;
    pp.num_q_heads = num_q_heads;
    pp.num_kv_heads = num_kv_heads;
    pp.group = g;
    pp.tokens_per_tile = tpt;
    pp.num_qtiles = (int)nqt;
    pp.block_size = block_size;
    pp.max_blocks_per_seq = max_blocks_per_seq;
    pp.num_blocks = num_blocks;
    pp.scale_log2 = scale * 1.4426950408889634f;
    const dim3 grid((unsigned)nqt, (unsigned)num_kv_heads, (unsigned)num_seqs);
    if (ps::take_injected_launch_error() != cudaSuccess) return PS_ERR_CUDA;
    ps_prefill_kernel<<<grid, kThreads, kSmemBytes, reinterpret_cast<cudaStream_t>(stream)>>>(tmQ, tmK, tmV, pp);
    if (cudaGetLastError() != cudaSuccess) return PS_ERR_CUDA;
    ps::note_launch();
    return PS_OK;
}
