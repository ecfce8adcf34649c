// ps_prefill.cu -- chunked-prefill attention over the paged KV cache on the
// 5th-generation tensor cores (tcgen05 + TMEM), 2-SM tiles, sm_103a.
//
// The prefill phase (PowerSlider Sec. 2.2) attends every new prompt token
// causally over its sequence's cache; unlike decode it is a dense
// contraction with high arithmetic intensity (Sec. 3 Obs. 2, App. B: the
// intensity grows with the number of tokens processed together).  Sequence s
// has L_s cached tokens whose last Q_s are the new (query) tokens; query i sits
// at position p = L_s - Q_s + i and sees keys 0 .. p.
//
// Tiling.  A query tile is 128 MMA rows: 128 / g consecutive query tokens
// times the g query heads of KV head j (row = token * g + head), so every K/V
// tile serves the whole group.  Two CTAs on a pair of SMs (a cluster of 2)
// take two adjacent query tiles of one (sequence, KV head) and run the
// contractions as one M = 256 tcgen05 MMA (cta_group::2): each CTA holds its
// own 128 query rows and half of every K/V tile -- keys 64 r .. 64 r + 63 of
// a 128-key K tile (K-major, stored [dim half][key][64]) and dims 64 r ..
// 64 r + 63 of all 128 keys of a V tile (MN-major, [key][64]) -- so each SM
// stages and reads half the K/V bytes a single-SM tile would, which is what
// the single-SM kernel ran short of (shared-memory bandwidth shared by the
// MMA operand reads and the TMA writes).  Keys stream through per-CTA rings
// of 16-key page slices addressed through the block table; each CTA's copies
// complete on the leader CTA's barriers (TMA .cta_group::2), so the leader
// issues the MMA for both once both halves have landed.  Both query tiles of
// a pair stream the keys the later tile needs; the earlier tile masks the
// rest.
//
// Warp roles (12 warps per CTA; warpgroup 0 gives registers to the two
// softmax warpgroups with setmaxnreg, 56 / 224 per thread):
//   warp 0     TMA: Q once per unit, then this CTA's half of each K tile into
//              a K ring.
//   warp 2     TMA: this CTA's half of each V tile into a V ring; the last
//              tile's rows past the needed keys are zeroed (its copy completes
//              locally first) before the leader is told.
//   warp 1     leader CTA only, one thread: S_n = Q K_n^T into TMEM score
//              buffer n & 1 of both CTAs (M = 256, N = 128, K = 128), and, once
//              both CTAs' softmax has written P_n, O_{n & 1} += P_n V_n with P
//              read from TMEM; tcgen05.commit multicasts each completion to
//              both CTAs' barriers.  A tile's K and V copies (both CTAs')
//              complete on one barrier, and the one commit after its P V
//              frees both stages: each commit and each barrier poll is issuer
//              time during which the tensor pipe runs dry, so the issuer keeps
//              one poll and two commits (S full, K/V free) per tile.
//   warp 3     idle (completes warpgroup 0).
//   warps 4-7  softmax group 0: the tiles of even global index n;
//   warps 8-11 softmax group 1: the tiles of odd n.  One TMEM lane (= one
//              row) per thread: load the score row, mask it causally, update
//              the running max m and sum l in fp32 (base 2, log2 e folded into
//              the scale), and write the bf16 probabilities over the first
//              half of the same S buffer (the A operand of the P V MMA).
// Each group thus runs an independent online softmax over every other key
// tile with its own accumulator (TMEM: S_0, S_1 at columns 0 and 128, O_0,
// O_1 at 256 and 384), so that one group computes while the other waits for
// its next score tile and the tensor core works on both: two softmax streams
// per SM sub-partition where one left the sub-partition idle during every
// wait.  At the end of a unit the group that did not run its last tile hands
// (m, l) of each row through shared memory to the group that did, which
// merges the halves -- O = (2^(m_0 - m) O_0 + 2^(m_1 - m) O_1) / (2^(m_0 - m)
// l_0 + 2^(m_1 - m) l_1), m = max(m_0, m_1) -- and writes the row, while the
// handing group (which owns the next unit's first tile) runs that tile's
// softmax.  P over S needs no barrier of its own: the Q K^T of
// tile n + 2 is issued after the P V of tile n, and tcgen05 MMAs of one
// thread run in order.  The softmax's instruction stream is what the MMA
// issue competes with on every SM sub-partition, so it is kept short: a
// three-input max, packed two-lane fp32 fma/add, and l summed from the fp32
// weights before they are rounded to bf16 for P V (the quotient O / l then
// differs from one with l summed from the rounded weights by a relative 2^-9
// at most).
// The rescale is lazy: a group's reference max m only moves when the tile
// max exceeds it by more than 2^8, so P <= 256 and no value leaves fp32/bf16
// range; the final O / l is the same quotient whichever reference max was
// used.

// Persistent clusters.  A launch has one cluster per pair of SMs; each runs
// a list of units -- (sequence, KV head, pair of query tiles) -- dealt out by
// work (descending, in a snake over the clusters), with the rings, the S/P
// buffers and their barrier phases running on from one unit to the next: the
// next unit's Q (double-buffered) and first K/V tiles load while the current
// unit finishes, and its first Q K^T and softmax run while the other group
// merges and writes out the current unit's rows.  (Batches with more units than fit a cluster's list run
// one unit per cluster.)
//
// Every mbarrier wait gives up after ~2 s of globaltimer, or at once when
// another role of its CTA has given up, and raises PS_DEVICE_TIMEOUT in the
// optional device status word; the producers then wait for their own copies,
// the MMA issuer for its own MMAs, both CTAs meet at a cluster barrier, and
// TMEM is freed on every path.

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
constexpr int kRows = 128;         // query rows per CTA (MMA M = 256 over the pair)
constexpr int kKeys = 128;         // MMA N of S, K of P.V: keys per tile
constexpr int kChunk = 16;         // keys per TMA box (one page slice)
#ifndef PS_PREFILL_STAGES
#define PS_PREFILL_STAGES 4
#endif
// K and V rings of the same depth: a tile's K and V land on one barrier and
// their stages are freed together, once the tile's P V is done.
constexpr int kStages = PS_PREFILL_STAGES;
constexpr int kThreads = 384;
// Registers per thread after the role split: warpgroup 0 (producers, MMA
// issuer) gives registers back, the two softmax warpgroups take them.  The sum
// must not exceed what the block is launched with (kThreads x the kernel's
// register count, checked on the host), or setmaxnreg.inc would wait forever.
constexpr int kRegsCtl = 56, kRegsSoftmax = 224;
static_assert(128 * kRegsCtl + 256 * kRegsSoftmax <= 65536, "register split");
constexpr int kHalfQ = kRows * 64 * 2;        // one 64-column half of the 128-row Q tile: 16 KiB
constexpr int kQBytes = 2 * kHalfQ;           // 32 KiB
constexpr int kPairKeys = kKeys / 2;          // keys of each K tile one CTA holds
constexpr int kKHalf = kPairKeys * 128;       // one 64-dim half of a CTA's K slice: 8 KiB
constexpr int kKStage = 2 * kKHalf;           // 16 KiB
constexpr int kVStage = kKeys * 128;          // 128 keys x this CTA's 64 dims: 16 KiB
constexpr int kOffQ = 0;                            // two Q buffers: the next unit's Q loads early
constexpr int kOffK = kOffQ + 2 * kQBytes;
constexpr int kOffV = kOffK + kStages * kKStage;
constexpr int kOffBar = kOffV + kStages * kVStage;
constexpr int kBarBytes = 512;
constexpr int kMaxUnitsPerCluster = 256;            // a cluster's unit list (persistent mode)
constexpr int kOffList = kOffBar + kBarBytes;
constexpr int kOffX = kOffList + kMaxUnitsPerCluster * 4;  // (m, l) of the handing group's rows for the merge
constexpr int kSmemBytes = 1024 + kOffX + kRows * 8;  // 1 KiB of alignment slack
// Persistent mode needs the whole batch's units (sequence x KV head x pair of
// query tiles) below this; the host launches one unit per cluster above it.
constexpr int kMaxPersistentUnits = 16384;
constexpr int kSchedBins = 64;                      // work bins of the schedule's counting sort
static_assert(kThreads * kSchedBins * 2 + 4 * kSchedBins * 4 <= kStages * kVStage, "schedule scratch");
static_assert(kSmemBytes <= 227 * 1024, "shared memory");
constexpr uint32_t kTmemCols = 512;
// TMEM columns (the same in both CTAs): S buffers at 0 and 128 (P, bf16 pairs
// packed in 32-bit columns, over the first 64 of each), O_0 and O_1 at 256 and 384.
constexpr uint32_t kColO = 256;
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
    int persistent;    // 1: grid of clusters, each running a list of units; 0: one unit per cluster
    int num_clusters;  // persistent mode: clusters in the grid
    long long test_stall_ns;  // > 0: injected stall (ps_test_inject), else 0
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
// D (both CTAs' TMEM) += A . B over the CTA pair: each CTA supplies its 128
// rows of A and its half (along N) of B at the same shared-memory offsets.
__device__ __forceinline__ void umma2(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}
// The same with A read from each CTA's tensor memory (row = TMEM lane, K
// packed in bf16 pairs along the columns: a K step of 16 is 8 columns).
__device__ __forceinline__ void umma2_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
        "r"(a_tmem), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}
// Arrive on the barrier at this offset in both CTAs of the pair once every
// MMA issued so far has completed.
__device__ __forceinline__ void umma_commit_pair(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(bar),
        "h"((uint16_t)3)
        : "memory");
}
__device__ __forceinline__ uint32_t cta_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
// Shared::cluster address of the same shared-memory location in CTA `rank`.
__device__ __forceinline__ uint32_t map_to(uint32_t addr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}
// Arrive on a barrier of either CTA of the pair.  The arrivals carry the
// default (CTA-scope release) semantics: what they order -- tensor-memory
// reads and writes finished with tcgen05.wait and fenced with
// tcgen05.fence::before_thread_sync, and TMA transfers counted by the
// barrier itself -- needs no cluster-scope release, which costs ~1-2 us of
// latency per arrival on this path.
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_bar) {
    asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(cluster_bar) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx_cluster(uint32_t cluster_bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cluster.b64 _, [%0], %1;" ::"r"(cluster_bar), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// TMA load into this CTA's shared memory whose completion is counted on a
// barrier of either CTA of the pair (`cluster_bar`), with an L2 policy.
__device__ __forceinline__ void tma_load_3d_pair(uint32_t dst, const CUtensorMap *tm, int c0, int c1, int c2,
                                                 uint32_t cluster_bar, uint64_t policy) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.cta_group::2.L2::cache_hint"
        " [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(c2), "r"(cluster_bar), "l"(policy)
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
// A whole 128-column score row in one load, and the 64 columns of packed P
// in one store: fewer tensor-memory instructions next to the MMAs.
__device__ __forceinline__ void tmem_ld128(uint32_t taddr, float *v) {
    uint32_t r[128];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x128.b32 {"
        "%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,"
        "%32,%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,"
        "%48,%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63,"
        "%64,%65,%66,%67,%68,%69,%70,%71,%72,%73,%74,%75,%76,%77,%78,%79,"
        "%80,%81,%82,%83,%84,%85,%86,%87,%88,%89,%90,%91,%92,%93,%94,%95,"
        "%96,%97,%98,%99,%100,%101,%102,%103,%104,%105,%106,%107,%108,%109,%110,%111,"
        "%112,%113,%114,%115,%116,%117,%118,%119,%120,%121,%122,%123,%124,%125,%126,%127"
        "}, [%128];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31]),
          "=r"(r[32]), "=r"(r[33]), "=r"(r[34]), "=r"(r[35]), "=r"(r[36]), "=r"(r[37]), "=r"(r[38]), "=r"(r[39]),
          "=r"(r[40]), "=r"(r[41]), "=r"(r[42]), "=r"(r[43]), "=r"(r[44]), "=r"(r[45]), "=r"(r[46]), "=r"(r[47]),
          "=r"(r[48]), "=r"(r[49]), "=r"(r[50]), "=r"(r[51]), "=r"(r[52]), "=r"(r[53]), "=r"(r[54]), "=r"(r[55]),
          "=r"(r[56]), "=r"(r[57]), "=r"(r[58]), "=r"(r[59]), "=r"(r[60]), "=r"(r[61]), "=r"(r[62]), "=r"(r[63]),
          "=r"(r[64]), "=r"(r[65]), "=r"(r[66]), "=r"(r[67]), "=r"(r[68]), "=r"(r[69]), "=r"(r[70]), "=r"(r[71]),
          "=r"(r[72]), "=r"(r[73]), "=r"(r[74]), "=r"(r[75]), "=r"(r[76]), "=r"(r[77]), "=r"(r[78]), "=r"(r[79]),
          "=r"(r[80]), "=r"(r[81]), "=r"(r[82]), "=r"(r[83]), "=r"(r[84]), "=r"(r[85]), "=r"(r[86]), "=r"(r[87]),
          "=r"(r[88]), "=r"(r[89]), "=r"(r[90]), "=r"(r[91]), "=r"(r[92]), "=r"(r[93]), "=r"(r[94]), "=r"(r[95]),
          "=r"(r[96]), "=r"(r[97]), "=r"(r[98]), "=r"(r[99]), "=r"(r[100]), "=r"(r[101]), "=r"(r[102]), "=r"(r[103]),
          "=r"(r[104]), "=r"(r[105]), "=r"(r[106]), "=r"(r[107]), "=r"(r[108]), "=r"(r[109]), "=r"(r[110]), "=r"(r[111]),
          "=r"(r[112]), "=r"(r[113]), "=r"(r[114]), "=r"(r[115]), "=r"(r[116]), "=r"(r[117]), "=r"(r[118]), "=r"(r[119]),
          "=r"(r[120]), "=r"(r[121]), "=r"(r[122]), "=r"(r[123]), "=r"(r[124]), "=r"(r[125]), "=r"(r[126]), "=r"(r[127])
        : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 128; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_st64u(uint32_t taddr, const uint32_t (&v)[64]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x64.b32 [%0], {"
        "%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32,"
        "%33,%34,%35,%36,%37,%38,%39,%40,%41,%42,%43,%44,%45,%46,%47,%48,"
        "%49,%50,%51,%52,%53,%54,%55,%56,%57,%58,%59,%60,%61,%62,%63,%64"
        "};"
        ::"r"(taddr), "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
          "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]), "r"(v[15]),
          "r"(v[16]), "r"(v[17]), "r"(v[18]), "r"(v[19]), "r"(v[20]), "r"(v[21]), "r"(v[22]), "r"(v[23]),
          "r"(v[24]), "r"(v[25]), "r"(v[26]), "r"(v[27]), "r"(v[28]), "r"(v[29]), "r"(v[30]), "r"(v[31]),
          "r"(v[32]), "r"(v[33]), "r"(v[34]), "r"(v[35]), "r"(v[36]), "r"(v[37]), "r"(v[38]), "r"(v[39]),
          "r"(v[40]), "r"(v[41]), "r"(v[42]), "r"(v[43]), "r"(v[44]), "r"(v[45]), "r"(v[46]), "r"(v[47]),
          "r"(v[48]), "r"(v[49]), "r"(v[50]), "r"(v[51]), "r"(v[52]), "r"(v[53]), "r"(v[54]), "r"(v[55]),
          "r"(v[56]), "r"(v[57]), "r"(v[58]), "r"(v[59]), "r"(v[60]), "r"(v[61]), "r"(v[62]), "r"(v[63])
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
__device__ __forceinline__ uint64_t pack2(float lo, float hi) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}
__device__ __forceinline__ void unpack2(uint64_t v, float &lo, float &hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}
// Two fp32 lanes at once (Blackwell packed FP32): a * b + c and a + b.
__device__ __forceinline__ uint64_t fma2(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}
__device__ __forceinline__ uint64_t add2(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ uint64_t mul2(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ float max3(float a, float b, float c) {
    float r;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(r) : "f"(a), "f"(b), "f"(c));
    return r;
}
__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ bool mbar_test(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// The softmax warps of a CTA that gave up (one of its waits ran out, here or
// in another role of the CTA) raise the abort flag of the other CTA of the
// pair too, so that every role there stops waiting at its next poll instead
// of at its own limit: every role of a CTA that gives up ends its loops, the
// softmax warps included.  Called once, where the softmax warps leave their
// loops: kept out of the waits and the control warps, whose code it would
// otherwise enlarge on the hot path.
__device__ __noinline__ void raise_peer_abort(volatile int *abort) {
    const uint32_t peer = map_to(saddr(const_cast<int *>(abort)), cta_rank() ^ 1u);
    asm volatile("st.shared::cluster.u32 [%0], %1;" ::"r"(peer), "r"(1) : "memory");
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
// The injected stall (tests only): a wait with the given limit on a barrier
// that nothing arrives on, giving up the way every wait does.
__device__ __forceinline__ bool stall_wait(uint32_t bar, unsigned long long limit_ns, volatile int *abort, unsigned *status) {
    const unsigned long long t0 = global_ns();
    bool ok = true;
    while (!mbar_try_wait(bar, 0u)) {
        if (*abort) { ok = false; break; }
        if (global_ns() - t0 > limit_ns) {
            *abort = 1;
            if (status) atomicOr(status, (unsigned)PS_DEVICE_TIMEOUT);
            ok = false;
            break;
        }
    }
    return __all_sync(0xffffffffu, ok);
}
// The waits of the producers and the softmax warps: the same bound, with a
// suspend-time hint, so that a warp whose phase has not completed sleeps in
// the barrier (woken when the phase completes, or after the hint) instead of
// spinning on the issue slots of the SM sub-partition it shares with a
// softmax warp that is computing.  The MMA issuer keeps spinning: its wake-up
// latency lies on the tile's critical path.
constexpr uint32_t kSuspendNs = 1000;
__device__ __forceinline__ bool mbar_try_wait_sleep(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity), "r"(kSuspendNs)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ bool wait_phase_sleep(uint32_t bar, uint32_t parity, volatile int *abort, unsigned *status) {
    const unsigned long long t0 = global_ns();
    while (!mbar_try_wait_sleep(bar, parity)) {
        if (*abort) return false;
        if (global_ns() - t0 > kWaitLimitNs) {
            *abort = 1;
            if (status) atomicOr(status, (unsigned)PS_DEVICE_TIMEOUT);
            return false;
        }
    }
    return true;
}
__device__ __forceinline__ bool warp_wait_sleep(uint32_t bar, uint32_t parity, volatile int *abort, unsigned *status) {
    return __all_sync(0xffffffffu, wait_phase_sleep(bar, parity, abort, status));
}
// Bounded wait without the abort shortcut: used to drain this thread's own
// copies and MMAs, which complete whatever the other roles did.
__device__ __forceinline__ void drain_phase(uint32_t bar, uint32_t parity) {
    const unsigned long long t0 = global_ns();
    while (!mbar_try_wait(bar, parity))
        if (global_ns() - t0 > kWaitLimitNs) return;
}


// Geometry of unit u (sequence s, KV head j, pair pi of query tiles) and its
// work in 128-key tiles; 0 for a unit with no query rows, or whose sequence is
// inconsistent (then `bad` is set).
struct Unit {
    int s, j, qt_hi, qs0, Q, L, kv_limit, ntiles;
};
__device__ __forceinline__ Unit unit_of(const PrefillParams &p, int u, int npairs, bool &bad) {
    Unit x;
    const int pi = u % npairs;
    x.j = (u / npairs) % p.num_kv_heads;
    x.s = u / (npairs * p.num_kv_heads);
    x.qt_hi = p.num_qtiles - 1 - 2 * pi;
    x.qs0 = __ldg(p.q_start + x.s);
    const int qs1 = __ldg(p.q_start + x.s + 1);
    x.Q = qs1 - x.qs0;
    x.L = __ldg(p.seq_lens + x.s);
    x.ntiles = 0;
    x.kv_limit = 0;
    bad = false;
    const int tpt = p.tokens_per_tile;
    if (max(x.qt_hi - 1, 0) * tpt >= x.Q) return x;  // neither tile of the pair has rows
    const long long cap = (long long)p.max_blocks_per_seq * p.block_size;
    if (x.Q < 0 || x.L < x.Q || (long long)x.L > cap || x.qs0 < 0 || qs1 > p.total_q) {
        bad = true;
        return x;
    }
    x.kv_limit = x.L - x.Q + min(x.Q, (x.qt_hi + 1) * tpt);  // keys the pair needs: [0, kv_limit)
    x.ntiles = (x.kv_limit + kKeys - 1) / kKeys;
    return x;
}

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    ps_prefill_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                      const __grid_constant__ CUtensorMap tmV, const PrefillParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *sm = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t rank = cta_rank();  // 0: the leader, which issues the MMAs
    const int g = p.group, tpt = p.tokens_per_tile;
    const int npairs = (p.num_qtiles + 1) / 2;
    int *ulist = reinterpret_cast<int *>(sm + kOffList);
    __shared__ int s_count, s_wmax;

    // ---- the cluster's units ------------------------------------------
    // One unit per cluster (grid order: heaviest pairs of query tiles first),
    // or, in persistent mode, every cluster of the grid runs a list: all
    // units sorted by work (descending, 64 bins, stable by unit index) and
    // dealt out in a snake (0 .. P-1, P-1 .. 0, ...), so that the clusters'
    // totals come out even.  Both CTAs of a cluster compute the same list.
    if (!p.persistent) {
        if (tid == 0) {
            const int u = (blockIdx.z * p.num_kv_heads + blockIdx.y) * npairs + (blockIdx.x >> 1);
            bool bad;
            const Unit x = unit_of(p, u, npairs, bad);
            if (bad && rank == 0 && p.status) atomicOr(p.status, (unsigned)PS_DEVICE_LEN_CLAMPED);
            ulist[0] = u;
            s_count = x.ntiles > 0 ? 1 : 0;
        }
    } else {
        const int U = p.num_seqs * p.num_kv_heads * npairs;  // <= kMaxPersistentUnits (host)
        const int P = p.num_clusters, me = (int)(blockIdx.x >> 1);
        const int a = (int)((long long)tid * U / kThreads), e = (int)((long long)(tid + 1) * U / kThreads);
        uint16_t *cnt = reinterpret_cast<uint16_t *>(sm + kOffV);                      // [kThreads][bins]
        int *bin_start = reinterpret_cast<int *>(sm + kOffV + kThreads * kSchedBins * 2);  // [bins]
        int *bin_total = bin_start + kSchedBins;
        if (tid == 0) { s_wmax = 1; s_count = 0; }
        for (int b = 0; b < kSchedBins; ++b) cnt[tid * kSchedBins + b] = 0;
        __syncthreads();
        int wmax = 1;
        for (int u = a; u < e; ++u) {
            bool bad;
            const Unit x = unit_of(p, u, npairs, bad);
            if (bad && blockIdx.x == 0 && p.status) atomicOr(p.status, (unsigned)PS_DEVICE_LEN_CLAMPED);
            wmax = max(wmax, x.ntiles);
        }
        atomicMax(&s_wmax, wmax);
        __syncthreads();
        wmax = s_wmax;
        auto bin_of = [&](int w) { return min(kSchedBins - 1, (int)((long long)(w - 1) * kSchedBins / wmax)); };
        for (int u = a; u < e; ++u) {
            bool bad;
            const Unit x = unit_of(p, u, npairs, bad);
            if (x.ntiles > 0) ++cnt[tid * kSchedBins + bin_of(x.ntiles)];
        }
        __syncthreads();
        if (tid < kSchedBins) {  // per bin: units of earlier threads (stable by unit index)
            int run = 0;
            for (int t = 0; t < kThreads; ++t) {
                const int c = cnt[t * kSchedBins + tid];
                cnt[t * kSchedBins + tid] = (uint16_t)run;
                run += c;
            }
            bin_total[tid] = run;
        }
        __syncthreads();
        if (tid == 0) {  // bins in descending work
            int acc = 0;
            for (int b = kSchedBins - 1; b >= 0; --b) {
                bin_start[b] = acc;
                acc += bin_total[b];
            }
            const int full = acc / P, rem = acc - full * P;
            s_count = full + ((full & 1) ? (P - 1 - me < rem) : (me < rem));
        }
        __syncthreads();
        for (int u = a; u < e; ++u) {
            bool bad;
            const Unit x = unit_of(p, u, npairs, bad);
            if (x.ntiles == 0) continue;
            const int b = bin_of(x.ntiles);
            const int r = bin_start[b] + cnt[tid * kSchedBins + b];
            ++cnt[tid * kSchedBins + b];
            const int round = r / P, pos = r - round * P;
            if (((round & 1) ? P - 1 - pos : pos) == me) ulist[round] = u;
        }
        // max_q_len below a chunk leaves that chunk's later rows uncovered.
        if (blockIdx.x == 0 && p.status)
            for (int s = tid; s < p.num_seqs; s += kThreads)
                if (__ldg(p.q_start + s + 1) - __ldg(p.q_start + s) > p.num_qtiles * tpt)
                    atomicOr(p.status, (unsigned)PS_DEVICE_LEN_CLAMPED);
    }
    if (!p.persistent && (blockIdx.x >> 1) == 0 && blockIdx.y == 0 && tid == 0 && rank == 0 && p.status) {
        const int Qs = __ldg(p.q_start + blockIdx.z + 1) - __ldg(p.q_start + blockIdx.z);
        if (Qs > p.num_qtiles * tpt) atomicOr(p.status, (unsigned)PS_DEVICE_LEN_CLAMPED);
    }
    __syncthreads();
    const int nunits = s_count;  // the same in both CTAs of the cluster
    if (nunits == 0) return;

    uint64_t *bars = reinterpret_cast<uint64_t *>(sm + kOffBar);
    auto bar_q = [&](int qb) { return saddr(bars + qb); };                                    // [2] leader's
    // K and V tile t: both CTAs' K and V copies complete on kvfull(t % kStages)
    // (the leader's); the tile's P V commit frees both stages through kvfree.
    auto bar_kvfull = [&](int st) { return saddr(bars + 2 + st); };           // [kStages], leader's
    auto bar_kvfree = [&](int st) { return saddr(bars + 2 + kStages + st); };  // [kStages]
    constexpr int kB = 2 + 2 * kStages;
    auto bar_sfull = [&](int b) { return saddr(bars + kB + b); };      // [2]
    auto bar_pfull = [&](int b) { return saddr(bars + kB + 2 + b); };  // [2] leader's
    const uint32_t bar_mma_end = saddr(bars + kB + 4);
    const uint32_t bar_vtail = saddr(bars + kB + 5);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + kB + 6);
    volatile int *abort = reinterpret_cast<volatile int *>(bars + kB + 7);
    auto bar_qfree = [&](int qb) { return saddr(bars + kB + 8 + qb); };  // [2]
    const uint32_t bar_ofree = saddr(bars + kB + 10);                    // leader's
    auto bar_xfull = [&](int q) { return saddr(bars + kB + 11 + q); };   // [4] (m, l) hand-off to the merging group, per lane quarter
    auto bar_xempty = [&](int q) { return saddr(bars + kB + 15 + q); };  // [4]
    const uint32_t bar_stall = saddr(bars + kB + 19);  // nothing arrives on it: the injected stall (tests only)
    static_assert((2 + 2 * kStages + 20) * 8 <= kBarBytes, "barrier area");

    if (tid == 0) {
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar_q(i), 2);  // one arrival (with its bytes) from each CTA
            mbar_init(bar_qfree(i), 1);
        }
        for (int i = 0; i < kStages; ++i) {
            mbar_init(bar_kvfull(i), 4);  // the K and the V arrival (with its bytes) of each CTA
            mbar_init(bar_kvfree(i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar_sfull(i), 1);
            mbar_init(bar_pfull(i), 8);  // the buffer's four softmax warps in each CTA
        }
        mbar_init(bar_mma_end, 1);
        mbar_init(bar_vtail, 1);
        mbar_init(bar_ofree, 8);  // both CTAs' merging softmax warps have read O
        mbar_init(bar_stall, 1);
        for (int q = 0; q < 4; ++q) {
            mbar_init(bar_xfull(q), 1);
            mbar_init(bar_xempty(q), 1);
        }
        *abort = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(saddr(tmem_slot)),
                     "r"(kTmemCols)
                     : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
    }
    // Both CTAs' barriers exist and their TMEM is allocated before either
    // CTA's copies or arrivals can reach the other (and the schedule scratch
    // in the V ring is no longer read).
    tc_fence_before();
    cluster_sync();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    const uint32_t sQ = saddr(sm + kOffQ), sK = saddr(sm + kOffK), sV = saddr(sm + kOffV);
    bool bad_unused;

    if (warp < 4) {
    asm volatile("setmaxnreg.dec.sync.aligned.u32 %0;" ::"n"(kRegsCtl));
    if (warp == 0 || warp == 2) {
        // ----------------------------------------------------- producers --
        const bool is_k = warp == 0;
        uint64_t keep;  // every K/V page is read by all query tiles of its (sequence, head)
        asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(keep));
        if (lane == 0) {
            asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(is_k ? &tmK : &tmV)) : "memory");
            if (is_k) asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmQ)) : "memory");
        }
        constexpr int stages = kStages;
        int issued = 0, tails = 0, units_q = 0;
        bool tail_pending = false, ok = true;
        for (int ui = 0; ok && ui < nunits; ++ui) {
            const Unit x = unit_of(p, ulist[ui], npairs, bad_unused);
            const int qt = x.qt_hi - (int)rank, tok0 = qt * tpt;
            const int *bt_row = p.block_table + (size_t)x.s * p.max_blocks_per_seq;
            if (is_k) {
                // Q of this unit into buffer ui & 1, once the Q K^T of unit ui - 2 is done.
                const int qb = ui & 1;
                if (ui >= 2 && !warp_wait_sleep(bar_qfree(qb), ((ui - 2) >> 1) & 1, abort, p.status)) { ok = false; break; }
                if (lane == 0) {
                    const uint32_t lq = map_to(bar_q(qb), 0);
                    mbar_expect_tx_cluster(lq, (uint32_t)(2 * 128 * g * tpt));
                    // Rows of a missing or empty tile read zeros or other rows; they are never written.
                    tma_load_3d_pair(sQ + qb * kQBytes, &tmQ, 0, x.j * g, x.qs0 + tok0, lq, keep);
                    tma_load_3d_pair(sQ + qb * kQBytes + kHalfQ, &tmQ, 64, x.j * g, x.qs0 + tok0, lq, keep);
                }
                units_q = ui + 1;
            }
            for (int n = 0; n < x.ntiles; ++n) {
                const int st = issued % stages, use = issued / stages;
                if (issued >= stages &&
                    !warp_wait_sleep(bar_kvfree(st), (use - 1) & 1, abort, p.status)) { ok = false; break; }
                const int base = n * kKeys;
                if (is_k) {
                    // Keys 64 rank .. 64 rank + 63 of the tile, both 64-dim halves:
                    // lanes 0-7 take (chunk lane & 3, half lane >> 2).
                    const int k0 = base + kPairKeys * (int)rank;
                    const int nc = max(0, min(kPairKeys / kChunk, (x.kv_limit - k0 + kChunk - 1) / kChunk));
                    const uint32_t full = map_to(bar_kvfull(st), 0);
                    if (lane == 0) mbar_expect_tx_cluster(full, (uint32_t)(nc * 2 * kChunk * 128));
                    __syncwarp();
                    const int c = lane & 3, half = lane >> 2;
                    if (lane < 8 && c < nc) {
                        const int t0 = k0 + c * kChunk;
                        const int lb = t0 / p.block_size;
                        const int b = __ldg(bt_row + lb);
                        int page = -1;  // out of range: TMA fills zeros
                        if (b >= 0 && (long long)b < p.num_blocks) page = b * p.num_kv_heads + x.j;
                        else if (p.status) atomicOr(p.status, (unsigned)PS_DEVICE_BAD_BLOCK);
                        tma_load_3d_pair(sK + st * kKStage + half * kKHalf + c * (kChunk * 128), &tmK, half * 64,
                                         t0 - lb * p.block_size, page, full, keep);
                    }
                    ++issued;
                } else {
                    // Dims 64 rank .. 64 rank + 63 of all keys of the tile: lane c takes chunk c.
                    const int valid = min(kKeys, x.kv_limit - base);
                    const int nc = (valid + kChunk - 1) / kChunk;
                    const bool tail = valid < kKeys;
                    const uint32_t full = map_to(bar_kvfull(st), 0);
                    if (lane == 0) {
                        if (tail) mbar_expect_tx(bar_vtail, (uint32_t)(nc * kChunk * 128));
                        else mbar_expect_tx_cluster(full, (uint32_t)(nc * kChunk * 128));
                    }
                    __syncwarp();
                    if (lane < nc) {
                        const int t0 = base + lane * kChunk;
                        const int lb = t0 / p.block_size;
                        const int b = __ldg(bt_row + lb);
                        int page = -1;
                        if (b >= 0 && (long long)b < p.num_blocks) page = b * p.num_kv_heads + x.j;
                        const uint32_t dst = sV + st * kVStage + lane * (kChunk * 128);
                        if (tail) tma_load_3d_hint(dst, &tmV, 64 * (int)rank, t0 - lb * p.block_size, page, bar_vtail, keep);
                        else tma_load_3d_pair(dst, &tmV, 64 * (int)rank, t0 - lb * p.block_size, page, full, keep);
                    }
                    ++issued;
                    if (tail) {
                        // The unit's last tile: its copy completes here first, then the
                        // rows past the needed keys (other tokens' data, or stale bytes)
                        // are zeroed -- P is zero there -- before the leader is told.
                        tail_pending = true;
                        if (!warp_wait_sleep(bar_vtail, tails & 1, abort, p.status)) { ok = false; break; }
                        tail_pending = false;
                        ++tails;
                        uint8_t *v = sm + kOffV + st * kVStage;
                        for (int e2 = lane; e2 < (kKeys - valid) * 8; e2 += 32)
                            *reinterpret_cast<uint4 *>(v + (valid + (e2 >> 3)) * 128 + (e2 & 7) * 16) = make_uint4(0, 0, 0, 0);
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) mbar_arrive_cluster(full);
                    }
                }
            }
        }
        // Drain: this CTA's copies must land before it can leave.  Copies that
        // count on the leader's barriers are covered by the leader's waits and
        // the final cluster barrier; the local ones are waited for here.
        if (tail_pending) drain_phase(bar_vtail, tails & 1);
        if (rank == 0) {
            for (int i = max(0, issued - stages); i < issued; ++i)
                drain_phase(bar_kvfull(i % stages), (i / stages) & 1);
            if (is_k)
                for (int ui = max(0, units_q - 2); ui < units_q; ++ui) drain_phase(bar_q(ui & 1), (ui >> 1) & 1);
        }
    } else if (warp == 1) {
        if (rank == 0) {
            // ---------------------------------------- MMA issuer (leader) --
            constexpr uint32_t idS = instr_desc(2 * kRows, kKeys, 0);
            constexpr uint32_t idO = instr_desc(2 * kRows, kD, 1);
            // Descriptor bases, once: a stage or K-step offset is an add to the
            // 14-bit start-address field (shared-memory addresses stay below 256 KiB).
            const uint64_t dQ = smem_desc(sQ, 16, 1024), dK = smem_desc(sK, 16, 1024), dV = smem_desc(sV, 16, 1024);
            bool ok = true;
            int t0 = 0;  // tiles of the earlier units (S/P buffers and K/V stages run on across units)
            for (int ui = 0; ok && ui < nunits; ++ui) {
                const Unit x = unit_of(p, ulist[ui], npairs, bad_unused);
                const int qb = ui & 1;
                if (!warp_wait(bar_q(qb), (ui >> 1) & 1, abort, p.status)) { ok = false; break; }
                const uint64_t dq = dQ + (uint64_t)((qb * kQBytes) >> 4);
                // A barrier poll costs a shared-memory round trip while the tensor
                // core streams operands: the next tile's K/V barrier is tested
                // before the current group's MMAs are issued (the result is used
                // after them), and waited for only if it had not completed.
                bool k_seen = false;
                for (int n = 0; ok && n <= x.ntiles; ++n) {
                    if (n < x.ntiles) {
                        const int t = t0 + n, st = t % kStages, b = t & 1;
                        if (!__all_sync(0xffffffffu, k_seen) && !warp_wait(bar_kvfull(st), (t / kStages) & 1, abort, p.status)) { ok = false; break; }
                        tc_fence_after();
                        if (lane == 0) {
                            const uint64_t kd = dK + (uint64_t)((st * kKStage) >> 4);
#pragma unroll
                            for (int kk = 0; kk < kD / 16; ++kk) {
                                umma2(tmem + b * kKeys, dq + (uint64_t)(((kk >> 2) * kHalfQ + (kk & 3) * 32) >> 4),
                                      kd + (uint64_t)(((kk >> 2) * kKHalf + (kk & 3) * 32) >> 4), idS, kk > 0);
                            }
                            umma_commit_pair(bar_sfull(b));
                            if (n == x.ntiles - 1) umma_commit_pair(bar_qfree(qb));  // Q buffer qb is free again
                        }
                        __syncwarp();
                    }
                    k_seen = false;
                    if (n >= 1) {
                        const int m = n - 1, t = t0 + m, st = t % kStages;
                        if (!warp_wait(bar_pfull(t & 1), (t >> 1) & 1, abort, p.status)) { ok = false; break; }
                        // The unit's first P V into each O buffer overwrites it: the
                        // previous unit's O_0 and O_1 must have been read out by both
                        // CTAs' merging softmax warps.
                        if (m == 0 && ui > 0 && !warp_wait(bar_ofree, (ui - 1) & 1, abort, p.status)) { ok = false; break; }
                        if (n + 1 < x.ntiles) {
                            const int tk = t0 + n + 1;
                            k_seen = mbar_test(bar_kvfull(tk % kStages), (tk / kStages) & 1);
                        }
                        tc_fence_after();
                        if (lane == 0) {
                            const uint32_t pt = tmem + (t & 1) * kKeys;  // P over S
                            const uint64_t vd = dV + (uint64_t)((st * kVStage) >> 4);
#pragma unroll
                            for (int kk = 0; kk < kKeys / 16; ++kk)
                                umma2_ts(tmem + kColO + (t & 1) * kD, pt + kk * 8, vd + (uint64_t)((kk * (16 * 128)) >> 4), idO,
                                         (m > 1 || kk > 0) ? 1u : 0u);
                            umma_commit_pair(bar_kvfree(st));  // this tile's P V done: its K and V stages are free
                        }
                        __syncwarp();
                    }
                }
                t0 += x.ntiles;
            }
            // Every MMA issued above has finished, in both CTAs, before TMEM
            // and shared memory go away.
            if (lane == 0) umma_commit_pair(bar_mma_end);
            __syncwarp();
        }
        drain_phase(bar_mma_end, 0);
    }
    } else {
        asm volatile("setmaxnreg.inc.sync.aligned.u32 %0;" ::"n"(kRegsSoftmax));
        // ------------------------------------------------------- softmax --
        const int G = warp >= 8 ? 1 : 0;  // key tiles of global index = G (mod 2)
        const int quarter = warp & 3;      // TMEM lanes 32 * quarter .. + 31
        const int r = quarter * 32 + lane;
        const uint32_t trow = tmem + ((uint32_t)(quarter * 32) << 16);
        const int tl = r / g, hl = r - tl * g;
        const float sl2 = p.scale_log2;
        float2 *xs = reinterpret_cast<float2 *>(sm + kOffX);
        bool ok = true;
        // Injected stall (tests only): group 0 of the leader CTA waits, before
        // its first score tile, on a barrier nothing arrives on, so the
        // leader's first P V never issues and the wait runs out the way a
        // real one would.
        if (p.test_stall_ns > 0 && G == 0 && rank == 0 &&
            !stall_wait(bar_stall, (unsigned long long)p.test_stall_ns, abort, p.status))
            ok = false;
        int t0 = 0;
        for (int ui = 0; ok && ui < nunits; ++ui) {
            const Unit x = unit_of(p, ulist[ui], npairs, bad_unused);
            const int qt = x.qt_hi - (int)rank, tok0 = qt * tpt;
            const bool row_valid = (tl < tpt) && (qt >= 0) && (tok0 + tl < x.Q);
            const int limit = row_valid ? (x.L - x.Q + tok0 + tl + 1) : x.kv_limit;
            float m_ref = -INFINITY;
            uint64_t l2 = pack2(0.f, 0.f);  // row sum, as two interleaved partial sums
            for (int n = ((t0 & 1) == G) ? 0 : 1; n < x.ntiles; n += 2) {
                const int t = t0 + n;
                if (!warp_wait_sleep(bar_sfull(G), (t >> 1) & 1, abort, p.status)) { ok = false; break; }
                tc_fence_after();
                float sv[kKeys];
                tmem_ld128(trow + G * kKeys, sv);
                tmem_wait_ld();
                tmem_loaded<kKeys>(sv);
                const int base = n * kKeys;
                if (base + kKeys > limit) {
#pragma unroll
                    for (int i = 0; i < kKeys; ++i)
                        if (base + i >= limit) sv[i] = -INFINITY;
                }
                // Two independent max chains over the halves of the row.
                float mxa = sv[0], mxb = sv[64];
#pragma unroll
                for (int i = 1; i + 1 < 64; i += 2) {
                    mxa = max3(mxa, sv[i], sv[i + 1]);
                    mxb = max3(mxb, sv[64 + i], sv[64 + i + 1]);
                }
                float mx = max3(mxa, mxb, fmaxf(sv[63], sv[127]));
                const float m_tile = mx * sl2;
                const bool grow = m_tile > m_ref + kRescaleLog2;
                const float alpha = grow ? ex2(m_ref - m_tile) : 1.f;
                if (n >= 2 && __any_sync(0xffffffffu, grow)) {
                    // O_G must hold this group's earlier tiles before it is rescaled.
                    if (!warp_wait_sleep(bar_kvfree((t - 2) % kStages), ((t - 2) / kStages) & 1, abort, p.status)) { ok = false; break; }
                    tc_fence_after();
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        float ov[32];
                        tmem_ld32(trow + kColO + G * kD + c * 32, ov);
                        tmem_wait_ld();
                        tmem_loaded<32>(ov);
#pragma unroll
                        for (int i = 0; i < 32; ++i) ov[i] *= alpha;
                        tmem_st32(trow + kColO + G * kD + c * 32, ov);
                    }
                    tmem_wait_st();
                }
                if (grow) {
                    l2 = mul2(l2, pack2(alpha, alpha));
                    m_ref = m_tile;
                }
                // A row whose keys in this group's tiles are all masked so far has
                // m_ref = -inf: its weights are 0 (not inf - inf).
                const float m_use = m_ref == -INFINITY ? 0.f : m_ref;
                const uint64_t sl2x2 = pack2(sl2, sl2), nm2 = pack2(-m_use, -m_use);
                // P (bf16 pairs) over the first 64 columns of this S buffer: the
                // P V of tile t - 2, the last reader of those columns, finished
                // before the Q K^T of tile t (whose completion was just waited for).
                uint32_t wp[64];
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    uint32_t *w = wp + c * 16;
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        const int i = c * 32 + 2 * e;
                        float x0, x1;
                        unpack2(fma2(pack2(sv[i], sv[i + 1]), sl2x2, nm2), x0, x1);
                        const float e0 = ex2(x0), e1 = ex2(x1);
                        const __nv_bfloat162 pr = __floats2bfloat162_rn(e0, e1);
                        l2 = add2(l2, pack2(e0, e1));
                        w[e] = *reinterpret_cast<const uint32_t *>(&pr);
                    }
                }
                tmem_st64u(trow + G * kKeys, wp);
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_cluster(map_to(bar_pfull(G), 0));
            }
            if (!ok) break;
            float la, lb;
            unpack2(l2, la, lb);
            // The group of the unit's last tile merges: the other group finished
            // its last tile a tile earlier and owns the next unit's first tile,
            // whose softmax then runs alongside the merge.
            const int tl_last = t0 + x.ntiles - 1;
            if (G != (tl_last & 1)) {
                // Hand (m, l) of these rows to the merging group.
                if (ui > 0 && !warp_wait_sleep(bar_xempty(quarter), (ui - 1) & 1, abort, p.status)) { ok = false; break; }
                xs[r] = make_float2(m_ref, la + lb);
                __syncwarp();
                if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar_xfull(quarter)) : "memory");
            } else {
                // This group's S-full wait of tile tl_last implies the P V of tile
                // tl_last - 2, so the barrier of the unit's last P V is at most one
                // phase behind: its parity wait cannot pass on an older phase.
                if (!warp_wait_sleep(bar_xfull(quarter), ui & 1, abort, p.status)) { ok = false; break; }
                if (!warp_wait_sleep(bar_kvfree(tl_last % kStages), (tl_last / kStages) & 1, abort, p.status)) { ok = false; break; }
                const float2 o1 = xs[r];
                __syncwarp();
                if (lane == 0) asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar_xempty(quarter)) : "memory");
                // The other group has tiles in this unit unless it has one tile
                // (which is this group's).
                const bool has1 = x.ntiles >= 2;
                const float m0 = m_ref, m1 = o1.x;
                const float m = fmaxf(m0, has1 ? m1 : -INFINITY);
                const float c0 = ex2(m0 - m), c1 = has1 ? ex2(m1 - m) : 0.f;
                const float inv = 1.f / ((la + lb) * c0 + o1.y * c1);
                const float f0 = c0 * inv, f1 = c1 * inv;
                tc_fence_after();
                // O = f0 O_G + f1 O_{1-G}, 32 dims at a time, straight to the output
                // row; then the leader may start the next unit's P V (which
                // overwrites both accumulators).
                uint16_t *orow = row_valid ? p.out + ((size_t)(x.qs0 + tok0 + tl) * p.num_q_heads + (size_t)x.j * g + hl) * kD : nullptr;
#pragma unroll 1
                for (int c = 0; c < 4; ++c) {
                    // Both accumulators are read; one this unit left unused holds
                    // stale values and is not used.
                    float a0[32], a1[32];
                    tmem_ld32(trow + kColO + G * kD + c * 32, a0);
                    tmem_ld32(trow + kColO + (G ^ 1) * kD + c * 32, a1);
                    tmem_wait_ld();
                    tmem_loaded<32>(a0);
                    tmem_loaded<32>(a1);
                    uint32_t w[16];
#pragma unroll
                    for (int e = 0; e < 16; ++e) {
                        float y0 = a0[2 * e] * f0, y1 = a0[2 * e + 1] * f0;
                        y0 = has1 ? fmaf(a1[2 * e], f1, y0) : y0;
                        y1 = has1 ? fmaf(a1[2 * e + 1], f1, y1) : y1;
                        const __nv_bfloat162 pr = __floats2bfloat162_rn(y0, y1);
                        w[e] = *reinterpret_cast<const uint32_t *>(&pr);
                    }
                    if (row_valid)
#pragma unroll
                        for (int v = 0; v < 4; ++v)
                            *reinterpret_cast<uint4 *>(orow + c * 32 + v * 8) = make_uint4(w[4 * v], w[4 * v + 1], w[4 * v + 2], w[4 * v + 3]);
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_cluster(map_to(bar_ofree, 0));
            }
            t0 += x.ntiles;
        }
        if (!ok && lane == 0) raise_peer_abort(abort);
    }
    // Neither CTA leaves (nor frees TMEM) while the other may still touch its
    // shared memory or the leader's MMAs may still run.
    tc_fence_before();
    __syncthreads();
    cluster_sync();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols) : "memory");
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
        !encode3d(&tmV, v_cache, (cuuint64_t)block_size, (cuuint64_t)(num_blocks * num_kv_heads), kChunk, 1))
        return PS_ERR_CUDA;
    // The shared-memory limit is a per-device function attribute: set it for
    // the current device on every call (cheap), so that a process driving
    // several GPUs works on each of them.
    if (cudaFuncSetAttribute(ps_prefill_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes) !=
        cudaSuccess)
        return PS_ERR_CUDA;
    cudaFuncAttributes fa;
    if (cudaFuncGetAttributes(&fa, ps_prefill_kernel) != cudaSuccess) return PS_ERR_CUDA;
    if (fa.numRegs * kThreads < 128 * kRegsCtl + 256 * kRegsSoftmax) return PS_ERR_UNSUPPORTED;

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
    // Units: (sequence, KV head, pair of adjacent query tiles).  Up to
    // kMaxPersistentUnits of them, one cluster of two CTAs per pair of SMs
    // runs a list of units (persistent); beyond, one cluster per unit.
    const long long npairs = (nqt + 1) / 2;
    const long long units = (long long)num_seqs * num_kv_heads * npairs;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return PS_ERR_CUDA;
    const int clusters = max(1, sms / 2);
    pp.persistent = (units <= kMaxPersistentUnits && (units + clusters - 1) / clusters <= kMaxUnitsPerCluster) ? 1 : 0;
    pp.num_clusters = clusters;
    pp.test_stall_ns = ps::take_injected_prefill_stall_ns();
    const dim3 grid = pp.persistent ? dim3((unsigned)(2 * clusters), 1, 1)
                                    : dim3((unsigned)(2 * npairs), (unsigned)num_kv_heads, (unsigned)num_seqs);
    if (ps::take_injected_launch_error() != cudaSuccess) return PS_ERR_CUDA;
    ps_prefill_kernel<<<grid, kThreads, kSmemBytes, reinterpret_cast<cudaStream_t>(stream)>>>(tmQ, tmK, tmV, pp);
    if (cudaGetLastError() != cudaSuccess) return PS_ERR_CUDA;
    ps::note_launch();
    return PS_OK;
}
