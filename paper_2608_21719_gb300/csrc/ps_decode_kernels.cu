// ps_decode_kernels.cu -- sm_103a kernel for batched paged GQA decode attention.
//
// One persistent launch per call: one CTA per SM, kWorkersPerCta independent
// worker warps per CTA.
//
// Work layout.  The KV work of the whole batch is one "tape" of 16-token
// tiles ordered by sequence, then KV head: segment (s, j) holds
// ceil(L_s / 16) tiles.  Every CTA rebuilds the per-sequence prefix sums of
// the tape in shared memory from seq_lens, and worker w of Ws takes the
// contiguous range [floor(w N / Ws), floor((w+1) N / Ws)) of the N tiles.
// The split is balanced to one tile whatever the mix of short answer-phase
// and long thinking-phase contexts (PowerSlider Sec. 2.2, Sec. 3 Obs. 3),
// needs no host knowledge of the lengths and no atomics, and depends only on
// the lengths and the grid, so results are bit-deterministic.
//
// Streaming.  A worker walks its range tile by tile.  Each tile's K and V
// arrive by TMA (cp.async.bulk.tensor, 128-byte swizzle, one box each,
// stored [64-column half][token][64]) in a per-warp ring of shared-memory
// stages completed on mbarriers; each
// (block, kv-head) page is read once for all g query heads of its group.
// Per tile the warp computes S^T = K Q^T and O^T += V^T P^T on the tensor
// cores (mma.sync m16n8k16, bf16 in, fp32 accumulate: tokens fill M = 16,
// the g <= 8 query heads fill N = 8) with an online softmax whose running
// max and sum stay in fp32 (scores in base 2, log2(e) folded into scale).
//
// Split-KV combine.  A piece of a segment that one range covers completely
// is normalised and written as bf16.  A piece cut by a range boundary leaves
// (m, l, acc) in the workspace and adds its tile count to the segment's
// counter; the warp that completes the count merges all pieces of the
// segment in tape order by the log-sum-exp rule
//   o = sum_c 2^(m_c - M) acc_c / sum_c 2^(m_c - M) l_c,  M = max_c m_c,
// and resets the counter for the next call.  A warp whose range ends inside
// a segment reads the segment's counter (acquire) when it starts its last
// tile; if every other piece is already counted, it is the segment's only
// possible merger and merges its own piece from registers, skipping the
// partial-state write, the fence and the atomic at the kernel's tail.
//
// No wait spins forever: every mbarrier wait gives up after ~2 s of
// globaltimer, raises PS_DEVICE_TIMEOUT in the workspace status word, drains
// the worker's outstanding copies with the same bound and returns.
#include <cuda_bf16.h>

#include <atomic>

#include "ps_internal.h"

namespace ps {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr unsigned long long kWaitLimitNs = 2000000000ull;
constexpr unsigned kFlagTimeout = 1u, kFlagBadBlock = 2u, kFlagLenClamped = 4u;

// ------------------------------------------------------------ PTX wrappers --

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
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

// Bounded wait for phase `parity` of an mbarrier; false after limit_ns
// (~2 s by default).
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity,
                                          unsigned long long limit_ns = kWaitLimitNs) {
    for (int i = 0; i < 256; ++i)
        if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    while (!mbar_try_wait(bar, parity))
        if (global_ns() - t0 > limit_ns) return false;
    return true;
}

__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap *tm, int c0, int c1, int c2, int c3,
                                            uint32_t bar) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4, %5}], [%6];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(tm)), "r"(c0), "r"(c1), "r"(c2), "r"(c3), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(bar)
        : "memory");
}

// 16-byte global -> shared copy that bypasses L1 (cp.async, completed by
// cp.async.wait_group in the issuing thread).
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}

__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
// Wait until at most N of this thread's committed cp.async groups are pending.
template <int N>
__device__ __forceinline__ void cp_async_wait_group() { asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory"); }

// Segment counter update with acquire-release semantics at GPU scope: it
// publishes this warp's partial state (written before it, ordered to lane 0
// by the warp barrier) and, for the warp that completes the count, makes
// every other piece's state visible.
__device__ __forceinline__ int atomic_add_acq_rel(int *p, int v) {
    int old;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}
__device__ __forceinline__ int load_acquire(const int *p) {
    int v;
    asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ void prefetch_l2(const void *p) {
    asm volatile("prefetch.global.L2 [%0];" ::"l"(p));
}

__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr)
                 : "memory");
}

__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t &r0, uint32_t &r1, uint32_t &r2, uint32_t &r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr)
                 : "memory");
}

__device__ __forceinline__ uint32_t movm_t(uint32_t x) {
    uint32_t y;
    asm volatile("movmatrix.sync.aligned.m8n8.trans.b16 %0, %1;" : "=r"(y) : "r"(x));
    return y;
}

// D = A(16x16 bf16, row) * B(16x8 bf16, col) + D, fp32 accumulate.
__device__ __forceinline__ void mma_bf16(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, "
        "{%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Pack two floats to bf16x2 (round to nearest even); `lo` lands in bits 0..15.
__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

__device__ __forceinline__ float bf16lo(uint32_t x) { return __uint_as_float(x << 16); }
__device__ __forceinline__ float bf16hi(uint32_t x) { return __uint_as_float(x & 0xffff0000u); }

__device__ __forceinline__ uint16_t f2bf(float x) { return __bfloat16_as_ushort(__float2bfloat16_rn(x)); }

// Byte offset of element (token, dim) inside a [half][16][64] tile written by
// TMA with 128-byte swizzle: the 16-byte chunk index within a 128-byte row is
// XORed with the row index mod 8 (stage buffers are 1024-byte aligned).
__device__ __forceinline__ uint32_t tile_off(int token, int dim) {
    return (uint32_t)((dim >> 6) * kHalfBytes + token * 128 + ((((dim & 63) >> 3) ^ (token & 7)) << 4));
}

// --------------------------------------------------------- tape cursor ----

struct Cursor {
    int s, h, st, ns;  // sequence, kv head, tile within segment, tiles in segment
};

__device__ __forceinline__ int tiles_of(int len) { return (len + kTileTokens - 1) / kTileTokens; }

__device__ __forceinline__ void advance(Cursor &c, const int *sL, int S, int Hkv) {
    if (++c.st < c.ns) return;
    c.st = 0;
    if (++c.h < Hkv) return;
    c.h = 0;
    do {
        ++c.s;
    } while (c.s < S && sL[c.s] == 0);
    c.ns = c.s < S ? tiles_of(sL[c.s]) : 0;
}

// Split of the tape into Ws contiguous static ranges of equal cost.  A warp
// loses time at each segment boundary inside its range (the cut piece's
// partial state and counter update, the next segment's query and
// block-table window), so a segment of ns tiles costs ns + c units, with
// c = kSegmentCost, and ranges are equal in units.  When ranges average
// fewer than 8c tiles (small, latency-bound batches) c is 0: the plain
// equal split.  Unit positions have a closed form: sequence s starts at
// U(s) = sP[s] + c * Hkv * s (an empty sequence costs c per head as well),
// segment h of it at U(s) + h * (ns + c), and its tiles take the first ns
// units.  Range r covers units [floor(r Utot / Ws), floor((r+1) Utot / Ws)).
// All of it is 32-bit: the host bounds Utot below 2^31 and the grid's
// workers below 2^15 (so r * (Utot mod Ws) < 2^30).
struct Partition {
    int N, Ws, S, Hkv, c, Utot, q0, r0;  // Utot = q0 * Ws + r0
    float ws_rcp, ws_per_unit;
    const int *sP, *sL;

    __device__ void init(int N_, int Ws_, int S_, int Hkv_, const int *sP_, const int *sL_) {
        N = N_; Ws = Ws_; S = S_; Hkv = Hkv_; sP = sP_; sL = sL_;
        c = (long long)N >= 8LL * kSegmentCost * Ws ? kSegmentCost : 0;
        Utot = seq_unit(S);
        q0 = Ws > 0 ? Utot / Ws : 0;
        r0 = Utot - q0 * Ws;
        ws_rcp = 1.f / (float)max(Ws, 1);
        ws_per_unit = (float)Ws / (float)max(Utot, 1);
    }
    __device__ int seq_unit(int s) const { return sP[s] + c * Hkv * s; }
    __device__ int segment_unit(int s, int h, int ns) const { return seq_unit(s) + h * (ns + c); }
    // floor(r Utot / Ws) = r q0 + floor(r r0 / Ws); the last quotient is below
    // Ws <= 2^15, so a float estimate is off by at most one and is corrected.
    __device__ int unit_begin(int r) const {
        const int x = r * r0;
        int q = (int)((float)x * ws_rcp);
        q += (q + 1) * Ws <= x ? 1 : 0;
        q -= q * Ws > x ? 1 : 0;
        return r * q0 + q;
    }
    // The range holding unit u: a float estimate, corrected exactly.
    __device__ int range_of_unit(int u) const {
        int r = min(Ws - 1, (int)((float)u * ws_per_unit));
        while (r + 1 < Ws && unit_begin(r + 1) <= u) ++r;
        while (r > 0 && unit_begin(r) > u) --r;
        return r;
    }
    // Where unit u falls (one lane): sequence s, head h, offset o in the
    // segment's ns + c units, and the number of tiles before u.
    struct Pos {
        int tile, s, h, o, ns;
    };
    __device__ Pos position(int u) const {
        Pos q;
        if (u >= Utot) {
            q.tile = N; q.s = S; q.h = 0; q.o = 0; q.ns = 0;
            return q;
        }
        int lo = 0, hi = S - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (seq_unit(mid) <= u) lo = mid; else hi = mid - 1;
        }
        q.s = lo;
        q.ns = tiles_of(sL[lo]);
        const int off = u - seq_unit(lo);  // < Hkv * (ns + c)
        const int d = q.ns + c;             // >= 1: the sequence holding u has units
        int h = (int)((float)off * __frcp_rn((float)d));  // h < Hkv: off by at most one
        h += (h + 1) * d <= off ? 1 : 0;
        h -= h * d > off ? 1 : 0;
        q.h = h;
        q.o = off - h * d;
        q.tile = sP[lo] + q.h * q.ns + min(q.o, q.ns);
        return q;
    }
    // The ranges r0..r1 holding segment (s, h) (tiles a .. a+ns-1), and
    // whether range r0 began at an earlier tile (then the segment's piece is
    // r0's second piece).  The merging warp's own range w = [b, e) is
    // usually r0 or r1, which needs no arithmetic.
    __device__ void merge_bounds(int s, int h, int ns, int w, int b, int e, int &r0, int &r1, int &cut0) const {
        const int a = sP[s] + h * ns;
        const int ua = segment_unit(s, h, ns);
        if (a >= b && a < e) {
            r0 = w;
            cut0 = b < a ? 1 : 0;
        } else {
            r0 = range_of_unit(ua);
            cut0 = position(unit_begin(r0)).tile < a ? 1 : 0;
        }
        r1 = (a + ns - 1 >= b && a + ns - 1 < e) ? w : range_of_unit(ua + ns - 1);
    }
};

// Merge `count` cut pieces of segment (s, h) into bf16 output rows by the
// log-sum-exp rule.  Piece i's workspace slot is slot_of(i), evaluated by the
// lane that owns piece i (i = lane + 32k, may diverge).  Pieces are read
// through L2 (other SMs wrote them).  For the weighted sums every lane owns
// dims [4*lane, 4*lane+4) of every head.
//
// The merge that completes a segment is usually the last thing its warp
// does, so its latency adds to the kernel's tail.  Two paths:
//  * staged (`stage` != nullptr: kStageArea bytes of this warp's shared
//    memory that nothing else uses during the call, and count <= 32): the
//    (m, l) pairs of all pieces and the accumulators of a batch of pieces are
//    copied in with cp.async, all in flight together, and every lane then
//    computes the maxima, weights and sums of l itself from broadcast reads,
//    so the chain has one L2 round trip per batch and no shuffles (which are
//    slow here while the other warps of the SM still stream);
//  * otherwise (the ring is still streaming, or more than 32 pieces): lanes
//    take one piece each for (m, l), reduce the maxima by shuffles, and read
//    the accumulators one piece after another.
// Both paths add the pieces' terms in piece order with the same operations,
// so the output bits do not depend on which warp merged, or where.
constexpr int kStageArea = kWorkerBytes;

// One piece's contribution to the merged sums (explicit fma).
__device__ __forceinline__ void accumulate_piece(float4 &acc, float &lsum, float e, float l, const float4 &a) {
    lsum = fmaf(e, l, lsum);
    acc.x = fmaf(e, a.x, acc.x); acc.y = fmaf(e, a.y, acc.y);
    acc.z = fmaf(e, a.z, acc.z); acc.w = fmaf(e, a.w, acc.w);
}

constexpr int kStageMlBytes = 32 * (int)kSlotMl * 4;  // (m, l) of up to 32 pieces

// The merging warp's own piece, still in registers (mma fragment layout:
// lane owns heads 2 (lane & 3) and 2 (lane & 3) + 1, dims mt 16 + lane / 4
// (+ 8)); m and l are the piece's running max and summed weights.
struct OwnPiece {
    const float (&acc)[8][4];
    float m0, m1, l0, l1;
};

template <typename SlotOf>
__device__ void merge_pieces_staged(const DecodeParams &p, int count, SlotOf slot_of, int s, int h, int lane,
                                    uint8_t *stage, int own, const OwnPiece &mine) {
    const int g = p.group;
    const int piece_bytes = g * kHeadDim * 4;
    const int per = min(32, (kStageArea - kStageMlBytes) / piece_bytes);  // pieces the area holds at once
    // All pieces in one batch when they fit (one L2 round trip); otherwise
    // batches of half the area, two in flight, so that the loads of one
    // overlap the sums of the other.
    const bool single = count <= per;
    const int bsz = single ? count : max(1, per / 2);
    const int nbatch = (count + bsz - 1) / bsz;
    const uint32_t ml_base = smem_addr(stage);
    const uint32_t acc_base = ml_base + kStageMlBytes + 16u * lane;
    const uint8_t *ml_st = stage;
    const uint8_t *acc_st = stage + kStageMlBytes + 16 * lane;
    const int my_slot = (lane < count && lane != own) ? (int)slot_of(lane) : 0;
    if (lane < count && lane != own) {
        const float *src = p.ws_ml + (size_t)my_slot * kSlotMl;
#pragma unroll
        for (int c = 0; c < (int)kSlotMl / 4; ++c) cp_async16(ml_base + (uint32_t)(lane * kSlotMl + 4 * c) * 4, src + 4 * c);
    }
    auto buf_first = [&](int b) -> int { return single ? 0 : (b & 1) * bsz; };  // piece position in the area
    auto issue_batch = [&](int b) {
        const int first = b * bsz, nb = min(bsz, count - first);
        for (int i = 0; i < nb; ++i) {
            const int piece = first + i;
            const int slot = __shfl_sync(kFull, my_slot, piece);
            if (piece == own) continue;
            const float *src = p.ws_acc + (size_t)slot * kSlotFloats + 4 * lane;
            for (int n = 0; n < g; ++n)
                cp_async16(acc_base + (uint32_t)((buf_first(b) + i) * g + n) * (kHeadDim * 4), src + n * kHeadDim);
        }
        cp_async_commit();
    };
    issue_batch(0);
    if (nbatch > 1) issue_batch(1);
    if (own >= 0) {
        // This warp's own piece comes from its registers (single batch only):
        // the (m, l) row and the accumulator, as the slot in the workspace
        // would hold them.
        float *ml_own = reinterpret_cast<float *>(stage + own * kSlotMl * 4);
        float *acc_own = reinterpret_cast<float *>(stage + kStageMlBytes + own * piece_bytes);
        const int h0 = 2 * (lane & 3), h1 = h0 + 1, drow = lane >> 2;
        if (lane < 4) {
            if (h0 < g) { ml_own[2 * h0] = mine.m0; ml_own[2 * h0 + 1] = mine.l0; }
            if (h1 < g) { ml_own[2 * h1] = mine.m1; ml_own[2 * h1 + 1] = mine.l1; }
        }
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
            const int d = mt * 16 + drow;
            if (h0 < g) {
                acc_own[h0 * kHeadDim + d] = mine.acc[mt][0];
                acc_own[h0 * kHeadDim + d + 8] = mine.acc[mt][2];
            }
            if (h1 < g) {
                acc_own[h1 * kHeadDim + d] = mine.acc[mt][1];
                acc_own[h1 * kHeadDim + d + 8] = mine.acc[mt][3];
            }
        }
    }
    if (nbatch > 1) cp_async_wait_group<1>();
    else cp_async_wait_group<0>();
    __syncwarp();  // (m, l) rows and batch 0 were copied by other lanes

    float M[kMaxGroup];
#pragma unroll
    for (int n = 0; n < kMaxGroup; ++n) M[n] = -INFINITY;
    for (int i = 0; i < count; ++i) {
        const float4 *ml = reinterpret_cast<const float4 *>(ml_st + i * kSlotMl * 4);
#pragma unroll
        for (int q4 = 0; q4 < kMaxGroup / 2; ++q4) {
            if (2 * q4 < g) {
                const float4 v = ml[q4];
                M[2 * q4] = fmaxf(M[2 * q4], v.x);
                M[2 * q4 + 1] = fmaxf(M[2 * q4 + 1], v.z);
            }
        }
    }
    float4 acc[kMaxGroup];
    float lsum[kMaxGroup];
#pragma unroll
    for (int n = 0; n < kMaxGroup; ++n) {
        acc[n] = make_float4(0.f, 0.f, 0.f, 0.f);
        lsum[n] = 0.f;
    }
    for (int b = 0; b < nbatch; ++b) {
        const int first = b * bsz, nb = min(bsz, count - first);
        if (b > 0) {
            if (b + 1 < nbatch) cp_async_wait_group<1>();
            else cp_async_wait_group<0>();
            __syncwarp();
        }
        for (int i = 0; i < nb; ++i) {
            const float4 *ml = reinterpret_cast<const float4 *>(ml_st + (first + i) * kSlotMl * 4);
            const uint8_t *src = acc_st + (size_t)(buf_first(b) + i) * piece_bytes;
#pragma unroll
            for (int q4 = 0; q4 < kMaxGroup / 2; ++q4) {
                if (2 * q4 >= g) continue;
                const float4 v = ml[q4];
#pragma unroll
                for (int k = 0; k < 2; ++k) {
                    const int n = 2 * q4 + k;
                    if (n < g) {
                        const float en = ex2((k ? v.z : v.x) - M[n]);
                        const float4 a = *reinterpret_cast<const float4 *>(src + n * (kHeadDim * 4));
                        accumulate_piece(acc[n], lsum[n], en, k ? v.w : v.y, a);
                    }
                }
            }
        }
        if (b + 2 < nbatch) {
            __syncwarp();  // every lane has read this buffer before it is refilled
            issue_batch(b + 2);
        }
    }
    uint16_t *o = p.out + ((size_t)s * p.num_q_heads + (size_t)h * g) * kHeadDim + 4 * lane;
#pragma unroll
    for (int n = 0; n < kMaxGroup; ++n) {
        if (n < g) {
            const float inv = 1.f / lsum[n];
            const uint32_t lo = (uint32_t)f2bf(acc[n].x * inv) | ((uint32_t)f2bf(acc[n].y * inv) << 16);
            const uint32_t hi = (uint32_t)f2bf(acc[n].z * inv) | ((uint32_t)f2bf(acc[n].w * inv) << 16);
            *reinterpret_cast<uint2 *>(o + n * kHeadDim) = make_uint2(lo, hi);
        }
    }
}

template <typename SlotOf>
__device__ void merge_pieces_direct(const DecodeParams &p, int count, SlotOf slot_of, int s, int h, int lane) {
    const int g = p.group;
    float M[kMaxGroup];
#pragma unroll
    for (int n = 0; n < kMaxGroup; ++n) M[n] = -INFINITY;
    for (int i = lane; i < count; i += 32) {
        const float4 *ml = reinterpret_cast<const float4 *>(p.ws_ml + slot_of(i) * kSlotMl);
#pragma unroll
        for (int q4 = 0; q4 < kMaxGroup / 2; ++q4) {
            const float4 v = __ldcg(ml + q4);
            M[2 * q4] = fmaxf(M[2 * q4], v.x);
            M[2 * q4 + 1] = fmaxf(M[2 * q4 + 1], v.z);
        }
    }
#pragma unroll
    for (int n = 0; n < kMaxGroup; ++n)
        if (n < g)
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) M[n] = fmaxf(M[n], __shfl_xor_sync(kFull, M[n], o));
    float4 acc[kMaxGroup];
    float lsum[kMaxGroup];
#pragma unroll
    for (int n = 0; n < kMaxGroup; ++n) {
        acc[n] = make_float4(0.f, 0.f, 0.f, 0.f);
        lsum[n] = 0.f;
    }
    for (int ib = 0; ib < count; ib += 32) {
        const int my_slot = ib + lane < count ? (int)slot_of(ib + lane) : 0;
        float e[kMaxGroup], l[kMaxGroup];  // weight and l of piece ib + lane
#pragma unroll
        for (int n = 0; n < kMaxGroup; ++n) e[n] = l[n] = 0.f;
        if (ib + lane < count) {
            const float4 *ml = reinterpret_cast<const float4 *>(p.ws_ml + (size_t)my_slot * kSlotMl);
#pragma unroll
            for (int q4 = 0; q4 < kMaxGroup / 2; ++q4) {
                if (2 * q4 >= g) continue;
                const float4 v = __ldcg(ml + q4);
                e[2 * q4] = ex2(v.x - M[2 * q4]);
                l[2 * q4] = v.y;
                if (2 * q4 + 1 < g) {
                    e[2 * q4 + 1] = ex2(v.z - M[2 * q4 + 1]);
                    l[2 * q4 + 1] = v.w;
                }
            }
        }
        const int cnt = min(32, count - ib);
        for (int i = 0; i < cnt; ++i) {
            const float *src = p.ws_acc + (size_t)__shfl_sync(kFull, my_slot, i) * kSlotFloats + 4 * lane;
            float4 v[kMaxGroup];
#pragma unroll
            for (int n = 0; n < kMaxGroup; ++n)
                if (n < g) v[n] = __ldcg(reinterpret_cast<const float4 *>(src + n * kHeadDim));
#pragma unroll
            for (int n = 0; n < kMaxGroup; ++n)
                if (n < g)
                    accumulate_piece(acc[n], lsum[n], __shfl_sync(kFull, e[n], i), __shfl_sync(kFull, l[n], i), v[n]);
        }
    }
    uint16_t *o = p.out + ((size_t)s * p.num_q_heads + (size_t)h * g) * kHeadDim + 4 * lane;
#pragma unroll
    for (int n = 0; n < kMaxGroup; ++n) {
        if (n < g) {
            const float inv = 1.f / lsum[n];
            const uint32_t lo = (uint32_t)f2bf(acc[n].x * inv) | ((uint32_t)f2bf(acc[n].y * inv) << 16);
            const uint32_t hi = (uint32_t)f2bf(acc[n].z * inv) | ((uint32_t)f2bf(acc[n].w * inv) << 16);
            *reinterpret_cast<uint2 *>(o + n * kHeadDim) = make_uint2(lo, hi);
        }
    }
}

template <typename SlotOf>
__device__ __forceinline__ void merge_pieces(const DecodeParams &p, int count, SlotOf slot_of, int s, int h, int lane,
                                             uint8_t *stage, const OwnPiece &mine) {
    if (stage != nullptr && count <= 32) merge_pieces_staged(p, count, slot_of, s, h, lane, stage, -1, mine);
    else merge_pieces_direct(p, count, slot_of, s, h, lane);
}

// --------------------------------------------------------------- kernel ----

__global__ void __launch_bounds__(kWorkersPerCta * 32, 1)
    ps_decode_kernel(const DecodeParams p, const __grid_constant__ CUtensorMap tmK,
                     const __grid_constant__ CUtensorMap tmV) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    uint64_t *bars = reinterpret_cast<uint64_t *>(smem + kWorkersPerCta * kWorkerBytes);
    int4 *metas = reinterpret_cast<int4 *>(bars + kWorkersPerCta * kStages);  // per stage: tile, piece
    int4 *pieces = metas + kWorkersPerCta * kStages;                          // per warp: ring of 4 pieces
    int *sP = reinterpret_cast<int *>(pieces + kWorkersPerCta * 4);           // [S + 1] tile prefix (x Hkv)
    int *sL = sP + p.num_seqs + 1;                                            // [S] clamped lengths
    __shared__ int warp_sums[kWorkersPerCta];
    __shared__ uint64_t stall_bar;  // nothing arrives on it: the injected stall (tests only)

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int S = p.num_seqs, Hkv = p.num_kv_heads, g = p.group, bs = p.block_size;
    unsigned *status = reinterpret_cast<unsigned *>(p.ws_header + kHdrStatus);

    // 1. Warm L2 with this CTA's slice of the block table, then build the
    //    clamped lengths and the exclusive prefix of tiles x kv-heads.
    {
        const size_t lines = ((size_t)S * p.max_blocks_per_seq * 4 + 127) / 128;
        for (size_t i = blockIdx.x + (size_t)tid * gridDim.x; i < lines; i += (size_t)blockDim.x * gridDim.x)
            prefetch_l2(reinterpret_cast<const char *>(p.block_table) + i * 128);
        const int nthr = blockDim.x;
        const int per = (S + nthr - 1) / nthr;
        const int lo = min(S, tid * per), hi = min(S, lo + per);
        int sum = 0;
        bool clamped = false;
        for (int i = lo; i < hi; ++i) {
            int L = p.seq_lens[i];
            if (L > p.len_cap) { L = p.len_cap; clamped = true; }
            if (L < 0) L = 0;
            sL[i] = L;
            sum += tiles_of(L) * Hkv;
        }
        if (clamped && blockIdx.x == 0) atomicOr(status, kFlagLenClamped);
        int incl = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(kFull, incl, o);
            if (lane >= o) incl += v;
        }
        if (lane == 31) warp_sums[warp] = incl;
        __syncthreads();
        int run = incl - sum;
        for (int i = 0; i < warp; ++i) run += warp_sums[i];
        for (int i = lo; i < hi; ++i) {
            sP[i] = run;
            run += tiles_of(sL[i]) * Hkv;
        }
        if (lo < hi && hi == S) sP[S] = run;
        if (lane == 0)
            for (int i = 0; i < kStages; ++i) mbar_init(smem_addr(&bars[warp * kStages + i]), 1);
        if (tid == 0) mbar_init(smem_addr(&stall_bar), 1);
        fence_mbar_init();
        __syncthreads();
    }
    // Empty sequences produce zero rows (CTA-strided over sequences).
    for (int s = blockIdx.x; s < S; s += gridDim.x) {
        if (sL[s] != 0) continue;
        uint32_t *o = reinterpret_cast<uint32_t *>(p.out + (size_t)s * p.num_q_heads * kHeadDim);
        for (int i = tid; i < p.num_q_heads * kHeadDim / 2; i += blockDim.x) o[i] = 0u;
    }

    // 2. Partition of the tape (identical in every CTA).
    Partition part;
    {
        const int N = sP[S];
        const int W = gridDim.x * kWorkersPerCta;
        const int cap = (N + p.min_stages - 1) / p.min_stages;
        part.init(N, N > 0 ? max(1, min(min(W, p.max_workers), cap)) : 0, S, Hkv, sP, sL);
    }
    const int w = warp * gridDim.x + blockIdx.x;  // CTAs first: a small Ws still spreads over SMs

    uint8_t *wbase = smem + warp * kWorkerBytes;
    uint8_t *qslots = wbase + kStages * kStageBytes;
    uint64_t *wbars = bars + warp * kStages;
    int4 *wmeta = metas + warp * kStages;
    int4 *wpieces = pieces + warp * 4;
    const int mbps = p.max_blocks_per_seq;

    // ---- issue side: TMA producer state (lane 0 issues, all lanes track) ----
    const bool issuing = w < part.Ws;
    int cur_rid = w, cur_b = 0, cur_e = 0, ip = 0;
    Cursor ic{0, 0, 0, 0};
    if (issuing) {
        // Lanes 0 and 1 find where the range starts and ends, at once.
        const Partition::Pos q = part.position(part.unit_begin(w + (lane & 1)));
        cur_b = __shfl_sync(kFull, q.tile, 0);
        cur_e = __shfl_sync(kFull, q.tile, 1);
        ip = cur_b;
        ic.s = __shfl_sync(kFull, q.s, 0);
        ic.h = __shfl_sync(kFull, q.h, 0);
        ic.st = __shfl_sync(kFull, q.o, 0);
        ic.ns = __shfl_sync(kFull, q.ns, 0);
        if (cur_b < cur_e && ic.st >= ic.ns) {
            // The start is in boundary units: the range begins at the next
            // segment (a range can also hold boundary units only).
            ic.st = 0;
            if (ic.ns > 0 && ic.h + 1 < Hkv) {
                ++ic.h;
            } else {
                ic.h = 0;
                do {
                    ++ic.s;
                } while (sL[ic.s] == 0);
                ic.ns = tiles_of(sL[ic.s]);
            }
        }
    }

    int issued = 0, pieces_issued = 0;
    int win_s = -1, win_j0 = 0, win_v = -1;  // block-table window, one entry per lane
    int pre_s = -1, pre_j0 = 0, pre_v = -1;  // prefetched next window
    // next tile to issue
    int nx_s = 0, nx_h = 0, nx_st = 0;
    bool nx_new = false, have_next = false;
    int4 nx_piece = make_int4(0, 0, 0, 0);

    auto fetch_window = [&](int s, int j0) -> int {
        const int j = j0 + lane;
        const int np = (sL[s] + bs - 1) / bs;
        return j < np ? __ldg(p.block_table + (size_t)s * mbps + j) : -1;
    };
    // Start loading the window that will most likely be needed after the current one.
    auto prefetch_next = [&](int s, int h) {
        int ns_ = -1, nj0 = 0;
        const int np = (sL[s] + bs - 1) / bs;
        if (win_j0 + 32 < np) {
            ns_ = s; nj0 = win_j0 + 32;
        } else if (h + 1 < Hkv) {
            ns_ = s; nj0 = 0;
        } else {
            int s2 = s + 1;
            while (s2 < S && sL[s2] == 0) ++s2;
            if (s2 < S) { ns_ = s2; nj0 = 0; }
        }
        if (ns_ < 0 || (ns_ == win_s && nj0 == win_j0) || (ns_ == pre_s && nj0 == pre_j0)) return;
        pre_s = ns_; pre_j0 = nj0;
        pre_v = fetch_window(ns_, nj0);
    };
    auto position_next = [&]() -> bool {
        if (!issuing || ip >= cur_e) return false;
        nx_s = ic.s; nx_h = ic.h; nx_st = ic.st;
        nx_new = ip == cur_b || ic.st == 0;
        nx_piece = make_int4(ic.s, ic.h, cur_rid, ip == cur_b ? 1 : 0);
        return true;
    };
    auto issue_next = [&]() {
        const int slot = issued % kStages;
        const int tok = nx_st * kTileTokens;
        const int j = tok / bs, tok0 = tok - j * bs, j0 = j & ~31;
        if (win_s != nx_s || win_j0 != j0) {
            if (pre_s == nx_s && pre_j0 == j0) {
                win_v = pre_v; pre_s = -1;
            } else {
                win_v = fetch_window(nx_s, j0);
            }
            win_s = nx_s; win_j0 = j0;
            prefetch_next(nx_s, nx_h);
        } else if (nx_new) {
            prefetch_next(nx_s, nx_h);
        }
        const int pb = __shfl_sync(kFull, win_v, j - j0);
        if (nx_new) ++pieces_issued;
        if (lane == 0) {
            int row = pb * Hkv + nx_h;
            if (pb < 0 || (long long)pb >= p.num_blocks) {
                row = -1;  // fully out of bounds: TMA fills zeros
                atomicOr(status, kFlagBadBlock);
            }
            if (nx_new) wpieces[(pieces_issued - 1) & 3] = nx_piece;
            wmeta[slot] = make_int4(nx_st, pieces_issued - 1, 0, 0);
            const uint32_t bar = smem_addr(&wbars[slot]);
            const uint32_t dst = smem_addr(wbase + slot * kStageBytes);
            const uint32_t qbytes = nx_new ? (uint32_t)(g * kHeadDim * 2) : 0u;
            fence_proxy_async_smem();
            mbar_arrive_expect_tx(bar, kStageBytes + qbytes);
            tma_load_4d(dst, &tmK, 0, tok0, 0, row, bar);
            tma_load_4d(dst + kTileBytes, &tmV, 0, tok0, 0, row, bar);
            if (nx_new) {
                const uint16_t *qsrc = p.q + ((size_t)nx_s * p.num_q_heads + (size_t)nx_h * g) * kHeadDim;
                bulk_load(smem_addr(qslots + ((pieces_issued - 1) % kQSlots) * kQSlotBytes), qsrc, qbytes, bar);
            }
        }
        ++issued;
        have_next = false;
        if (++ip < cur_e) advance(ic, sL, S, Hkv);
    };

    // ---- consume side state ----
    int cur_piece = -1, c_tiles = 0;
    int4 cpi = make_int4(0, 0, 0, 0);
    uint32_t qf[16];
    float acc[8][4];
    float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
    const int h0 = 2 * (lane & 3), h1 = h0 + 1;
    const int trow = lane >> 2;  // token row of this lane in the S^T fragment
    const int drow = lane >> 2;  // dim row of this lane in the O^T fragment

    auto refill = [&](int consumed) {
        while (issued - consumed < kStages) {
            if (!have_next) {
                have_next = position_next();
                if (!have_next) break;
            }
            if (nx_new && pieces_issued >= cur_piece + 1 + kQSlots) break;  // query slot still in use
            issue_next();
        }
    };

    // Finish the consume side's current piece: write its output, or leave its
    // partial state and count its tiles, merging the segment if it was last.
    // `others_done` (-1: not known) is the segment's tile count as read with
    // acquire semantics while the range's last tile was consumed: when it
    // already holds every tile but this piece's, no other warp can complete
    // the count, so this warp is the segment's only merger and merges its
    // own piece straight from its registers (no partial state, fence or
    // atomic on the critical path of the kernel's tail).
    auto finalize = [&](bool ring_idle, int others_done) {
        float L0 = l0, L1 = l1;
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
            L0 += __shfl_xor_sync(kFull, L0, o);
            L1 += __shfl_xor_sync(kFull, L1, o);
        }
        const int s = cpi.x, h = cpi.y;
        const int ns = tiles_of(sL[s]);
        if (c_tiles == ns) {
            // One worker covered the whole segment: write the bf16 output rows.
            uint16_t *o = p.out + ((size_t)s * p.num_q_heads + (size_t)h * g) * kHeadDim;
            const float i0 = 1.f / L0, i1 = 1.f / L1;
#pragma unroll
            for (int mt = 0; mt < 8; ++mt) {
                const int d = mt * 16 + drow;
                if (h0 < g) {
                    o[h0 * kHeadDim + d] = f2bf(acc[mt][0] * i0);
                    o[h0 * kHeadDim + d + 8] = f2bf(acc[mt][2] * i0);
                }
                if (h1 < g) {
                    o[h1 * kHeadDim + d] = f2bf(acc[mt][1] * i1);
                    o[h1 * kHeadDim + d + 8] = f2bf(acc[mt][3] * i1);
                }
            }
            return;
        }
        int *cnt = p.seg_done + (size_t)s * Hkv + h;
        const OwnPiece mine{acc, m0, m1, L0, L1};
        // Range r0 + i holds one piece of the segment: its first piece (slot
        // 2r) unless the range began at an earlier tile.  Only r0 can.
        int r0, r1, cut0;
        if (ring_idle && others_done >= 0 && others_done + c_tiles == ns) {
            part.merge_bounds(s, h, ns, cur_rid, cur_b, cur_e, r0, r1, cut0);
            const int count = r1 - r0 + 1;
            const int per = min(32, (kStageArea - kStageMlBytes) / (g * kHeadDim * 4));
            if (count <= per) {
                auto slot_of = [&](int i) -> size_t { return 2 * (size_t)(r0 + i) + (i == 0 ? cut0 : 0); };
                merge_pieces_staged(p, count, slot_of, s, h, lane, wbase, cur_rid - r0, mine);
                if (lane == 0) *cnt = 0;  // nobody else touches it in this call
                return;
            }
        }
        // Cut by a range boundary: leave (m, l, acc) in the range's slot.
        const size_t slotid = 2 * (size_t)cpi.z + (cpi.w ? 0 : 1);
        float *A = p.ws_acc + slotid * kSlotFloats;
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
            const int d = mt * 16 + drow;
            if (h0 < g) {
                A[h0 * kHeadDim + d] = acc[mt][0];
                A[h0 * kHeadDim + d + 8] = acc[mt][2];
            }
            if (h1 < g) {
                A[h1 * kHeadDim + d] = acc[mt][1];
                A[h1 * kHeadDim + d + 8] = acc[mt][3];
            }
        }
        if (lane < 4) {
            float *ML = p.ws_ml + slotid * kSlotMl;
            ML[2 * h0] = m0; ML[2 * h0 + 1] = L0;
            ML[2 * h1] = m1; ML[2 * h1 + 1] = L1;
        }
        __threadfence();
        __syncwarp();
        int done = 0;
        if (lane == 0) done = atomic_add_acq_rel(cnt, c_tiles) + c_tiles;
        done = __shfl_sync(kFull, done, 0);
        if (done != ns) return;
        // This warp completed the segment (lane 0's acquire, ordered before
        // the other lanes' reads by the shuffle's warp barrier): merge its
        // pieces in tape order.
        part.merge_bounds(s, h, ns, cur_rid, cur_b, cur_e, r0, r1, cut0);
        __syncwarp();
        auto slot_of = [&](int i) -> size_t { return 2 * (size_t)(r0 + i) + (i == 0 ? cut0 : 0); };
        merge_pieces(p, r1 - r0 + 1, slot_of, s, h, lane, ring_idle ? wbase : nullptr, mine);
        if (lane == 0) *cnt = 0;
    };

    int consumed = 0, others_done = -1;
    refill(0);
    if (p.test_stall_ns > 0 && issued > 0 &&
        !__all_sync(kFull, mbar_wait(smem_addr(&stall_bar), 0u, (unsigned long long)p.test_stall_ns))) {
        // Injected stall: handled like a wait that ran out below, before any
        // tile is consumed.
        if (lane == 0) atomicOr(status, kFlagTimeout);
        for (int k = 0; k < issued; ++k) mbar_wait(smem_addr(&wbars[k % kStages]), (uint32_t)((k / kStages) & 1));
        consumed = issued;
    }
    while (consumed < issued) {
        const int slot = consumed % kStages;
        const bool arrived = mbar_wait(smem_addr(&wbars[slot]), (uint32_t)((consumed / kStages) & 1));
        if (!__all_sync(kFull, arrived)) {
            if (lane == 0) atomicOr(status, kFlagTimeout);
            // Drain this worker's outstanding copies (bounded) before leaving.
            for (int k = consumed + 1; k < issued; ++k)
                mbar_wait(smem_addr(&wbars[k % kStages]), (uint32_t)((k / kStages) & 1));
            cur_piece = -1;
            break;
        }
        __syncwarp();
        const int4 meta = wmeta[slot];
        const int st = meta.x, pord = meta.y;
        if (pord != cur_piece) {
            if (cur_piece >= 0) finalize(false, -1);
            cur_piece = pord;
            cpi = wpieces[pord & 3];
            const uint32_t qs = smem_addr(qslots + (pord % kQSlots) * kQSlotBytes);
#pragma unroll
            for (int kp = 0; kp < 4; ++kp)
                ldsm_x4(qs + (lane & 7) * (kHeadDim * 2) + (32 * kp + 8 * (lane >> 3)) * 2, qf[4 * kp], qf[4 * kp + 1],
                        qf[4 * kp + 2], qf[4 * kp + 3]);
            if ((lane >> 2) >= g) {
#pragma unroll
                for (int i = 0; i < 16; ++i) qf[i] = 0u;
            }
            c_tiles = 0;
            m0 = m1 = -INFINITY;
            l0 = l1 = 0.f;
#pragma unroll
            for (int mt = 0; mt < 8; ++mt) acc[mt][0] = acc[mt][1] = acc[mt][2] = acc[mt][3] = 0.f;
        }
        const uint8_t *stage = wbase + slot * kStageBytes;
        const uint32_t sK = smem_addr(stage), sV = sK + kTileBytes;
        const int Ls = sL[cpi.x];
        const int ns = tiles_of(Ls);
        if (lane == 0 && consumed + 1 == issued && !(issuing && ip < cur_e) && c_tiles + 1 != ns)
            // The range's last tile, and its piece is cut: read how much of
            // the segment the other warps have finished (used by finalize).
            others_done = load_acquire(p.seg_done + (size_t)cpi.x * Hkv + cpi.y);
        if (p.k_new != nullptr && st == ns - 1) {
            // Fused append: the last token of the segment is the current one.
            // Its K and V rows come from k_new / v_new (the cache slot still
            // holds stale data in the tile TMA just delivered) and are also
            // stored into the cache.  Lanes 0-15 move the K row, 16-31 the V
            // row, one 16-byte chunk each.
            const int tpos = Ls - 1;
            const int r = tpos - (ns - 1) * kTileTokens;
            const bool isv = lane >= 16;
            const int ci = lane & 15, half = ci >> 3, c = ci & 7;
            const size_t row = ((size_t)cpi.x * Hkv + cpi.y) * kHeadDim + (size_t)ci * 8;
            const uint4 val = *reinterpret_cast<const uint4 *>((isv ? p.v_new : p.k_new) + row);
            uint8_t *tile = const_cast<uint8_t *>(stage) + (isv ? kTileBytes : 0);
            *reinterpret_cast<uint4 *>(tile + half * kHalfBytes + r * 128 + ((c ^ (r & 7)) << 4)) = val;
            const int pb = __ldg(p.block_table + (size_t)cpi.x * mbps + tpos / bs);
            if (pb >= 0 && (long long)pb < p.num_blocks) {
                uint16_t *dst = (isv ? p.v_cache_w : p.k_cache_w) +
                                (((size_t)pb * Hkv + cpi.y) * bs + tpos % bs) * kHeadDim + (size_t)ci * 8;
                *reinterpret_cast<uint4 *>(dst) = val;
            }
            fence_proxy_async_smem();
            __syncwarp();
        }

        // S^T (16 tokens x 8 heads) = K (16 x 128) . Q^T (128 x 8), two accumulation chains.
        float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
        {
            const int tok = (lane & 7) + ((lane >> 3) & 1) * 8;
            const int dsub = (lane >> 4) * 8;
#pragma unroll
            for (int kk = 0; kk < 8; ++kk) {
                uint32_t a0, a1, a2, a3;
                ldsm_x4(sK + tile_off(tok, kk * 16 + dsub), a0, a1, a2, a3);
                if (kk & 1) mma_bf16(sb, a0, a1, a2, a3, qf[2 * kk], qf[2 * kk + 1]);
                else mma_bf16(sa, a0, a1, a2, a3, qf[2 * kk], qf[2 * kk + 1]);
            }
        }
        const int n_valid = st == ns - 1 ? Ls - (ns - 1) * kTileTokens : kTileTokens;
        float x0 = (sa[0] + sb[0]) * p.scale_log2, x1 = (sa[1] + sb[1]) * p.scale_log2;
        float x2 = (sa[2] + sb[2]) * p.scale_log2, x3 = (sa[3] + sb[3]) * p.scale_log2;
        if (trow >= n_valid) x0 = x1 = -INFINITY;
        if (trow + 8 >= n_valid) x2 = x3 = -INFINITY;
        if (n_valid < kTileTokens) {
            // Tail of the sequence: zero the V rows past the last token so that
            // 0-weights never meet stale or NaN data in the P.V product.
            const int rows = kTileTokens - n_valid;
            uint8_t *vt = const_cast<uint8_t *>(stage) + kTileBytes;
            for (int i = lane; i < rows * 16; i += 32) {
                const int r = n_valid + (i >> 4), half = (i >> 3) & 1, c = i & 7;
                *reinterpret_cast<uint4 *>(vt + half * kHalfBytes + r * 128 + c * 16) = make_uint4(0, 0, 0, 0);
            }
            // These generic-proxy writes must be ordered before the TMA that
            // later refills this stage.
            fence_proxy_async_smem();
            __syncwarp();
        }
        float mx0 = fmaxf(x0, x2), mx1 = fmaxf(x1, x3);
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {
            mx0 = fmaxf(mx0, __shfl_xor_sync(kFull, mx0, o));
            mx1 = fmaxf(mx1, __shfl_xor_sync(kFull, mx1, o));
        }
        const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);  // finite: a tile has >= 1 valid token
        const float al0 = ex2(m0 - mn0), al1 = ex2(m1 - mn1);
        m0 = mn0;
        m1 = mn1;
        const uint32_t P01 = pack_bf16(ex2(x0 - mn0), ex2(x1 - mn1));  // token trow
        const uint32_t P23 = pack_bf16(ex2(x2 - mn0), ex2(x3 - mn1));  // token trow + 8
        l0 = l0 * al0 + bf16lo(P01) + bf16lo(P23);
        l1 = l1 * al1 + bf16hi(P01) + bf16hi(P23);
#pragma unroll
        for (int mt = 0; mt < 8; ++mt) {
            acc[mt][0] *= al0; acc[mt][1] *= al1; acc[mt][2] *= al0; acc[mt][3] *= al1;
        }
        // P^T fragments (k = token, n = head) by transposing the bf16 score tiles.
        const uint32_t pb0 = movm_t(P01), pb1 = movm_t(P23);

        // O^T (128 x 8) += V^T (128 x 16) . P^T (16 x 8)
        {
            const int j = lane >> 3;
            const int tok = (lane & 7) + (j >> 1) * 8;
            const int dsub = (j & 1) * 8;
#pragma unroll
            for (int mt = 0; mt < 8; ++mt) {
                uint32_t a0, a1, a2, a3;
                ldsm_x4_t(sV + tile_off(tok, mt * 16 + dsub), a0, a1, a2, a3);
                mma_bf16(acc[mt], a0, a1, a2, a3, pb0, pb1);
            }
        }
        ++c_tiles;
        ++consumed;
        refill(consumed);
    }
    // Every copy into the ring has landed: it can stage the final merge.
    others_done = __shfl_sync(kFull, others_done, 0);
    if (cur_piece >= 0) finalize(true, others_done);
}

}  // namespace

cudaError_t launch_decode(const DecodeParams &p, const CUtensorMap &tmK, const CUtensorMap &tmV, int grid_ctas,
                          size_t smem_bytes, cudaStream_t stream) {
    // Allow the kernel the largest dynamic shared memory the device offers
    // (its opt-in limit less the kernel's static shared memory).  The limit is
    // a property of the device and this binary and is computed once; the
    // attribute belongs to the current context and is set on every call, so
    // a context created after cudaDeviceReset() gets it too.  Every caller
    // sets the same value, so concurrent calls cannot leave a smaller one.
    static std::atomic<int> attr_limit[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    int limit = attr_limit[dev].load(std::memory_order_acquire);
    if (limit == 0) {
        int optin = 0;
        cudaFuncAttributes fa;
        if ((e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev)) != cudaSuccess ||
            (e = cudaFuncGetAttributes(&fa, ps_decode_kernel)) != cudaSuccess)
            return e;
        limit = optin - (int)fa.sharedSizeBytes;
        attr_limit[dev].store(limit, std::memory_order_release);
    }
    if (smem_bytes > (size_t)limit) return cudaErrorInvalidValue;
    if ((e = cudaFuncSetAttribute(ps_decode_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, limit)) !=
        cudaSuccess)
        return e;
    if ((e = take_injected_launch_error()) != cudaSuccess) return e;
    DecodeParams q = p;
    q.test_stall_ns = take_injected_stall_ns();
    ps_decode_kernel<<<grid_ctas, kWorkersPerCta * 32, smem_bytes, stream>>>(q, tmK, tmV);
    return cudaGetLastError();
}

}  // namespace ps
