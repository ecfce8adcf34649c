// ps_kv_transfer.cu -- KV hand-off between stage pools: pack a set of
// sequences' paged K/V into contiguous per-sequence buffers, and unpack such
// buffers into another pool through its block table (PowerSlider Sec. 5: a
// reasoning request's KV cache moves from the thinking pool to the answer
// pool; the transport itself is out of scope, this is the on-GPU gather and
// scatter on either side of it).
//
// Packed layout of sequence i (element offset offsets[i], a multiple of 8):
// K[j][t][:] for kv head j < Hkv and token t < L_i, then V in the same order.
//
// One persistent launch: every CTA builds the prefix of (pages x kv heads)
// over the sequences in shared memory; warps take (sequence, kv head, page)
// units grid-strided and copy the page's valid rows (one contiguous run of
// rows x head_dim x 2 bytes on each side) with 16-byte streaming loads and
// stores, all of a unit's loads in flight before its stores.  The copy is
// bound by HBM read + write bandwidth.
#include <cuda_runtime.h>

#include <cstdint>

#include "ps_decode.h"
#include "ps_internal.h"

namespace {

constexpr int kXferWarps = 8;
constexpr int kXferCtasPerSm = 2;
constexpr int kXferMaxSeqs = 4096;
constexpr int kChunk = 8;  // 16-byte vectors per lane per batch

struct XferParams {
    const uint16_t *k_cache;  // pack: source pool; unpack: unused
    const uint16_t *v_cache;
    uint16_t *k_pool;         // unpack: destination pool; pack: unused
    uint16_t *v_pool;
    const uint16_t *packed_src;  // unpack source
    uint16_t *packed_dst;        // pack destination
    const long long *offsets;
    const int *block_table;
    const int *seq_lens;
    unsigned *status;          // optional PS_DEVICE_* flags
    int num_seqs, num_kv_heads, head_dim, block_size, max_blocks_per_seq;
    long long num_blocks;
};

template <bool kPack>
__global__ void __launch_bounds__(kXferWarps * 32) ps_kv_transfer_kernel(const XferParams p) {
    extern __shared__ int xsm[];
    int *sP = xsm;                   // [S + 1] prefix of pages x Hkv
    int *sL = xsm + p.num_seqs + 1;  // [S] clamped lengths
    __shared__ int wsum[kXferWarps];
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int S = p.num_seqs, Hkv = p.num_kv_heads, bs = p.block_size, d = p.head_dim;
    const int cap = p.max_blocks_per_seq * bs;
    {
        const int per = (S + blockDim.x - 1) / blockDim.x;
        const int lo = min(S, tid * per), hi = min(S, lo + per);
        int sum = 0;
        bool bad = false;
        for (int i = lo; i < hi; ++i) {
            int L = p.seq_lens[i];
            if (L > cap) { L = cap; bad = true; }
            if (L < 0) L = 0;
            if ((p.offsets[i] & 7) != 0) { L = 0; bad = true; }  // 16-byte rows need 8-element alignment
            sL[i] = L;
            sum += (L + bs - 1) / bs * Hkv;
        }
        if (bad && p.status && blockIdx.x == 0) atomicOr(p.status, PS_DEVICE_LEN_CLAMPED);
        int incl = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        if (lane == 31) wsum[warp] = incl;
        __syncthreads();
        int run = incl - sum;
        for (int i = 0; i < warp; ++i) run += wsum[i];
        for (int i = lo; i < hi; ++i) {
            sP[i] = run;
            run += (sL[i] + bs - 1) / bs * Hkv;
        }
        if (lo < hi && hi == S) sP[S] = run;
        __syncthreads();
    }
    const int units = sP[S];
    const int vec_per_row = d / 8;  // 16-byte vectors per token row
    for (int u = blockIdx.x * kXferWarps + warp; u < units; u += gridDim.x * kXferWarps) {
        int lo = 0, hi = S - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (sP[mid] <= u) lo = mid; else hi = mid - 1;
        }
        const int i = lo, L = sL[i];
        const int np = (L + bs - 1) / bs;
        const int off = u - sP[i];
        const int j = off / np, pg = off - j * np;
        const int rows = min(bs, L - pg * bs);
        const int b = __ldg(p.block_table + (size_t)i * p.max_blocks_per_seq + pg);
        if (b < 0 || (long long)b >= p.num_blocks) {
            if (lane == 0 && p.status) atomicOr(p.status, PS_DEVICE_BAD_BLOCK);
            continue;
        }
        const size_t page = (((size_t)b * Hkv + j) * bs) * d;                     // pool element offset
        const size_t kp = (size_t)p.offsets[i] + ((size_t)j * L + (size_t)pg * bs) * d;  // packed element offset
        const size_t vp = kp + (size_t)Hkv * L * d;
        const int nvec = rows * vec_per_row;
        for (int base = 0; base < nvec; base += 32 * kChunk) {
            uint4 ka[kChunk], va[kChunk];
#pragma unroll
            for (int c = 0; c < kChunk; ++c) {
                const int e = base + c * 32 + lane;
                if (e < nvec) {
                    if (kPack) {
                        ka[c] = __ldcs(reinterpret_cast<const uint4 *>(p.k_cache + page) + e);
                        va[c] = __ldcs(reinterpret_cast<const uint4 *>(p.v_cache + page) + e);
                    } else {
                        ka[c] = __ldcs(reinterpret_cast<const uint4 *>(p.packed_src + kp) + e);
                        va[c] = __ldcs(reinterpret_cast<const uint4 *>(p.packed_src + vp) + e);
                    }
                }
            }
#pragma unroll
            for (int c = 0; c < kChunk; ++c) {
                const int e = base + c * 32 + lane;
                if (e < nvec) {
                    if (kPack) {
                        __stcs(reinterpret_cast<uint4 *>(p.packed_dst + kp) + e, ka[c]);
                        __stcs(reinterpret_cast<uint4 *>(p.packed_dst + vp) + e, va[c]);
                    } else {
                        __stcs(reinterpret_cast<uint4 *>(p.k_pool + page) + e, ka[c]);
                        __stcs(reinterpret_cast<uint4 *>(p.v_pool + page) + e, va[c]);
                    }
                }
            }
        }
    }
}

bool aligned_to(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

ps_status_t check_xfer(const void *a, const void *b, const void *c, const long long *offsets, const int *bt,
                       const int *sl, int num_seqs, int num_kv_heads, int head_dim, int block_size,
                       int max_blocks_per_seq, long long num_blocks) {
    if (!a || !b || !c || !offsets || !bt || !sl) return PS_ERR_INVALID_ARG;
    if (!aligned_to(a, 16) || !aligned_to(b, 16) || !aligned_to(c, 16) || !aligned_to(offsets, 8) ||
        !aligned_to(bt, 4) || !aligned_to(sl, 4))
        return PS_ERR_INVALID_ARG;
    if (num_seqs <= 0 || num_kv_heads <= 0 || head_dim <= 0 || block_size <= 0 || max_blocks_per_seq <= 0 ||
        num_blocks <= 0)
        return PS_ERR_INVALID_ARG;
    if (head_dim % 8 != 0 || num_seqs > kXferMaxSeqs) return PS_ERR_UNSUPPORTED;
    const long long cap = (long long)max_blocks_per_seq * block_size;
    if (cap > INT32_MAX || (long long)num_seqs * max_blocks_per_seq * num_kv_heads > INT32_MAX)
        return PS_ERR_UNSUPPORTED;
    return PS_OK;
}

template <bool kPack>
ps_status_t launch_xfer(const XferParams &xp, void *stream) {
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
        return PS_ERR_CUDA;
    const size_t smem = (size_t)(2 * xp.num_seqs + 1) * sizeof(int);
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(ps_kv_transfer_kernel<kPack>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) !=
            cudaSuccess)
        return PS_ERR_CUDA;
    if (ps::take_injected_launch_error() != cudaSuccess) return PS_ERR_CUDA;
    ps_kv_transfer_kernel<kPack><<<sms * kXferCtasPerSm, kXferWarps * 32, smem, reinterpret_cast<cudaStream_t>(stream)>>>(xp);
    if (cudaGetLastError() != cudaSuccess) return PS_ERR_CUDA;
    ps::note_launch();
    return PS_OK;
}

}  // namespace

extern "C" ps_status_t ps_kv_pack(const void *k_cache, const void *v_cache, const int *block_table,
                                  int max_blocks_per_seq, const int *seq_lens, int num_seqs, int num_kv_heads,
                                  int head_dim, int block_size, long long num_blocks, const long long *dst_offsets,
                                  void *dst, unsigned int *device_status, void *stream) {
    ps_status_t e = check_xfer(k_cache, v_cache, dst, dst_offsets, block_table, seq_lens, num_seqs, num_kv_heads,
                               head_dim, block_size, max_blocks_per_seq, num_blocks);
    if (e != PS_OK) return e;
    XferParams xp = {};
    xp.k_cache = static_cast<const uint16_t *>(k_cache);
    xp.v_cache = static_cast<const uint16_t *>(v_cache);
    xp.packed_dst = static_cast<uint16_t *>(dst);
    xp.offsets = dst_offsets;
    xp.block_table = block_table;
    xp.seq_lens = seq_lens;
    xp.status = device_status;
    xp.num_seqs = num_seqs;
    xp.num_kv_heads = num_kv_heads;
    xp.head_dim = head_dim;
    xp.block_size = block_size;
    xp.max_blocks_per_seq = max_blocks_per_seq;
    xp.num_blocks = num_blocks;
    return launch_xfer<true>(xp, stream);
}

extern "C" ps_status_t ps_kv_unpack(const void *src, const long long *src_offsets, const int *block_table,
                                    int max_blocks_per_seq, const int *seq_lens, int num_seqs, int num_kv_heads,
                                    int head_dim, int block_size, long long num_blocks, void *k_cache, void *v_cache,
                                    unsigned int *device_status, void *stream) {
    ps_status_t e = check_xfer(k_cache, v_cache, src, src_offsets, block_table, seq_lens, num_seqs, num_kv_heads,
                               head_dim, block_size, max_blocks_per_seq, num_blocks);
    if (e != PS_OK) return e;
    XferParams xp = {};
    xp.k_pool = static_cast<uint16_t *>(k_cache);
    xp.v_pool = static_cast<uint16_t *>(v_cache);
    xp.packed_src = static_cast<const uint16_t *>(src);
    xp.offsets = src_offsets;
    xp.block_table = block_table;
    xp.seq_lens = seq_lens;
    xp.status = device_status;
    xp.num_seqs = num_seqs;
    xp.num_kv_heads = num_kv_heads;
    xp.head_dim = head_dim;
    xp.block_size = block_size;
    xp.max_blocks_per_seq = max_blocks_per_seq;
    xp.num_blocks = num_blocks;
    return launch_xfer<false>(xp, stream);
}
