// ps_decode_noalloc.cu -- decode attention for callers that cannot allocate.
//
// Some callers have no way to hand the library a workspace: a host engine
// whose device memory is owned by an allocator the plugin may not call,
// a foreign-function caller that only holds the tensors it passes in, or a
// serving process that accounts every byte up front and forbids any
// allocation after start-up.  ps_decode_attention_noalloc() serves them.  It
// runs the same kernel as ps_decode_attention_planned() with a fully static
// split, and keeps the split-KV scratch (counters and partial softmax
// states) in the fixed device array below instead of a caller workspace.
// Nothing here calls cudaMalloc, cudaFree or any allocating routine.
//
// The array costs every GPU that loads the library kNoallocScratchBytes of
// device memory until the process exits.  All calls share it, and it keeps
// whatever the previous call left there, so each call first clears the part
// that must start at zero; two calls that overlap on the GPU (different
// streams, or different host threads) race on it and give wrong results.
#include <cuda.h>
#include <cuda_runtime.h>

#include <cmath>
#include <cstdint>
#include <mutex>

#include "ps_decode.h"
#include "ps_internal.h"

namespace {

constexpr size_t kNoallocScratchBytes = (size_t)PS_NOALLOC_SCRATCH_BYTES;

// The scratch itself.  Host code must not use this name as an address: it is
// a host-side stand-in for the device symbol.  The device address comes from
// cudaGetSymbolAddress() below.
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoallocScratchBytes];

// Device address of the scratch array in the current context.  It is
// resolved on every call rather than cached: the address belongs to the
// context, and after cudaDeviceReset() (or with another context current) a
// cached one would point at memory that is no longer this array's.  The
// lookup is cheap next to the launch.  Under lazy module loading (the CUDA
// default) the first lookup on a device is also what loads this module and
// commits the array's memory on that device.
cudaError_t scratch_address(void **out) {
    void *ptr = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&ptr, g_noalloc_scratch);
    if (e != cudaSuccess) return e;
    *out = ptr;
    return cudaSuccess;
}

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn tiled_encoder() {
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

// Same 4-D view of a paged cache the planned path uses: dims (64, slot, half,
// block x kv-head) with the half stride inside the slot stride, box
// 64 x 16 x 2 x 1, 128-byte swizzle.
bool encode_cache(CUtensorMap *tm, const void *base, int block_size, long long num_blocks, int num_kv_heads) {
    EncodeTiledFn fn = tiled_encoder();
    if (!fn) return false;
    cuuint64_t dims[4] = {64, (cuuint64_t)block_size, 2, (cuuint64_t)num_blocks * (cuuint64_t)num_kv_heads};
    cuuint64_t strides[3] = {(cuuint64_t)ps::kHeadDim * 2, 64 * 2, (cuuint64_t)block_size * ps::kHeadDim * 2};
    cuuint32_t box[4] = {64, (cuuint32_t)ps::kTileTokens, 2, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    return fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides, box, estr,
              CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
              CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool is_aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

}  // namespace

extern "C" ps_status_t ps_decode_attention_noalloc(const void *q, const void *k_cache, const void *v_cache,
                                                   const int *block_table, const int *seq_lens, void *out,
                                                   int num_seqs, int num_q_heads, int num_kv_heads, int head_dim,
                                                   int block_size, int max_blocks_per_seq, long long num_blocks,
                                                   float scale, void *stream) {
    using namespace ps;
    if (!q || !k_cache || !v_cache || !block_table || !seq_lens || !out) return PS_ERR_INVALID_ARG;
    if (!is_aligned(q, 16) || !is_aligned(k_cache, 16) || !is_aligned(v_cache, 16) || !is_aligned(out, 16) ||
        !is_aligned(block_table, 4) || !is_aligned(seq_lens, 4))
        return PS_ERR_INVALID_ARG;
    if (!std::isfinite(scale)) return PS_ERR_INVALID_ARG;
    // The same shape check as the planned path (supported set and the 32-bit
    // bounds of the device split).
    const ps_status_t shape = check_decode_shape(num_seqs, num_q_heads, num_kv_heads, head_dim, block_size,
                                                 max_blocks_per_seq, num_blocks);
    if (shape != PS_OK) return shape;
    const long long len_cap = (long long)max_blocks_per_seq * block_size;

    // The per-segment counters alone may already exceed the array.
    if (kWsHeaderBytes + (size_t)num_seqs * num_kv_heads * 4 > kNoallocScratchBytes) return PS_ERR_UNSUPPORTED;
    int dev = 0, sms = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
        return PS_ERR_CUDA;
    // Scratch layout: the planned path's workspace layout (header,
    // per-segment counters, two partial slots per worker range).
    const WorkspaceLayout lay = workspace_layout(num_seqs, num_kv_heads, sms * kWorkersPerCta);
    if (lay.total > kNoallocScratchBytes) return PS_ERR_UNSUPPORTED;  // beyond the fixed scratch array

    void *scratch = nullptr;
    if (scratch_address(&scratch) != cudaSuccess) return PS_ERR_CUDA;
    CUtensorMap tmK, tmV;
    if (!encode_cache(&tmK, k_cache, block_size, num_blocks, num_kv_heads) ||
        !encode_cache(&tmV, v_cache, block_size, num_blocks, num_kv_heads))
        return PS_ERR_CUDA;

    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    uint8_t *ws = static_cast<uint8_t *>(scratch);
    // Counters and the status word must start at zero; the previous call's
    // contents are still in the array.
    if (cudaMemsetAsync(ws, 0, lay.acc_off, st) != cudaSuccess) return PS_ERR_CUDA;

    DecodeParams dp;
    dp.q = static_cast<const uint16_t *>(q);
    dp.block_table = block_table;
    dp.seq_lens = seq_lens;
    dp.out = static_cast<uint16_t *>(out);
    dp.ws_header = reinterpret_cast<int *>(ws);
    dp.seg_done = reinterpret_cast<int *>(ws + lay.seg_done_off);
    dp.ws_acc = reinterpret_cast<float *>(ws + lay.acc_off);
    dp.ws_ml = reinterpret_cast<float *>(ws + lay.ml_off);
    dp.num_seqs = num_seqs;
    dp.num_q_heads = num_q_heads;
    dp.num_kv_heads = num_kv_heads;
    dp.group = num_q_heads / num_kv_heads;
    dp.block_size = block_size;
    dp.max_blocks_per_seq = max_blocks_per_seq;
    dp.num_blocks = num_blocks;
    dp.len_cap = (int)len_cap;
    dp.max_workers = sms * kWorkersPerCta;
    dp.min_stages = kDefaultMinStages;
    dp.scale_log2 = (float)((double)scale * 1.4426950408889634);
    dp.k_new = dp.v_new = nullptr;
    dp.k_cache_w = dp.v_cache_w = nullptr;
    if (launch_decode(dp, tmK, tmV, sms, partial_smem_bytes(num_seqs), st) != cudaSuccess) return PS_ERR_CUDA;
    return PS_OK;
}
