// ps_internal.h -- constants and launch parameters shared by the host side
// (ps_decode_host.cpp) and the kernels (ps_decode_kernels.cu).  Not part of
// the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace ps {

// Shapes the kernels are written for.
constexpr int kHeadDim = 128;
constexpr int kMaxGroup = 8;        // query heads per KV head (mma N = 8)
constexpr int kMaxSeqs = 4096;      // per-CTA length/prefix tables live in smem
constexpr int kTileTokens = 16;     // tokens per streamed K/V tile (mma M = 16)

// Streaming configuration of the partial kernel.
constexpr int kWorkersPerCta = 4;   // independent warps, each its own KV stream
constexpr int kStages = 5;          // K/V tiles in flight per warp
constexpr int kQSlots = 2;          // query tiles staged per warp
constexpr int kDefaultMinStages = 8;

// Shared-memory geometry.  A 16-token x 128-dim bf16 tile is loaded as two
// 64-column halves by TMA with 128-byte swizzle: [half][token][64].
constexpr int kHalfBytes = kTileTokens * 64 * 2;          // 2048
constexpr int kTileBytes = 2 * kHalfBytes;                // 4096 (K or V)
constexpr int kStageBytes = 2 * kTileBytes;               // 8192 (K + V)
constexpr int kQSlotBytes = kMaxGroup * kHeadDim * 2;     // 2048
constexpr int kWorkerBytes = kStages * kStageBytes + kQSlots * kQSlotBytes;

// Workspace layout (bytes from the workspace base).
constexpr size_t kWsHeaderBytes = 256;   // int32 words, see kHdr*
constexpr int kHdrStatus = 0;            // PS_DEVICE_* flags (atomicOr)
constexpr int kHdrTotalStages = 1;       // N: 16-token tiles over all (seq, kv-head)
constexpr int kHdrWorkers = 2;           // W: workers the partition used
constexpr size_t kSlotFloats = (size_t)kMaxGroup * kHeadDim;  // acc of one partial
constexpr size_t kSlotMl = (size_t)kMaxGroup * 2;              // (m, l) of one partial

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct WorkspaceLayout {
    size_t prefix_off, acc_off, ml_off, total;
};

inline WorkspaceLayout workspace_layout(int num_seqs, int total_workers) {
    WorkspaceLayout w;
    w.prefix_off = kWsHeaderBytes;
    w.acc_off = align_up(w.prefix_off + (size_t)(num_seqs + 1) * 4, 256);
    const size_t slots = 2 * (size_t)total_workers;
    w.ml_off = align_up(w.acc_off + slots * kSlotFloats * 4, 256);
    w.total = align_up(w.ml_off + slots * kSlotMl * 4, 256);
    return w;
}

inline size_t partial_smem_bytes(int num_seqs) {
    return 1024 /* alignment slack */ + (size_t)kWorkersPerCta * kWorkerBytes +
           (size_t)kWorkersPerCta * kStages * 8 + (size_t)(2 * num_seqs + 1) * 4;
}

struct PartialParams {
    const uint16_t *q;          // bf16 [S][Hq][128]
    const int *block_table;     // [S][mbps]
    const int *seq_lens;        // [S]
    uint16_t *out;              // bf16 [S][Hq][128]
    int *ws_header;
    int *ws_prefix;             // [S + 1]
    float *ws_acc;              // [2W][8][128]
    float *ws_ml;               // [2W][8][2]
    int num_seqs, num_q_heads, num_kv_heads, group, block_size, max_blocks_per_seq;
    long long num_blocks;
    int len_cap;                // max_blocks_per_seq * block_size
    int max_workers;            // cap on W
    int min_stages;             // floor on a worker's share
    float scale_log2;           // scale * log2(e)
};

struct CombineParams {
    uint16_t *out;
    const int *ws_header;
    const int *ws_prefix;
    const float *ws_acc;
    const float *ws_ml;
    int num_seqs, num_q_heads, num_kv_heads, group;
};

// Launchers (ps_decode_kernels.cu).  Return cudaSuccess or the launch error.
cudaError_t launch_partial(const PartialParams &p, const CUtensorMap &tmK, const CUtensorMap &tmV,
                           int grid_ctas, size_t smem_bytes, cudaStream_t stream);
cudaError_t launch_combine(const CombineParams &p, cudaStream_t stream);

}  // namespace ps
