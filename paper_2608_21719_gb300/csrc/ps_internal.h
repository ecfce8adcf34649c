// ps_internal.h -- constants and launch parameters shared by the host side
// (ps_decode_host.cpp) and the kernel (ps_decode_kernels.cu).  Not part of
// the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "ps_decode.h"

namespace ps {

// Shapes the kernel is written for.
constexpr int kHeadDim = 128;
constexpr int kMaxGroup = 8;        // query heads per KV head (mma N = 8)
constexpr int kMaxSeqs = 4096;      // per-CTA length/prefix tables live in smem
constexpr int kTileTokens = 16;     // tokens per streamed K/V tile (mma M = 16)

// Streaming configuration: one CTA per SM, kWorkersPerCta independent warps,
// each with a ring of kStages K/V tiles.  Eight warps per SM are needed to
// hide the per-tile latency of one warp; two stages each keep ~15 MB in
// flight over the GPU, well above what HBM3e needs.
#ifndef PS_WORKERS_PER_CTA
#define PS_WORKERS_PER_CTA 8
#endif
#ifndef PS_STAGES
#define PS_STAGES 2
#endif
constexpr int kWorkersPerCta = PS_WORKERS_PER_CTA;
constexpr int kStages = PS_STAGES;
#ifndef PS_QSLOTS
#define PS_QSLOTS 2
#endif
constexpr int kQSlots = PS_QSLOTS;       // query tiles staged per warp
// Weight of a segment boundary in the static split, in tiles: a warp loses
// ~2-3 tiles' time at each one (measured); 4 was the best of 0-6 on the four
// large workloads together (the response is not smooth: boundary placement
// matters as well).
#ifndef PS_SEGMENT_COST
#define PS_SEGMENT_COST 4
#endif
constexpr int kSegmentCost = PS_SEGMENT_COST;
constexpr int kMaxGridCtas = 4096;             // keeps the split's 32-bit arithmetic exact
constexpr int kDefaultMinStages = 2;     // smallest share of a worker, in tiles (tuned on the 4-sequence workload)

// Shared-memory geometry.  A 16-token x 128-dim bf16 tile is loaded as two
// 64-column halves by TMA with 128-byte swizzle: [half][token][64].
constexpr int kHalfBytes = kTileTokens * 64 * 2;          // 2048
constexpr int kTileBytes = 2 * kHalfBytes;                // 4096 (K or V)
constexpr int kStageBytes = 2 * kTileBytes;               // 8192 (K + V)
constexpr int kQSlotBytes = kMaxGroup * kHeadDim * 2;     // 2048
constexpr int kWorkerBytes = kStages * kStageBytes + kQSlots * kQSlotBytes;
static_assert(kWorkerBytes % 1024 == 0, "stage buffers must stay 1024-byte aligned");

// Workspace layout (bytes from the workspace base).
constexpr size_t kWsHeaderBytes = 256;   // int32 words, see kHdr*
constexpr int kHdrStatus = 0;            // PS_DEVICE_* flags (atomicOr)
constexpr size_t kSlotFloats = (size_t)kMaxGroup * kHeadDim;  // acc of one partial piece
constexpr size_t kSlotMl = (size_t)kMaxGroup * 2;              // (m, l) of one partial piece
inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct WorkspaceLayout {
    size_t seg_done_off, acc_off, ml_off, total;
};

// Partial-piece slots: two per worker range (its first and its last piece;
// the pieces between them cover whole segments and need no slot).
inline size_t max_slots(int total_workers) { return 2 * (size_t)total_workers; }

inline WorkspaceLayout workspace_layout(int num_seqs, int num_kv_heads, int total_workers) {
    WorkspaceLayout w;
    const size_t segs = (size_t)num_seqs * num_kv_heads;
    w.seg_done_off = kWsHeaderBytes;
    w.acc_off = align_up(w.seg_done_off + segs * 4, 256);
    const size_t slots = max_slots(total_workers);
    w.ml_off = align_up(w.acc_off + slots * kSlotFloats * 4, 256);
    w.total = align_up(w.ml_off + slots * kSlotMl * 4, 256);
    return w;
}

constexpr size_t kMaxSmemPerCta = 227 * 1024;  // opt-in limit of one CTA on sm_100/sm_103

inline size_t partial_smem_bytes(int num_seqs) {
    return 1024 /* alignment slack */ + (size_t)kWorkersPerCta * kWorkerBytes +
           (size_t)kWorkersPerCta * (kStages * (8 + 16) + 4 * 16) + (size_t)(2 * num_seqs + 1) * 4;
}

// Host-side shape check shared by every decode entry point (planned and
// workspace-free), so that both reject exactly the same shapes.  Besides the
// supported set it bounds what the device split computes in 32 bits: tile
// counts, the split's cost units (tiles plus kSegmentCost per segment
// boundary, Partition::seq_unit) and TMA row coordinates.
inline ps_status_t check_decode_shape(int num_seqs, int num_q_heads, int num_kv_heads, int head_dim,
                                      int block_size, int max_blocks_per_seq, long long num_blocks) {
    if (num_seqs <= 0 || num_q_heads <= 0 || num_kv_heads <= 0 || head_dim <= 0 || block_size <= 0 ||
        max_blocks_per_seq <= 0 || num_blocks <= 0)
        return PS_ERR_INVALID_ARG;
    if (num_q_heads % num_kv_heads != 0) return PS_ERR_INVALID_ARG;
    if (head_dim != kHeadDim) return PS_ERR_UNSUPPORTED;
    if (num_q_heads / num_kv_heads > kMaxGroup) return PS_ERR_UNSUPPORTED;
    if (block_size % kTileTokens != 0 || block_size > 256) return PS_ERR_UNSUPPORTED;
    if (num_seqs > kMaxSeqs || partial_smem_bytes(num_seqs) > kMaxSmemPerCta) return PS_ERR_UNSUPPORTED;
    const long long len_cap = (long long)max_blocks_per_seq * block_size;
    const long long tiles = (long long)num_seqs * ((len_cap + kTileTokens - 1) / kTileTokens) * num_kv_heads;
    const long long units = tiles + (long long)kSegmentCost * num_kv_heads * num_seqs;
    if (len_cap > INT32_MAX || units > INT32_MAX) return PS_ERR_UNSUPPORTED;
    if (num_blocks * num_kv_heads > INT32_MAX) return PS_ERR_UNSUPPORTED;
    return PS_OK;
}

struct DecodeParams {
    const uint16_t *q;          // bf16 [S][Hq][128]
    const int *block_table;     // [S][mbps]
    const int *seq_lens;        // [S]
    uint16_t *out;              // bf16 [S][Hq][128]
    int *ws_header;
    int *seg_done;              // [S][Hkv] tiles finished per segment (self-resetting)
    float *ws_acc;              // [slots][8][128]
    float *ws_ml;               // [slots][8][2]
    int num_seqs, num_q_heads, num_kv_heads, group, block_size, max_blocks_per_seq;
    long long num_blocks;
    int len_cap;                // max_blocks_per_seq * block_size
    int max_workers;            // cap on workers
    int min_stages;             // floor on a worker's share
    float scale_log2;           // scale * log2(e)
    // Fused append (all null for plain decode attention): the current token's
    // K and V, bf16 [S][Hkv][128], written into its cache slot and attended.
    const uint16_t *k_new, *v_new;
    uint16_t *k_cache_w, *v_cache_w;
    long long test_stall_ns;    // > 0: injected stall (ps_test_inject), else 0
};

// Launcher (ps_decode_kernels.cu).  Returns cudaSuccess or the launch error.
// Adds one to the library's launch counter (ps_decode_launch_count()).
void note_launch();

// One-shot faults set by ps_test_inject(): the CUDA error the next launch
// reports instead of launching (cudaSuccess: none), and the stall the next
// decode or prefill launch makes (0: none).  Each call consumes what it
// returns.
cudaError_t take_injected_launch_error();
long long take_injected_stall_ns();
long long take_injected_prefill_stall_ns();

cudaError_t launch_decode(const DecodeParams &p, const CUtensorMap &tmK, const CUtensorMap &tmV, int grid_ctas,
                          size_t smem_bytes, cudaStream_t stream);

}  // namespace ps
