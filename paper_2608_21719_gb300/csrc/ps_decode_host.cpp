// ps_decode_host.cpp -- the C ABI of include/ps_decode.h: argument checks,
// plans, stream bindings, TMA descriptor encoding and the launch.
#include <cuda.h>
#include <cuda_runtime.h>

#include <atomic>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>
#include <new>
#include <unordered_map>

#include "ps_decode.h"
#include "ps_internal.h"

using namespace ps;

struct ps_decode_plan {
    uint32_t magic;
    int num_seqs, num_q_heads, num_kv_heads, head_dim, block_size, max_blocks_per_seq;
    long long num_blocks;
    int num_sms, grid_ctas, max_workers, min_stages;
    size_t smem_bytes;
    WorkspaceLayout ws;
    void *workspace = nullptr;
    size_t workspace_size = 0;
    bool status_needs_clear = false;
    // TMA descriptors for the last (k_cache, v_cache) pair seen.
    const void *tm_k_ptr = nullptr, *tm_v_ptr = nullptr;
    alignas(64) CUtensorMap tmK;
    alignas(64) CUtensorMap tmV;
    cudaEvent_t ev_start = nullptr, ev_end = nullptr;
};

namespace {

constexpr uint32_t kPlanMagic = 0x50534450u;  // "PSDP"
std::atomic<unsigned long long> g_launches{0};
std::mutex g_bind_mu;
std::unordered_map<void *, ps_decode_plan *> g_bindings;

bool live(const ps_decode_plan *p) { return p != nullptr && p->magic == kPlanMagic; }

bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
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

// 4-D view of a paged cache: dim0 = 64 dims of a half row (contiguous), dim1 =
// slot within the block (256-byte stride), dim2 = half of the row (128-byte
// stride), dim3 = (block, kv-head) page.  A box of 64 dims x 16 slots x 2
// halves x 1 page lands in shared memory as one 128-byte-swizzled tile laid
// out [half][slot][64], so one copy fetches a 16-token tile of K or V.
ps_status_t encode_cache_map(CUtensorMap *tm, const void *base, const ps_decode_plan *p) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return PS_ERR_CUDA;
    cuuint64_t dims[4] = {64, (cuuint64_t)p->block_size, 2, (cuuint64_t)p->num_blocks * (cuuint64_t)p->num_kv_heads};
    cuuint64_t strides[3] = {(cuuint64_t)kHeadDim * 2, 64 * 2, (cuuint64_t)p->block_size * kHeadDim * 2};
    cuuint32_t box[4] = {64, (cuuint32_t)kTileTokens, 2, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    CUresult r = fn(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? PS_OK : PS_ERR_CUDA;
}

ps_status_t run_planned(ps_decode_plan *p, const void *q, const void *k, const void *v, const int *bt,
                        const int *sl, void *out, float scale, void *stream, const void *k_new = nullptr,
                        const void *v_new = nullptr) {
    if (!q || !k || !v || !bt || !sl || !out) return PS_ERR_INVALID_ARG;
    if ((k_new == nullptr) != (v_new == nullptr)) return PS_ERR_INVALID_ARG;
    if (k_new && (!aligned(k_new, 16) || !aligned(v_new, 16))) return PS_ERR_INVALID_ARG;
    if (!aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) || !aligned(bt, 4) || !aligned(sl, 4) ||
        !aligned(out, 16))
        return PS_ERR_INVALID_ARG;
    if (!std::isfinite(scale)) return PS_ERR_INVALID_ARG;
    if (!p->workspace || p->workspace_size < p->ws.total) return PS_ERR_WORKSPACE;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);

    if (p->tm_k_ptr != k) {
        ps_status_t e = encode_cache_map(&p->tmK, k, p);
        if (e != PS_OK) return e;
        p->tm_k_ptr = k;
    }
    if (p->tm_v_ptr != v) {
        ps_status_t e = encode_cache_map(&p->tmV, v, p);
        if (e != PS_OK) return e;
        p->tm_v_ptr = v;
    }
    uint8_t *ws = static_cast<uint8_t *>(p->workspace);
    if (p->status_needs_clear) {
        // The status word and the per-segment counters start at zero; the
        // kernel returns the counters to zero at the end of every call.
        if (cudaMemsetAsync(ws, 0, p->ws.acc_off, st) != cudaSuccess) return PS_ERR_CUDA;
        p->status_needs_clear = false;
    }

    DecodeParams dp;
    dp.q = static_cast<const uint16_t *>(q);
    dp.block_table = bt;
    dp.seq_lens = sl;
    dp.out = static_cast<uint16_t *>(out);
    dp.ws_header = reinterpret_cast<int *>(ws);
    dp.seg_done = reinterpret_cast<int *>(ws + p->ws.seg_done_off);
    dp.ws_acc = reinterpret_cast<float *>(ws + p->ws.acc_off);
    dp.ws_ml = reinterpret_cast<float *>(ws + p->ws.ml_off);
    dp.num_seqs = p->num_seqs;
    dp.num_q_heads = p->num_q_heads;
    dp.num_kv_heads = p->num_kv_heads;
    dp.group = p->num_q_heads / p->num_kv_heads;
    dp.block_size = p->block_size;
    dp.max_blocks_per_seq = p->max_blocks_per_seq;
    dp.num_blocks = p->num_blocks;
    dp.len_cap = p->max_blocks_per_seq * p->block_size;
    dp.max_workers = p->max_workers;
    dp.min_stages = p->min_stages;
    dp.scale_log2 = (float)((double)scale * 1.4426950408889634);
    dp.k_new = static_cast<const uint16_t *>(k_new);
    dp.v_new = static_cast<const uint16_t *>(v_new);
    dp.k_cache_w = k_new ? static_cast<uint16_t *>(const_cast<void *>(k)) : nullptr;
    dp.v_cache_w = k_new ? static_cast<uint16_t *>(const_cast<void *>(v)) : nullptr;

    if (p->ev_start && cudaEventRecord(p->ev_start, st) != cudaSuccess) return PS_ERR_CUDA;
    if (launch_decode(dp, p->tmK, p->tmV, p->grid_ctas, p->smem_bytes, st) != cudaSuccess) return PS_ERR_CUDA;
    g_launches.fetch_add(1, std::memory_order_relaxed);
    if (p->ev_end && cudaEventRecord(p->ev_end, st) != cudaSuccess) return PS_ERR_CUDA;
    return PS_OK;
}

}  // namespace

void ps::note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

namespace {
std::atomic<int> g_inject_launch_error{0};
std::atomic<long long> g_inject_stall_ns{0};
std::atomic<long long> g_inject_prefill_stall_ns{0};
}  // namespace

cudaError_t ps::take_injected_launch_error() {
    return static_cast<cudaError_t>(g_inject_launch_error.exchange(0, std::memory_order_acq_rel));
}

long long ps::take_injected_stall_ns() { return g_inject_stall_ns.exchange(0, std::memory_order_acq_rel); }

long long ps::take_injected_prefill_stall_ns() {
    return g_inject_prefill_stall_ns.exchange(0, std::memory_order_acq_rel);
}

ps_status_t ps_test_inject(int kind, long long value) {
    switch (kind) {
        case PS_INJECT_LAUNCH_ERROR:
            if (value < 0 || value > 10000) return PS_ERR_INVALID_ARG;
            g_inject_launch_error.store((int)value, std::memory_order_release);
            return PS_OK;
        case PS_INJECT_DECODE_STALL:
            if (value != 0 && (value < 1000 || value > 1000000000)) return PS_ERR_INVALID_ARG;
            g_inject_stall_ns.store(value, std::memory_order_release);
            return PS_OK;
        case PS_INJECT_PREFILL_STALL:
            if (value != 0 && (value < 1000 || value > 1000000000)) return PS_ERR_INVALID_ARG;
            g_inject_prefill_stall_ns.store(value, std::memory_order_release);
            return PS_OK;
        default:
            return PS_ERR_INVALID_ARG;
    }
}

extern "C" {

ps_status_t ps_decode_plan_create_ex(int num_seqs, int num_q_heads, int num_kv_heads, int head_dim, int block_size,
                                     int max_blocks_per_seq, long long num_blocks, int num_sms, int max_workers,
                                     int min_stages_per_worker, ps_decode_plan_t **plan, size_t *workspace_bytes) {
    if (!plan || !workspace_bytes) return PS_ERR_INVALID_ARG;
    *plan = nullptr;
    *workspace_bytes = 0;
    if (num_sms < 0 || max_workers < 0 || min_stages_per_worker < 0) return PS_ERR_INVALID_ARG;
    if (num_sms > kMaxGridCtas) return PS_ERR_UNSUPPORTED;
    ps_status_t e = check_decode_shape(num_seqs, num_q_heads, num_kv_heads, head_dim, block_size, max_blocks_per_seq,
                                num_blocks);
    if (e != PS_OK) return e;
    if (num_sms == 0) {
        int dev = 0;
        if (cudaGetDevice(&dev) != cudaSuccess) return PS_ERR_CUDA;
        if (cudaDeviceGetAttribute(&num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || num_sms <= 0)
            return PS_ERR_CUDA;
    }
    ps_decode_plan *p = new (std::nothrow) ps_decode_plan();
    if (!p) return PS_ERR_INVALID_ARG;
    p->magic = kPlanMagic;
    p->num_seqs = num_seqs;
    p->num_q_heads = num_q_heads;
    p->num_kv_heads = num_kv_heads;
    p->head_dim = head_dim;
    p->block_size = block_size;
    p->max_blocks_per_seq = max_blocks_per_seq;
    p->num_blocks = num_blocks;
    p->num_sms = num_sms;
    p->grid_ctas = num_sms;
    const int total_workers = p->grid_ctas * kWorkersPerCta;
    p->max_workers = (max_workers > 0 && max_workers < total_workers) ? max_workers : total_workers;
    p->min_stages = min_stages_per_worker > 0 ? min_stages_per_worker : kDefaultMinStages;
    p->smem_bytes = partial_smem_bytes(num_seqs);
    p->ws = workspace_layout(num_seqs, num_kv_heads, total_workers);
    *plan = p;
    *workspace_bytes = p->ws.total;
    return PS_OK;
}

ps_status_t ps_decode_plan_create(int num_seqs, int num_q_heads, int num_kv_heads, int head_dim, int block_size,
                                  int max_blocks_per_seq, long long num_blocks, ps_decode_plan_t **plan,
                                  size_t *workspace_bytes) {
    return ps_decode_plan_create_ex(num_seqs, num_q_heads, num_kv_heads, head_dim, block_size, max_blocks_per_seq,
                                    num_blocks, 0, 0, 0, plan, workspace_bytes);
}

ps_status_t ps_decode_plan_set_workspace(ps_decode_plan_t *plan, void *workspace, size_t bytes) {
    if (!live(plan) || !workspace || !aligned(workspace, 256)) return PS_ERR_INVALID_ARG;
    if (bytes < plan->ws.total) return PS_ERR_WORKSPACE;
    plan->workspace = workspace;
    plan->workspace_size = bytes;
    plan->status_needs_clear = true;
    return PS_OK;
}

ps_status_t ps_decode_plan_bind(ps_decode_plan_t *plan, void *stream) {
    std::lock_guard<std::mutex> lk(g_bind_mu);
    if (plan == nullptr) {
        g_bindings.erase(stream);
        return PS_OK;
    }
    if (!live(plan)) return PS_ERR_INVALID_ARG;
    g_bindings[stream] = plan;
    return PS_OK;
}

ps_status_t ps_decode_plan_destroy(ps_decode_plan_t *plan) {
    if (plan == nullptr) return PS_OK;
    if (!live(plan)) return PS_ERR_INVALID_ARG;
    {
        std::lock_guard<std::mutex> lk(g_bind_mu);
        for (auto it = g_bindings.begin(); it != g_bindings.end();)
            it = (it->second == plan) ? g_bindings.erase(it) : std::next(it);
    }
    plan->magic = 0;
    delete plan;
    return PS_OK;
}

ps_status_t ps_decode_plan_info(const ps_decode_plan_t *plan, ps_decode_plan_info_t *info) {
    if (!live(plan) || !info) return PS_ERR_INVALID_ARG;
    info->num_seqs = plan->num_seqs;
    info->num_q_heads = plan->num_q_heads;
    info->num_kv_heads = plan->num_kv_heads;
    info->head_dim = plan->head_dim;
    info->block_size = plan->block_size;
    info->max_blocks_per_seq = plan->max_blocks_per_seq;
    info->num_blocks = plan->num_blocks;
    info->num_sms = plan->num_sms;
    info->grid_ctas = plan->grid_ctas;
    info->workers_per_cta = kWorkersPerCta;
    info->stages_per_worker = kStages;
    info->max_workers = plan->max_workers;
    info->min_stages_per_worker = plan->min_stages;
    info->workspace_bytes = plan->ws.total;
    info->smem_bytes = plan->smem_bytes;
    return PS_OK;
}

ps_status_t ps_decode_attention_planned(const ps_decode_plan_t *plan, const void *q, const void *k_cache,
                                        const void *v_cache, const int *block_table, const int *seq_lens, void *out,
                                        float scale, void *stream) {
    if (!live(plan)) return PS_ERR_NO_PLAN;
    return run_planned(const_cast<ps_decode_plan *>(plan), q, k_cache, v_cache, block_table, seq_lens, out, scale,
                       stream);
}

ps_status_t ps_decode_append_attention_planned(const ps_decode_plan_t *plan, const void *q, const void *k_new,
                                               const void *v_new, void *k_cache, void *v_cache,
                                               const int *block_table, const int *seq_lens, void *out, float scale,
                                               void *stream) {
    if (!live(plan)) return PS_ERR_NO_PLAN;
    if (!k_new || !v_new) return PS_ERR_INVALID_ARG;
    return run_planned(const_cast<ps_decode_plan *>(plan), q, k_cache, v_cache, block_table, seq_lens, out, scale,
                       stream, k_new, v_new);
}

ps_status_t ps_decode_attention(const void *q, const void *k_cache, const void *v_cache, const int *block_table,
                                const int *seq_lens, void *out, int num_seqs, int num_q_heads, int num_kv_heads,
                                int head_dim, int block_size, float scale, void *stream) {
    ps_decode_plan *p = nullptr;
    {
        std::lock_guard<std::mutex> lk(g_bind_mu);
        auto it = g_bindings.find(stream);
        if (it != g_bindings.end()) p = it->second;
    }
    if (!live(p)) return PS_ERR_NO_PLAN;
    if (p->num_seqs != num_seqs || p->num_q_heads != num_q_heads || p->num_kv_heads != num_kv_heads ||
        p->head_dim != head_dim || p->block_size != block_size)
        return PS_ERR_NO_PLAN;
    return run_planned(p, q, k_cache, v_cache, block_table, seq_lens, out, scale, stream);
}

ps_status_t ps_decode_plan_set_timing_events(ps_decode_plan_t *plan, void *ev_start, void *ev_end) {
    if (!live(plan)) return PS_ERR_INVALID_ARG;
    plan->ev_start = reinterpret_cast<cudaEvent_t>(ev_start);
    plan->ev_end = reinterpret_cast<cudaEvent_t>(ev_end);
    return PS_OK;
}

ps_status_t ps_decode_plan_read_device_status(ps_decode_plan_t *plan, void *stream, unsigned int *flags) {
    if (!live(plan) || !flags) return PS_ERR_INVALID_ARG;
    if (!plan->workspace) return PS_ERR_WORKSPACE;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (plan->status_needs_clear) {
        *flags = 0;
        return PS_OK;
    }
    unsigned int h = 0;
    if (cudaMemcpyAsync(&h, plan->workspace, sizeof h, cudaMemcpyDeviceToHost, st) != cudaSuccess) return PS_ERR_CUDA;
    if (cudaStreamSynchronize(st) != cudaSuccess) return PS_ERR_CUDA;
    if (cudaMemsetAsync(plan->workspace, 0, sizeof h, st) != cudaSuccess) return PS_ERR_CUDA;
    *flags = h;
    return PS_OK;
}

unsigned long long ps_decode_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

const char *ps_status_string(ps_status_t s) {
    switch (s) {
        case PS_OK: return "ok";
        case PS_ERR_INVALID_ARG: return "invalid argument";
        case PS_ERR_UNSUPPORTED: return "unsupported shape";
        case PS_ERR_NO_PLAN: return "no matching plan bound to the stream";
        case PS_ERR_WORKSPACE: return "workspace missing or too small";
        case PS_ERR_CUDA: return "CUDA call failed";
        default: return "unknown status";
    }
}

int ps_decode_abi_version(void) { return 100; }

}  // extern "C"
