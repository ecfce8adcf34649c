/*
 * ps_decode.h -- C ABI of the GB300 (sm_103a) paged decode-attention library.
 *
 * The library computes batched decode-phase attention for the thinking and
 * answer tokens of reasoning LLM serving (PowerSlider, Sec. 2.2: decode emits
 * one token per sequence per step and is bound by reading the KV cache; App.
 * B.2 Eq. (bytes-layer) charges it 2BSd bytes of KV per layer).  Every query
 * head h of sequence s attends over all L_s cached tokens of that sequence:
 *
 *   o[s][h] = sum_{t < L_s} softmax_t(scale * q[s][h] . K_s[t]) V_s[t]
 *
 * with grouped-query heads (g = num_q_heads / num_kv_heads query heads share
 * KV head h / g) and a paged KV cache addressed through a block table.
 *
 * ---------------------------------------------------------------- layouts --
 *  q           bf16  [num_seqs][num_q_heads][head_dim]              contiguous
 *  k_cache     bf16  [num_blocks][num_kv_heads][block_size][head_dim] contiguous
 *  v_cache     bf16  same layout as k_cache
 *  block_table int32 [num_seqs][max_blocks_per_seq] row-major; token t of
 *              sequence s is slot t % block_size of physical block
 *              block_table[s][t / block_size].  Entries past the last block a
 *              sequence uses are never read.
 *  seq_lens    int32 [num_seqs]; number of cached tokens of each sequence,
 *              the current token included.  0 is allowed (output row = 0).
 *  out         bf16  [num_seqs][num_q_heads][head_dim]; fully overwritten,
 *              round-to-nearest-even from fp32.
 *
 * ----------------------------------------------------------- conventions --
 *  - Every tensor pointer is a DEVICE pointer owned by the caller; the library
 *    never allocates or frees device memory.  q, k_cache, v_cache and out
 *    must be 16-byte aligned; block_table and seq_lens 4-byte aligned.
 *  - Calls are asynchronous and ordered on the given CUDA stream
 *    (cudaStream_t passed as void*; NULL is the legacy default stream).
 *  - Supported shapes: head_dim == 128; 1 <= num_q_heads / num_kv_heads <= 8;
 *    block_size a multiple of 16 in [16, 256]; 1 <= num_seqs <= 4096.
 *    Other shapes return PS_ERR_UNSUPPORTED.
 *  - Device-side values are not validated on the host.  A seq_lens value
 *    above max_blocks_per_seq * block_size is clamped to it, and a block id
 *    outside [0, num_blocks) reads zeros; both set a flag readable with
 *    ps_decode_plan_read_device_status().  Nothing faults.
 *  - Split-KV workspace: the caller allocates ps_decode_plan_create()'s
 *    workspace_bytes of device memory and hands it to the plan.  It holds
 *    the partial (max, sum, weighted-value) states of cut pieces plus a few
 *    counters that every call leaves at zero.  One workspace must not be
 *    used by two calls that can run concurrently; after a call that raised
 *    PS_DEVICE_TIMEOUT, hand the workspace to the plan again
 *    (ps_decode_plan_set_workspace) so that its counters are re-zeroed.
 *  - Results are bit-deterministic: the split of the work depends only on
 *    the sequence lengths and the plan, never on scheduling.
 *  - A plan is not thread-safe: use it from one host thread at a time.
 */
#ifndef PS_DECODE_H
#define PS_DECODE_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int ps_status_t;

#define PS_OK 0
#define PS_ERR_INVALID_ARG (-1) /* null pointer, bad dimension, misalignment */
#define PS_ERR_UNSUPPORTED (-2) /* valid but outside the shapes listed above */
#define PS_ERR_NO_PLAN (-3)     /* no plan bound to the stream, or dims differ */
#define PS_ERR_WORKSPACE (-4)   /* workspace missing or smaller than planned */
#define PS_ERR_CUDA (-5)        /* a CUDA runtime/driver call failed */

/* Flags of the device status word (ps_decode_plan_read_device_status). */
#define PS_DEVICE_TIMEOUT 1u       /* an in-kernel wait ran out; output invalid */
#define PS_DEVICE_BAD_BLOCK 2u     /* a block id outside [0, num_blocks) was read */
#define PS_DEVICE_LEN_CLAMPED 4u   /* a seq_lens entry exceeded the block-table row */

typedef struct ps_decode_plan ps_decode_plan_t; /* opaque, host-owned */

/* Read-only description of a plan, for tests and measurement. */
typedef struct ps_decode_plan_info {
    int num_seqs, num_q_heads, num_kv_heads, head_dim, block_size;
    int max_blocks_per_seq;
    long long num_blocks;
    int num_sms;               /* SMs the grid is sized for */
    int grid_ctas;             /* CTAs of the split-KV partial kernel */
    int workers_per_cta;       /* independent streaming warps per CTA */
    int stages_per_worker;     /* 16-token K/V tiles in flight per warp */
    int max_workers;           /* cap on the number of equal ranges the work is split into */
    int min_stages_per_worker; /* floor on a worker's share, in 16-token tiles */
    size_t workspace_bytes;
    size_t smem_bytes;         /* dynamic shared memory of the partial kernel */
} ps_decode_plan_info_t;

/*
 * Plan a decode-attention shape.  The plan fixes the grid of the kernel (one
 * CTA per SM, eight streaming warps each) and sizes the workspace that
 * carries the partial (max, sum, weighted-value) states of split-KV pieces
 * to the log-sum-exp merge.  No device memory is allocated.
 *
 *   max_blocks_per_seq  row stride of block_table (entries)
 *   num_blocks          physical blocks in k_cache / v_cache (TMA bounds)
 *   plan                out: new plan; free with ps_decode_plan_destroy()
 *   workspace_bytes     out: device bytes the caller must provide
 *
 * Queries the current CUDA device for its SM count.  Errors:
 * PS_ERR_INVALID_ARG (null out-pointers, non-positive dims, num_q_heads not a
 * multiple of num_kv_heads), PS_ERR_UNSUPPORTED (shape outside the supported
 * set), PS_ERR_CUDA (no device).
 */
ps_status_t ps_decode_plan_create(int num_seqs, int num_q_heads, int num_kv_heads, int head_dim,
                                  int block_size, int max_blocks_per_seq, long long num_blocks,
                                  ps_decode_plan_t **plan, size_t *workspace_bytes);

/*
 * As ps_decode_plan_create(), with explicit knobs (0 = default for each):
 *   num_sms                SM count to size the grid for (0: query the device;
 *                          a positive value needs no GPU, e.g. for host tests;
 *                          at most 4096, else PS_ERR_UNSUPPORTED)
 *   max_workers            upper bound on the number of contiguous ranges of
 *                          equal cost the batch's KV stream is split into
 *                          (1 = one warp does everything, no split)
 *   min_stages_per_worker  smallest range, in 16-token tiles
 *                          (1 = split as finely as the workers allow)
 */
ps_status_t ps_decode_plan_create_ex(int num_seqs, int num_q_heads, int num_kv_heads, int head_dim,
                                     int block_size, int max_blocks_per_seq, long long num_blocks,
                                     int num_sms, int max_workers, int min_stages_per_worker,
                                     ps_decode_plan_t **plan, size_t *workspace_bytes);

/* Give the plan its caller-owned device workspace (>= workspace_bytes, 256-byte
 * aligned).  The first call after this zeroes the workspace's counters and
 * status word on that call's stream.  Errors: PS_ERR_INVALID_ARG,
 * PS_ERR_WORKSPACE. */
ps_status_t ps_decode_plan_set_workspace(ps_decode_plan_t *plan, void *workspace, size_t bytes);

/* Bind the plan to a stream so that ps_decode_attention() on that stream
 * uses it (the 13-argument call has no block-table stride and no workspace
 * of its own).  Binding NULL plan removes the stream's binding.  A stream has
 * at most one plan; rebinding replaces it.  Errors: none besides
 * PS_ERR_INVALID_ARG for a destroyed plan. */
ps_status_t ps_decode_plan_bind(ps_decode_plan_t *plan, void *stream);

/* Destroy a plan and drop every stream binding to it.  NULL is a no-op. */
ps_status_t ps_decode_plan_destroy(ps_decode_plan_t *plan);

/* Fill *info with the plan's shape and launch configuration. */
ps_status_t ps_decode_plan_info(const ps_decode_plan_t *plan, ps_decode_plan_info_t *info);

/*
 * Decode attention with the plan bound to `stream` (ps_decode_plan_bind).
 * Launches one kernel on `stream`: the split-KV streaming pass with the
 * log-sum-exp merge of cut pieces fused into it.  scale is applied to q . k
 * before the softmax (1/sqrt(head_dim) for standard attention; any finite
 * value is accepted).
 *
 * Errors: PS_ERR_NO_PLAN when no plan is bound to `stream` or its
 * (num_seqs, num_q_heads, num_kv_heads, head_dim, block_size) differ from the
 * arguments; PS_ERR_WORKSPACE when the plan has no workspace;
 * PS_ERR_INVALID_ARG for null/misaligned pointers or a non-finite scale;
 * PS_ERR_CUDA when a launch fails.  Nothing is launched on error.
 */
ps_status_t ps_decode_attention(const void *q, const void *k_cache, const void *v_cache,
                                const int *block_table, const int *seq_lens, void *out,
                                int num_seqs, int num_q_heads, int num_kv_heads, int head_dim,
                                int block_size, float scale, void *stream);

/* The same computation with an explicit plan (no stream binding needed).
 * CUDA graphs: a call can be captured into a graph on `stream` once the plan
 * has made one call outside capture with the same k_cache / v_cache (that
 * call encodes the TMA descriptors on the host and clears the workspace's
 * status word); replays then read whatever the captured pointers hold. */
ps_status_t ps_decode_attention_planned(const ps_decode_plan_t *plan, const void *q,
                                        const void *k_cache, const void *v_cache,
                                        const int *block_table, const int *seq_lens, void *out,
                                        float scale, void *stream);

/*
 * One whole decode step of attention: append the current token's key and
 * value to the paged cache and attend over every cached token including it
 * (PowerSlider Sec. 2.2: each decode step adds one token per sequence and
 * reads the whole KV cache).  One kernel launch.
 *
 *   k_new, v_new  bf16 [num_seqs][num_kv_heads][head_dim], 16-byte aligned:
 *                 the current token's key and value
 *   k_cache, v_cache  as in ps_decode_attention(), written in place: for
 *                 every sequence with seq_lens[s] > 0, slot
 *                 (seq_lens[s]-1) % block_size of block
 *                 block_table[s][(seq_lens[s]-1) / block_size] receives the
 *                 new rows (the caller has already counted the new token in
 *                 seq_lens and reserved its block).  Nothing else in the
 *                 cache is written.
 * The result equals writing the rows first and then calling
 * ps_decode_attention().  Errors as ps_decode_attention_planned(), plus
 * PS_ERR_INVALID_ARG for a null or misaligned k_new / v_new.
 */
ps_status_t ps_decode_append_attention_planned(const ps_decode_plan_t *plan, const void *q, const void *k_new,
                                               const void *v_new, void *k_cache, void *v_cache,
                                               const int *block_table, const int *seq_lens, void *out,
                                               float scale, void *stream);

/*
 * KV hand-off between stage pools (PowerSlider Sec. 5: a reasoning request's
 * KV cache moves from the thinking pool to the answer pool).  These are the
 * on-GPU gather and scatter on either side of the transfer; the transport is
 * the caller's.  Neither needs a plan.
 *
 * Packed layout of sequence i, starting at element offset offsets[i] (int64,
 * device array, a multiple of 8): K[j][t][0..head_dim) for kv head
 * j < num_kv_heads and token t < seq_lens[i], then V in the same order, i.e.
 * 2 * num_kv_heads * seq_lens[i] * head_dim bf16 elements.
 *
 * ps_kv_pack copies slot (block_table[i][t / block_size], j, t % block_size)
 * of k_cache / v_cache to packed position (j, t).  ps_kv_unpack copies packed
 * position (j, t) to that slot of the destination pool (block_table being the
 * receiver's); slots of the pool that no packed token maps to are not written.
 *
 *   caches, dst/src  bf16, 16-byte aligned; cache layout as for decode
 *   block_table      int32 [num_seqs][max_blocks_per_seq]
 *   seq_lens         int32 [num_seqs] (values above max_blocks_per_seq *
 *                    block_size are clamped; a sequence whose offset is not a
 *                    multiple of 8 is skipped; both raise
 *                    PS_DEVICE_LEN_CLAMPED)
 *   num_blocks       blocks in the pool; out-of-pool ids skip their page and
 *                    raise PS_DEVICE_BAD_BLOCK
 *   device_status    optional device word that receives PS_DEVICE_* flags
 * Supported: head_dim a multiple of 8, 1 <= num_seqs <= 4096.  Errors:
 * PS_ERR_INVALID_ARG, PS_ERR_UNSUPPORTED, PS_ERR_CUDA.
 */
ps_status_t ps_kv_pack(const void *k_cache, const void *v_cache, const int *block_table,
                       int max_blocks_per_seq, const int *seq_lens, int num_seqs, int num_kv_heads,
                       int head_dim, int block_size, long long num_blocks, const long long *dst_offsets,
                       void *dst, unsigned int *device_status, void *stream);

ps_status_t ps_kv_unpack(const void *src, const long long *src_offsets, const int *block_table,
                         int max_blocks_per_seq, const int *seq_lens, int num_seqs, int num_kv_heads,
                         int head_dim, int block_size, long long num_blocks, void *k_cache, void *v_cache,
                         unsigned int *device_status, void *stream);

/*
 * Chunked-prefill attention over the paged cache (PowerSlider Sec. 2.2: the
 * prefill phase processes the new prompt tokens together and is compute-bound,
 * Sec. 3 Obs. 2).  Sequence s owns query rows q_start[s] .. q_start[s+1]-1;
 * they are the LAST Q_s = q_start[s+1] - q_start[s] of its seq_lens[s] cached
 * tokens (their K/V are already in the cache), and query i of the sequence,
 * at position p = seq_lens[s] - Q_s + i, attends to the cached tokens 0 .. p:
 *
 *   out[q_start[s] + i][h] = sum_{t <= p} softmax_t(scale * q . K_s[t]) V_s[t]
 *
 * with KV head h / g as for decode.  Q.K^T and P.V run on the tensor cores
 * (tcgen05, fp32 accumulation in tensor memory); P is rounded to bf16.
 *
 *   q, out       bf16 [total_q_tokens][num_q_heads][head_dim], 16-byte aligned
 *   k_cache, v_cache, block_table  as for ps_decode_attention()
 *   seq_lens     int32 [num_seqs], tokens in the cache including the new ones
 *   q_start      int32 [num_seqs + 1], q_start[0] = 0, non-decreasing,
 *                q_start[num_seqs] <= total_q_tokens (all three on the device)
 *   max_q_len    an upper bound on Q_s over the batch (sizes the grid; the
 *                query tiles past a sequence's Q_s do nothing; a chunk longer
 *                than max_q_len has its rows past it left unwritten and raises
 *                PS_DEVICE_LEN_CLAMPED).  With max_q_len, num_seqs or
 *                total_q_tokens 0 the call launches nothing and returns PS_OK
 *                (no row is written and no flag raised).
 *   device_status  optional device word that receives PS_DEVICE_* flags
 * A sequence with Q_s > seq_lens[s], a negative Q_s, a length above
 * max_blocks_per_seq * block_size or rows outside [0, total_q_tokens) is
 * skipped (its rows are not written) and raises PS_DEVICE_LEN_CLAMPED; an
 * out-of-pool block id reads zeros and raises PS_DEVICE_BAD_BLOCK; a stalled
 * pipeline gives up after ~2 s and raises PS_DEVICE_TIMEOUT.
 * Supported: head_dim 128, g = num_q_heads / num_kv_heads <= 16, block_size a
 * multiple of 16, num_seqs <= 65535.  Needs no workspace.  Errors:
 * PS_ERR_INVALID_ARG (null or misaligned pointer, bad sizes, non-finite
 * scale), PS_ERR_UNSUPPORTED, PS_ERR_CUDA.
 */
ps_status_t ps_prefill_attention(const void *q, const void *k_cache, const void *v_cache, const int *block_table,
                                 const int *seq_lens, const int *q_start, void *out, int num_seqs,
                                 int total_q_tokens, int max_q_len, int num_q_heads, int num_kv_heads,
                                 int head_dim, int block_size, int max_blocks_per_seq, long long num_blocks,
                                 float scale, unsigned int *device_status, void *stream);

/*
 * Measurement hook: when events are set (cudaEvent_t as void*, NULL to
 * clear), every call records ev_start right before its kernel and ev_end
 * right after it, on the call's stream.
 */
ps_status_t ps_decode_plan_set_timing_events(ps_decode_plan_t *plan, void *ev_start, void *ev_end);

/* Copy the device status word (PS_DEVICE_* flags raised by calls since the
 * last read) to *flags, synchronising `stream`, then clear it.  Errors:
 * PS_ERR_WORKSPACE (no workspace), PS_ERR_CUDA. */
ps_status_t ps_decode_plan_read_device_status(ps_decode_plan_t *plan, void *stream,
                                              unsigned int *flags);

/*
 * Decode attention for callers that cannot allocate device memory.  (The
 * paper has no counterpart; this is a deployment convenience.)
 *
 * Some callers can pass the library their tensors but cannot give it a
 * workspace: plugins whose host engine owns every device allocation, callers
 * over a foreign-function interface that hold only the buffers they pass in,
 * or serving processes that budget all device memory at start-up and forbid
 * allocations afterwards.  This entry point needs no plan and no workspace:
 * the split-KV scratch lives in a fixed device array inside the library of
 * PS_NOALLOC_SCRATCH_BYTES, which every GPU that loads the library holds
 * until the process exits.  It calls no cudaMalloc, cudaFree or other
 * allocating routine.
 *
 * Arguments are those of ps_decode_attention() plus the two a plan would
 * otherwise supply: max_blocks_per_seq (the block_table row stride) and
 * num_blocks (physical blocks in k_cache / v_cache).  The work is split
 * statically, with the same kernel and the same numerics as the planned path.
 *
 * - Every call looks up the scratch array's device address in the current
 *   context, so a call after cudaDeviceReset() or under another context uses
 *   that context's copy.  The first call on each device does the set-up:
 *   under CUDA's default lazy module loading it loads the library's module
 *   there, which commits the array's PS_NOALLOC_SCRATCH_BYTES of device
 *   memory at that moment, and it sets the kernel's shared-memory limit.  A
 *   server that forbids allocation after start-up should therefore make one
 *   call on each device during start-up (or set CUDA_MODULE_LOADING=EAGER),
 *   and that first call must come before any stream capture.
 * - Every call shares the one array and first clears its counters on
 *   `stream`.  Calls that overlap on the GPU (other streams, other host
 *   threads) race on the array and produce wrong results: serialise them.
 * - Shapes whose scratch need exceeds PS_NOALLOC_SCRATCH_BYTES (2 partial
 *   states of 8 x 130 floats per streaming warp, plus 4 bytes per
 *   (sequence, kv-head)) return PS_ERR_UNSUPPORTED before anything is
 *   launched.
 * - Launches through this entry point are not counted by
 *   ps_decode_launch_count(), and there is no device status word to read.
 * Errors: PS_ERR_INVALID_ARG, PS_ERR_UNSUPPORTED, PS_ERR_CUDA.
 */
#define PS_NOALLOC_SCRATCH_BYTES (16u << 20)
ps_status_t ps_decode_attention_noalloc(const void *q, const void *k_cache, const void *v_cache,
                                        const int *block_table, const int *seq_lens, void *out,
                                        int num_seqs, int num_q_heads, int num_kv_heads, int head_dim,
                                        int block_size, int max_blocks_per_seq, long long num_blocks,
                                        float scale, void *stream);

/*
 * Fault injection, for tests of the error paths (process-wide, one shot,
 * value 0 clears; nothing here faults, traps or hangs the GPU):
 *   PS_INJECT_LAUNCH_ERROR  the library's next kernel launch, from any entry
 *                           point, is not made; the call returns PS_ERR_CUDA
 *                           as if the launch had reported CUDA error `value`
 *                           (1 .. 10000).
 *   PS_INJECT_DECODE_STALL  the next decode-attention launch makes every
 *                           streaming warp first wait, for `value` ns
 *                           (1000 .. 1000000000), on an mbarrier that nothing
 *                           arrives on.  The wait runs out as a real stall
 *                           would: the kernel raises PS_DEVICE_TIMEOUT, lets
 *                           the copies it has in flight land and exits
 *                           without writing any output (which is then
 *                           invalid).  Recovery is the documented one.
 *   PS_INJECT_PREFILL_STALL the next chunked-prefill launch makes one
 *                           softmax warpgroup of every CTA pair first wait,
 *                           for `value` ns (1000 .. 1000000000), on an
 *                           mbarrier that nothing arrives on.  The wait runs out as a real
 *                           stall would: both CTAs of every pair give up,
 *                           PS_DEVICE_TIMEOUT is raised, the copies in flight
 *                           land, tensor memory is freed and the kernel exits
 *                           without writing output.  The next call is normal.
 * Errors: PS_ERR_INVALID_ARG for an unknown kind or a value out of range.
 */
#define PS_INJECT_LAUNCH_ERROR 1
#define PS_INJECT_DECODE_STALL 2
#define PS_INJECT_PREFILL_STALL 3
ps_status_t ps_test_inject(int kind, long long value);

/* Number of kernels this library has launched in this process through the
 * decode, fused-append, prefill and KV hand-off entry points (the
 * workspace-free entry point is not counted). */
unsigned long long ps_decode_launch_count(void);

/* Static description of a status code. */
const char *ps_status_string(ps_status_t status);

/* ABI version of this header (major * 100 + minor). */
int ps_decode_abi_version(void);

#ifdef __cplusplus
}
#endif

#endif /* PS_DECODE_H */
