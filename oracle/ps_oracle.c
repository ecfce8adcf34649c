/*
 * ps_oracle.c -- plain fp64 CPU reference for batched decode-phase attention
 * over a paged KV cache with grouped-query heads.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the oracle that the CUDA path is
 * checked against.  Only the test suite, the smoke check in
 * __graft_entry__.py and the CPU-baseline leg of bench.py may load it.  It
 * shares no code, header, table or helper with the CUDA library, and it never
 * reads anything the CUDA library produced.
 *
 * What is computed (PowerSlider, Sec. 2.2: a decode step emits one new token
 * per sequence and attends over every cached token of that sequence; the KV
 * cache is the dominant byte stream, App. B.2 Eq. (bytes-layer), term 2BSd):
 *
 *   for each sequence s and query head h, with g = Hq / Hkv and KV head
 *   j = h / g (contiguous grouping),
 *
 *     x_t  = scale * sum_d q[s][h][d] * K_s[t][d],        t = 0 .. L_s - 1
 *     o[s][h][:] = sum_t exp(x_t - max_u x_u) V_s[t][:] / sum_t exp(x_t - max_u x_u)
 *
 *   where the logical token t of sequence s lives in physical block
 *   b = block_table[s][t / bs], slot t % bs, and
 *     K_s[t][:] = k_cache[b][j][t % bs][:]   (layout [num_blocks][Hkv][bs][d])
 *     V_s[t][:] = v_cache[b][j][t % bs][:].
 *   L_s = 0 gives an all-zero output row.
 *
 * Every input element is a bfloat16 bit pattern; it is widened exactly to
 * double, and all arithmetic is double precision with libm exp().  Nothing
 * is blocked, fused or reordered: each (s, h) row is a direct transcription
 * of the definition above.
 *
 * ps_oracle_decode_attention_split() computes the same quantity by cutting
 * each sequence's context into fixed chunks, keeping per chunk the running
 * maximum m_c, the sum l_c = sum exp(x - m_c) and the weighted value sum
 * acc_c, and merging the chunks with the log-sum-exp rule
 *   o = sum_c exp(m_c - M) acc_c / sum_c exp(m_c - M) l_c,  M = max_c m_c.
 * It exists so that the split-invariance of the definition can be pinned in
 * the tests; it is not a different method.
 *
 * Pins (tests/test_oracle_pins.py): brute-force dense attention on logical
 * arrays, closed forms (single token, constant V, zero query, equal keys),
 * invariance to physical block relabelling, invariance to chunking,
 * GQA == MHA with repeated KV heads, and torch's fp64 scaled-dot-product
 * attention on tiny dense shapes.
 *
 * ps_oracle_prefill_attention() is the chunked-prefill counterpart (query
 * tokens that are the last Q_s cached tokens, causal); its pins are dense
 * causal brute force, torch's fp64 causal scaled-dot-product attention on
 * whole prompts, bit-exact equality with the decode oracle when Q_s = 1, and
 * blindness to tokens after each query's position.
 *
 * ps_oracle_kv_pack()/ps_oracle_kv_unpack() are the KV hand-off gather and
 * scatter (pure data movement, pinned bit-exact).
 *
 * Error codes: 0 ok; -1 invalid argument; -2 a block id outside
 * [0, num_blocks) is referenced; -3 a sequence length exceeds
 * max_blocks_per_seq * block_size; -4 out of host memory.
 */
#include <math.h>
#include <pthread.h>
#include <stdatomic.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

static double bf16_bits_to_double(uint16_t bits)
{
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

typedef struct {
    const uint16_t *q;
    const uint16_t *k_cache;
    const uint16_t *v_cache;
    const int32_t *block_table;
    const int32_t *seq_lens;
    int num_seqs, num_q_heads, num_kv_heads, head_dim, block_size;
    int max_blocks_per_seq;
    long long num_blocks;
    double scale;
    int chunk_tokens; /* 0: no chunking */
    double *out;
    atomic_int next_row;
    atomic_int status;
} job_t;

/* Address of the first element of token t of sequence s, KV head j. */
static const uint16_t *token_row(const job_t *jb, const uint16_t *cache, int s, int j, int t, int *err)
{
    int32_t b = jb->block_table[(size_t)s * jb->max_blocks_per_seq + t / jb->block_size];
    if (b < 0 || (long long)b >= jb->num_blocks) {
        *err = -2;
        return NULL;
    }
    size_t page = (size_t)b * jb->num_kv_heads + (size_t)j;
    return cache + (page * jb->block_size + (size_t)(t % jb->block_size)) * jb->head_dim;
}

/* One output row by the plain definition. */
static int row_plain(job_t *jb, int s, int h, double *logits)
{
    const int d = jb->head_dim;
    const int g = jb->num_q_heads / jb->num_kv_heads;
    const int j = h / g;
    const int L = jb->seq_lens[s];
    const uint16_t *qv = jb->q + ((size_t)s * jb->num_q_heads + h) * d;
    double *o = jb->out + ((size_t)s * jb->num_q_heads + h) * d;
    int err = 0;

    for (int i = 0; i < d; ++i) o[i] = 0.0;
    if (L == 0) return 0;

    double m = -INFINITY;
    for (int t = 0; t < L; ++t) {
        const uint16_t *kr = token_row(jb, jb->k_cache, s, j, t, &err);
        if (err) return err;
        double dot = 0.0;
        for (int i = 0; i < d; ++i) dot += bf16_bits_to_double(qv[i]) * bf16_bits_to_double(kr[i]);
        logits[t] = jb->scale * dot;
        if (logits[t] > m) m = logits[t];
    }
    double z = 0.0;
    for (int t = 0; t < L; ++t) {
        double w = exp(logits[t] - m);
        z += w;
        const uint16_t *vr = token_row(jb, jb->v_cache, s, j, t, &err);
        if (err) return err;
        for (int i = 0; i < d; ++i) o[i] += w * bf16_bits_to_double(vr[i]);
    }
    for (int i = 0; i < d; ++i) o[i] /= z;
    return 0;
}

/* The same row through per-chunk (m, l, acc) states merged by log-sum-exp. */
static int row_split(job_t *jb, int s, int h, double *logits, double *acc_all, double *m_all, double *l_all)
{
    const int d = jb->head_dim;
    const int g = jb->num_q_heads / jb->num_kv_heads;
    const int j = h / g;
    const int L = jb->seq_lens[s];
    const int C = jb->chunk_tokens;
    const uint16_t *qv = jb->q + ((size_t)s * jb->num_q_heads + h) * d;
    double *o = jb->out + ((size_t)s * jb->num_q_heads + h) * d;
    int err = 0;

    for (int i = 0; i < d; ++i) o[i] = 0.0;
    if (L == 0) return 0;

    const int nchunks = (L + C - 1) / C;
    for (int c = 0; c < nchunks; ++c) {
        const int t0 = c * C;
        const int t1 = (t0 + C < L) ? t0 + C : L;
        double *acc = acc_all + (size_t)c * d;
        double m = -INFINITY;
        for (int t = t0; t < t1; ++t) {
            const uint16_t *kr = token_row(jb, jb->k_cache, s, j, t, &err);
            if (err) return err;
            double dot = 0.0;
            for (int i = 0; i < d; ++i) dot += bf16_bits_to_double(qv[i]) * bf16_bits_to_double(kr[i]);
            logits[t] = jb->scale * dot;
            if (logits[t] > m) m = logits[t];
        }
        double l = 0.0;
        for (int i = 0; i < d; ++i) acc[i] = 0.0;
        for (int t = t0; t < t1; ++t) {
            double w = exp(logits[t] - m);
            l += w;
            const uint16_t *vr = token_row(jb, jb->v_cache, s, j, t, &err);
            if (err) return err;
            for (int i = 0; i < d; ++i) acc[i] += w * bf16_bits_to_double(vr[i]);
        }
        m_all[c] = m;
        l_all[c] = l;
    }
    double M = -INFINITY;
    for (int c = 0; c < nchunks; ++c)
        if (m_all[c] > M) M = m_all[c];
    double z = 0.0;
    for (int c = 0; c < nchunks; ++c) {
        double w = exp(m_all[c] - M);
        z += w * l_all[c];
        for (int i = 0; i < d; ++i) o[i] += w * acc_all[(size_t)c * d + i];
    }
    for (int i = 0; i < d; ++i) o[i] /= z;
    return 0;
}

static void *worker(void *arg)
{
    job_t *jb = (job_t *)arg;
    int maxL = 0;
    for (int s = 0; s < jb->num_seqs; ++s)
        if (jb->seq_lens[s] > maxL) maxL = jb->seq_lens[s];
    double *logits = (double *)malloc(sizeof(double) * (size_t)(maxL > 0 ? maxL : 1));
    double *acc = NULL, *ms = NULL, *ls = NULL;
    if (jb->chunk_tokens > 0) {
        size_t nc = (size_t)(maxL + jb->chunk_tokens - 1) / (size_t)jb->chunk_tokens + 1;
        acc = (double *)malloc(sizeof(double) * nc * (size_t)jb->head_dim);
        ms = (double *)malloc(sizeof(double) * nc);
        ls = (double *)malloc(sizeof(double) * nc);
    }
    if (!logits || (jb->chunk_tokens > 0 && (!acc || !ms || !ls))) {
        atomic_store(&jb->status, -4);
        free(logits); free(acc); free(ms); free(ls);
        return NULL;
    }
    const int rows = jb->num_seqs * jb->num_q_heads;
    for (;;) {
        int r = atomic_fetch_add(&jb->next_row, 1);
        if (r >= rows || atomic_load(&jb->status) != 0) break;
        int s = r / jb->num_q_heads, h = r % jb->num_q_heads;
        int e = jb->chunk_tokens > 0 ? row_split(jb, s, h, logits, acc, ms, ls) : row_plain(jb, s, h, logits);
        if (e) {
            int zero = 0;
            atomic_compare_exchange_strong(&jb->status, &zero, e);
            break;
        }
    }
    free(logits); free(acc); free(ms); free(ls);
    return NULL;
}

static int run(job_t *jb, int num_threads)
{
    if (!jb->q || !jb->k_cache || !jb->v_cache || !jb->block_table || !jb->seq_lens || !jb->out) return -1;
    if (jb->num_seqs < 0 || jb->num_q_heads <= 0 || jb->num_kv_heads <= 0 || jb->head_dim <= 0 ||
        jb->block_size <= 0 || jb->max_blocks_per_seq < 0 || jb->num_blocks < 0 ||
        jb->num_q_heads % jb->num_kv_heads != 0 || jb->chunk_tokens < 0)
        return -1;
    for (int s = 0; s < jb->num_seqs; ++s) {
        if (jb->seq_lens[s] < 0) return -1;
        if ((long long)jb->seq_lens[s] > (long long)jb->max_blocks_per_seq * jb->block_size) return -3;
    }
    atomic_init(&jb->next_row, 0);
    atomic_init(&jb->status, 0);
    if (num_threads < 1) num_threads = 1;
    if (num_threads > 1024) num_threads = 1024;
    pthread_t *tids = (pthread_t *)malloc(sizeof(pthread_t) * (size_t)num_threads);
    if (!tids) return -4;
    int started = 0;
    for (int i = 0; i < num_threads; ++i) {
        if (pthread_create(&tids[i], NULL, worker, jb) != 0) break;
        ++started;
    }
    if (started == 0) worker(jb);
    for (int i = 0; i < started; ++i) pthread_join(tids[i], NULL);
    free(tids);
    return atomic_load(&jb->status);
}

int ps_oracle_decode_attention(const uint16_t *q, const uint16_t *k_cache, const uint16_t *v_cache,
                               const int32_t *block_table, const int32_t *seq_lens, int num_seqs,
                               int num_q_heads, int num_kv_heads, int head_dim, int block_size,
                               int max_blocks_per_seq, long long num_blocks, double scale,
                               int num_threads, double *out)
{
    job_t jb;
    memset(&jb, 0, sizeof jb);
    jb.q = q; jb.k_cache = k_cache; jb.v_cache = v_cache;
    jb.block_table = block_table; jb.seq_lens = seq_lens;
    jb.num_seqs = num_seqs; jb.num_q_heads = num_q_heads; jb.num_kv_heads = num_kv_heads;
    jb.head_dim = head_dim; jb.block_size = block_size; jb.max_blocks_per_seq = max_blocks_per_seq;
    jb.num_blocks = num_blocks; jb.scale = scale; jb.chunk_tokens = 0; jb.out = out;
    return run(&jb, num_threads);
}

int ps_oracle_decode_attention_split(const uint16_t *q, const uint16_t *k_cache, const uint16_t *v_cache,
                                     const int32_t *block_table, const int32_t *seq_lens, int num_seqs,
                                     int num_q_heads, int num_kv_heads, int head_dim, int block_size,
                                     int max_blocks_per_seq, long long num_blocks, double scale,
                                     int chunk_tokens, int num_threads, double *out)
{
    if (chunk_tokens <= 0) return -1;
    job_t jb;
    memset(&jb, 0, sizeof jb);
    jb.q = q; jb.k_cache = k_cache; jb.v_cache = v_cache;
    jb.block_table = block_table; jb.seq_lens = seq_lens;
    jb.num_seqs = num_seqs; jb.num_q_heads = num_q_heads; jb.num_kv_heads = num_kv_heads;
    jb.head_dim = head_dim; jb.block_size = block_size; jb.max_blocks_per_seq = max_blocks_per_seq;
    jb.num_blocks = num_blocks; jb.scale = scale; jb.chunk_tokens = chunk_tokens; jb.out = out;
    return run(&jb, num_threads);
}

/*
 * KV hand-off between stage pools (PowerSlider Sec. 5: a request's KV cache
 * moves from the thinking pool to the answer pool; only the on-GPU gather and
 * scatter are modelled here, not the transport).
 *
 * Packed layout of sequence i (element offset dst_offsets[i]):
 *   K[j][t][:] for j < Hkv, t < L_i, then V[j][t][:] in the same order,
 * i.e. 2 * Hkv * L_i * d contiguous bf16 elements.
 *
 * ps_oracle_kv_pack copies cache slot (block_table[i][t / bs], j, t % bs) to
 * packed position (j, t); ps_oracle_kv_unpack copies it back through another
 * block table.  Both return 0, -1 (invalid argument) or -2 (block id outside
 * the pool); unpack leaves every slot it does not own untouched.
 */
static int kv_addr(const int32_t *bt, int mbps, long long nb, int hkv, int bs, int d, int i, int j, int t,
                   size_t *off)
{
    int32_t b = bt[(size_t)i * mbps + t / bs];
    if (b < 0 || (long long)b >= nb) return -2;
    *off = (((size_t)b * hkv + (size_t)j) * bs + (size_t)(t % bs)) * d;
    return 0;
}

int ps_oracle_kv_pack(const uint16_t *k_cache, const uint16_t *v_cache, const int32_t *block_table,
                      int max_blocks_per_seq, const int32_t *seq_lens, int num_seqs, int num_kv_heads,
                      int head_dim, int block_size, long long num_blocks, const long long *dst_offsets,
                      uint16_t *dst)
{
    if (!k_cache || !v_cache || !block_table || !seq_lens || !dst_offsets || !dst || num_seqs < 0 ||
        num_kv_heads <= 0 || head_dim <= 0 || block_size <= 0)
        return -1;
    for (int i = 0; i < num_seqs; ++i) {
        const int L = seq_lens[i];
        if (L < 0 || (long long)L > (long long)max_blocks_per_seq * block_size) return -1;
        uint16_t *kd = dst + dst_offsets[i];
        uint16_t *vd = kd + (size_t)num_kv_heads * L * head_dim;
        for (int j = 0; j < num_kv_heads; ++j)
            for (int t = 0; t < L; ++t) {
                size_t off;
                int e = kv_addr(block_table, max_blocks_per_seq, num_blocks, num_kv_heads, block_size, head_dim,
                                i, j, t, &off);
                if (e) return e;
                size_t p = ((size_t)j * L + t) * head_dim;
                memcpy(kd + p, k_cache + off, sizeof(uint16_t) * (size_t)head_dim);
                memcpy(vd + p, v_cache + off, sizeof(uint16_t) * (size_t)head_dim);
            }
    }
    return 0;
}

int ps_oracle_kv_unpack(const uint16_t *src, const long long *src_offsets, const int32_t *block_table,
                        int max_blocks_per_seq, const int32_t *seq_lens, int num_seqs, int num_kv_heads,
                        int head_dim, int block_size, long long num_blocks, uint16_t *k_cache, uint16_t *v_cache)
{
    if (!k_cache || !v_cache || !block_table || !seq_lens || !src_offsets || !src || num_seqs < 0 ||
        num_kv_heads <= 0 || head_dim <= 0 || block_size <= 0)
        return -1;
    for (int i = 0; i < num_seqs; ++i) {
        const int L = seq_lens[i];
        if (L < 0 || (long long)L > (long long)max_blocks_per_seq * block_size) return -1;
        const uint16_t *ks = src + src_offsets[i];
        const uint16_t *vs = ks + (size_t)num_kv_heads * L * head_dim;
        for (int j = 0; j < num_kv_heads; ++j)
            for (int t = 0; t < L; ++t) {
                size_t off;
                int e = kv_addr(block_table, max_blocks_per_seq, num_blocks, num_kv_heads, block_size, head_dim,
                                i, j, t, &off);
                if (e) return e;
                size_t p = ((size_t)j * L + t) * head_dim;
                memcpy(k_cache + off, ks + p, sizeof(uint16_t) * (size_t)head_dim);
                memcpy(v_cache + off, vs + p, sizeof(uint16_t) * (size_t)head_dim);
            }
    }
    return 0;
}

/*
 * Chunked-prefill attention over the paged cache (PowerSlider Sec. 2.2: the
 * prefill phase processes many prompt tokens at once and is compute-bound,
 * Sec. 3 Obs. 2).  Sequence s holds L_s = seq_lens[s] cached tokens, the last
 * Q_s = q_start[s+1] - q_start[s] of which are the new (query) tokens; query i
 * of sequence s sits at position p = L_s - Q_s + i and attends causally to the
 * cached tokens t = 0 .. p:
 *
 *   out[q_start[s] + i][h] = sum_{t<=p} softmax_t(scale * q . K_s[t]) V_s[t]
 *
 * with KV head h / g and the same paged layout as decode.  q and out are
 * [total query tokens][Hq][d].  With Q_s = 1 for every sequence this is
 * exactly ps_oracle_decode_attention.  Error codes as for decode; -1 also for
 * Q_s > L_s or a decreasing q_start.
 */
typedef struct {
    const uint16_t *q, *k_cache, *v_cache;
    const int32_t *block_table, *seq_lens, *q_start;
    int num_seqs, num_q_heads, num_kv_heads, head_dim, block_size, max_blocks_per_seq;
    long long num_blocks;
    double scale;
    double *out;
    int total_q;
    atomic_int next_row;
    atomic_int status;
} prefill_job_t;

static int prefill_row(prefill_job_t *jb, int s, int i, int h, double *logits)
{
    const int d = jb->head_dim;
    const int g = jb->num_q_heads / jb->num_kv_heads;
    const int j = h / g;
    const int L = jb->seq_lens[s];
    const int Q = jb->q_start[s + 1] - jb->q_start[s];
    const int p = L - Q + i;
    const size_t row = (size_t)(jb->q_start[s] + i) * jb->num_q_heads + h;
    const uint16_t *qv = jb->q + row * d;
    double *o = jb->out + row * d;
    job_t view;  /* reuse the decode address helper */
    memset(&view, 0, sizeof view);
    view.block_table = jb->block_table;
    view.num_kv_heads = jb->num_kv_heads;
    view.head_dim = d;
    view.block_size = jb->block_size;
    view.max_blocks_per_seq = jb->max_blocks_per_seq;
    view.num_blocks = jb->num_blocks;
    int err = 0;
    for (int e = 0; e < d; ++e) o[e] = 0.0;
    double m = -INFINITY;
    for (int t = 0; t <= p; ++t) {
        const uint16_t *kr = token_row(&view, jb->k_cache, s, j, t, &err);
        if (err) return err;
        double dot = 0.0;
        for (int e = 0; e < d; ++e) dot += bf16_bits_to_double(qv[e]) * bf16_bits_to_double(kr[e]);
        logits[t] = jb->scale * dot;
        if (logits[t] > m) m = logits[t];
    }
    double z = 0.0;
    for (int t = 0; t <= p; ++t) {
        double w = exp(logits[t] - m);
        z += w;
        const uint16_t *vr = token_row(&view, jb->v_cache, s, j, t, &err);
        if (err) return err;
        for (int e = 0; e < d; ++e) o[e] += w * bf16_bits_to_double(vr[e]);
    }
    for (int e = 0; e < d; ++e) o[e] /= z;
    return 0;
}

static void *prefill_worker(void *arg)
{
    prefill_job_t *jb = (prefill_job_t *)arg;
    int maxL = 1;
    for (int s = 0; s < jb->num_seqs; ++s)
        if (jb->seq_lens[s] > maxL) maxL = jb->seq_lens[s];
    double *logits = (double *)malloc(sizeof(double) * (size_t)maxL);
    if (!logits) {
        atomic_store(&jb->status, -4);
        return NULL;
    }
    const int rows = jb->total_q * jb->num_q_heads;
    for (;;) {
        int r = atomic_fetch_add(&jb->next_row, 1);
        if (r >= rows || atomic_load(&jb->status) != 0) break;
        const int tok = r / jb->num_q_heads, h = r % jb->num_q_heads;
        int s = 0;
        while (jb->q_start[s + 1] <= tok) ++s;
        int e = prefill_row(jb, s, tok - jb->q_start[s], h, logits);
        if (e) {
            int zero = 0;
            atomic_compare_exchange_strong(&jb->status, &zero, e);
            break;
        }
    }
    free(logits);
    return NULL;
}

int ps_oracle_prefill_attention(const uint16_t *q, const uint16_t *k_cache, const uint16_t *v_cache,
                                const int32_t *block_table, const int32_t *seq_lens, const int32_t *q_start,
                                int num_seqs, int num_q_heads, int num_kv_heads, int head_dim, int block_size,
                                int max_blocks_per_seq, long long num_blocks, double scale, int num_threads,
                                double *out)
{
    if (!q || !k_cache || !v_cache || !block_table || !seq_lens || !q_start || !out || num_seqs < 0 ||
        num_q_heads <= 0 || num_kv_heads <= 0 || head_dim <= 0 || block_size <= 0 ||
        num_q_heads % num_kv_heads != 0 || q_start[0] != 0)
        return -1;
    for (int s = 0; s < num_seqs; ++s) {
        const int Q = q_start[s + 1] - q_start[s];
        if (Q < 0 || Q > seq_lens[s]) return -1;
        if ((long long)seq_lens[s] > (long long)max_blocks_per_seq * block_size) return -3;
    }
    prefill_job_t jb;
    memset(&jb, 0, sizeof jb);
    jb.q = q; jb.k_cache = k_cache; jb.v_cache = v_cache;
    jb.block_table = block_table; jb.seq_lens = seq_lens; jb.q_start = q_start;
    jb.num_seqs = num_seqs; jb.num_q_heads = num_q_heads; jb.num_kv_heads = num_kv_heads;
    jb.head_dim = head_dim; jb.block_size = block_size; jb.max_blocks_per_seq = max_blocks_per_seq;
    jb.num_blocks = num_blocks; jb.scale = scale; jb.out = out; jb.total_q = q_start[num_seqs];
    atomic_init(&jb.next_row, 0);
    atomic_init(&jb.status, 0);
    if (num_threads < 1) num_threads = 1;
    if (num_threads > 1024) num_threads = 1024;
    pthread_t *tids = (pthread_t *)malloc(sizeof(pthread_t) * (size_t)num_threads);
    if (!tids) return -4;
    int started = 0;
    for (int i = 0; i < num_threads; ++i) {
        if (pthread_create(&tids[i], NULL, prefill_worker, &jb) != 0) break;
        ++started;
    }
    if (started == 0) prefill_worker(&jb);
    for (int i = 0; i < started; ++i) pthread_join(tids[i], NULL);
    free(tids);
    return atomic_load(&jb.status);
}
