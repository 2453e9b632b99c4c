/*
 * fp64 CPU oracle for one mixed prefill/decode attention step over a paged
 * KV cache, plus the KV append that precedes it.
 *
 * TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and the CPU
 * baseline legs of bench.py may load this library. It shares no code, header
 * or constant with the CUDA path under paper_2606_04415_gb300/.
 *
 * What it computes. The paper (FlexNPU) defines the two phases that share a
 * device (prefill processes the prompt, decode emits one token at a time,
 * Sec. 1 and Sec. 2.3) and co-locates them on one KV pool (Sec. 3.4, "Memory
 * Locality"); it prints no attention formula. The arithmetic below is the
 * textbook scaled-dot-product attention with a causal mask at absolute
 * positions, written out with no blocking, fusion or reordering:
 *
 *   for sequence s, query i in [0, q_s), query head h:
 *     pos   = ctx_s - q_s + i                (ctx counts this step's tokens)
 *     kvh   = h / (Hq / Hkv)                 (contiguous GQA grouping)
 *     key j in [0, pos]: blk = bt[s][j / bs], off = j % bs
 *     s_j   = scale * <q, K[blk][off][kvh]>
 *     m     = max_j s_j,  l = sum_j exp(s_j - m)
 *     O     = sum_j exp(s_j - m) V[blk][off][kvh] / l
 *     LSE   = m + ln l
 *
 * For the latent (MLA) layout, K rows are [blk][off][0:d_qk] of the single
 * latent cache and V rows are the first d_v columns of the same rows.
 * Inputs are bf16 bit patterns, widened exactly to double.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

static double bf16_to_double(uint16_t b) {
    uint32_t u = ((uint32_t)b) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* KV append: copy row t of `rows` into slot slot_mapping[t] of `cache` for
 * every t with slot_mapping[t] >= 0. A row is `row_elems` bf16 values (one
 * slot of the cache: Hkv*d for split K/V caches, d_qk for the latent cache).
 * Returns 0, or -1 if a slot is >= num_slots (nothing is copied then). */
int oracle_kv_append(const uint16_t *rows, const int64_t *slot_mapping,
                     int64_t num_tokens, int64_t row_elems,
                     uint16_t *cache, int64_t num_slots) {
    for (int64_t t = 0; t < num_tokens; ++t)
        if (slot_mapping[t] >= num_slots) return -1;
    for (int64_t t = 0; t < num_tokens; ++t) {
        int64_t s = slot_mapping[t];
        if (s < 0) continue;
        memcpy(cache + s * row_elems, rows + t * row_elems,
               (size_t)row_elems * sizeof(uint16_t));
    }
    return 0;
}

typedef struct {
    int32_t num_seqs;
    const int32_t *query_len, *context_len, *block_table;
    int32_t bt_stride;
    int32_t hq, hkv, dqk, dv, bs, latent;
    double scale;
    const uint16_t *q, *k_cache, *v_cache;
} attn_args;

static const uint16_t *key_row(const attn_args *a, int32_t s, int32_t j, int32_t kvh) {
    int64_t blk = a->block_table[(int64_t)s * a->bt_stride + j / a->bs];
    int64_t slot = blk * a->bs + j % a->bs;
    if (a->latent) return a->k_cache + slot * a->dqk;
    return a->k_cache + (slot * a->hkv + kvh) * a->dqk;
}

static const uint16_t *value_row(const attn_args *a, int32_t s, int32_t j, int32_t kvh) {
    int64_t blk = a->block_table[(int64_t)s * a->bt_stride + j / a->bs];
    int64_t slot = blk * a->bs + j % a->bs;
    if (a->latent) return a->k_cache + slot * a->dqk; /* V = first dv columns */
    return a->v_cache + (slot * a->hkv + kvh) * a->dv;
}

/* One output row: query token t (of sequence s, index i in its chunk), head h.
 * `score` has room for ctx_s doubles. Writes dv outputs, the LSE, and, if
 * `weights` is not NULL, the pos+1 softmax weights exp(s_j - LSE). */
static void attend_row(const attn_args *a, int32_t s, int32_t i, int64_t t, int32_t h,
                       double *score, double *o, double *lse, double *weights) {
    const int32_t pos = a->context_len[s] - a->query_len[s] + i;
    const int32_t kvh = h / (a->hq / a->hkv);
    const uint16_t *qrow = a->q + (t * a->hq + h) * a->dqk;
    double m = -INFINITY;
    for (int32_t j = 0; j <= pos; ++j) {
        const uint16_t *k = key_row(a, s, j, kvh);
        double dot = 0.0;
        for (int32_t c = 0; c < a->dqk; ++c) dot += bf16_to_double(qrow[c]) * bf16_to_double(k[c]);
        score[j] = a->scale * dot;
        if (score[j] > m) m = score[j];
    }
    double l = 0.0;
    for (int32_t c = 0; c < a->dv; ++c) o[c] = 0.0;
    for (int32_t j = 0; j <= pos; ++j) {
        double e = exp(score[j] - m);
        l += e;
        const uint16_t *v = value_row(a, s, j, kvh);
        for (int32_t c = 0; c < a->dv; ++c) o[c] += e * bf16_to_double(v[c]);
    }
    for (int32_t c = 0; c < a->dv; ++c) o[c] /= l;
    *lse = m + log(l);
    if (weights)
        for (int32_t j = 0; j <= pos; ++j) weights[j] = exp(score[j] - *lse);
}

/* Mixed-batch attention. Queries are packed sequence by sequence.
 * q: bf16 [T, hq, dqk]; k_cache: bf16 [num_blocks, bs, hkv, dqk] (latent:
 * [num_blocks, bs, dqk]); v_cache: bf16 [num_blocks, bs, hkv, dv] (latent:
 * ignored). out: double [n_rows, hq, dv], lse: double [n_rows, hq], where the
 * rows are all T tokens (tokens == NULL) or the listed token indices.
 * scale <= 0 means 1/sqrt(dqk). Returns 0, or -1 on bad arguments. */
int oracle_attention(int32_t num_seqs, const int32_t *query_len, const int32_t *context_len,
                     const int32_t *block_table, int32_t bt_stride,
                     int32_t hq, int32_t hkv, int32_t dqk, int32_t dv, int32_t bs,
                     int32_t latent, double scale,
                     const uint16_t *q, const uint16_t *k_cache, const uint16_t *v_cache,
                     const int64_t *tokens, int64_t n_tokens,
                     double *out, double *lse, int32_t num_threads) {
    if (num_seqs < 0 || hq <= 0 || hkv <= 0 || hq % hkv || dqk <= 0 || dv <= 0 || bs <= 0)
        return -1;
    if (latent && (hkv != 1 || dv > dqk)) return -1;
    attn_args a = {num_seqs, query_len, context_len, block_table, bt_stride,
                   hq, hkv, dqk, dv, bs, latent,
                   scale > 0 ? scale : 1.0 / sqrt((double)dqk), q, k_cache, v_cache};
    int64_t T = 0;
    int32_t max_ctx = 1;
    for (int32_t s = 0; s < num_seqs; ++s) {
        if (query_len[s] < 1 || context_len[s] < query_len[s]) return -1;
        T += query_len[s];
        if (context_len[s] > max_ctx) max_ctx = context_len[s];
    }
    int32_t *seq_of = (int32_t *)malloc(sizeof(int32_t) * (size_t)(T ? T : 1));
    int32_t *idx_of = (int32_t *)malloc(sizeof(int32_t) * (size_t)(T ? T : 1));
    for (int32_t s = 0, t = 0; s < num_seqs; ++s)
        for (int32_t i = 0; i < query_len[s]; ++i, ++t) { seq_of[t] = s; idx_of[t] = i; }
    const int64_t rows = tokens ? n_tokens : T;
    for (int64_t r = 0; tokens && r < rows; ++r)
        if (tokens[r] < 0 || tokens[r] >= T) { free(seq_of); free(idx_of); return -1; }
#ifdef _OPENMP
    if (num_threads > 0) omp_set_num_threads(num_threads);
#else
    (void)num_threads;
#endif
#pragma omp parallel
    {
        double *score = (double *)malloc(sizeof(double) * (size_t)max_ctx);
#pragma omp for schedule(dynamic, 1)
        for (int64_t rh = 0; rh < rows * hq; ++rh) {
            int64_t r = rh / hq;
            int32_t h = (int32_t)(rh % hq);
            int64_t t = tokens ? tokens[r] : r;
            attend_row(&a, seq_of[t], idx_of[t], t, h, score,
                       out + (r * hq + h) * dv, lse + r * hq + h, NULL);
        }
        free(score);
    }
    free(seq_of);
    free(idx_of);
    return 0;
}

/* Softmax weights of one row (token t, head h): writes pos+1 doubles into
 * `weights` (room for context_len of t's sequence) and returns pos+1, or -1. */
int64_t oracle_softmax_weights(int32_t num_seqs, const int32_t *query_len, const int32_t *context_len,
                               const int32_t *block_table, int32_t bt_stride,
                               int32_t hq, int32_t hkv, int32_t dqk, int32_t dv, int32_t bs,
                               int32_t latent, double scale,
                               const uint16_t *q, const uint16_t *k_cache, const uint16_t *v_cache,
                               int64_t t, int32_t h, double *weights) {
    if (hq <= 0 || hkv <= 0 || hq % hkv || h < 0 || h >= hq || t < 0) return -1;
    attn_args a = {num_seqs, query_len, context_len, block_table, bt_stride,
                   hq, hkv, dqk, dv, bs, latent,
                   scale > 0 ? scale : 1.0 / sqrt((double)dqk), q, k_cache, v_cache};
    int64_t start = 0;
    for (int32_t s = 0; s < num_seqs; ++s) {
        if (t < start + query_len[s]) {
            int32_t i = (int32_t)(t - start);
            double *score = (double *)malloc(sizeof(double) * (size_t)context_len[s]);
            double *o = (double *)malloc(sizeof(double) * (size_t)dv);
            double lse;
            attend_row(&a, s, i, t, h, score, o, &lse, weights);
            free(score);
            free(o);
            return (int64_t)(context_len[s] - query_len[s] + i) + 1;
        }
        start += query_len[s];
    }
    return -1;
}

int oracle_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
