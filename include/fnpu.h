/*
 * fnpu.h -- C ABI of the GB300 mixed prefill/decode paged-attention step.
 *
 * One serving step in which prefill chunks and decode queries share the
 * device and one paged KV pool (the dynamic PD co-location of Sec. 3.4):
 * prefill is compute-heavy and decode is bound by KV-cache reads (Sec. 1,
 * Sec. 3.3, Fig. 1-2), so the step interleaves both kinds of work on the same
 * SMs. A step is
 *
 *   fnpu_kv_append          store the step's new K/V rows in their paged slots
 *   fnpu_mixed_attn_plan    (host) classify sequences by phase and build the
 *                           work list -- the phase-aware dispatch of Sec. 3.4
 *   fnpu_mixed_attn_run     causal attention of every query over its sequence's
 *                           cached keys, one launch on the caller's stream
 *   fnpu_mixed_step         the append and the attention of a step in one call
 *
 * As in the paper's control path (Sec. 3.2), calls pass metadata and pointers
 * only: tensors stay in device memory owned by the caller; the library never
 * copies them. All entry points are asynchronous on the given CUDA stream
 * (cudaStream_t passed as void*; NULL = legacy default stream) and return an
 * fnpu_status; none aborts or prints.
 *
 * Math (the paper gives none; this is textbook attention): for sequence s with
 * query_len q and context_len ctx (ctx counts this step's q new tokens), query
 * i in [0, q) sits at absolute position pos = ctx - q + i and attends to keys
 * j = 0..pos of its sequence. Query head h reads kv head h / (Hq / Hkv).
 *   S_j = scale * <Q[t,h,:], K_j>;  O[t,h,:] = sum_j softmax(S)_j V_j;
 *   LSE[t,h] = ln sum_j exp(S_j)          (natural log, fp32)
 * Key j of sequence s lives in block block_table[s][j / bs] at offset j % bs.
 * Scores and softmax are fp32; QK^T and PV take bf16 operands and fp32
 * accumulation; O is rounded to bf16 (nearest-even).
 *
 * Layouts (row-major, contiguous, bf16 = 16-bit brain float):
 *   q        bf16 [T, Hq, d_qk]      queries packed sequence by sequence
 *   k_cache  bf16 [num_blocks, bs, Hkv, d_qk]
 *   v_cache  bf16 [num_blocks, bs, Hkv, d_v]
 *   latent (v_in_k_latent = 1, MLA): k_cache bf16 [num_blocks, bs, d_qk],
 *            Hkv = 1, V = the first d_v columns of each K row, v_cache NULL
 *   out      bf16 [T, Hq, d_v];  lse fp32 [T, Hq]
 * All device pointers must be 16-byte aligned.
 */
#ifndef FNPU_H_
#define FNPU_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    FNPU_OK = 0,
    FNPU_EINVAL = -1,          /* bad argument; nothing was launched */
    FNPU_EUNSUPPORTED = -2,    /* valid but not implemented (head dims etc.) */
    FNPU_ECUDA = -3,           /* a CUDA runtime call failed */
    FNPU_EDEVICE_TIMEOUT = -4, /* a bounded device-side wait gave up, or a kernel
                                  found its shared memory misaligned and did nothing */
    FNPU_ENOMEM = -5,          /* device or host allocation failed */
    FNPU_EDEVICE_RANGE = -6    /* a kernel met an out-of-range slot, context length or
                                  block id and skipped it */
} fnpu_status;

typedef struct {
    int32_t num_q_heads;   /* Hq, a multiple of num_kv_heads */
    int32_t num_kv_heads;  /* Hkv (1 for the latent layout) */
    int32_t head_dim_qk;   /* supported: 64, 128 (split K/V); 576 (latent); 192 (expanded
                              latent rows, see fnpu_mla_expand: prefill plans only) */
    int32_t head_dim_v;    /* = head_dim_qk for split K/V; 512 for latent; 128 with 192 */
    int32_t block_size;    /* tokens per KV block (16 or 64 ...), >= 1 */
    int32_t num_blocks;    /* blocks in the pool */
    int32_t v_in_k_latent; /* 1: MLA latent cache, V aliases K[:, :d_v] */
    float softmax_scale;   /* <= 0 selects 1/sqrt(head_dim_qk) */
    int32_t kv_fp8;        /* 1: the pools hold the FP8 (e4m3) cache format below; 0: bf16 */
} fnpu_attn_desc;

/*
 * FP8 KV cache (kv_fp8 = 1). Decode is bound by KV-cache reads (Sec. 1,
 * Sec. 3.3); one-byte values halve them. The paper quantises its DeepSeek-R1
 * deployment to 8 bits (Sec. 4.1) but gives no cache format; this is the
 * library's. Supported for split K/V with Hkv = 4, d_qk = d_v = 128,
 * block_size = 16, Hq / Hkv <= 8 (decode, prefill and mixed plans; the plan
 * stages an f16 copy of its prefill sequences' blocks and queries for the
 * tensor-core prefill, so values must lie within the f16 range); anything
 * else returns FNPU_EUNSUPPORTED.
 *   Quantisation, per stored row (one slot, one kv head, 128 values):
 *     scale = amax |x| / 448 in fp32 (1 for a zero row), code = the e4m3 value
 *     nearest to x / scale (fp32 quotient; ties to the even code; magnitudes
 *     above 448 saturate to 448; a zero code is stored with a clear sign bit).
 *     The stored value is value(code) * scale.
 *   Pools: k_cache and v_cache are byte arrays of num_blocks blocks of 8448
 *   bytes (16-byte aligned). Within a block, with c = (j mod 8) / 2 and
 *   r = (j mod 2) + 2 (j / 8) for j in 0..15:
 *     K: codes [16 slots][4 heads][128], column 16 k + j of a row at byte
 *        32 c + 4 k + r; then fp32 scales [16 slots][4 heads] at byte 8192
 *     V: codes [4 heads][128 columns][16 slots], slot j of a column at
 *        byte 4 c + r; then fp32 scales [16 slots][4 heads] at byte 8192
 *   The attention products take f16 operands (e4m3 values are exact in f16;
 *   queries must lie within the f16 range) and fp32 accumulation.
 */

typedef struct fnpu_plan fnpu_plan; /* opaque, owned by the library */

/* Plan options (all zero = defaults). */
typedef struct {
    int32_t decode_split_keys; /* keys per decode split item; 0 = chosen by the planner */
    int32_t decode_share_pct;  /* share of resident work slots that take decode work
                                  first in the phase-aware schedule; 0 = planner default */
    int32_t num_sms;           /* SMs to plan for; 0 = the current device's count */
    int32_t flags;             /* FNPU_PLAN_* bits */
} fnpu_plan_opts;

#define FNPU_PLAN_SEPARATE_LAUNCHES 1 /* run prefill and decode as separate launches */
#define FNPU_PLAN_NO_TCGEN05 2        /* prefill on the mma.sync path (comparison only) */
#define FNPU_PLAN_GREEN_CONTEXTS 4    /* co-located step: prefill and decode in green contexts
                                         over disjoint SM partitions (the decode share rounded
                                         up to the device's partition granularity); plan
                                         fails with FNPU_EUNSUPPORTED where they cannot be made */
#define FNPU_PLAN_FUSED_APPEND 8      /* fnpu_mixed_step: where the prefill runs on the tcgen05
                                         kernel over a bf16 cache (not in green contexts), its
                                         CTAs write the prefill-path rows themselves and a small
                                         kernel writes the decode rows, instead of one append
                                         kernel ahead of the run. Results are the same bit for
                                         bit; on the Qwen co-located and prefill-only steps it
                                         measured slower than the default (the append kernel's
                                         time is hidden by the prefill grid's dependent launch) */

/*
 * KV append: for each token t in [0, num_tokens) with slot_mapping[t] >= 0,
 * copy k_new[t] (Hkv*d_qk values; latent: d_qk values) into slot
 * slot_mapping[t] of k_cache and v_new[t] (Hkv*d_v values) into the same slot
 * of v_cache, bit-exactly. Slot s means block s / bs, offset s % bs. Negative
 * slots are padding and are skipped. Must run before fnpu_mixed_attn_run of
 * the same step: a step's queries see their own new keys.
 *   desc          attention shape (host pointer)
 *   k_new, v_new  device bf16 [num_tokens, Hkv, d]; v_new NULL for latent
 *   slot_mapping  device int64 [num_tokens]
 *   k_cache, v_cache  device pools as above; v_cache NULL for latent
 * With kv_fp8 = 1 each new row is quantised into the FP8 format above (codes
 * and scale); the result is bit-exact with that definition.
 * Errors: FNPU_EINVAL on NULL pointers or bad shape (nothing launched). A slot
 * >= num_blocks*bs cannot be seen on the host; the kernel skips it and raises
 * the device error flag, reported as FNPU_EDEVICE_RANGE by fnpu_check().
 * Duplicate non-negative slots are a caller error (result unspecified).
 */
int fnpu_kv_append(const fnpu_attn_desc *desc, const void *k_new, const void *v_new,
                   const int64_t *slot_mapping, int32_t num_tokens,
                   void *k_cache, void *v_cache, void *stream);

/*
 * Build the work list for one step. Host arrays, all of length num_seqs:
 *   query_len[s] >= 1, context_len[s] >= query_len[s],
 *   phase[s] = 0 (prefill chunk) or 1 (decode),
 *   block_table: int32 [num_seqs, block_table_stride]; only the first
 *   ceil(context_len[s] / bs) entries of row s are read, each < num_blocks.
 * The phase decides only which queue a sequence's work enters (prefill tiles
 * on the tensor-core path, decode split items on the bandwidth path), never
 * the result. A decode of several tokens (query_len[s] > 1, as in speculative
 * verification) is causal attention of a short chunk on its context and
 * takes the prefill path; one-token decodes take the decode path. The plan copies everything it needs (the block table included)
 * to its own device workspace with one asynchronous copy on `stream`; the
 * host arrays may be freed on return. The plan stays valid for any number of
 * runs with the same metadata and caches of the same shape.
 * Errors: FNPU_EINVAL for any violated condition above, FNPU_EUNSUPPORTED for
 * head dims or groupings without a kernel, FNPU_ENOMEM, FNPU_ECUDA.
 * *out is set only on success.
 */
int fnpu_mixed_attn_plan(const fnpu_attn_desc *desc, int32_t num_seqs,
                         const int32_t *query_len, const int32_t *context_len,
                         const uint8_t *phase, const int32_t *block_table,
                         int32_t block_table_stride, void *stream, fnpu_plan **out);

/* As fnpu_mixed_attn_plan, with options (opts may be NULL). */
int fnpu_mixed_attn_plan_ex(const fnpu_attn_desc *desc, int32_t num_seqs,
                            const int32_t *query_len, const int32_t *context_len,
                            const uint8_t *phase, const int32_t *block_table,
                            int32_t block_table_stride, const fnpu_plan_opts *opts,
                            void *stream, fnpu_plan **out);

/*
 * Re-plan: rebuild `plan` for a new step's metadata (same descriptor; the
 * arguments as for fnpu_mixed_attn_plan_ex), keeping what the plan already
 * holds -- its streams, events and green contexts, two pinned staging
 * buffers used in turn, and its device workspace, which is reallocated only
 * when the new step needs more than it holds (then with a quarter of
 * headroom, after waiting for the device). In a serving loop whose metadata
 * changes every step (the phase-aware dispatch of Sec. 3.4 plans every step
 * anew) this makes the plan host work alone: no allocation, stream or event
 * creation in the steady state. Green contexts are rebuilt only when the
 * decode share asks for a different partition.
 * The metadata upload is enqueued on `stream`. Runs of the plan already
 * enqueued on `stream` finish before it; runs enqueued on other streams must
 * be ordered before this call's upload by the caller. The plan's error flag
 * is kept (fnpu_plan_check still reports a failed earlier run).
 * Errors: as fnpu_mixed_attn_plan_ex; on FNPU_EINVAL or FNPU_EUNSUPPORTED
 * from the argument checks the plan is unchanged; after any other error it
 * must be re-planned successfully or destroyed before it runs again.
 */
int fnpu_mixed_attn_replan(fnpu_plan *plan, int32_t num_seqs, const int32_t *query_len,
                           const int32_t *context_len, const uint8_t *phase, const int32_t *block_table,
                           int32_t block_table_stride, const fnpu_plan_opts *opts, void *stream);

/*
 * Attention for every query of the planned step. q, k_cache, v_cache, out,
 * lse are device pointers in the layouts above (v_cache NULL for latent;
 * with kv_fp8 = 1, k_cache and v_cache are the FP8 byte pools).
 * Enqueues the work on `stream` and returns without synchronising. Runs of
 * one plan must not overlap on the GPU (they share the plan's split scratch).
 * Errors: FNPU_EINVAL (NULL pointers), FNPU_ECUDA (launch failure).
 */
int fnpu_mixed_attn_run(const fnpu_plan *plan, const void *q, const void *k_cache,
                        const void *v_cache, void *out, float *lse, void *stream);

/*
 * A whole step: fnpu_kv_append of the step's new rows followed by
 * fnpu_mixed_attn_run, with the same arguments and the same results bit for
 * bit (the shared KV pool of both phases, Sec. 3.4). k_new, v_new and
 * slot_mapping are as for fnpu_kv_append, with the plan's token count; their
 * rows are the planned step's tokens in order. By default the two calls are
 * made in turn. With FNPU_PLAN_FUSED_APPEND, where the plan's prefill runs on
 * the tcgen05 kernel over a bf16 cache (and not in green contexts), that
 * kernel's CTAs write the prefill-path rows themselves before they read the
 * cache (a cooperative launch: they wait for one another, bounded), and a
 * small kernel writes the decode rows ahead of the decode kernel. An
 * out-of-range slot raises the library-wide flag (fnpu_check), as
 * fnpu_kv_append does; a bounded wait that runs out raises the plan's flag.
 * Errors: FNPU_EINVAL (NULL or misaligned pointers), FNPU_ECUDA.
 */
int fnpu_mixed_step(const fnpu_plan *plan, const void *k_new, const void *v_new, const int64_t *slot_mapping,
                    const void *q, void *k_cache, void *v_cache, void *out, float *lse, void *stream);


/* Synchronise `stream`, then read and clear the plan's device error flag:
 * FNPU_OK, FNPU_EDEVICE_TIMEOUT or FNPU_ECUDA. After FNPU_EDEVICE_TIMEOUT the
 * outputs of the failed run are undefined; the plan's work queues and split
 * counters are reset, so the plan can be run again. */
int fnpu_plan_check(const fnpu_plan *plan, void *stream);

/* Synchronise `stream`, then read and clear the library-wide device error
 * flag of the current device (set by fnpu_kv_append on an out-of-range slot,
 * and by fnpu_decode_attn_noalloc on a context length or block id out of
 * range): FNPU_OK, FNPU_EDEVICE_RANGE or FNPU_ECUDA. */
int fnpu_check(void *stream);

/* Release the plan and its device workspace. Waits for the plan's stream
 * work to finish first. NULL is ignored. */
void fnpu_plan_destroy(fnpu_plan *plan);

/* Plan statistics for reporting (host copies; any out pointer may be NULL):
 * number of prefill tiles, decode split items, kernel launches per run, and
 * bytes of device workspace the plan holds. */
int fnpu_plan_info(const fnpu_plan *plan, int32_t *prefill_items, int32_t *decode_items,
                   int32_t *launches_per_run, int64_t *workspace_bytes);

/*
 * Dispatch-ratio feedback (Sec. 3.4: the phase-aware dispatcher sets the
 * share of the device that serves decode from the measured pressure of each
 * phase). A serving loop plans step n with fnpu_plan_opts.decode_share_pct =
 * s_n, runs it, reads the phase times, and plans step n + 1 with the share
 * the controller returns.
 *
 * fnpu_plan_phase_ms: for a co-located plan (both phases present, launched
 * side by side), the device time from the start of the last run of `plan` to
 * the end of its prefill work (*prefill_ms) and to the end of its decode work
 * including the split merge (*decode_ms). Blocks until that run has ended.
 *   Errors: FNPU_EINVAL for NULL arguments or a plan that has not run yet;
 *   FNPU_EUNSUPPORTED for a plan that does not co-locate (one phase only,
 *   latent attention, or FNPU_PLAN_SEPARATE_LAUNCHES).
 *
 * fnpu_dispatch_next_share: host arithmetic only. From the share share_pct
 * (1..99, percent of SMs, as decode_share_pct) and the phase times it gave,
 * the share for the next step: with decode time taken as proportional to
 * 1 / share and prefill time to 1 / (100 - share), the share at which both
 * phases would end together, approached halfway (at least one point while
 * that share is a point or more away) and clamped to [1, 50]; kept when
 * |decode - prefill| <= tolerance * the larger, or when the share is within
 * a point of the balance share.
 *   Errors: FNPU_EINVAL for a NULL out pointer, a share outside 1..99, a
 *   time that is not positive, or a negative tolerance.
 */
int fnpu_plan_phase_ms(const fnpu_plan *plan, float *prefill_ms, float *decode_ms);
int fnpu_dispatch_next_share(int32_t share_pct, float prefill_ms, float decode_ms, float tolerance,
                             int32_t *next_share_pct);

/*
 * The decode share (percent of the SMs whose CTAs start on decode, rounded,
 * at least 1) that a co-located plan uses: the one it was given, or the
 * planner's own choice when decode_share_pct was 0. A serving loop starts its
 * feedback from it. The planner models each prefill CTA as ending at its load
 * of the longest-first schedule of the prefill items, and the decode as
 * streaming on its own SMs from the start and on each prefill SM once that
 * SM's CTA has ended; it takes the share with the shortest modelled step.
 *   Errors: FNPU_EINVAL for NULL arguments; FNPU_EUNSUPPORTED for a plan that
 *   does not co-locate.
 */
int fnpu_plan_decode_share(const fnpu_plan *plan, int32_t *share_pct);

/*
 * Decode attention without any allocation. The paper has no counterpart:
 * this entry point exists for callers that may not call cudaMalloc at all,
 * for instance code that must stay inside memory another framework reserved
 * up front, or a serving process whose device memory is fixed once at start.
 * A plan cannot serve them, because fnpu_mixed_attn_plan allocates a device
 * workspace. This call computes the same GQA-packed split-KV decode as the
 * decode items of fnpu_mixed_attn_run, but keeps its split scratch (partial
 * outputs, partial log-sum-exps, merge counters) in one fixed array of
 * FNPU_NOALLOC_SCRATCH_BYTES inside the library, which every GPU that loads
 * the library holds until the process exits. It calls no cudaMalloc, no
 * cudaFree and no allocating library routine.
 *
 * Every sequence is a decode: query_len = 1, and sequence s's query is row s.
 *   context_len   device int32 [num_seqs], each in [1, max_context_len]
 *                 (counts the new token)
 *   block_table   device int32 [num_seqs, block_table_stride], stride >=
 *                 ceil(max_context_len / block_size)
 *   max_context_len  host bound on context_len; it sizes the grid
 *   split_keys    keys per split, a multiple of 64; 0 selects 512
 *   q             device bf16 [num_seqs, Hq, d]; out bf16 [num_seqs, Hq, d];
 *                 lse fp32 [num_seqs, Hq]; k_cache / v_cache as above
 * Supports split K/V caches with d_qk = d_v in {64, 128} and Hq/Hkv <= 8.
 * The context lengths and block ids are device data, so the kernel checks
 * them: a sequence whose context_len lies outside [1, max_context_len] is
 * skipped (its out and lse rows are left as they were), and a block id
 * outside [0, num_blocks) is never loaded (the sequence's result is then
 * undefined); either raises the library-wide device error flag, which
 * fnpu_check reports as FNPU_EDEVICE_RANGE. No load leaves the block-table
 * rows or the pools.
 * Errors: FNPU_EINVAL for bad arguments and for requests whose scratch
 * (4 B per counter, plus 4 B * (Hq/Hkv) * (d + 1) per split, for
 * num_seqs * Hkv * ceil(max_context_len / split_keys) splits) exceeds
 * FNPU_NOALLOC_SCRATCH_BYTES; FNPU_EUNSUPPORTED for other shapes and for
 * the FP8 cache (kv_fp8 = 1: plan-based runs only);
 * FNPU_ECUDA. Nothing is launched on error.
 * The first call on a device looks up the scratch array's device address
 * (cudaGetSymbolAddress) while that device is current; make that first call
 * before any stream capture. All calls share the one array, which keeps the
 * last call's contents; each call clears its merge counters itself with
 * cudaMemsetAsync on `stream`. Calls that overlap on the GPU (on different
 * streams, or with no ordering between them) race on the array and must not
 * be issued.
 */
#define FNPU_NOALLOC_SCRATCH_BYTES (16u << 20)
int fnpu_decode_attn_noalloc(const fnpu_attn_desc *desc, int32_t num_seqs,
                             const int32_t *context_len, const int32_t *block_table,
                             int32_t block_table_stride, int32_t max_context_len,
                             int32_t split_keys, const void *q, const void *k_cache,
                             const void *v_cache, void *out, float *lse, void *stream);

/* Static description of a status code; never NULL. */
const char *fnpu_status_str(int status);

/* Text of the last failed CUDA call on this thread ("" if none), e.g. to
 * explain an FNPU_ECUDA; never NULL, valid until the next library call. */
const char *fnpu_last_cuda_error(void);

/* Library version, major * 10000 + minor * 100 + patch. */
int fnpu_version(void);

/*
 * MLA without absorption (prefill): expand latent cache rows into per-head
 * keys and values, so that a prefill chunk can run as ordinary multi-head
 * attention (d_qk = 192, d_v = 128, Hkv = Hq) through fnpu_mixed_attn_plan /
 * _run over k_out / v_out seen as a paged cache. For row i with latent row
 * L = latent_cache[slots[i]] (c = L[0:512], r = L[512:576]) and head h:
 *   k_out[i, h, 0:128]   = c W_UK[h]      k_out[i, h, 128:192] = r
 *   v_out[i, h, :]       = c W_UV[h]
 * products in fp32, rounded to bf16 (nearest-even). This is the decompressed
 * form of the latent attention of Sec. 4.1's DeepSeek-R1 deployment: with
 * q = [q_nope, q_rope], q_nope . (c W_UK[h]) = (W_UK[h] q_nope) . c, so both
 * forms give the same scores; the absorbed kernel of fnpu_mixed_attn_run
 * attends over the latent rows directly.
 *   desc          the latent cache: v_in_k_latent = 1, Hkv = 1, d_qk = 576,
 *                 d_v = 512, block_size, num_blocks; num_q_heads = heads to expand
 *   latent_cache  device bf16 [num_blocks, block_size, 576]
 *   slots         device int64 [n]: latent slot of row i; negative = a zero row
 *   w_uk, w_uv    device bf16 [Hq, 512, 128] (row-major per head)
 *   workspace     device, at least n * 512 * 2 bytes (scratch; caller-owned)
 *   k_out         device bf16 [n, Hq, 192];  v_out device bf16 [n, Hq, 128]
 * Two kernels of this library on the stream: a gather of the c parts into
 * the workspace (and of the r parts into every head's key), then one
 * tcgen05 GEMM (per CTA 128 rows x one head's 128 key and 128 value
 * columns, an fp32 accumulator in tensor memory) for both products.
 * Errors: FNPU_EINVAL for NULL or misaligned pointers (16 bytes; slots 8),
 * n < 0 or a desc that is not a latent cache; FNPU_EUNSUPPORTED for other
 * latent widths; FNPU_ECUDA if a CUDA call fails. A slot >=
 * num_blocks * block_size gives a zero row and raises the device error
 * flag (FNPU_EDEVICE_RANGE from fnpu_check); a bounded wait of the GEMM
 * that gives up leaves its rows undefined and makes fnpu_check return
 * FNPU_EDEVICE_TIMEOUT.
 */
int fnpu_mla_expand(const fnpu_attn_desc *desc, const void *latent_cache, const int64_t *slots, int32_t n,
                    const void *w_uk, const void *w_uv, void *workspace, void *k_out, void *v_out,
                    void *stream);

#ifdef __cplusplus
}
#endif

#endif /* FNPU_H_ */
