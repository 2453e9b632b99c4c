// Internal structures shared between the host planner and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/fnpu.h"

namespace fnpu {

// One decode split item: keys [key_begin, key_end) of sequence `seq` at the
// sequence's single query position, for kv head `kvh` and its G query heads
// (per-head kernel) or for every kv head (all-heads kernel, kvh = 0). Splits
// of one group share `group` (their merge counter) and write partial results
// to scratch rows part_base + split. The item also carries its sequence's
// query token and block-table row and the ids of its first four blocks, so
// that a kernel can issue its first copies after one load.
struct DecodeItem {
    int32_t seq, kvh, key_begin, key_end;
    int32_t split, num_splits, part_base, group;
    int32_t q_start, bt_row, pad0, pad1;
    int32_t blk[4];  // block_table[bt_row][key_begin / bs + i], 0 past the item
};
static_assert(sizeof(DecodeItem) == 64, "DecodeItem layout");

// One prefill tile: query rows [row_begin, row_begin + rows) of sequence
// `seq`'s chunk for query head `head` (the mma.sync path) or for kv head
// `head` with all its query heads packed (the tcgen05 path). The tcgen05 path
// may split the keys of a tile: the item then covers 64-key tiles
// [kt_begin, kt_end) only, writes its partial result to scratch row
// part_base + split and the last split of the tile to finish (merge counter
// `group`) combines all num_splits of them. Unsplit items have
// num_splits == 1 and cover every key their rows can see.
struct PrefillItem {
    int32_t seq, head, row_begin, rows;
    int32_t kt_begin, kt_end, split, num_splits;
    int32_t part_base, group;
    int32_t q_start, prefix, ctx_len, bt_row;  // the sequence's SeqInfo, so one load decodes an item
    int32_t pad0, pad1;
};
static_assert(sizeof(PrefillItem) == 64, "PrefillItem layout");

// One latent-attention (MLA) work item: query heads [64 hb, 64 hb + 64) of
// query row `row` of sequence `seq` (a prefill or a decode row alike) over
// keys [key_begin, key_end); splits of one (token, head block) share `group`
// and write partials to scratch rows part_base + split.
struct MlaItem {
    int32_t seq, row, hb, key_begin;
    int32_t key_end, split, num_splits, part_base;
    int32_t group, pad0, pad1, pad2;
};
static_assert(sizeof(MlaItem) == 48, "MlaItem layout");

// The key splits of one decode token, merged by a separate kernel (TMA
// decode path): partial rows part_base .. part_base + num_splits - 1.
struct MergeGroup {
    int32_t token, num_splits, part_base, pad;
};
static_assert(sizeof(MergeGroup) == 16, "MergeGroup layout");

// Per-sequence metadata on the device.
struct SeqInfo {
    int32_t q_start;  // first query token of the sequence in q/out/lse
    int32_t q_len;
    int32_t ctx_len;  // includes this step's q_len new tokens
    int32_t bt_row;   // row of the sequence in the device block table
};
static_assert(sizeof(SeqInfo) == 16, "SeqInfo layout");

struct AttnParams {
    const void *q;        // bf16 [T, Hq, dqk]
    const void *k_cache;  // bf16 [nb, bs, Hkv, dqk] (latent: [nb, bs, dqk])
    const void *v_cache;  // bf16 [nb, bs, Hkv, dv]  (latent: == k_cache)
    void *out;            // bf16 [T, Hq, dv]
    float *lse;           // fp32 [T, Hq]
    const SeqInfo *seqs;
    const int32_t *block_table;  // [num_seqs, bt_stride]
    int32_t bt_stride;
    int32_t num_q_heads, num_kv_heads, group, block_size, num_blocks;
    int64_t num_tokens;
    int32_t head_dim_qk, head_dim_v;
    int64_t k_slot_stride;  // elements between consecutive slots of k_cache
    int64_t v_slot_stride;
    float scale_log2;       // softmax scale * log2(e)
    // decode split-KV
    const DecodeItem *ditems;
    int32_t num_ditems;
    float *part_o;          // fp32 [num_parts, group, dv]
    float *part_lse;        // fp32 [num_parts, group] (log2 domain)
    int32_t *counters;      // [num_groups], zero between runs (per-head decode kernel)
    const MergeGroup *mgroups;  // TMA decode path: split tokens to merge after the decode kernel
    int32_t num_mgroups;
    // prefill
    const PrefillItem *pitems;
    int32_t num_pitems;
    float *ppart_o;         // fp32 split-prefill partials, per partial: [2 tiles][dv / 4][128 rows] float4
    float *ppart_lse;       // fp32 [num_pparts, 2, 128] (log2 domain)
    int32_t *pcounters;     // [num_pgroups, 8] one per softmax warp, zero between runs
    // latent attention (MLA): one work list for both phases
    const MlaItem *mitems;
    int32_t num_mitems;
    int32_t *err;           // device error flag of the plan
    int32_t *sched;         // persistent work queues: [0..1] prefill, [2..3] decode (next item, finished CTAs)
    // the step's append of the prefill-path rows inside the tcgen05 prefill
    // (fnpu_mixed_step): fa_count null = none. Tokens fa_tokens[0 .. n) of
    // k_new / v_new go to their slots; a grid-wide count (zero between runs)
    // says when every CTA has written its share.
    const uint4 *fa_k_new;
    const uint4 *fa_v_new;
    const int64_t *fa_slots;
    const int32_t *fa_tokens;
    uint4 *fa_k_cache;
    uint4 *fa_v_cache;
    int32_t *fa_count;
    int *fa_range_err;      // the library-wide error flag (bit 0: a slot past the pool)
    int32_t fa_num_tokens, fa_k_chunks, fa_v_chunks;
    int64_t fa_num_slots;
};

// cuTensorMapEncodeTiled, looked up once through the runtime's driver entry
// point (the library does not link the driver library); null if unavailable.
typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *,
                                  CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                  CUtensorMapFloatOOBfill);
EncodeTiledFn tensor_map_encoder();

// Record a failed CUDA call for fnpu_last_cuda_error(); returns FNPU_ECUDA.
int cuda_fail(cudaError_t e, const char *where);
#define FNPU_CUDA_TRY(call)                                   \
    do {                                                      \
        cudaError_t e_ = (call);                              \
        if (e_ != cudaSuccess) return ::fnpu::cuda_fail(e_, #call); \
    } while (0)

// Launchers (defined in the .cu files).
int launch_kv_append(const fnpu_attn_desc *d, const void *k_new, const void *v_new,
                     const int64_t *slots, int32_t num_tokens, void *k_cache, void *v_cache,
                     void *stream);
// the same append for the tokens tokens[0 .. n) of k_new / v_new only
int launch_kv_append_list(const fnpu_attn_desc *d, const void *k_new, const void *v_new, const int64_t *slots,
                          const int32_t *tokens, int32_t n, void *k_cache, void *v_cache, void *stream);
int read_and_clear_global_error(void *stream, int *flag);
// Device address of the library-wide error flag on the current device (looked
// up once per device), for kernels of other translation units that raise it.
int global_error_address(int **out);
// MLA expansion: gather the c parts of latent rows (512 + 64 columns) into ws
// [n, 512] and broadcast their r parts into columns 128..191 of k_out [n, heads, 192]
int launch_mla_gather(const void *latent, const int64_t *slots, int32_t n, int64_t num_slots, int32_t heads,
                      void *ws, void *k_out, void *stream);
// FP8 (e4m3) cache: append (quantising) and decode (split-KV, TMA-fed)
int launch_kv_append_fp8(const fnpu_attn_desc *d, const void *k_new, const void *v_new,
                         const int64_t *slots, int32_t num_tokens, void *k_cache, void *v_cache,
                         void *stream);
int launch_decode_fp8(const AttnParams &p, void *stream, int max_ctas);
int launch_prefill_fp8(const AttnParams &p, void *stream);
// Staging of the FP8 cache for the tcgen05 prefill: job j dequantises source
// block `src` (valid slots) into f16 block `dst` of k_f16 / v_f16 (plain
// layout [16 slots][4 heads][128]); the queries are converted bf16 -> f16.
struct Fp8StageJob {
    int32_t dst, src, valid, pad;
};
int launch_fp8_stage(const void *k_pool, const void *v_pool, const Fp8StageJob *jobs, int32_t num_jobs, void *k_f16,
                     void *v_f16, const void *q_bf16, void *q_f16, int64_t q_values, void *stream);
bool decode_fp8_supported(int d_qk, int d_v, int hkv, int group, int block_size);
int launch_decode_mma(const AttnParams &p, void *stream);
int launch_decode_tma(const AttnParams &p, void *stream, int max_ctas);
bool decode_tma_supported(int d_qk, int d_v, int hkv, int group, int block_size);
int launch_prefill_mma(const AttnParams &p, void *stream);
int launch_mla(const AttnParams &p, void *stream);
// tcgen05 latent attention: items are (token, d_v half, key range) of 128 heads
int launch_mla_tc(const AttnParams &p, void *stream);
bool mla_tc_supported(int d_qk, int d_v, int hq, int hkv, int block_size);
int mla_tc_keys_per_tile();
// log-sum-exp merge of the split tokens listed in p.mgroups (partials [part, Hq, dv])
int launch_split_merge(const AttnParams &p, void *stream);
bool mla_supported(int d_qk, int d_v, int hq, int hkv);
int mla_heads_per_item();
// started (a cudaEvent_t, may be null): recorded once every CTA has begun;
// f16: Q, K and V are f16 (d = 128 only), else bf16; pdl: a programmatic
// dependent launch of the kernel before it on `stream`. With p.fa_count set
// the CTAs first write the prefill-path rows of the step (a cooperative
// launch: they wait for one another before reading the cache).
int launch_prefill_tc(const AttnParams &p, void *stream, int max_ctas, void *started = nullptr, bool f16 = false,
                      bool pdl = false);
bool prefill_tc_supported(int d_qk, int d_v, int block_size, int group);
int prefill_tc_rows_per_item(int group);
int prefill_tc_keys_per_tile();

}  // namespace fnpu
