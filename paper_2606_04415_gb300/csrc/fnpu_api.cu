// Host side of the C ABI: argument validation, the phase-aware planner and
// the launch sequence of a run.
//
// The planner is the GPU counterpart of the paper's phase-aware dispatch
// (Sec. 3.4): requests are classified by phase into a prefill queue (tensor
// work, tiles of query rows) and a decode queue (bandwidth work, split-KV
// items), and the mix of the two decides how the device is shared. The plan
// carries metadata only; tensors stay with the caller (Sec. 3.2).
#include <math.h>
#include <stdlib.h>
#include <stdio.h>
#include <string.h>

#include <algorithm>
#include <cmath>
#include <mutex>
#include <set>
#include <type_traits>
#include <utility>
#include <vector>

#include <cuda.h>

#include "fnpu_internal.h"

struct fnpu_plan {
    fnpu_attn_desc desc;
    float scale;
    int32_t num_seqs = 0;
    int64_t num_tokens = 0;
    int32_t bt_width = 0;
    int32_t num_sms = 0;
    int32_t flags = 0;
    bool use_tc = false;
    bool use_dt = false;
    bool use_mla = false;  // latent attention: one work list for both phases
    bool use_mla_tc = false;  // ... on the tcgen05 kernel (items of 128 heads and one d_v half)
    int32_t num_mitems = 0;
    fnpu::MlaItem *d_mitems = nullptr;
    int32_t num_mgroups = 0;  // split decode tokens merged by the merge kernel
    fnpu::MergeGroup *d_mgroups = nullptr;  // decode on the TMA-fed persistent kernel (items cover all kv heads)
    int32_t num_ditems = 0, num_pitems = 0, num_groups = 0, num_parts = 0;
    // device workspace: the error flag and work queues at offset 0 (kept
    // across re-plans), then metadata and scratch; it grows only when a
    // re-plan needs more than ws_cap bytes
    void *d_ws = nullptr;
    size_t ws_bytes = 0, ws_cap = 0;
    // pinned staging of the metadata upload, two buffers used in turn; the
    // event after each upload says when its buffer may be rewritten
    void *h_stage[2] = {nullptr, nullptr};
    size_t stage_cap[2] = {0, 0};
    cudaEvent_t e_upload[2] = {nullptr, nullptr};
    int32_t stage_turn = 0;
    fnpu::SeqInfo *d_seqs = nullptr;
    int32_t *d_bt = nullptr;
    fnpu::DecodeItem *d_ditems = nullptr;
    // FP8 cache with tcgen05 prefill: the prefill sequences' blocks dequantised
    // to f16 (num_jobs blocks, block table of tbt_width columns) and the
    // queries in f16, staged before the prefill kernel
    int32_t num_jobs = 0, tbt_width = 1, num_tblocks = 0;
    fnpu::Fp8StageJob *d_jobs = nullptr;
    int32_t *d_tbt = nullptr;
    void *d_tq = nullptr, *d_tk = nullptr, *d_tv = nullptr;
    fnpu::PrefillItem *d_pitems = nullptr;
    int32_t *d_counters = nullptr;
    int32_t *d_err = nullptr;
    // the step's tokens by queue (tcgen05 prefill plans): rows the prefill
    // grid appends itself in fnpu_mixed_step, and the decode rows
    int32_t *d_ftok = nullptr, *d_dtok = nullptr;
    int32_t num_ftok = 0, num_dtok = 0;
    float *d_part_lse = nullptr;
    float *d_part_o = nullptr;
    int32_t *d_pcounters = nullptr;
    float *d_ppart_lse = nullptr;
    float *d_ppart_o = nullptr;
    int32_t num_pparts = 0, num_pgroups = 0;
    // co-location (Sec. 3.4): prefill CTAs on pre_ctas SMs and decode CTAs on
    // the others, launched on two library streams forked from and joined back
    // into the caller's stream; e_started fires once all prefill CTAs began
    bool coloc = false;
    int32_t pre_ctas = 0;
    cudaStream_t s_pre = nullptr, s_dec = nullptr;
    cudaEvent_t e_fork = nullptr, e_started = nullptr, e_pre = nullptr, e_dec = nullptr;
    // FNPU_PLAN_GREEN_CONTEXTS: the two streams belong to green contexts over
    // disjoint SM partitions (dec_sms SMs for decode, pre_ctas for prefill)
    CUgreenCtx g_pre = nullptr, g_dec = nullptr;
    int32_t dec_sms = 0;
    int32_t green_k = -1;  // decode SMs asked of the current green contexts
    int32_t green_pre = 0;  // SMs of their prefill partition
};

namespace fnpu {

thread_local char g_last_cuda_error[256] = "";

int cuda_fail(cudaError_t e, const char *where) {
    snprintf(g_last_cuda_error, sizeof(g_last_cuda_error), "%s: %s", where, cudaGetErrorString(e));
    cudaGetLastError();  // clear non-sticky errors
    return FNPU_ECUDA;
}

namespace {

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Driver entry points of green contexts (SM partitions), looked up once.
struct GreenApi {
    CUresult (*device_get)(CUdevice *, int) = nullptr;
    CUresult (*get_resource)(CUdevice, CUdevResource *, CUdevResourceType) = nullptr;
    CUresult (*split)(CUdevResource *, unsigned int *, const CUdevResource *, CUdevResource *, unsigned int,
                      unsigned int) = nullptr;
    CUresult (*gen_desc)(CUdevResourceDesc *, CUdevResource *, unsigned int) = nullptr;
    CUresult (*create)(CUgreenCtx *, CUdevResourceDesc, CUdevice, unsigned int) = nullptr;
    CUresult (*destroy)(CUgreenCtx) = nullptr;
    CUresult (*stream_create)(CUstream *, CUgreenCtx, unsigned int, int) = nullptr;
    bool ok = false;
};

const GreenApi &green_api() {
    static std::once_flag once;
    static GreenApi g;
    std::call_once(once, [] {
        auto get = [](const char *name, auto &fn) {
            void *ptr = nullptr;
            cudaDriverEntryPointQueryResult q;
            if (cudaGetDriverEntryPointByVersion(name, &ptr, 13000, cudaEnableDefault, &q) == cudaSuccess &&
                q == cudaDriverEntryPointSuccess)
                fn = reinterpret_cast<std::remove_reference_t<decltype(fn)>>(ptr);
            return fn != nullptr;
        };
        g.ok = get("cuDeviceGet", g.device_get) && get("cuDeviceGetDevResource", g.get_resource) &&
               get("cuDevSmResourceSplitByCount", g.split) && get("cuDevResourceGenerateDesc", g.gen_desc) &&
               get("cuGreenCtxCreate", g.create) && get("cuGreenCtxDestroy", g.destroy) &&
               get("cuGreenCtxStreamCreate", g.stream_create);
        cudaGetLastError();
    });
    return g;
}

// The co-location streams (and green contexts) of a plan.
void destroy_streams(fnpu_plan *pl) {
    if (pl->s_pre) cudaStreamDestroy(pl->s_pre);
    if (pl->s_dec) cudaStreamDestroy(pl->s_dec);
    if (pl->g_pre) green_api().destroy(pl->g_pre);
    if (pl->g_dec) green_api().destroy(pl->g_dec);
    pl->g_pre = pl->g_dec = nullptr;
    pl->s_pre = pl->s_dec = nullptr;
    pl->green_k = -1;
}

void destroy_sync_objects(fnpu_plan *pl) {
    destroy_streams(pl);
    if (pl->e_started) cudaEventDestroy(pl->e_started);
    if (pl->e_dec) cudaEventDestroy(pl->e_dec);
    if (pl->e_fork) cudaEventDestroy(pl->e_fork);
    if (pl->e_pre) cudaEventDestroy(pl->e_pre);
    pl->e_fork = pl->e_started = pl->e_pre = pl->e_dec = nullptr;
}

// Everything a plan owns; the plan itself is deleted by the caller.
void release_plan(fnpu_plan *pl) {
    destroy_sync_objects(pl);
    for (int i = 0; i < 2; ++i) {
        if (pl->e_upload[i]) cudaEventDestroy(pl->e_upload[i]);
        if (pl->h_stage[i]) cudaFreeHost(pl->h_stage[i]);
        pl->e_upload[i] = nullptr;
        pl->h_stage[i] = nullptr;
        pl->stage_cap[i] = 0;
    }
    if (pl->d_ws) cudaFree(pl->d_ws);
    pl->d_ws = nullptr;
    pl->ws_cap = 0;
}

// Modelled rates of the two phases (measured on the co-located Qwen2.5-7B
// step): a prefill CTA finishes one 128-key tile of both Q tiles (d = 128)
// in about 1.5 us; a decode SM streams about 69 GB/s of KV cache and the
// whole device about 4 TB/s.
constexpr double kTileSec = 1.5e-6;
constexpr double kDecodeSmBps = 69e9;
constexpr double kDecodeAllBps = 4.0e12;

// (stop_at: the run may end as soon as the makespan reaches it; loads, if
// given, receives the final number of workers per load)
int64_t lpt_makespan(const std::vector<int32_t> &hist, int32_t m, int64_t stop_at = INT64_MAX,
                     std::vector<int32_t> *loads = nullptr);
std::vector<int32_t> cost_histogram(const std::vector<int64_t> &costs);

// SMs that start on decode while the others run prefill: the prefill CTAs on
// sms - k SMs take the items longest first, so each ends at its load of the
// LPT schedule of the item costs on sms - k workers, the last at the makespan
// Tp. Decode streams at min(all, per SM x SMs it holds) on the k SMs from the
// start and on each prefill SM from the moment its CTA ends (its CTAs take
// the SMs the prefill leaves), until the decode bytes are read at Td. The k
// with the shortest modelled step max(Tp, Td) wins, the largest such k on
// ties (more decode done while the prefill lasts).
int32_t choose_decode_sms(const std::vector<int64_t> &item_tiles, double tile_scale, int64_t dec_bytes,
                          int32_t sms) {
    const std::vector<int32_t> hist = cost_histogram(item_tiles);
    const double unit = tile_scale * kTileSec;  // seconds per cost unit
    std::vector<int32_t> loads;
    // (prefill end, decode end) with k decode SMs
    auto phases = [&](int32_t k) {
        const double tp = static_cast<double>(lpt_makespan(hist, sms - k, INT64_MAX, &loads)) * unit;
        double left = static_cast<double>(dec_bytes), t = 0.0;
        int32_t n = k;
        for (size_t ld = 0; ld <= loads.size() && left > 0.0; ++ld) {
            // decode on n SMs until the next prefill CTAs end (at load ld)
            const double next = ld < loads.size() ? static_cast<double>(ld) * unit : 1e30;
            if (ld < loads.size() && loads[ld] == 0) continue;
            const double rate = std::min(kDecodeAllBps, n * kDecodeSmBps);
            if (next > t) {
                const double run = std::min(next - t, left / rate);
                left -= run * rate;
                t += run;
            }
            if (ld < loads.size()) n += loads[ld];
        }
        return std::make_pair(tp, t);
    };
    // The prefill end grows with k and the decode end shrinks, so the step
    // max(Tp, Td) is shortest near the smallest k whose decode ends within
    // the prefill: found by bisection, then the k around it are compared
    // (the LPT makespan is not strictly monotone in the number of workers)
    const int32_t kmax = std::max<int32_t>(sms / 2, 1);
    int32_t lo = 1, hi = kmax;
    while (lo < hi) {
        const int32_t mid = (lo + hi) / 2;
        const auto ph = phases(mid);
        if (ph.second <= ph.first) hi = mid;
        else lo = mid + 1;
    }
    int32_t best_k = 1;
    double best_t = -1.0;
    for (int32_t k = std::max<int32_t>(1, lo - 4); k <= std::min<int32_t>(kmax, lo + 4); ++k) {
        const auto ph = phases(k);
        const double step = std::max(ph.first, ph.second);
        if (best_t < 0 || step <= best_t) {
            best_t = step;
            best_k = k;
        }
    }
    return best_k;
}

// Two packed Q tiles of one kv head (the tcgen05 prefill unit) before its key
// range is split.
struct TcUnit {
    int32_t seq, kvh, r0, rows;
    int32_t ntiles;     // 64-key tiles its rows can see
    int32_t max_start;  // last tile a split may start at: every row must see a key of every split
};

// Cost model of a prefill work item in units of one 128-key tile of both Q
// tiles: switching items (loading Q, draining the pipeline, the epilogue) and,
// for a split item, writing its partial result and the merge.
constexpr int64_t kTcItemCost = 2;
constexpr int64_t kTcMergeCost = 4;

// First tile of split j of n over ntiles tiles (split n is the end).
int32_t split_bound(int32_t ntiles, int32_t n, int32_t j) {
    return static_cast<int32_t>((static_cast<int64_t>(ntiles) * j) / n);
}

// Item costs (positive integers, in tiles) as a histogram: hist[c] items of
// cost c.
std::vector<int32_t> cost_histogram(const std::vector<int64_t> &costs) {
    int64_t cmax = 0;
    for (int64_t c : costs) cmax = std::max(cmax, c);
    std::vector<int32_t> hist(static_cast<size_t>(cmax) + 1, 0);
    for (int64_t c : costs) ++hist[static_cast<size_t>(std::max<int64_t>(c, 0))];
    return hist;
}

// Longest-processing-time-first makespan of the items of `hist` on m workers:
// the items longest first, each to the least loaded worker. The loads are
// integers and the least load never decreases (the worker that takes an item
// had the least load), so a count of workers per load value with a pointer
// that only moves up finds the least loaded workers; the items of one cost go
// to them together (workers are interchangeable, so the loads evolve as with
// one item at a time). No load exceeds the mean plus the largest item, which
// bounds the counts. Linear in distinct costs + loads.
int64_t lpt_makespan(const std::vector<int32_t> &hist, int32_t m, int64_t stop_at, std::vector<int32_t> *loads) {
    m = std::max<int32_t>(m, 1);
    int64_t total = 0, n = 0;
    for (size_t c = 0; c < hist.size(); ++c) {
        total += static_cast<int64_t>(c) * hist[c];
        n += hist[c];
    }
    if (n == 0) {
        if (loads) loads->assign(1, m);
        return 0;
    }
    const int64_t cmax = static_cast<int64_t>(hist.size()) - 1;
    const size_t bound = static_cast<size_t>(total / m + cmax + 1);
    thread_local std::vector<int32_t> cnt;
    cnt.assign(bound + 1, 0);
    cnt[0] = m;
    size_t p = 0;
    int64_t span = 0;
    for (int64_t c = cmax; c >= 0; --c) {
        int64_t k = hist[static_cast<size_t>(c)];
        while (k > 0) {
            while (cnt[p] == 0) ++p;
            const int64_t t = std::min<int64_t>(cnt[p], k);
            cnt[p] -= static_cast<int32_t>(t);
            cnt[p + static_cast<size_t>(c)] += static_cast<int32_t>(t);
            span = std::max<int64_t>(span, static_cast<int64_t>(p) + c);
            k -= t;
            if (span >= stop_at) return span;  // the caller only wants spans below stop_at
        }
    }
    if (loads) loads->assign(cnt.begin(), cnt.begin() + static_cast<std::ptrdiff_t>(span) + 1);
    return span;
}

// Indices of `cost` by decreasing cost, equal costs in index order (a stable
// longest-first order). The costs here are small non-negative integers, so a
// counting sort does it in linear time; a wide range falls back to a stable
// sort.
std::vector<int32_t> longest_first(const std::vector<int64_t> &cost) {
    const size_t n = cost.size();
    std::vector<int32_t> order(n);
    int64_t cmax = 0;
    for (int64_t c : cost) cmax = std::max(cmax, c);
    if (cmax <= 4 * static_cast<int64_t>(n) + 4096) {
        std::vector<int32_t> start(static_cast<size_t>(cmax) + 2, 0);  // bucket cmax - c, largest cost first
        for (int64_t c : cost) ++start[static_cast<size_t>(cmax - c) + 1];
        for (size_t b = 1; b < start.size(); ++b) start[b] += start[b - 1];
        for (size_t i = 0; i < n; ++i) order[static_cast<size_t>(start[static_cast<size_t>(cmax - cost[i])]++)] = static_cast<int32_t>(i);
    } else {
        for (size_t i = 0; i < n; ++i) order[i] = static_cast<int32_t>(i);
        std::stable_sort(order.begin(), order.end(), [&](int32_t a, int32_t b) { return cost[a] > cost[b]; });
    }
    return order;
}

// Number of key splits per unit. A persistent CTA per SM takes items longest
// first, so the step lasts about as long as the LPT schedule of the items.
// Splitting the largest units evens that schedule out but costs a partial
// write and a merge, so the piece-size cap is chosen among a few candidates
// by the modelled makespan.
std::vector<int32_t> choose_prefill_splits(const std::vector<TcUnit> &units, int32_t sms) {
    int64_t total = 0, maxc = 0;
    for (const TcUnit &u : units) {
        total += u.ntiles;
        maxc = std::max<int64_t>(maxc, u.ntiles);
    }
    std::vector<int64_t> caps = {maxc};
    for (int k = 2; k <= 8; ++k) caps.push_back((maxc + k - 1) / k);
    // (cap below: pieces shorter than 4 tiles cost more than they balance)
    for (int j = 1; j <= 8; ++j) caps.push_back((total + static_cast<int64_t>(sms) * j - 1) / (static_cast<int64_t>(sms) * j));
    std::vector<int32_t> best(units.size(), 1), ns(units.size(), 1);
    int64_t best_span = -1;
    {  // drop repeated candidates, keeping the first of each (ties go to the earlier one)
        std::vector<int64_t> uniq;
        for (int64_t c : caps)
            if (std::find(uniq.begin(), uniq.end(), c) == uniq.end()) uniq.push_back(c);
        caps.swap(uniq);
    }
    std::vector<int32_t> hist(static_cast<size_t>(maxc + kTcItemCost + kTcMergeCost) + 1);
    // the most splits a unit can take (at most 16): its last split must start
    // at or before max_start, and that start, floor(ntiles (n - 1) / n), does
    // not decrease with n, so the feasible counts are 1 .. nmax
    std::vector<int32_t> nmax(units.size(), 1);
    for (size_t i = 0; i < units.size(); ++i) {
        int32_t n = std::min<int32_t>(16, std::max<int32_t>(units[i].ntiles, 1));  // no empty piece
        while (n > 1 && split_bound(units[i].ntiles, n, n - 1) > units[i].max_start) --n;
        nmax[i] = n;
    }
    // split_units[c]: units longer than c tiles that may split. Under a cap
    // of c exactly these split, each into two pieces or more, and a unit cut
    // into n >= 2 pieces costs at least kTcItemCost + 2 kTcMergeCost more than
    // whole; with the total of the unsplit items that bounds a candidate's
    // total from below before its splits are worked out
    std::vector<int32_t> split_units(static_cast<size_t>(maxc) + 2, 0);
    for (size_t i = 0; i < units.size(); ++i)
        if (nmax[i] >= 2) ++split_units[static_cast<size_t>(units[i].ntiles) - 1];
    for (int64_t c = maxc - 1; c >= 0; --c) split_units[static_cast<size_t>(c)] += split_units[static_cast<size_t>(c) + 1];
    const int64_t whole = total + static_cast<int64_t>(units.size()) * kTcItemCost;
    std::vector<int32_t> prev;
    for (int64_t cap : caps) {
        if (cap < 4) continue;
        if (best_span >= 0) {
            const int64_t nsplit = cap >= maxc ? 0 : split_units[static_cast<size_t>(cap)];
            if (nsplit == 0) continue;  // no unit splits: the first candidate's items
            const int64_t lb = whole + nsplit * (kTcItemCost + 2 * kTcMergeCost);
            if ((lb + sms - 1) / sms >= best_span) continue;
        }
        // ceil(ntiles / cap) = floor((ntiles - 1) / cap) + 1 in double, exact
        // for tile counts (below 2^26): a quotient that is not an integer has a
        // fraction of at least 1 / cap, above 1e-8, and the product errs by far
        // less than the 1e-9 added (the conversion truncates, = floor here)
        const double inv = 1.0 / static_cast<double>(cap);
        // (no schedule on sms workers is shorter than ceil(total / sms), so a
        // candidate whose total already reaches the best span is skipped)
        // (units come in runs with equal tile counts and split limits, one
        // per kv head of a row block: such a unit repeats the one before)
        int64_t tot = 0;
        for (size_t i = 0; i < units.size(); ++i) {
            int32_t n;
            if (i > 0 && units[i].ntiles == units[i - 1].ntiles && nmax[i] == nmax[i - 1]) {
                n = ns[i - 1];
            } else {
                const int32_t q = static_cast<int32_t>((units[i].ntiles - 1) * inv + 1e-9) + 1;
                n = std::min(q, nmax[i]);
            }
            ns[i] = n;
            tot += units[i].ntiles + static_cast<int64_t>(n) * (kTcItemCost + (n > 1 ? kTcMergeCost : 0));
        }
        if (ns == prev) continue;  // the same splits as the candidate before
        prev = ns;
        if (best_span >= 0 && (tot + sms - 1) / sms >= best_span) continue;
        std::fill(hist.begin(), hist.end(), 0);
        for (size_t i = 0; i < units.size(); ++i) {
            // n pieces of floor(ntiles / n) or one more tiles (split_bound
            // rounds down), the longer ones ntiles mod n of them
            const int32_t n = ns[i], nt = units[i].ntiles, q = nt / n, r = nt % n;
            const int32_t extra = kTcItemCost + (n > 1 ? kTcMergeCost : 0);
            hist[static_cast<size_t>(q + 1 + extra)] += r;
            hist[static_cast<size_t>(q + extra)] += n - r;
        }
        const int64_t span = lpt_makespan(hist, sms, best_span < 0 ? INT64_MAX : best_span);
        if (best_span < 0 || span < best_span) {
            best_span = span;
            best = ns;
        }
    }
    return best;
}

}  // namespace

EncodeTiledFn tensor_map_encoder() {
    static std::once_flag once;
    static EncodeTiledFn fn = nullptr;
    std::call_once(once, [] {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(ptr);
    });
    return fn;
}

namespace {

bool shape_ok(const fnpu_attn_desc *d, int *status) {
    *status = FNPU_EINVAL;
    if (!d) return false;
    if (d->num_q_heads <= 0 || d->num_kv_heads <= 0 || d->num_q_heads % d->num_kv_heads) return false;
    if (d->head_dim_qk <= 0 || d->head_dim_v <= 0 || d->block_size <= 0 || d->num_blocks <= 0)
        return false;
    if (d->kv_fp8 != 0 && d->kv_fp8 != 1) return false;
    if (d->v_in_k_latent) {
        if (d->num_kv_heads != 1 || d->head_dim_v > d->head_dim_qk) return false;
    }
    if ((static_cast<int64_t>(d->head_dim_qk) * 2) % 16 || (static_cast<int64_t>(d->head_dim_v) * 2) % 16)
        return false;
    *status = FNPU_OK;
    return true;
}

// The FP8 cache format exists for Hkv = 4, d = 128, 16-slot blocks, G <= 8.
bool fp8_shape(const fnpu_attn_desc *d) {
    return !d->v_in_k_latent && decode_fp8_supported(d->head_dim_qk, d->head_dim_v, d->num_kv_heads,
                                                     d->num_q_heads / d->num_kv_heads, d->block_size);
}

// Kernels exist for split K/V with d in {64, 128} (decode needs G <= 8) and
// for the latent layout with d_qk = 576, d_v = 512 and a multiple of 64 heads.
// The FP8 cache has one decode and one prefill kernel for its one shape; the
// per-head keys (192 columns) and values (128) of a decompressed latent cache
// have a prefill kernel only.
int kernel_support(const fnpu_attn_desc *d, bool has_decode, bool has_prefill) {
    (void)has_prefill;
    if (d->kv_fp8) return fp8_shape(d) ? FNPU_OK : FNPU_EUNSUPPORTED;
    if (!d->v_in_k_latent && d->head_dim_qk == 192 && d->head_dim_v == 128)
        return has_decode ? FNPU_EUNSUPPORTED : FNPU_OK;
    if (d->v_in_k_latent)
        return mla_supported(d->head_dim_qk, d->head_dim_v, d->num_q_heads, d->num_kv_heads) ? FNPU_OK
                                                                                               : FNPU_EUNSUPPORTED;
    if (d->head_dim_qk != d->head_dim_v) return FNPU_EUNSUPPORTED;
    if (d->head_dim_qk != 64 && d->head_dim_qk != 128) return FNPU_EUNSUPPORTED;
    if (has_decode && d->num_q_heads / d->num_kv_heads > 8) return FNPU_EUNSUPPORTED;
    return FNPU_OK;
}

}  // namespace
}  // namespace fnpu

namespace fnpu {
namespace {
// The tcgen05 prefill launch; over the FP8 cache, first the f16 staging of
// the prefill sequences' blocks and of the queries, and the prefill reads those.
// With pdl a bf16 prefill grid is a programmatic dependent launch of the
// kernel before it on `stream` (the step's append): its CTAs set up while that
// kernel drains, and its loaders wait for it before the first read.
int launch_prefill(const fnpu_plan *pl, const AttnParams &p, void *stream, int ctas, void *started,
                   bool pdl = false) {
    if (!pl->desc.kv_fp8) return launch_prefill_tc(p, stream, ctas, started, false, pdl);
    const int rc = launch_fp8_stage(p.k_cache, p.v_cache, pl->d_jobs, pl->num_jobs, pl->d_tk, pl->d_tv, p.q, pl->d_tq,
                                    p.num_tokens * p.num_q_heads * p.head_dim_qk, stream);
    if (rc != FNPU_OK) return rc;
    AttnParams pp = p;
    pp.q = pl->d_tq;
    pp.k_cache = pl->d_tk;
    pp.v_cache = pl->d_tv;
    pp.block_table = pl->d_tbt;
    pp.bt_stride = pl->tbt_width;
    pp.num_blocks = pl->num_tblocks;
    return launch_prefill_tc(pp, stream, ctas, started, true);
}
}  // namespace
}  // namespace fnpu

using namespace fnpu;

extern "C" {

const char *fnpu_status_str(int s) {
    switch (s) {
        case FNPU_OK: return "ok";
        case FNPU_EINVAL: return "invalid argument";
        case FNPU_EUNSUPPORTED: return "unsupported shape";
        case FNPU_ECUDA: return "CUDA runtime error";
        case FNPU_EDEVICE_TIMEOUT: return "device-side wait timed out";
        case FNPU_ENOMEM: return "out of memory";
        case FNPU_EDEVICE_RANGE: return "device met an out-of-range slot";
        default: return "unknown status";
    }
}

int fnpu_version(void) { return 100; }

const char *fnpu_last_cuda_error(void) { return g_last_cuda_error; }

int fnpu_kv_append(const fnpu_attn_desc *desc, const void *k_new, const void *v_new,
                   const int64_t *slot_mapping, int32_t num_tokens, void *k_cache, void *v_cache,
                   void *stream) {
    int st;
    if (!shape_ok(desc, &st)) return st;
    if (num_tokens < 0) return FNPU_EINVAL;
    if (num_tokens == 0) return FNPU_OK;
    const bool latent = desc->v_in_k_latent != 0;
    if (!k_new || !slot_mapping || !k_cache) return FNPU_EINVAL;
    if (!latent && (!v_new || !v_cache)) return FNPU_EINVAL;
    const uintptr_t mis = reinterpret_cast<uintptr_t>(k_new) | reinterpret_cast<uintptr_t>(k_cache) |
                          (latent ? 0 : (reinterpret_cast<uintptr_t>(v_new) |
                                         reinterpret_cast<uintptr_t>(v_cache)));
    if (mis & 15u) return FNPU_EINVAL;
    if (reinterpret_cast<uintptr_t>(slot_mapping) & 7u) return FNPU_EINVAL;
    if (desc->kv_fp8) {
        if (!fp8_shape(desc)) return FNPU_EUNSUPPORTED;
        return launch_kv_append_fp8(desc, k_new, v_new, slot_mapping, num_tokens, k_cache, v_cache, stream);
    }
    return launch_kv_append(desc, k_new, v_new, slot_mapping, num_tokens, k_cache, v_cache, stream);
}

int fnpu_check(void *stream) {
    int flag = 0;
    const int rc = read_and_clear_global_error(stream, &flag);
    if (rc != FNPU_OK) return rc;
    if (flag & 4) return FNPU_EDEVICE_TIMEOUT;  // a bounded wait of the MLA expansion gave up
    return flag ? FNPU_EDEVICE_RANGE : FNPU_OK;
}

int fnpu_mixed_attn_plan(const fnpu_attn_desc *desc, int32_t num_seqs, const int32_t *query_len,
                         const int32_t *context_len, const uint8_t *phase,
                         const int32_t *block_table, int32_t block_table_stride, void *stream,
                         fnpu_plan **out) {
    return fnpu_mixed_attn_plan_ex(desc, num_seqs, query_len, context_len, phase, block_table,
                                   block_table_stride, nullptr, stream, out);
}

}  // extern "C"

namespace {

// Validated shape of one step's metadata.
struct StepMeta {
    int64_t T = 0;
    int32_t width = 1;
    bool has_decode = false, has_prefill = false;
};

// Host checks of a plan's arguments: nothing is launched or allocated.
int validate_meta(const fnpu_attn_desc *desc, int32_t num_seqs, const int32_t *query_len,
                  const int32_t *context_len, const uint8_t *phase, const int32_t *block_table,
                  int32_t block_table_stride, const fnpu_plan_opts &o, StepMeta *m) {
    int st;
    if (!shape_ok(desc, &st)) return st;
    if (num_seqs < 0) return FNPU_EINVAL;
    if (num_seqs > 0 && (!query_len || !context_len || !phase || !block_table)) return FNPU_EINVAL;
    if (o.decode_split_keys < 0 || o.decode_share_pct < 0 || o.decode_share_pct > 100 || o.num_sms < 0)
        return FNPU_EINVAL;
    const int32_t bs = desc->block_size;
    StepMeta r;
    for (int32_t s = 0; s < num_seqs; ++s) {
        const int32_t q = query_len[s], c = context_len[s];
        if (q < 1 || c < q) return FNPU_EINVAL;
        if (phase[s] > 1) return FNPU_EINVAL;
        // a decode step of several tokens (speculative verification) is causal
        // attention of a short chunk: its rows take the prefill path
        r.has_decode |= phase[s] == 1 && q == 1;
        r.has_prefill |= phase[s] == 0 || q > 1;
        const int32_t nb = (c + bs - 1) / bs;
        if (nb > block_table_stride) return FNPU_EINVAL;
        const int32_t *row = block_table + static_cast<int64_t>(s) * block_table_stride;
        int32_t lo = INT32_MAX, hi = INT32_MIN;  // (a min/max pass over the row vectorises)
        for (int32_t j = 0; j < nb; ++j) {
            lo = std::min(lo, row[j]);
            hi = std::max(hi, row[j]);
        }
        if (nb > 0 && (lo < 0 || hi >= desc->num_blocks)) return FNPU_EINVAL;
        r.width = std::max(r.width, nb);
        r.T += q;
    }
    if (r.T > INT32_MAX) return FNPU_EINVAL;
    if (num_seqs > 0) {
        const int ks = kernel_support(desc, r.has_decode, r.has_prefill);
        if (ks != FNPU_OK) return ks;
    }
    *m = r;
    return FNPU_OK;
}

int plan_sms(const fnpu_plan_opts &o, int *sms) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return FNPU_ECUDA;
    *sms = o.num_sms;
    if (*sms == 0 && cudaDeviceGetAttribute(sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return FNPU_ECUDA;
    return FNPU_OK;
}

// Build (or rebuild) the work list of a validated step into `pl`, reusing
// whatever streams, events, staging buffers and workspace it already holds.
// On an error after validation the plan must be re-planned or destroyed.
int plan_fill(fnpu_plan *pl, const fnpu_attn_desc *desc, int32_t num_seqs, const int32_t *query_len,
              const int32_t *context_len, const uint8_t *phase, const int32_t *block_table,
              int32_t block_table_stride, const fnpu_plan_opts &o, const StepMeta &meta, int sms,
              void *stream) {
    const int32_t bs = desc->block_size;
    const int64_t T = meta.T;
    const int32_t width = meta.width;
    pl->desc = *desc;
    pl->scale = desc->softmax_scale > 0.f ? desc->softmax_scale
                                          : static_cast<float>(1.0 / sqrt(static_cast<double>(desc->head_dim_qk)));
    pl->num_seqs = num_seqs;
    pl->num_jobs = 0;  // (FP8 staging, set below when the plan has some)
    pl->tbt_width = 1;
    pl->num_tblocks = 0;
    pl->num_tokens = T;
    pl->bt_width = width;
    pl->num_sms = sms;
    pl->flags = o.flags;
    pl->use_mla = desc->v_in_k_latent != 0;
    pl->use_mla_tc = pl->use_mla && !(o.flags & FNPU_PLAN_NO_TCGEN05) &&
                     mla_tc_supported(desc->head_dim_qk, desc->head_dim_v, desc->num_q_heads, desc->num_kv_heads, bs);
    pl->use_dt = !pl->use_mla && decode_tma_supported(desc->head_dim_qk, desc->head_dim_v, desc->num_kv_heads,
                                                      desc->num_q_heads / desc->num_kv_heads, bs);
    pl->use_tc = !pl->use_mla && !(o.flags & FNPU_PLAN_NO_TCGEN05) &&
                 prefill_tc_supported(desc->head_dim_qk, desc->head_dim_v, bs,
                                      desc->num_q_heads / desc->num_kv_heads);

    const int32_t G = desc->num_q_heads / desc->num_kv_heads;
    // working lists, kept per thread across plans so that a re-plan
    // allocates nothing once they have grown to the step's size
    thread_local std::vector<SeqInfo> seqs;
    thread_local std::vector<DecodeItem> ditems;
    thread_local std::vector<PrefillItem> pitems;
    thread_local std::vector<std::pair<int64_t, int32_t>> pcost;  // (cost, index) for LPT order
    thread_local std::vector<TcUnit> tc_units;
    thread_local std::vector<MergeGroup> mgroups;
    seqs.assign(static_cast<size_t>(num_seqs), SeqInfo{});
    ditems.clear();
    pitems.clear();
    pcost.clear();
    tc_units.clear();
    mgroups.clear();

    // decode split length: a TMA decode item streams every kv head of its
    // keys, and about two equal items per SM already keep HBM saturated, while
    // every further item adds a partial result to write and merge and a
    // switch in its CTA: measured on 64 decodes of 512..4096 keys, attention
    // takes 61 us with 512-key items (322 items), 65 us with 256 and 68 us
    // with 128. The per-head kernel aims at about 3 waves of 2 CTAs per SM.
    // the queue a sequence's work enters: decode items for one-token decodes
    auto decode_queue = [&](int32_t s) { return phase[s] == 1 && query_len[s] == 1; };
    // a decode item with its sequence's fields and its first four block ids
    auto decode_item = [&](int32_t s, int32_t kvh, int32_t kb, int32_t ke, int32_t sp, int32_t ns, int32_t base,
                           int32_t grp) {
        DecodeItem it{s, kvh, kb, ke, sp, ns, base, grp, seqs[s].q_start, seqs[s].bt_row, 0, 0, {0, 0, 0, 0}};
        for (int32_t i = 0; i < 4 && kb / bs + i <= (ke - 1) / bs; ++i)
            it.blk[i] = block_table[static_cast<int64_t>(s) * block_table_stride + kb / bs + i];
        return it;
    };
    int64_t dec_keys = 0;
    for (int32_t s = 0; s < num_seqs; ++s)
        if (decode_queue(s))
            dec_keys += static_cast<int64_t>(context_len[s]) * (pl->use_dt ? 1 : desc->num_kv_heads);
    int32_t split = o.decode_split_keys;
    if (split == 0) {
        const int64_t target = (pl->use_dt ? 2LL : 6LL) * sms;
        int64_t sk = (dec_keys + target - 1) / std::max<int64_t>(target, 1);
        sk = (sk + 63) / 64 * 64;
        split = static_cast<int32_t>(std::min<int64_t>(std::max<int64_t>(sk, pl->use_dt ? 128 : 256), 4096));
    }

    // latent attention: every query row (prefill or decode) is 64-head blocks
    // over its visible keys, split into pieces of at most mla_split keys so
    // that about three CTAs per SM share the work; longest first
    thread_local std::vector<MlaItem> mitems;
    mitems.clear();
    int32_t mla_split = 0;
    int32_t mla_split_tiles = 0;
    if (pl->use_mla_tc) {
        // two CTAs (d_v halves) per piece, 64-key tiles; a token is cut only
        // when it alone would exceed half of an SM's mean share of the tiles
        // (then pieces of whole tiles, at least 16 of them)
        const int32_t kt = mla_tc_keys_per_tile();
        int64_t tiles = 0;
        for (int32_t s = 0; s < num_seqs; ++s)
            for (int32_t i = 0; i < query_len[s]; ++i)
                tiles += 2 * ((context_len[s] - query_len[s] + i + 1 + kt - 1) / kt);
        const int64_t half_mean = (tiles + 2LL * sms - 1) / (2LL * sms);
        mla_split_tiles = static_cast<int32_t>(std::min<int64_t>(std::max<int64_t>(half_mean, 16), 1 << 20));
    } else if (pl->use_mla) {
        int64_t rows_keys = 0;
        for (int32_t s = 0; s < num_seqs; ++s) {
            const int64_t q = query_len[s], p0 = context_len[s] - query_len[s];
            rows_keys += q * p0 + q * (q + 1) / 2;
        }
        rows_keys *= desc->num_q_heads / mla_heads_per_item();
        const int64_t target = 3LL * sms;
        int64_t sk = (rows_keys + target - 1) / target;
        sk = std::max<int64_t>((sk + 255) / 256 * 256, 1024);
        mla_split = static_cast<int32_t>(std::min<int64_t>(sk, 1 << 20));
    }

    int32_t qs = 0, parts = 0, groups = 0;
    for (int32_t s = 0; s < num_seqs; ++s) {
        seqs[s] = SeqInfo{qs, query_len[s], context_len[s], s};
        const int32_t q = query_len[s], c = context_len[s];
        if (pl->use_mla_tc) {
            const int32_t kt = mla_tc_keys_per_tile();
            for (int32_t i = 0; i < q; ++i) {
                const int32_t keys = c - q + i + 1;
                const int32_t nt = (keys + kt - 1) / kt;
                const int32_t ns = (nt + mla_split_tiles - 1) / mla_split_tiles;
                const int32_t per = (nt + ns - 1) / ns;  // tiles per piece
                const int32_t base = ns > 1 ? parts : 0;
                if (ns > 1) {
                    mgroups.push_back(MergeGroup{qs + i, ns, parts, 0});
                    parts += ns;
                }
                for (int32_t sp = 0; sp < ns; ++sp)
                    for (int32_t h = 0; h < 2; ++h)  // the two d_v halves, next to each other
                        mitems.push_back(MlaItem{s, i, h, sp * per * kt, std::min(keys, (sp + 1) * per * kt), sp, ns,
                                                 base, 0, 0, 0, 0});
            }
        } else if (pl->use_mla) {
            const int32_t nhb = desc->num_q_heads / mla_heads_per_item();
            for (int32_t i = 0; i < q; ++i) {
                const int32_t keys = c - q + i + 1;
                const int32_t ns = (keys + mla_split - 1) / mla_split;
                const int32_t sk = (keys + ns - 1) / ns;  // even pieces
                for (int32_t hb = 0; hb < nhb; ++hb) {
                    const int32_t base = ns > 1 ? parts : 0, grp = ns > 1 ? groups : 0;
                    if (ns > 1) {
                        parts += ns;
                        groups += 1;
                    }
                    for (int32_t sp = 0; sp < ns; ++sp)
                        mitems.push_back(MlaItem{s, i, hb, sp * sk, std::min(keys, (sp + 1) * sk), sp, ns, base, grp,
                                                 0, 0, 0});
                }
            }
        } else if (decode_queue(s) && pl->use_dt) {
            // items over all kv heads; a split sequence is merged by the merge
            // kernel (at most 256 splits: its scratch grows with them)
            const int32_t sk = std::max(split, (c + 256 * 64 - 1) / (256 * 64) * 64);
            const int32_t ns = (c + sk - 1) / sk;
            const int32_t base = ns > 1 ? parts : 0;
            if (ns > 1) {
                mgroups.push_back(MergeGroup{qs, ns, parts, 0});
                parts += ns;
            }
            for (int32_t sp = 0; sp < ns; ++sp) {
                const int32_t kb = sp * sk, ke = std::min(c, kb + sk);
                ditems.push_back(decode_item(s, 0, kb, ke, sp, ns, base, 0));
            }
        } else if (decode_queue(s)) {
            const int32_t ns = (c + split - 1) / split;
            for (int32_t kvh = 0; kvh < desc->num_kv_heads; ++kvh) {
                const int32_t grp = groups++;
                const int32_t base = ns > 1 ? parts : 0;
                if (ns > 1) parts += ns;
                for (int32_t sp = 0; sp < ns; ++sp) {
                    const int32_t kb = sp * split, ke = std::min(c, kb + split);
                    ditems.push_back(decode_item(s, kvh, kb, ke, sp, ns, base, grp));
                }
            }
        } else if (pl->use_tc) {
            // tcgen05 tiles: two Q tiles of P positions x G heads of one kv
            // head; their key splits are chosen once all tiles are known
            const int32_t prefix = c - q;
            const int32_t P2 = prefill_tc_rows_per_item(G), KT = prefill_tc_keys_per_tile();
            for (int32_t r0 = 0; r0 < q; r0 += P2) {
                const int32_t rows = std::min(P2, q - r0);
                const int32_t ntiles = (prefix + r0 + rows + KT - 1) / KT;
                for (int32_t kvh = 0; kvh < desc->num_kv_heads; ++kvh)
                    tc_units.push_back(TcUnit{s, kvh, r0, rows, ntiles, (prefix + r0) / KT});
            }
        } else {
            const int32_t prefix = c - q;
            for (int32_t r0 = 0; r0 < q; r0 += 64) {
                const int32_t rows = std::min(64, q - r0);
                for (int32_t h = 0; h < desc->num_q_heads; ++h) {
                    pcost.emplace_back(static_cast<int64_t>(prefix) + r0 + rows,
                                       static_cast<int32_t>(pitems.size()));
                    pitems.push_back(PrefillItem{s, h, r0, rows, 0, 0, 0, 1, 0, 0, qs, prefix, c, s, 0, 0});
                }
            }
        }
        qs += query_len[s];
    }
    // co-location: the decode CTAs take a share of the SMs while the prefill
    // CTAs hold the rest
    pl->coloc = pl->use_tc && pl->use_dt && !tc_units.empty() && !ditems.empty() &&
                !(o.flags & FNPU_PLAN_SEPARATE_LAUNCHES);
    pl->pre_ctas = sms;
    if (pl->coloc) {
        int64_t dec_bytes = 0;
        for (const DecodeItem &it : ditems)
            dec_bytes += static_cast<int64_t>(it.key_end - it.key_begin) * desc->num_kv_heads *
                         (desc->kv_fp8 ? desc->head_dim_qk + desc->head_dim_v + 8
                                       : (desc->head_dim_qk + desc->head_dim_v) * 2);
        std::vector<int64_t> item_tiles;
        for (const TcUnit &u : tc_units) item_tiles.push_back(u.ntiles + kTcItemCost);
        std::sort(item_tiles.begin(), item_tiles.end(), [](int64_t a, int64_t b) { return a > b; });
        const double tile_scale = (desc->head_dim_qk + desc->head_dim_v) / 256.0;  // relative to d = 128
        const int32_t k = o.decode_share_pct > 0
                              ? std::min(sms - 1, std::max(1, (sms * o.decode_share_pct + 50) / 100))
                              : choose_decode_sms(item_tiles, tile_scale, dec_bytes, sms);
        pl->pre_ctas = sms - k;
        if ((o.flags & FNPU_PLAN_GREEN_CONTEXTS) && pl->g_pre && pl->green_k == k) {
            pl->pre_ctas = pl->green_pre;  // the partitions of the last plan fit this share
        } else if (o.flags & FNPU_PLAN_GREEN_CONTEXTS) {
            // enforce the split in hardware: a green context of at least k SMs
            // (rounded up to the partition granularity) for decode and one of
            // the remaining SMs for prefill, each with its own stream
            destroy_streams(pl);
            const GreenApi &g = green_api();
            int dev = 0;
            CUdevice cudev = 0;
            CUdevResource all{}, part{}, rest{};
            CUdevResourceDesc d_dec = nullptr, d_pre = nullptr;
            unsigned int ngroups = 1;
            CUstream st_dec = nullptr, st_pre = nullptr;
            const bool made = g.ok && cudaGetDevice(&dev) == cudaSuccess && g.device_get(&cudev, dev) == CUDA_SUCCESS &&
                              g.get_resource(cudev, &all, CU_DEV_RESOURCE_TYPE_SM) == CUDA_SUCCESS &&
                              static_cast<int32_t>(all.sm.smCount) == sms &&
                              g.split(&part, &ngroups, &all, &rest, 0, static_cast<unsigned int>(k)) == CUDA_SUCCESS &&
                              ngroups == 1 && rest.sm.smCount > 0 && g.gen_desc(&d_dec, &part, 1) == CUDA_SUCCESS &&
                              g.gen_desc(&d_pre, &rest, 1) == CUDA_SUCCESS &&
                              g.create(&pl->g_dec, d_dec, cudev, CU_GREEN_CTX_DEFAULT_STREAM) == CUDA_SUCCESS &&
                              g.create(&pl->g_pre, d_pre, cudev, CU_GREEN_CTX_DEFAULT_STREAM) == CUDA_SUCCESS &&
                              g.stream_create(&st_dec, pl->g_dec, CU_STREAM_NON_BLOCKING, 0) == CUDA_SUCCESS &&
                              g.stream_create(&st_pre, pl->g_pre, CU_STREAM_NON_BLOCKING, 0) == CUDA_SUCCESS;
            pl->s_dec = reinterpret_cast<cudaStream_t>(st_dec);
            pl->s_pre = reinterpret_cast<cudaStream_t>(st_pre);
            if (!made) {
                cudaGetLastError();
                destroy_streams(pl);
                return FNPU_EUNSUPPORTED;
            }
            pl->dec_sms = static_cast<int32_t>(part.sm.smCount);
            pl->pre_ctas = pl->green_pre = static_cast<int32_t>(rest.sm.smCount);
            pl->green_k = k;
        } else if (pl->g_pre) {
            destroy_streams(pl);  // plain streams are made below
        }
    }
    int32_t pparts = 0, pgroups = 0;
    if (!tc_units.empty()) {
        const std::vector<int32_t> ns = choose_prefill_splits(tc_units, pl->pre_ctas);
        for (size_t u = 0; u < tc_units.size(); ++u) {
            const TcUnit &t = tc_units[u];
            const int32_t n = ns[u];
            const int32_t base = n > 1 ? pparts : 0, grp = n > 1 ? pgroups : 0;
            if (n > 1) {
                pparts += n;
                pgroups += 1;
            }
            for (int32_t j = 0; j < n; ++j) {
                const int32_t kb = split_bound(t.ntiles, n, j), ke = split_bound(t.ntiles, n, j + 1);
                pcost.emplace_back(static_cast<int64_t>(ke - kb) + kTcItemCost + (n > 1 ? kTcMergeCost : 0),
                                   static_cast<int32_t>(pitems.size()));
                pitems.push_back(PrefillItem{t.seq, t.kvh, t.r0, t.rows, kb, ke, j, n, base, grp,
                                             seqs[t.seq].q_start, seqs[t.seq].ctx_len - seqs[t.seq].q_len,
                                             seqs[t.seq].ctx_len, seqs[t.seq].bt_row, 0, 0});
            }
        }
    }
    // FP8 cache, tcgen05 prefill: every prefill sequence's blocks get an f16
    // copy (its own block-table row over the staged blocks)
    std::vector<Fp8StageJob> jobs;
    std::vector<int32_t> tbt;
    if (desc->kv_fp8 && pl->use_tc && !tc_units.empty()) {
        std::vector<char> pre(num_seqs, 0);
        for (const TcUnit &u : tc_units) pre[u.seq] = 1;
        int32_t tw = 1;
        for (int32_t s = 0; s < num_seqs; ++s)
            if (pre[s]) tw = std::max(tw, (context_len[s] + bs - 1) / bs);
        tbt.assign(static_cast<size_t>(std::max(num_seqs, 1)) * tw, 0);
        for (int32_t s = 0; s < num_seqs; ++s) {
            if (!pre[s]) continue;
            const int32_t nb = (context_len[s] + bs - 1) / bs;
            for (int32_t j = 0; j < nb; ++j) {
                const int32_t dst = static_cast<int32_t>(jobs.size());
                jobs.push_back(Fp8StageJob{dst, block_table[static_cast<int64_t>(s) * block_table_stride + j],
                                           std::min(bs, context_len[s] - j * bs), 0});
                tbt[static_cast<size_t>(s) * tw + j] = dst;
            }
        }
        pl->num_jobs = static_cast<int32_t>(jobs.size());
        pl->tbt_width = tw;
        pl->num_tblocks = std::max(pl->num_jobs, 1);
    }

    // longest prefill tiles first; decode items longest first as well (the
    // items are gathered in these orders straight into the upload below)
    std::vector<int32_t> porder, dorder;
    {
        thread_local std::vector<int64_t> cost;
        cost.assign(pitems.size(), 0);
        for (const auto &pc : pcost) cost[static_cast<size_t>(pc.second)] = pc.first;
        porder = longest_first(cost);
        cost.resize(ditems.size());
        for (size_t i = 0; i < ditems.size(); ++i) cost[i] = ditems[i].key_end - ditems[i].key_begin;
        dorder = longest_first(cost);
    }

    std::stable_sort(mitems.begin(), mitems.end(), [](const MlaItem &a, const MlaItem &b) {
        return (a.key_end - a.key_begin) > (b.key_end - b.key_begin);
    });
    pl->num_mitems = static_cast<int32_t>(mitems.size());
    pl->num_mgroups = static_cast<int32_t>(mgroups.size());
    pl->num_ditems = static_cast<int32_t>(ditems.size());
    pl->num_pitems = static_cast<int32_t>(pitems.size());
    pl->num_groups = groups;
    pl->num_parts = parts;
    pl->num_pparts = pparts;
    pl->num_pgroups = pgroups;
    // the step's tokens by queue, for the append inside the prefill grid
    thread_local std::vector<int32_t> ftok, dtok;
    ftok.clear();
    dtok.clear();
    if ((o.flags & FNPU_PLAN_FUSED_APPEND) && pl->use_tc && !pl->use_mla && !pitems.empty()) {
        for (int32_t s = 0; s < num_seqs; ++s)
            for (int32_t i = 0; i < query_len[s]; ++i) (decode_queue(s) ? dtok : ftok).push_back(seqs[s].q_start + i);
    }
    pl->num_ftok = static_cast<int32_t>(ftok.size());
    pl->num_dtok = static_cast<int32_t>(dtok.size());
    if (pl->coloc) {
        // made once per plan and kept across re-plans (green streams above)
        int lo = 0, hi = 0;
        const bool mk_streams = !pl->s_pre;
        if ((mk_streams && cudaDeviceGetStreamPriorityRange(&lo, &hi) != cudaSuccess) ||
            (mk_streams && cudaStreamCreateWithPriority(&pl->s_pre, cudaStreamNonBlocking, hi) != cudaSuccess) ||
            (mk_streams && cudaStreamCreateWithPriority(&pl->s_dec, cudaStreamNonBlocking, lo) != cudaSuccess) ||
            (!pl->e_fork && cudaEventCreateWithFlags(&pl->e_fork, cudaEventDefault) != cudaSuccess) ||
            (!pl->e_started && cudaEventCreateWithFlags(&pl->e_started, cudaEventDisableTiming) != cudaSuccess) ||
            (!pl->e_pre && cudaEventCreateWithFlags(&pl->e_pre, cudaEventDefault) != cudaSuccess) ||
            (!pl->e_dec && cudaEventCreateWithFlags(&pl->e_dec, cudaEventDefault) != cudaSuccess)) {
            cudaGetLastError();
            return FNPU_ECUDA;
        }
    }

    // workspace: the error flag and work queues (kept across re-plans), the
    // metadata (uploaded), then scratch (never read before written)
    size_t off = 0;
    // err [0], work queues [2..5], the count of the append inside the prefill grid [6]
    const size_t o_err = off; off = align_up(off + sizeof(int32_t) * 8, 256);
    const size_t o_meta = off;
    const size_t o_seqs = off; off = align_up(off + sizeof(SeqInfo) * std::max(num_seqs, 1), 256);
    const size_t o_bt = off; off = align_up(off + sizeof(int32_t) * static_cast<size_t>(std::max(num_seqs, 1)) * width, 256);
    const size_t o_di = off; off = align_up(off + sizeof(DecodeItem) * std::max<size_t>(ditems.size(), 1), 256);
    const size_t o_mi = off; off = align_up(off + sizeof(MlaItem) * std::max<size_t>(mitems.size(), 1), 256);
    const size_t o_mg = off; off = align_up(off + sizeof(MergeGroup) * std::max<size_t>(mgroups.size(), 1), 256);
    const size_t o_pi = off; off = align_up(off + sizeof(PrefillItem) * std::max<size_t>(pitems.size(), 1), 256);
    const size_t o_cnt = off; off = align_up(off + sizeof(int32_t) * std::max(groups, 1), 256);
    const size_t o_pcnt = off; off = align_up(off + sizeof(int32_t) * 8 * static_cast<size_t>(std::max(pgroups, 1)), 256);
    const size_t o_jobs = off; off = align_up(off + sizeof(Fp8StageJob) * std::max<size_t>(jobs.size(), 1), 256);
    const size_t o_tbt = off; off = align_up(off + sizeof(int32_t) * std::max<size_t>(tbt.size(), 1), 256);
    const size_t o_ftok = off; off = align_up(off + sizeof(int32_t) * std::max<size_t>(ftok.size(), 1), 256);
    const size_t o_dtok = off; off = align_up(off + sizeof(int32_t) * std::max<size_t>(dtok.size(), 1), 256);
    const size_t meta_bytes = off;
    // query heads per partial
    const int32_t part_rows = pl->use_mla_tc ? desc->num_q_heads
                              : pl->use_mla  ? mla_heads_per_item()
                                             : (pl->use_dt ? desc->num_q_heads : G);
    const size_t o_plse = off; off = align_up(off + sizeof(float) * static_cast<size_t>(std::max(parts, 1)) * part_rows, 256);
    const size_t o_po = off; off = align_up(off + sizeof(float) * static_cast<size_t>(std::max(parts, 1)) * part_rows * desc->head_dim_v, 256);
    const size_t o_pplse = off; off = align_up(off + sizeof(float) * 256 * static_cast<size_t>(std::max(pparts, 1)), 256);
    const size_t o_ppo = off; off = align_up(off + sizeof(float) * 256 * static_cast<size_t>(std::max(pparts, 1)) * desc->head_dim_v, 256);
    // FP8 staging: f16 copies of the prefill sequences' blocks and the queries
    const size_t stage_blk = static_cast<size_t>(bs) * desc->num_kv_heads * desc->head_dim_qk * 2;
    const size_t o_tk = off; off = align_up(off + (pl->num_jobs ? stage_blk * pl->num_tblocks : 0), 256);
    const size_t o_tv = off; off = align_up(off + (pl->num_jobs ? stage_blk * pl->num_tblocks : 0), 256);
    const size_t o_tq = off;
    off = align_up(off + (pl->num_jobs ? static_cast<size_t>(T) * desc->num_q_heads * desc->head_dim_qk * 2 : 0), 256);
    pl->ws_bytes = off;

    // device workspace: allocated once, grown only when a re-plan needs more
    // (after the work already queued on the device has finished)
    int32_t carried_err = 0;
    bool fresh = false;
    if (pl->ws_bytes > pl->ws_cap) {
        const bool growing = pl->d_ws != nullptr;
        if (growing) {
            if (cudaDeviceSynchronize() != cudaSuccess ||
                cudaMemcpy(&carried_err, pl->d_ws, sizeof(int32_t), cudaMemcpyDeviceToHost) != cudaSuccess) {
                cudaGetLastError();
                return FNPU_ECUDA;
            }
            cudaFree(pl->d_ws);
            pl->d_ws = nullptr;
            pl->ws_cap = 0;
        }
        const size_t cap = growing ? pl->ws_bytes + pl->ws_bytes / 4 : pl->ws_bytes;
        if (cudaMalloc(&pl->d_ws, cap) != cudaSuccess) {
            cudaGetLastError();
            pl->d_ws = nullptr;
            return FNPU_ENOMEM;
        }
        pl->ws_cap = cap;
        fresh = true;
    }
    // pinned staging: two buffers in turn; wait (if at all) only for the
    // upload that last used this one
    const int turn = pl->stage_turn;
    if (pl->e_upload[turn] && cudaEventSynchronize(pl->e_upload[turn]) != cudaSuccess) {
        cudaGetLastError();
        return FNPU_ECUDA;
    }
    if (pl->stage_cap[turn] < meta_bytes) {
        if (pl->h_stage[turn]) cudaFreeHost(pl->h_stage[turn]);
        pl->h_stage[turn] = nullptr;
        pl->stage_cap[turn] = 0;
        const size_t cap = meta_bytes + meta_bytes / 4;
        if (cudaMallocHost(&pl->h_stage[turn], cap) != cudaSuccess) {
            cudaGetLastError();
            pl->h_stage[turn] = nullptr;
            return FNPU_ENOMEM;
        }
        pl->stage_cap[turn] = cap;
    }
    if (!pl->e_upload[turn] && cudaEventCreateWithFlags(&pl->e_upload[turn], cudaEventDisableTiming) != cudaSuccess) {
        cudaGetLastError();
        return FNPU_ECUDA;
    }
    uint8_t *h = static_cast<uint8_t *>(pl->h_stage[turn]);
    // only the error flag and work queues and the merge counters must start at
    // zero; every other region is written below where a kernel reads it (the
    // block-table columns past a sequence's blocks are never read)
    memset(h + o_err, 0, o_meta - o_err);
    memset(h + o_cnt, 0, o_jobs - o_cnt);
    reinterpret_cast<int32_t *>(h + o_err)[0] = carried_err;
    if (num_seqs) memcpy(h + o_seqs, seqs.data(), sizeof(SeqInfo) * num_seqs);
    for (int32_t s = 0; s < num_seqs; ++s)
        memcpy(h + o_bt + sizeof(int32_t) * static_cast<size_t>(s) * width,
               block_table + static_cast<int64_t>(s) * block_table_stride,
               sizeof(int32_t) * static_cast<size_t>((context_len[s] + bs - 1) / bs));
    {
        DecodeItem *dst = reinterpret_cast<DecodeItem *>(h + o_di);
        for (size_t i = 0; i < dorder.size(); ++i) dst[i] = ditems[static_cast<size_t>(dorder[i])];
    }
    if (!mitems.empty()) memcpy(h + o_mi, mitems.data(), sizeof(MlaItem) * mitems.size());
    if (!mgroups.empty()) memcpy(h + o_mg, mgroups.data(), sizeof(MergeGroup) * mgroups.size());
    if (!jobs.empty()) memcpy(h + o_jobs, jobs.data(), sizeof(Fp8StageJob) * jobs.size());
    if (!tbt.empty()) memcpy(h + o_tbt, tbt.data(), sizeof(int32_t) * tbt.size());
    if (!ftok.empty()) memcpy(h + o_ftok, ftok.data(), sizeof(int32_t) * ftok.size());
    if (!dtok.empty()) memcpy(h + o_dtok, dtok.data(), sizeof(int32_t) * dtok.size());
    {
        PrefillItem *dst = reinterpret_cast<PrefillItem *>(h + o_pi);
        for (size_t i = 0; i < porder.size(); ++i) dst[i] = pitems[static_cast<size_t>(porder[i])];
    }

    uint8_t *d = static_cast<uint8_t *>(pl->d_ws);
    pl->d_seqs = reinterpret_cast<SeqInfo *>(d + o_seqs);
    pl->d_bt = reinterpret_cast<int32_t *>(d + o_bt);
    pl->d_ditems = reinterpret_cast<DecodeItem *>(d + o_di);
    pl->d_mitems = reinterpret_cast<MlaItem *>(d + o_mi);
    pl->d_mgroups = reinterpret_cast<MergeGroup *>(d + o_mg);
    pl->d_pitems = reinterpret_cast<PrefillItem *>(d + o_pi);
    pl->d_counters = reinterpret_cast<int32_t *>(d + o_cnt);
    pl->d_err = reinterpret_cast<int32_t *>(d + o_err);
    pl->d_part_lse = reinterpret_cast<float *>(d + o_plse);
    pl->d_part_o = reinterpret_cast<float *>(d + o_po);
    pl->d_pcounters = reinterpret_cast<int32_t *>(d + o_pcnt);
    pl->d_ppart_lse = reinterpret_cast<float *>(d + o_pplse);
    pl->d_ppart_o = reinterpret_cast<float *>(d + o_ppo);
    pl->d_jobs = reinterpret_cast<Fp8StageJob *>(d + o_jobs);
    pl->d_tbt = reinterpret_cast<int32_t *>(d + o_tbt);
    pl->d_ftok = reinterpret_cast<int32_t *>(d + o_ftok);
    pl->d_dtok = reinterpret_cast<int32_t *>(d + o_dtok);
    pl->d_tk = d + o_tk;
    pl->d_tv = d + o_tv;
    pl->d_tq = d + o_tq;
    // a fresh workspace gets its error flag and queues (zero) with the
    // metadata; a reused one keeps them (the queues are zero between runs)
    const size_t up0 = fresh ? o_err : o_meta;
    cudaStream_t cs = static_cast<cudaStream_t>(stream);
    if (cudaMemcpyAsync(d + up0, h + up0, meta_bytes - up0, cudaMemcpyHostToDevice, cs) != cudaSuccess ||
        cudaEventRecord(pl->e_upload[turn], cs) != cudaSuccess) {
        cudaGetLastError();
        return FNPU_ECUDA;
    }
    pl->stage_turn = turn ^ 1;
    return FNPU_OK;
}

}  // namespace

extern "C" {

int fnpu_mixed_attn_plan_ex(const fnpu_attn_desc *desc, int32_t num_seqs, const int32_t *query_len,
                            const int32_t *context_len, const uint8_t *phase,
                            const int32_t *block_table, int32_t block_table_stride,
                            const fnpu_plan_opts *opts, void *stream, fnpu_plan **out) {
    if (!out) return FNPU_EINVAL;
    fnpu_plan_opts o = {};
    if (opts) o = *opts;
    StepMeta m;
    int rc = validate_meta(desc, num_seqs, query_len, context_len, phase, block_table, block_table_stride, o, &m);
    if (rc != FNPU_OK) return rc;
    int sms = 0;
    rc = plan_sms(o, &sms);
    if (rc != FNPU_OK) return rc;
    fnpu_plan *pl = new (std::nothrow) fnpu_plan();
    if (!pl) return FNPU_ENOMEM;
    rc = plan_fill(pl, desc, num_seqs, query_len, context_len, phase, block_table, block_table_stride, o, m, sms,
                   stream);
    if (rc != FNPU_OK) {
        release_plan(pl);
        delete pl;
        return rc;
    }
    *out = pl;
    return FNPU_OK;
}

int fnpu_mixed_attn_replan(fnpu_plan *pl, int32_t num_seqs, const int32_t *query_len, const int32_t *context_len,
                           const uint8_t *phase, const int32_t *block_table, int32_t block_table_stride,
                           const fnpu_plan_opts *opts, void *stream) {
    if (!pl) return FNPU_EINVAL;
    fnpu_plan_opts o = {};
    if (opts) o = *opts;
    StepMeta m;
    int rc = validate_meta(&pl->desc, num_seqs, query_len, context_len, phase, block_table, block_table_stride, o,
                           &m);
    if (rc != FNPU_OK) return rc;  // the plan is unchanged
    int sms = 0;
    rc = plan_sms(o, &sms);
    if (rc != FNPU_OK) return rc;
    const fnpu_attn_desc desc = pl->desc;
    return plan_fill(pl, &desc, num_seqs, query_len, context_len, phase, block_table, block_table_stride, o, m, sms,
                     stream);
}

}  // extern "C"

namespace fnpu {
namespace {

// The kernels' arguments for one run of a plan (pointers checked by the caller).
AttnParams run_params(const fnpu_plan *pl, const void *q, const void *k_cache, const void *v_cache, void *out,
                      float *lse) {
    const bool latent = pl->desc.v_in_k_latent != 0;
    AttnParams p = {};
    const fnpu_attn_desc &d = pl->desc;
    p.q = q;
    p.k_cache = k_cache;
    p.v_cache = latent ? k_cache : v_cache;
    p.out = out;
    p.lse = lse;
    p.seqs = pl->d_seqs;
    p.block_table = pl->d_bt;
    p.bt_stride = pl->bt_width;
    p.num_q_heads = d.num_q_heads;
    p.num_kv_heads = d.num_kv_heads;
    p.group = d.num_q_heads / d.num_kv_heads;
    p.block_size = d.block_size;
    p.num_blocks = d.num_blocks;
    p.num_tokens = pl->num_tokens;
    p.head_dim_qk = d.head_dim_qk;
    p.head_dim_v = d.head_dim_v;
    p.k_slot_stride = latent ? d.head_dim_qk : static_cast<int64_t>(d.num_kv_heads) * d.head_dim_qk;
    p.v_slot_stride = latent ? d.head_dim_qk : static_cast<int64_t>(d.num_kv_heads) * d.head_dim_v;
    p.scale_log2 = pl->scale * 1.4426950408889634f;
    p.ditems = pl->d_ditems;
    p.mitems = pl->d_mitems;
    p.mgroups = pl->d_mgroups;
    p.num_mgroups = pl->num_mgroups;
    p.num_mitems = pl->num_mitems;
    p.num_ditems = pl->num_ditems;
    p.part_o = pl->d_part_o;
    p.part_lse = pl->d_part_lse;
    p.counters = pl->d_counters;
    p.pitems = pl->d_pitems;
    p.num_pitems = pl->num_pitems;
    p.ppart_o = pl->d_ppart_o;
    p.ppart_lse = pl->d_ppart_lse;
    p.pcounters = pl->d_pcounters;
    p.err = pl->d_err;
    p.sched = pl->d_err + 2;
    return p;
}

bool run_pointers_ok(const fnpu_plan *pl, const void *q, const void *k_cache, const void *v_cache, const void *out,
                     const float *lse) {
    const bool latent = pl->desc.v_in_k_latent != 0;
    if (!q || !k_cache || !out || !lse || (!latent && !v_cache)) return false;
    const uintptr_t mis = reinterpret_cast<uintptr_t>(q) | reinterpret_cast<uintptr_t>(k_cache) |
                          reinterpret_cast<uintptr_t>(out) | reinterpret_cast<uintptr_t>(lse) |
                          (latent ? 0 : reinterpret_cast<uintptr_t>(v_cache));
    return (mis & 15u) == 0;
}

// The decode kernel of a plan and its merge, on `stream`.
int launch_decode(const fnpu_plan *pl, const AttnParams &p, void *stream, int ctas) {
    return pl->desc.kv_fp8 ? launch_decode_fp8(p, stream, ctas) : launch_decode_tma(p, stream, ctas);
}

// Both phases side by side: pre_ctas persistent prefill CTAs (one per SM, the
// tensor pipe; a decode CTA does not fit beside one) and decode CTAs on the
// other SMs (HBM). The decode stream waits for the event that fires once
// every prefill CTA has begun, so the decode grid only takes the SMs left
// over: with both grids pending at once the hardware may place either first,
// and stream priority alone does not settle it. Decode CTAs beyond the free
// SMs start on the SMs that the prefill leaves as its queue runs dry; the
// decode merge follows the decode grid on its stream, beside the prefill.
int run_colocated(const fnpu_plan *pl, const AttnParams &p, void *stream) {
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const bool green = pl->g_pre != nullptr;  // partitions enforced: no placement order to keep
    FNPU_CUDA_TRY(cudaEventRecord(pl->e_fork, s));
    if (!green) {
        // The prefill grid goes on the caller's stream (a fork to a library
        // stream costs the wait across streams before it starts), as a
        // programmatic dependent of the kernel before it (the step's append):
        // its CTAs take their SMs and set up while that kernel drains. The
        // decode stream waits for the fork (everything before the prefill is
        // done) and for the prefill grid's launch-completion event. (Over the
        // FP8 cache the staging kernel comes before the prefill, which is then
        // an ordinary launch: as the staging's dependent, the prefill's
        // launch-completion event held the decode back by some 65 us.)
        FNPU_CUDA_TRY(cudaStreamWaitEvent(pl->s_dec, pl->e_fork, 0));
        int rc = launch_prefill(pl, p, s, pl->pre_ctas, pl->e_started, !pl->desc.kv_fp8);
        if (rc == FNPU_OK) {
            FNPU_CUDA_TRY(cudaStreamWaitEvent(pl->s_dec, pl->e_started, 0));
            rc = launch_decode(pl, p, pl->s_dec, 3 * pl->num_sms);
        }
        FNPU_CUDA_TRY(cudaEventRecord(pl->e_pre, s));
        FNPU_CUDA_TRY(cudaEventRecord(pl->e_dec, pl->s_dec));
        FNPU_CUDA_TRY(cudaStreamWaitEvent(s, pl->e_dec, 0));
        return rc;
    }
    // green contexts: each phase on its partition's stream, both from the fork
    FNPU_CUDA_TRY(cudaStreamWaitEvent(pl->s_pre, pl->e_fork, 0));
    int rc = launch_prefill(pl, p, pl->s_pre, pl->pre_ctas, nullptr);
    if (rc == FNPU_OK) {
        FNPU_CUDA_TRY(cudaStreamWaitEvent(pl->s_dec, pl->e_fork, 0));
        rc = launch_decode(pl, p, pl->s_dec, 3 * pl->dec_sms);
    }
    FNPU_CUDA_TRY(cudaEventRecord(pl->e_pre, pl->s_pre));
    FNPU_CUDA_TRY(cudaEventRecord(pl->e_dec, pl->s_dec));
    FNPU_CUDA_TRY(cudaStreamWaitEvent(s, pl->e_pre, 0));
    FNPU_CUDA_TRY(cudaStreamWaitEvent(s, pl->e_dec, 0));
    return rc;
}

// A whole step whose tcgen05 prefill grid appends the prefill-path rows
// itself (p.fa_*): the decode rows go in by a small kernel ahead of the
// decode kernel, on the decode's stream. Co-located: the prefill grid on the
// caller's stream, the decode stream after the fork and the prefill grid's
// launch, as in run_colocated. Otherwise the phases one after the other.
int run_step_fused(const fnpu_plan *pl, const AttnParams &p, const void *k_new, const void *v_new,
                   const int64_t *slots, void *k_cache, void *v_cache, void *stream) {
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (pl->coloc) {
        FNPU_CUDA_TRY(cudaEventRecord(pl->e_fork, s));
        FNPU_CUDA_TRY(cudaStreamWaitEvent(pl->s_dec, pl->e_fork, 0));
        int rc = launch_prefill(pl, p, s, pl->pre_ctas, pl->e_started, false);
        if (rc == FNPU_OK) {
            FNPU_CUDA_TRY(cudaStreamWaitEvent(pl->s_dec, pl->e_started, 0));
            rc = launch_kv_append_list(&pl->desc, k_new, v_new, slots, pl->d_dtok, pl->num_dtok, k_cache, v_cache,
                                       pl->s_dec);
        }
        if (rc == FNPU_OK) rc = launch_decode(pl, p, pl->s_dec, 3 * pl->num_sms);
        FNPU_CUDA_TRY(cudaEventRecord(pl->e_pre, s));
        FNPU_CUDA_TRY(cudaEventRecord(pl->e_dec, pl->s_dec));
        FNPU_CUDA_TRY(cudaStreamWaitEvent(s, pl->e_dec, 0));
        return rc;
    }
    int rc = launch_kv_append_list(&pl->desc, k_new, v_new, slots, pl->d_dtok, pl->num_dtok, k_cache, v_cache, s);
    if (rc == FNPU_OK && pl->num_ditems > 0)
        rc = pl->use_dt ? launch_decode_tma(p, stream, 3 * pl->num_sms) : launch_decode_mma(p, stream);
    if (rc != FNPU_OK) return rc;
    return launch_prefill(pl, p, stream, pl->num_sms, nullptr, false);
}

}  // namespace
}  // namespace fnpu

extern "C" {

int fnpu_mixed_attn_run(const fnpu_plan *pl, const void *q, const void *k_cache, const void *v_cache,
                        void *out, float *lse, void *stream) {
    if (!pl) return FNPU_EINVAL;
    if (pl->num_tokens == 0) return FNPU_OK;
    if (!run_pointers_ok(pl, q, k_cache, v_cache, out, lse)) return FNPU_EINVAL;
    const AttnParams p = run_params(pl, q, k_cache, v_cache, out, lse);
    if (pl->use_mla) return pl->use_mla_tc ? launch_mla_tc(p, stream) : launch_mla(p, stream);
    if (pl->coloc) return run_colocated(pl, p, stream);
    int rc = pl->desc.kv_fp8 ? launch_decode_fp8(p, stream, 3 * pl->num_sms)
             : pl->use_dt    ? launch_decode_tma(p, stream, 3 * pl->num_sms)
                             : launch_decode_mma(p, stream);
    if (rc != FNPU_OK) return rc;
    if (pl->use_tc) return launch_prefill(pl, p, stream, pl->num_sms, nullptr, true);
    return pl->desc.kv_fp8 ? launch_prefill_fp8(p, stream) : launch_prefill_mma(p, stream);
}

int fnpu_mixed_step(const fnpu_plan *pl, const void *k_new, const void *v_new, const int64_t *slot_mapping,
                    const void *q, void *k_cache, void *v_cache, void *out, float *lse, void *stream) {
    if (!pl) return FNPU_EINVAL;
    if (pl->num_tokens == 0) return FNPU_OK;
    const bool latent = pl->desc.v_in_k_latent != 0;
    if (!k_new || !slot_mapping || (!latent && !v_new)) return FNPU_EINVAL;
    if (((reinterpret_cast<uintptr_t>(k_new) | (latent ? 0 : reinterpret_cast<uintptr_t>(v_new))) & 15u) ||
        (reinterpret_cast<uintptr_t>(slot_mapping) & 7u))
        return FNPU_EINVAL;
    if (!run_pointers_ok(pl, q, k_cache, v_cache, out, lse)) return FNPU_EINVAL;
    const int32_t n = static_cast<int32_t>(pl->num_tokens);
    // the prefill grid takes the prefill rows where the plan asks for it and
    // the prefill is the tcgen05 kernel over a bf16 cache (green-context
    // plans keep the two calls)
    const bool fused = (pl->flags & FNPU_PLAN_FUSED_APPEND) && pl->use_tc && !pl->use_mla && !pl->desc.kv_fp8 &&
                       pl->num_ftok > 0 && !pl->g_pre;
    if (!fused) {
        const int rc = fnpu_kv_append(&pl->desc, k_new, v_new, slot_mapping, n, k_cache, v_cache, stream);
        if (rc != FNPU_OK) return rc;
        return fnpu_mixed_attn_run(pl, q, k_cache, v_cache, out, lse, stream);
    }
    AttnParams p = run_params(pl, q, k_cache, v_cache, out, lse);
    int *range_err = nullptr;
    const int rc = global_error_address(&range_err);
    if (rc != FNPU_OK) return rc;
    p.fa_k_new = static_cast<const uint4 *>(k_new);
    p.fa_v_new = static_cast<const uint4 *>(v_new);
    p.fa_slots = slot_mapping;
    p.fa_tokens = pl->d_ftok;
    p.fa_k_cache = static_cast<uint4 *>(k_cache);
    p.fa_v_cache = static_cast<uint4 *>(v_cache);
    p.fa_count = pl->d_err + 6;  // zero between runs (the last CTA out resets it)
    p.fa_range_err = range_err;
    p.fa_num_tokens = pl->num_ftok;
    p.fa_k_chunks = static_cast<int32_t>(static_cast<int64_t>(pl->desc.num_kv_heads) * pl->desc.head_dim_qk * 2 / 16);
    p.fa_v_chunks = static_cast<int32_t>(static_cast<int64_t>(pl->desc.num_kv_heads) * pl->desc.head_dim_v * 2 / 16);
    p.fa_num_slots = static_cast<int64_t>(pl->desc.num_blocks) * pl->desc.block_size;
    return run_step_fused(pl, p, k_new, v_new, slot_mapping, k_cache, v_cache, stream);
}

int fnpu_plan_check(const fnpu_plan *pl, void *stream) {
    if (!pl) return FNPU_EINVAL;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(s) != cudaSuccess) return FNPU_ECUDA;
    int32_t v = 0;
    if (cudaMemcpy(&v, pl->d_err, sizeof(v), cudaMemcpyDeviceToHost) != cudaSuccess) return FNPU_ECUDA;
    if (v != 0) {
        const int32_t zero[8] = {0, 0, 0, 0, 0, 0, 0, 0};  // also resets the persistent work queues
        if (cudaMemcpy(pl->d_err, zero, sizeof(zero), cudaMemcpyHostToDevice) != cudaSuccess)
            return FNPU_ECUDA;
        // an aborted run can leave split-merge counters behind
        if (cudaMemset(pl->d_counters, 0, sizeof(int32_t) * std::max(pl->num_groups, 1)) != cudaSuccess ||
            cudaMemset(pl->d_pcounters, 0, sizeof(int32_t) * 8 * std::max(pl->num_pgroups, 1)) != cudaSuccess ||
            cudaDeviceSynchronize() != cudaSuccess)
            return FNPU_ECUDA;
        return FNPU_EDEVICE_TIMEOUT;
    }
    return FNPU_OK;
}

void fnpu_plan_destroy(fnpu_plan *pl) {
    if (!pl) return;
    cudaDeviceSynchronize();
    release_plan(pl);
    delete pl;
}

int fnpu_plan_info(const fnpu_plan *pl, int32_t *prefill_items, int32_t *decode_items,
                   int32_t *launches_per_run, int64_t *workspace_bytes) {
    if (!pl) return FNPU_EINVAL;
    // latent attention has one work list for both phases, reported as prefill items
    if (prefill_items) *prefill_items = pl->num_pitems + pl->num_mitems;
    if (decode_items) *decode_items = pl->num_ditems;
    if (launches_per_run)
        *launches_per_run = (pl->num_pitems > 0) + (pl->num_ditems > 0) + (pl->num_mitems > 0) + (pl->num_mgroups > 0) +
                            (pl->num_jobs > 0 ? 1 : 0);  // FP8 staging: blocks and queries to f16
    if (workspace_bytes) *workspace_bytes = static_cast<int64_t>(pl->ws_cap);
    return FNPU_OK;
}

// The decode share of a co-located plan, as a rounded percent of the SMs.
int fnpu_plan_decode_share(const fnpu_plan *pl, int32_t *share_pct) {
    if (!pl || !share_pct) return FNPU_EINVAL;
    if (!pl->coloc || pl->num_sms <= 0) return FNPU_EUNSUPPORTED;
    const int32_t k = pl->num_sms - pl->pre_ctas;
    *share_pct = std::max<int32_t>(1, (200 * k + pl->num_sms) / (2 * pl->num_sms));  // rounded percent
    return FNPU_OK;
}

// Phase times of the last co-located run: the fork, prefill-end and
// decode-end events of the plan's two streams carry device timestamps.
int fnpu_plan_phase_ms(const fnpu_plan *pl, float *prefill_ms, float *decode_ms) {
    if (!pl || !prefill_ms || !decode_ms) return FNPU_EINVAL;
    if (!pl->coloc) return FNPU_EUNSUPPORTED;
    if (cudaEventSynchronize(pl->e_pre) != cudaSuccess || cudaEventSynchronize(pl->e_dec) != cudaSuccess)
        return cuda_fail(cudaGetLastError(), "cudaEventSynchronize (phase times)");
    float a = 0.f, b = 0.f;
    if (cudaEventElapsedTime(&a, pl->e_fork, pl->e_pre) != cudaSuccess ||
        cudaEventElapsedTime(&b, pl->e_fork, pl->e_dec) != cudaSuccess) {
        cudaGetLastError();  // no run of this plan has been recorded yet
        return FNPU_EINVAL;
    }
    *prefill_ms = a;
    *decode_ms = b;
    return FNPU_OK;
}

// Dispatch-ratio feedback (Sec. 3.4): while each phase holds its own SMs,
// decode time goes about as 1 / s and prefill time as 1 / (1 - s) for a
// decode share s of the SMs, so times d and p measured at share s give
// D = d s and P = p (1 - s), and both phases would end together at
// s* = D / (D + P). The next share moves halfway there (a damped step, as the
// prefill time is a step function of its SM count), at least one point while
// s* is a point or more away, and stays within [1, 50] percent.
int fnpu_dispatch_next_share(int32_t share_pct, float prefill_ms, float decode_ms, float tolerance,
                             int32_t *next_share_pct) {
    if (!next_share_pct || share_pct < 1 || share_pct > 99 || !(prefill_ms > 0.f) || !(decode_ms > 0.f) ||
        !(tolerance >= 0.f))
        return FNPU_EINVAL;
    auto clamp = [](int32_t v) { return std::min<int32_t>(50, std::max<int32_t>(1, v)); };
    const double p = prefill_ms, d = decode_ms;
    if (std::fabs(d - p) <= tolerance * std::max(d, p)) {
        *next_share_pct = clamp(share_pct);
        return FNPU_OK;
    }
    const double s = share_pct / 100.0;
    const double dd = d * s, pp = p * (1.0 - s);
    const double target = dd / (dd + pp);
    int32_t next = static_cast<int32_t>(std::lround(100.0 * (s + 0.5 * (target - s))));
    if (next == share_pct && std::fabs(100.0 * target - share_pct) >= 1.0) next += d > p ? 1 : -1;
    *next_share_pct = clamp(next);
    return FNPU_OK;
}

}  // extern "C"
