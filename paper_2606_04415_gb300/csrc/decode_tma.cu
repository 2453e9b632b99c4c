// Decode split-KV attention fed by TMA through an mbarrier ring
// (Hkv = 4 kv heads, d = 64 or 128, G <= 8 query heads per kv head, block
// size a multiple of 16).
//
// Decode is bound by KV-cache reads (Sec. 1, Sec. 3.3, Fig. 2). The kernel is
// kept small -- five warps, at most 128 registers a thread, 64 KB of shared
// memory for d = 128 -- so that three CTAs share an SM and a few SMs alone
// can stream decode work while the others run prefill (Sec. 3.4).
//   * Persistent CTAs take items -- a sequence's key range, longest first --
//     CTA b item b first, then from an atomic queue one item ahead of use (the
//     last CTA out resets it); the next item's descriptor, block ids and
//     query are loaded during the current item, so an item boundary costs no
//     memory round trip, and a descriptor carries the item's query token,
//     block-table row and first four block ids, so that a CTA issues its
//     first copies one load after it starts. (Taking two items ahead left
//     CTAs idle when items were few: the first CTAs reserved them all.)
//   * A 2-stage ring of 16-key stages holds K and V of all four kv heads. A
//     producer warp issues the TMA copies (four boxes of 16 slots x 4 heads x
//     64 columns for d = 128) as soon as a stage is free; issuing them from a
//     compute warp cost that warp about as much as its arithmetic. The tensor map
//     lists the slot dimension before the kv-head dimension, so a box lands
//     head-major (16 consecutive slots of one head form 16 rows) and the
//     128-byte swizzle is keyed by the slot: ldmatrix over eight consecutive
//     slots of one head is conflict-free.
//   * Each warp owns one kv head and runs the GQA-packed mma.sync scheme
//     (S^T = K Q^T with the 16 keys in M and the G query heads in N; P^T by
//     movmatrix; O^T += V^T P^T), releasing a stage with one mbarrier arrival.
//   * V rows past the item's keys are zeroed by their warp before the PV
//     product, so stale slots never reach it.
//   * A split writes its partial result (Eq. 1 restricted to its keys, with
//     its log-sum-exp); a second small kernel merges the splits of every
//     sequence, one warp per (token, query head), all in parallel. Merging in
//     the last split instead took one dependent round trip per two splits and
//     capped the splits per sequence, and with few splits the items were too
//     coarse to share the bandwidth evenly among the CTAs.
// Every mbarrier wait is bounded and raises the plan's error flag on timeout.
#include <math.h>

#include "common.cuh"
#include "tc.cuh"

namespace fnpu {
namespace {

constexpr int kHkv = 4;
constexpr int kKeys = 16;        // keys per stage
constexpr int kStages = 2;
constexpr int kWarps = 4;        // compute warps, one per kv head
constexpr int kThreads = 32 * (kWarps + 1);  // + the TMA producer warp
constexpr int kHalfBytes = kHkv * kKeys * 128;  // all heads, one 64-column half

template <int D>
struct DtCfg {
    static constexpr int kTileBytes = (D / 64) * kHalfBytes;  // K or V of one stage
    static constexpr int kStageBytes = 2 * kTileBytes;
    static constexpr int kBarOff = kStages * kStageBytes;
    // full[S] empty[S]
    static constexpr int kNumBars = 2 * kStages;
    // + item ring [4] and the abort flag
    static constexpr int kSmemBytes = kBarOff + 8 * kNumBars + 32;
};

struct DtMaps {
    CUtensorMap k, v;
};

// shared-memory offset of (slot, kv head, 16-byte chunk) inside a K or V tile
__device__ __forceinline__ uint32_t dt_off(int slot, int head, int chunk) {
    return static_cast<uint32_t>((chunk >> 3) * kHalfBytes + (head * kKeys + slot) * 128 +
                                 (((chunk & 7) ^ (slot & 7)) << 4));
}

// What a warp keeps of one item.
struct DtGeo {
    int t;          // query token
    int bt_row;
    int kb, ke;     // keys [kb, ke)
    int split, ns, part_base, group;
    int b0, b1, b2, b3;  // ids of the item's first four blocks
};

template <int D>
__device__ __forceinline__ void load_q(const AttnParams &p, int t, int head, int g8, int c,
                                       uint32_t (&qb)[D / 16][2]) {
    const __nv_bfloat16 *qrow = static_cast<const __nv_bfloat16 *>(p.q) +
                                (static_cast<int64_t>(t) * p.num_q_heads + head * p.group) * D;
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
        if (g8 < p.group) {
            qb[kk][0] = __ldg(reinterpret_cast<const uint32_t *>(qrow + g8 * D + kk * 16 + 2 * c));
            qb[kk][1] = __ldg(reinterpret_cast<const uint32_t *>(qrow + g8 * D + kk * 16 + 8 + 2 * c));
        } else {
            qb[kk][0] = qb[kk][1] = 0u;
        }
    }
}

// block ids of the item's blocks, relative block `lane` in lane `lane`
__device__ __forceinline__ int load_blk_lane(const AttnParams &p, const DtGeo &g, int lane) {
    const int b0 = g.kb / p.block_size;
    const int nblk = (g.ke - 1) / p.block_size - b0 + 1;
    return lane < nblk ? __ldg(p.block_table + static_cast<int64_t>(g.bt_row) * p.bt_stride + b0 + lane) : 0;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 3)
    decode_tma_kernel(const AttnParams p, const __grid_constant__ DtMaps maps) {
    using Cfg = DtCfg<D>;
    extern __shared__ __align__(1024) uint8_t smem[];
    const uint32_t s_base = smem_u32(smem);
    const uint32_t s_bars = s_base + Cfg::kBarOff;
    auto FULL = [&](int s) { return s_bars + 8 * s; };
    auto EMPTY = [&](int s) { return s_bars + 8 * (kStages + s); };
    int *ring = reinterpret_cast<int *>(smem + Cfg::kBarOff + 8 * Cfg::kNumBars);  // [4]
    volatile int *abort_flag = ring + 4;
    int *sched = p.sched + 2;  // this kernel's work queue: next item, finished CTAs

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n_items = p.num_ditems;
    pdl_trigger();  // the merge grid may be placed once these CTAs are; it waits for them to finish
    if ((s_base & 1023u) != 0) {  // the swizzled tiles need 1024-byte alignment
        if (tid == 0) atomicOr(p.err, 2);
        return;
    }
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(FULL(s), 1);
            tc::mbar_init(EMPTY(s), kWarps);
        }
        ring[0] = blockIdx.x;  // the first item without the queue (grid <= items); the queue serves the rest
        *abort_flag = 0;
        tc::fence_mbar_init();
    }
    if (warp == kWarps && lane == 0) {
        tc::prefetch_tmap(&maps.k);
        tc::prefetch_tmap(&maps.v);
    }
    __syncthreads();

    auto wait = [&](uint32_t bar, uint32_t parity) -> bool {
        if (tc::mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if (tc::mbar_wait(bar, parity)) return true;
        *abort_flag = 1;
        atomicOr(p.err, 1);
        return false;
    };
    auto geo_of = [&](const DecodeItem &it) {
        DtGeo g;
        g.t = it.q_start;
        g.bt_row = it.bt_row;
        g.b0 = it.blk[0];
        g.b1 = it.blk[1];
        g.b2 = it.blk[2];
        g.b3 = it.blk[3];
        g.kb = it.key_begin;
        g.ke = it.key_end;
        g.split = it.split;
        g.ns = it.num_splits;
        g.part_base = it.part_base;
        g.group = it.group;
        return g;
    };

    const int head = warp;
    const int g8 = lane >> 2, c = lane & 3;
    const int lj = lane >> 3, lr = lane & 7;
    const int G = p.group;
    const int Hq = p.num_q_heads;
    const int bs = p.block_size;
    __nv_bfloat16 *out = static_cast<__nv_bfloat16 *>(p.out);

    // issue stage `j` of item `g` into ring position `gs` (producer warp, whole warp)
    auto issue = [&](const DtGeo &g, int j, int blk_lane, int gs) -> bool {
        const int st = gs % kStages;
        if (gs >= kStages && !wait(EMPTY(st), ((gs / kStages) - 1) & 1)) return false;
        const int key0 = g.kb + j * kKeys;
        const int rel = key0 / bs - g.kb / bs;  // warp-uniform
        int blk;
        if (rel < 4) {  // from the item itself: the lanes' block-id loads may still be in flight
            blk = rel == 0 ? g.b0 : rel == 1 ? g.b1 : rel == 2 ? g.b2 : g.b3;
        } else {
            blk = __shfl_sync(0xffffffffu, blk_lane, rel & 31);
            if (rel >= 32) blk = __ldg(p.block_table + static_cast<int64_t>(g.bt_row) * p.bt_stride + key0 / bs);
        }
        const uint32_t sK = s_base + st * Cfg::kStageBytes, sV = sK + Cfg::kTileBytes;
        tc::mbar_arrive_expect_tx_warp(FULL(st), Cfg::kStageBytes);
#pragma unroll
        for (int h = 0; h < D / 64; ++h) {
            tc::tma_load_4d_warp(sK + h * kHalfBytes, &maps.k, FULL(st), h * 64, key0 % bs, 0, blk);
            tc::tma_load_4d_warp(sV + h * kHalfBytes, &maps.v, FULL(st), h * 64, key0 % bs, 0, blk);
        }
        return true;
    };

    if (warp == kWarps) {
        // ---------------------------------------------------- TMA producer
        // Runs up to kStages stages ahead of the compute warps. It takes the
        // next item from the queue at the start of the current one (one item
        // ahead, so that the queue still balances the CTAs), publishes its
        // index in the item ring before it issues stage 2 of the current item
        // (the compute warps read it after that stage has landed), and loads
        // the next item's descriptor, then a stage later its block ids, so
        // that no dependent memory round trip sits between stages. An item's
        // first four blocks come with its descriptor.
        int gs = 0;
        bool ok = true;
        int idx = ring[0];
        DecodeItem it{};
        if (idx < n_items) it = p.ditems[idx];
        DtGeo cur = geo_of(it);
        int blk_lane = idx < n_items ? load_blk_lane(p, cur, lane) : 0;
        for (int k = 0; ok && idx < n_items; ++k) {
            int a = 0;
            if (lane == 0) a = static_cast<int>(gridDim.x) + atomicAdd(sched, 1);  // the next item
            const int ntiles = (cur.ke - cur.kb + kKeys - 1) / kKeys;
            const int spub = ntiles > 2 ? 2 : ntiles - 1;
            const int s1 = spub + 1 < ntiles ? spub + 1 : spub;
            int idx_n = n_items;
            DecodeItem nit{};
            DtGeo nxt{};
            int blk_lane_n = 0;
            for (int i = 0; i < ntiles; ++i, ++gs) {
                if (i == spub) {
                    idx_n = __shfl_sync(0xffffffffu, a, 0);
                    if (lane == 0) *reinterpret_cast<volatile int *>(ring + ((k + 1) & 3)) = idx_n;
                    __syncwarp();  // before the arrival of this stage, which releases it
                    if (idx_n < n_items) nit = p.ditems[idx_n];
                }
                if (!issue(cur, i, blk_lane, gs)) { ok = false; break; }
                if (idx_n < n_items && i == s1) {
                    nxt = geo_of(nit);
                    blk_lane_n = load_blk_lane(p, nxt, lane);
                }
            }
            if (!ok) break;
            idx = idx_n;
            cur = nxt;
            blk_lane = blk_lane_n;
        }
    } else if (ring[0] < n_items) {
        int idx = ring[0];
        DtGeo cur;
        {
            cur = geo_of(p.ditems[idx]);
        }
        uint32_t qb[D / 16][2];
        load_q<D>(p, cur.t, head, g8, c, qb);
        bool ok = true;
        int g = 0;  // ring position of the current item's first stage
        for (int k = 0; ok; ++k) {
            const int ntiles = (cur.ke - cur.kb + kKeys - 1) / kKeys;
            const int spub = ntiles > 2 ? 2 : ntiles - 1;  // the stage after which the next index is readable
            int idx_n = n_items;
            bool has_next = false;
            DecodeItem nit{};
            DtGeo nxt{};
            uint32_t qn[D / 16][2];

            float o[D / 16][4];
#pragma unroll
            for (int mt = 0; mt < D / 16; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
            float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
            const int nkeys = cur.ke - cur.kb;
            for (int i = 0; i < ntiles; ++i) {
                const int gs = g + i;
                const int st = gs % kStages;
                if (!wait(FULL(st), (gs / kStages) & 1)) { ok = false; break; }
                if (i == spub) {  // the producer published it before issuing this stage
                    idx_n = *reinterpret_cast<volatile int *>(ring + ((k + 1) & 3));
                    has_next = idx_n < n_items;
                    if (has_next) nit = p.ditems[idx_n];
                }
                const uint32_t sK = s_base + st * Cfg::kStageBytes, sV = sK + Cfg::kTileBytes;
                const int nv = nkeys - i * kKeys;  // valid keys in this stage (>= 1)
                const bool tail = nv < kKeys;
                if (tail) {  // zero this head's V rows past the item's keys
                    for (int e = lane; e < (kKeys - nv) * 8 * (D / 64); e += 32) {
                        const int hh = e / ((kKeys - nv) * 8), rem = e % ((kKeys - nv) * 8);
                        const int sl = nv + rem / 8, ch = rem % 8;
                        *reinterpret_cast<uint4 *>(smem + st * Cfg::kStageBytes + Cfg::kTileBytes + hh * kHalfBytes +
                                                   (head * kKeys + sl) * 128 + ch * 16) = make_uint4(0u, 0u, 0u, 0u);
                    }
                    __syncwarp();
                }
                float s[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    uint32_t a0, a1, a2, a3;
                    ldmatrix_x4(a0, a1, a2, a3, sK + dt_off(lr + 8 * (lj & 1), head, 2 * kk + (lj >> 1)));
                    mma_bf16_16816(s, a0, a1, a2, a3, qb[kk][0], qb[kk][1]);
                }
                const bool v0 = g8 < nv, v1 = g8 + 8 < nv;
                const float x0 = v0 ? s[0] * p.scale_log2 : -INFINITY;
                const float x1 = v0 ? s[1] * p.scale_log2 : -INFINITY;
                const float x2 = v1 ? s[2] * p.scale_log2 : -INFINITY;
                const float x3 = v1 ? s[3] * p.scale_log2 : -INFINITY;
                float t0 = fmaxf(x0, x2), t1 = fmaxf(x1, x3);
                t0 = warp_max_xor(t0, 4); t0 = warp_max_xor(t0, 8); t0 = warp_max_xor(t0, 16);
                t1 = warp_max_xor(t1, 4); t1 = warp_max_xor(t1, 8); t1 = warp_max_xor(t1, 16);
                const float mn0 = fmaxf(m0, t0), mn1 = fmaxf(m1, t1);
                const float b0 = (mn0 == -INFINITY) ? 0.f : mn0;
                const float b1 = (mn1 == -INFINITY) ? 0.f : mn1;
                const float al0 = fast_exp2(m0 - b0), al1 = fast_exp2(m1 - b1);
                const float p0 = fast_exp2(x0 - b0), p1 = fast_exp2(x1 - b1);
                const float p2 = fast_exp2(x2 - b0), p3 = fast_exp2(x3 - b1);
                l0 = l0 * al0 + p0 + p2;
                l1 = l1 * al1 + p1 + p3;
                m0 = mn0;
                m1 = mn1;
#pragma unroll
                for (int mt = 0; mt < D / 16; ++mt) {
                    o[mt][0] *= al0; o[mt][1] *= al1; o[mt][2] *= al0; o[mt][3] *= al1;
                }
                const uint32_t pb0 = movmatrix_trans(pack_bf16x2(p0, p1));
                const uint32_t pb1 = movmatrix_trans(pack_bf16x2(p2, p3));
#pragma unroll
                for (int mt = 0; mt < D / 16; ++mt) {
                    uint32_t a0, a1, a2, a3;
                    ldmatrix_x4_trans(a0, a1, a2, a3, sV + dt_off(lr + 8 * (lj >> 1), head, 2 * mt + (lj & 1)));
                    mma_bf16_16816(o[mt], a0, a1, a2, a3, pb0, pb1);
                }
                if (tail) tc::fence_proxy_async_smem();  // order the zeroing before the next TMA write
                __syncwarp();
                tc::mbar_arrive_warp(EMPTY(st));
                // the next item's query: a stage after its descriptor (at once for
                // a short item)
                if (has_next && i == (spub + 1 < ntiles ? spub + 1 : spub)) {
                    nxt = geo_of(nit);
                    load_q<D>(p, nxt.t, head, g8, c, qn);
                }
            }
            if (!ok) break;
            l0 += __shfl_xor_sync(0xffffffffu, l0, 4);
            l0 += __shfl_xor_sync(0xffffffffu, l0, 8);
            l0 += __shfl_xor_sync(0xffffffffu, l0, 16);
            l1 += __shfl_xor_sync(0xffffffffu, l1, 4);
            l1 += __shfl_xor_sync(0xffffffffu, l1, 8);
            l1 += __shfl_xor_sync(0xffffffffu, l1, 16);
            const float inv0 = 1.f / l0, inv1 = 1.f / l1;
            const int h0 = 2 * c, h1 = 2 * c + 1;  // this lane's query heads within the group
            if (cur.ns == 1) {
#pragma unroll
                for (int mt = 0; mt < D / 16; ++mt) {
                    const int d0 = mt * 16 + g8;
                    if (h0 < G) {
                        __nv_bfloat16 *r = out + (static_cast<int64_t>(cur.t) * Hq + head * G + h0) * D;
                        r[d0] = __float2bfloat16_rn(o[mt][0] * inv0);
                        r[d0 + 8] = __float2bfloat16_rn(o[mt][2] * inv0);
                    }
                    if (h1 < G) {
                        __nv_bfloat16 *r = out + (static_cast<int64_t>(cur.t) * Hq + head * G + h1) * D;
                        r[d0] = __float2bfloat16_rn(o[mt][1] * inv1);
                        r[d0 + 8] = __float2bfloat16_rn(o[mt][3] * inv1);
                    }
                }
                if (g8 == 0) {
                    if (h0 < G) p.lse[static_cast<int64_t>(cur.t) * Hq + head * G + h0] = (m0 + log2f(l0)) * kLn2;
                    if (h1 < G) p.lse[static_cast<int64_t>(cur.t) * Hq + head * G + h1] = (m1 + log2f(l1)) * kLn2;
                }
            } else {
                const int64_t part = cur.part_base + cur.split;
#pragma unroll
                for (int mt = 0; mt < D / 16; ++mt) {
                    const int d0 = mt * 16 + g8;
                    if (h0 < G) {
                        float *r = p.part_o + (part * Hq + head * G + h0) * D;
                        r[d0] = o[mt][0] * inv0;
                        r[d0 + 8] = o[mt][2] * inv0;
                    }
                    if (h1 < G) {
                        float *r = p.part_o + (part * Hq + head * G + h1) * D;
                        r[d0] = o[mt][1] * inv1;
                        r[d0 + 8] = o[mt][3] * inv1;
                    }
                }
                if (g8 == 0) {
                    if (h0 < G) p.part_lse[part * Hq + head * G + h0] = m0 + log2f(l0);
                    if (h1 < G) p.part_lse[part * Hq + head * G + h1] = m1 + log2f(l1);
                }
            }
            if (!has_next) break;
            g += ntiles;
            cur = nxt;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) { qb[kk][0] = qn[kk][0]; qb[kk][1] = qn[kk][1]; }
        }
    }

    __syncthreads();
    if (tid == 0) {  // the last CTA out resets the work queue for the next run
        __threadfence();
        if (atomicAdd(sched + 1, 1) == static_cast<int>(gridDim.x) - 1) {
            sched[0] = 0;
            sched[1] = 0;
            __threadfence();
        }
    }
}

// Merge of the key splits of one query token: out = sum_s w_s O_s / sum_s w_s,
// w_s = 2^(lse_s - max), lse = max + log2(sum w) (the log-sum-exp combination
// of partial softmax results). One warp per (split token, query head), lanes
// holding float4 columns lane, lane + 32, ... of the row. The splits go in
// chunks of 32: a chunk's log-sum-exps take one load per lane, its weights
// reach the other lanes by shuffle, and a running maximum rescales what
// earlier chunks summed; the partial rows stream with 16 float4 per lane in
// flight, so a token of up to 32 splits costs a few memory round trips.
constexpr int kMergeWarps = 4;

template <int D>
__global__ void __launch_bounds__(32 * kMergeWarps) split_merge_kernel(const AttnParams p) {
    constexpr int kV = D / 4;                 // float4 per row
    constexpr int kC = (kV + 31) / 32;        // float4 columns per lane
    constexpr int kB = 16 / kC;               // partial rows in flight
    const int wg = blockIdx.x * kMergeWarps + (threadIdx.x >> 5), lane = threadIdx.x & 31;
    const int Hq = p.num_q_heads;
    pdl_wait();  // the partial results of the grid before
    if (wg >= p.num_mgroups * Hq) return;
    const MergeGroup mg = p.mgroups[wg / Hq];
    const int h = wg % Hq;
    const int ns = mg.num_splits, base = mg.part_base;
    const float4 *po = reinterpret_cast<const float4 *>(p.part_o);
    float M = -INFINITY, L = 0.f;
    float4 acc[kC];
#pragma unroll
    for (int c = 0; c < kC; ++c) acc[c] = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int c0 = 0; c0 < ns; c0 += 32) {
        const int nc = ns - c0 < 32 ? ns - c0 : 32;
        const float my = lane < nc ? __ldcg(p.part_lse + static_cast<int64_t>(base + c0 + lane) * Hq + h) : -INFINITY;
        float cm = my;
#pragma unroll
        for (int o2 = 16; o2 > 0; o2 >>= 1) cm = fmaxf(cm, __shfl_xor_sync(0xffffffffu, cm, o2));
        const float Mn = fmaxf(M, cm);
        const float a = fast_exp2(M - Mn);  // 0 for the first chunk (M = -inf)
        const float w = fast_exp2(my - Mn);  // this lane's split weight, 0 past the chunk
        float cl = w;
#pragma unroll
        for (int o2 = 16; o2 > 0; o2 >>= 1) cl += __shfl_xor_sync(0xffffffffu, cl, o2);
        L = L * a + cl;
#pragma unroll
        for (int c = 0; c < kC; ++c) {
            acc[c].x *= a; acc[c].y *= a; acc[c].z *= a; acc[c].w *= a;
        }
        M = Mn;
        // lanes past the row (D = 64) read a duplicate column and drop it
        const float4 *row = po + (static_cast<int64_t>(base + c0) * Hq + h) * kV + (lane & (kV < 32 ? kV - 1 : 31));
        for (int j0 = 0; j0 < nc; j0 += kB) {
            float4 v[kB][kC];
#pragma unroll
            for (int u = 0; u < kB; ++u)
                if (j0 + u < nc) {
#pragma unroll
                    for (int c = 0; c < kC; ++c) v[u][c] = __ldcg(row + static_cast<int64_t>(j0 + u) * Hq * kV + 32 * c);
                }
#pragma unroll
            for (int u = 0; u < kB; ++u) {
                if (j0 + u < nc) {
                    const float wj = __shfl_sync(0xffffffffu, w, j0 + u);
#pragma unroll
                    for (int c = 0; c < kC; ++c) {
                        acc[c].x += wj * v[u][c].x; acc[c].y += wj * v[u][c].y;
                        acc[c].z += wj * v[u][c].z; acc[c].w += wj * v[u][c].w;
                    }
                }
            }
        }
    }
    const float il = 1.f / L;
    __nv_bfloat16 *orow = static_cast<__nv_bfloat16 *>(p.out) + (static_cast<int64_t>(mg.token) * Hq + h) * D;
#pragma unroll
    for (int c = 0; c < kC; ++c) {
        if (32 * c + lane < kV) {
            uint2 pk;
            pk.x = pack_bf16x2(acc[c].x * il, acc[c].y * il);
            pk.y = pack_bf16x2(acc[c].z * il, acc[c].w * il);
            *reinterpret_cast<uint2 *>(orow + (32 * c + lane) * 4) = pk;
        }
    }
    if (lane == 0) p.lse[static_cast<int64_t>(mg.token) * Hq + h] = (M + log2f(L)) * kLn2;
}

// 4-D map over a paged cache [num_blocks, bs, Hkv, d] with the slot dimension
// listed before the kv-head dimension: a box (64 columns, 16 slots, Hkv heads,
// 1 block) lands in shared memory head-major.
bool encode_slot_major_map(CUtensorMap *m, const void *base, int d, int hkv, int bs, int nblocks) {
    EncodeTiledFn enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t dims[4] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(bs), static_cast<cuuint64_t>(hkv),
                          static_cast<cuuint64_t>(nblocks)};
    cuuint64_t strides[3] = {static_cast<cuuint64_t>(hkv) * d * 2, static_cast<cuuint64_t>(d) * 2,
                             static_cast<cuuint64_t>(bs) * hkv * d * 2};
    cuuint32_t box[4] = {64, static_cast<cuuint32_t>(kKeys), static_cast<cuuint32_t>(hkv), 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D>
int launch_dt(const AttnParams &p, cudaStream_t st, int max_ctas) {
    using Cfg = DtCfg<D>;
    DtMaps maps;
    if (!encode_slot_major_map(&maps.k, p.k_cache, D, p.num_kv_heads, p.block_size, p.num_blocks) ||
        !encode_slot_major_map(&maps.v, p.v_cache, D, p.num_kv_heads, p.block_size, p.num_blocks))
        return cuda_fail(cudaErrorInvalidValue, "cuTensorMapEncodeTiled (decode)");
    FNPU_CUDA_TRY(cudaFuncSetAttribute(decode_tma_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Cfg::kSmemBytes));
    FNPU_CUDA_TRY(cudaFuncSetAttribute(decode_tma_kernel<D>, cudaFuncAttributePreferredSharedMemoryCarveout,
                                       cudaSharedmemCarveoutMaxShared));
    const int grid = p.num_ditems < max_ctas ? p.num_ditems : max_ctas;
    FNPU_CUDA_TRY(launch_ex(decode_tma_kernel<D>, grid, kThreads, Cfg::kSmemBytes, st, false, nullptr, p, maps));
    return FNPU_OK;
}

}  // namespace

bool decode_tma_supported(int d_qk, int d_v, int hkv, int group, int block_size) {
    return d_qk == d_v && (d_qk == 64 || d_qk == 128) && hkv == kHkv && group <= 8 && block_size % kKeys == 0;
}

int launch_decode_tma(const AttnParams &p, void *stream, int max_ctas) {
    if (p.num_ditems == 0) return FNPU_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    int rc = FNPU_EUNSUPPORTED;
    switch (p.head_dim_qk) {
        case 64: rc = launch_dt<64>(p, st, max_ctas); break;
        case 128: rc = launch_dt<128>(p, st, max_ctas); break;
        default: break;
    }
    if (rc != FNPU_OK) return rc;
    return launch_split_merge(p, stream);
}

int launch_split_merge(const AttnParams &p, void *stream) {
    if (p.num_mgroups == 0) return FNPU_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int blocks = (p.num_mgroups * p.num_q_heads + kMergeWarps - 1) / kMergeWarps;
    void (*kernel)(AttnParams) = nullptr;
    switch (p.head_dim_v) {
        case 64: kernel = split_merge_kernel<64>; break;
        case 128: kernel = split_merge_kernel<128>; break;
        case 512: kernel = split_merge_kernel<512>; break;
        default: return FNPU_EUNSUPPORTED;
    }
    // a dependent launch: its CTAs take the SMs that the CTAs of the grid
    // before leave and wait there for that grid's writes
    FNPU_CUDA_TRY(launch_ex(kernel, blocks, 32 * kMergeWarps, 0, st, true, nullptr, p));
    return FNPU_OK;
}

}  // namespace fnpu
