// Decode split-KV attention fed by TMA through an mbarrier ring
// (Hkv = 4 kv heads, d = 64 or 128, G <= 8 query heads per kv head, block
// size a multiple of 16).
//
// Decode is bound by KV-cache reads (Sec. 1, Sec. 3.3, Fig. 2). The kernel is
// kept small -- four warps, at most 128 registers a thread, 64 KB of shared
// memory for d = 128 -- so that up to three CTAs share an SM and a few SMs
// alone can stream decode work while the others run prefill (Sec. 3.4).
//   * Persistent CTAs take items -- a sequence's key range, longest first --
//     from an atomic queue two items ahead of use (the last CTA out resets it);
//     the next item's descriptor, block ids and query are loaded during the
//     current item, so an item boundary costs no memory round trip.
//   * A 2-stage ring of 16-key stages holds K and V of all four kv heads. Warp
//     0 issues the TMA copies of the stage after the one it is about to read:
//     four boxes of 16 slots x 4 heads x 64 columns for d = 128. The tensor map
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
//     its log-sum-exp); the last split of a (sequence, kv head) to finish
//     merges all of them. The release fence and the counter update of an item
//     are deferred to the second stage of the next item, when the partial
//     stores have long completed, and a merge they trigger to the end of it.
// Every mbarrier wait is bounded and raises the plan's error flag on timeout.
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "tc.cuh"

namespace fnpu {
namespace {

constexpr int kHkv = 4;
constexpr int kKeys = 16;        // keys per stage
constexpr int kStages = 2;
constexpr int kWarps = 4;        // one per kv head
constexpr int kThreads = 32 * kWarps;
constexpr int kHalfBytes = kHkv * kKeys * 128;  // all heads, one 64-column half

template <int D>
struct DtCfg {
    static constexpr int kTileBytes = (D / 64) * kHalfBytes;  // K or V of one stage
    static constexpr int kStageBytes = 2 * kTileBytes;
    static constexpr int kBarOff = kStages * kStageBytes;
    // full[S] empty[S] itemdone[2]
    static constexpr int kNumBars = 2 * kStages + 2;
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
__global__ void __launch_bounds__(kThreads, 4)
    decode_tma_kernel(const AttnParams p, const __grid_constant__ DtMaps maps) {
    using Cfg = DtCfg<D>;
    extern __shared__ __align__(1024) uint8_t smem[];
    const uint32_t s_base = smem_u32(smem);
    const uint32_t s_bars = s_base + Cfg::kBarOff;
    auto FULL = [&](int s) { return s_bars + 8 * s; };
    auto EMPTY = [&](int s) { return s_bars + 8 * (kStages + s); };
    auto ITEMDONE = [&](int b) { return s_bars + 8 * (2 * kStages + b); };
    int *ring = reinterpret_cast<int *>(smem + Cfg::kBarOff + 8 * Cfg::kNumBars);  // [4]
    volatile int *abort_flag = ring + 4;
    int *sched = p.sched + 2;  // this kernel's work queue: next item, finished CTAs

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n_items = p.num_ditems;
    if ((s_base & 1023u) != 0) {  // the swizzled tiles need 1024-byte alignment
        if (tid == 0) atomicOr(p.err, 2);
        return;
    }
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(FULL(s), 1);
            tc::mbar_init(EMPTY(s), kWarps);
        }
        tc::mbar_init(ITEMDONE(0), kWarps);
        tc::mbar_init(ITEMDONE(1), kWarps);
        ring[0] = atomicAdd(sched, 1);
        ring[1] = atomicAdd(sched, 1);
        *abort_flag = 0;
        tc::fence_mbar_init();
    }
    if (warp == 0 && lane == 0) {
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
    auto geo_of = [&](const DecodeItem &it, const SeqInfo &si) {
        DtGeo g;
        g.t = si.q_start;
        g.bt_row = si.bt_row;
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

    // issue stage `j` of item `g` into ring position `gs` (warp 0, whole warp)
    auto issue = [&](const DtGeo &g, int j, int blk_lane, int gs) -> bool {
        const int st = gs % kStages;
        if (gs >= kStages && !wait(EMPTY(st), ((gs / kStages) - 1) & 1)) return false;
        const int key0 = g.kb + j * kKeys;
        const int rel = key0 / bs - g.kb / bs;
        int blk = __shfl_sync(0xffffffffu, blk_lane, rel & 31);
        if (rel >= 32) blk = __ldg(p.block_table + static_cast<int64_t>(g.bt_row) * p.bt_stride + key0 / bs);
        const uint32_t sK = s_base + st * Cfg::kStageBytes, sV = sK + Cfg::kTileBytes;
        tc::mbar_arrive_expect_tx_warp(FULL(st), Cfg::kStageBytes);
#pragma unroll
        for (int h = 0; h < D / 64; ++h) {
            tc::tma_load_4d_warp(sK + h * kHalfBytes, &maps.k, FULL(st), h * 64, key0 % bs, 0, blk);
            tc::tma_load_4d_warp(sV + h * kHalfBytes, &maps.v, FULL(st), h * 64, key0 % bs, 0, blk);
        }
        return true;
    };

    // merge of the splits of (sequence of token t, this kv head), by the last split
    auto merge = [&](int t, int ns, int base) {
        float M[8], L[8];
#pragma unroll
        for (int h = 0; h < 8; ++h) { M[h] = -INFINITY; L[h] = 0.f; }
        for (int sp = lane; sp < ns; sp += 32) {
            const float *pl = p.part_lse + static_cast<int64_t>(base + sp) * Hq + head * G;
#pragma unroll
            for (int h = 0; h < 8; ++h)
                if (h < G) M[h] = fmaxf(M[h], __ldcg(pl + h));
        }
#pragma unroll
        for (int h = 0; h < 8; ++h)
#pragma unroll
            for (int o2 = 16; o2 > 0; o2 >>= 1) M[h] = fmaxf(M[h], __shfl_xor_sync(0xffffffffu, M[h], o2));
        for (int sp = lane; sp < ns; sp += 32) {
            const float *pl = p.part_lse + static_cast<int64_t>(base + sp) * Hq + head * G;
#pragma unroll
            for (int h = 0; h < 8; ++h)
                if (h < G) L[h] += fast_exp2(__ldcg(pl + h) - M[h]);
        }
#pragma unroll
        for (int h = 0; h < 8; ++h)
#pragma unroll
            for (int o2 = 16; o2 > 0; o2 >>= 1) L[h] += __shfl_xor_sync(0xffffffffu, L[h], o2);
        if (lane < D / 4) {
            float4 acc[8];
#pragma unroll
            for (int h = 0; h < 8; ++h) acc[h] = make_float4(0.f, 0.f, 0.f, 0.f);
            const float4 *po = reinterpret_cast<const float4 *>(p.part_o);
#pragma unroll 2
            for (int sp = 0; sp < ns; ++sp) {
                const int64_t row = static_cast<int64_t>(base + sp) * Hq + head * G;
#pragma unroll
                for (int h = 0; h < 8; ++h) {
                    if (h < G) {
                        const float w = fast_exp2(__ldcg(p.part_lse + row + h) - M[h]);
                        const float4 v = __ldcg(po + (row + h) * (D / 4) + lane);
                        acc[h].x += w * v.x; acc[h].y += w * v.y; acc[h].z += w * v.z; acc[h].w += w * v.w;
                    }
                }
            }
#pragma unroll
            for (int h = 0; h < 8; ++h) {
                if (h < G) {
                    const float il = 1.f / L[h];
                    uint2 pk;
                    pk.x = pack_bf16x2(acc[h].x * il, acc[h].y * il);
                    pk.y = pack_bf16x2(acc[h].z * il, acc[h].w * il);
                    *reinterpret_cast<uint2 *>(out + (static_cast<int64_t>(t) * Hq + head * G + h) * D + lane * 4) = pk;
                }
            }
        }
        if (lane < G) {
            float Ml = M[0], Ll = L[0];
#pragma unroll
            for (int h = 1; h < 8; ++h)
                if (lane == h) { Ml = M[h]; Ll = L[h]; }
            p.lse[static_cast<int64_t>(t) * Hq + head * G + lane] = (Ml + log2f(Ll)) * kLn2;
        }
    };

    // A finished split's counter update waits until its partial stores have
    // completed (a stage into the next item); a merge it triggers runs at the
    // end of that next item, when the accumulators are free.
    bool pend = false, mrg = false;
    int pend_t = 0, pend_ns = 0, pend_base = 0, pend_group = 0;
    auto settle = [&]() {
        if (!pend) return;
        pend = false;
        __threadfence();  // this warp's partial stores before the counter update
        __syncwarp();
        int last = 0;
        if (lane == 0) last = atomicAdd(p.counters + pend_group * kHkv + head, 1) == pend_ns - 1;
        mrg = __shfl_sync(0xffffffffu, last, 0) != 0;
    };
    auto merge_if_last = [&]() {
        if (!mrg) return;
        mrg = false;
        __threadfence();
        merge(pend_t, pend_ns, pend_base);
        if (lane == 0) p.counters[pend_group * kHkv + head] = 0;  // ready for the next run
    };

    int idx = ring[0];
    if (idx < n_items) {
        DtGeo cur;
        {
            const DecodeItem it = p.ditems[idx];
            cur = geo_of(it, p.seqs[it.seq]);
        }
        uint32_t qb[D / 16][2];
        load_q<D>(p, cur.t, head, g8, c, qb);
        int blk_lane = warp == 0 ? load_blk_lane(p, cur, lane) : 0;
        bool ok = true;
        if (warp == 0) ok = issue(cur, 0, blk_lane, 0);
        int g = 0;  // ring position of the current item's first stage
        for (int k = 0; ok; ++k) {
            const int ntiles = (cur.ke - cur.kb + kKeys - 1) / kKeys;
            const int idx_n = ring[(k + 1) & 3];
            const bool has_next = idx_n < n_items;
            int a_next = 0;
            if (warp == 0 && lane == 0) a_next = atomicAdd(sched, 1);  // the item after next
            DecodeItem nit{};
            if (has_next) nit = p.ditems[idx_n];
            SeqInfo nsi{};
            DtGeo nxt{};
            uint32_t qn[D / 16][2];
            int blk_lane_n = 0;

            float o[D / 16][4];
#pragma unroll
            for (int mt = 0; mt < D / 16; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
            float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
            const int nkeys = cur.ke - cur.kb;
            bool nready = false;
            for (int i = 0; i < ntiles; ++i) {
                const int gs = g + i;
                const int st = gs % kStages;
                // the next item: its sequence row after stage 0, its block ids
                // and query from stage 2 on (or before its first stage is issued)
                if (has_next && !nready && (i == 2 || i == ntiles - 1)) {
                    if (i == 0) nsi = p.seqs[nit.seq];
                    nxt = geo_of(nit, nsi);
                    load_q<D>(p, nxt.t, head, g8, c, qn);
                    if (warp == 0) blk_lane_n = load_blk_lane(p, nxt, lane);
                    nready = true;
                }
                if (warp == 0) {
                    if (i + 1 < ntiles) ok = issue(cur, i + 1, blk_lane, gs + 1);
                    else if (has_next) ok = issue(nxt, 0, blk_lane_n, gs + 1);
                    if (!ok) break;
                }
                if (!wait(FULL(st), (gs / kStages) & 1)) { ok = false; break; }
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
                if (i == 0 && has_next && !nready) nsi = p.seqs[nit.seq];
                if (i == 1) settle();  // the previous item's counter, now that its stores are done
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
            settle();  // (the previous item, if this one had a single stage)
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
            merge_if_last();  // the previous item's merge, with this item's accumulators stored
            if (cur.ns > 1) {
                pend = true;
                pend_t = cur.t;
                pend_ns = cur.ns;
                pend_base = cur.part_base;
                pend_group = cur.group;
            }
            // publish the item after next, then step to the next item
            if (warp == 0 && lane == 0) ring[(k + 2) & 3] = a_next;
            __syncwarp();
            tc::mbar_arrive_warp(ITEMDONE(k & 1));
            if (!wait(ITEMDONE(k & 1), (k >> 1) & 1)) break;
            if (!has_next) break;
            g += ntiles;
            cur = nxt;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) { qb[kk][0] = qn[kk][0]; qb[kk][1] = qn[kk][1]; }
            blk_lane = blk_lane_n;
        }
        if (!*abort_flag) {
            settle();
            merge_if_last();
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

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *,
                                  CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                  CUtensorMapFloatOOBfill);

EncodeTiledFn dt_encoder() {
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

// 4-D map over a paged cache [num_blocks, bs, Hkv, d] with the slot dimension
// listed before the kv-head dimension: a box (64 columns, 16 slots, Hkv heads,
// 1 block) lands in shared memory head-major.
bool encode_slot_major_map(CUtensorMap *m, const void *base, int d, int hkv, int bs, int nblocks) {
    EncodeTiledFn enc = dt_encoder();
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
    decode_tma_kernel<D><<<grid, kThreads, Cfg::kSmemBytes, st>>>(p, maps);
    FNPU_CUDA_TRY(cudaGetLastError());
    return FNPU_OK;
}

}  // namespace

bool decode_tma_supported(int d_qk, int d_v, int hkv, int group, int block_size) {
    return d_qk == d_v && (d_qk == 64 || d_qk == 128) && hkv == kHkv && group <= 8 && block_size % kKeys == 0;
}

int launch_decode_tma(const AttnParams &p, void *stream, int max_ctas) {
    if (p.num_ditems == 0) return FNPU_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    switch (p.head_dim_qk) {
        case 64: return launch_dt<64>(p, st, max_ctas);
        case 128: return launch_dt<128>(p, st, max_ctas);
        default: return FNPU_EUNSUPPORTED;
    }
}

}  // namespace fnpu
