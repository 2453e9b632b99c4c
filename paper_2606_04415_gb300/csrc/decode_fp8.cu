// Decode split-KV attention over an FP8 (e4m3) KV cache (Hkv = 4 kv heads,
// d = 128, G <= 8 query heads per kv head, blocks of 16 slots).
//
// Decode is bound by KV-cache reads (Sec. 1, Sec. 3.3, Fig. 2); one-byte codes
// halve them. The cache format is this library's (include/fnpu.h): per block,
// K codes [16 slots][4 heads][128] with the columns of a row permuted, V
// codes [4 heads][128][16 slots] (transposed, slots permuted), each followed
// by fp32 scales [16 slots][4 heads]; a stored value is code * scale.
//
// The kernel keeps the structure of the bf16 TMA decode kernel (persistent
// CTAs on an atomic queue one item ahead, a producer warp, one compute warp
// per kv head, GQA-packed m16n8k16 products S^T = K Q^T and O^T += V^T P^T, a
// split-merge kernel after it). What differs:
//   * A 16-key stage is one block: a 4-D box of K codes lands head-major
//     (slot dimension listed before the head dimension, 128-byte swizzle),
//     one bulk copy brings the block's V codes ([head][column][16 slots]) with
//     the V scales behind them, and another the K scales (a tensor box of
//     the V codes would be 512 rows of 16 bytes; the bulk copy is one request).
//   * The products run in f16: e4m3 values are exact in f16, the query is
//     converted once per item, and the codes go through cvt e4m3x2 -> f16x2.
//     The column permutation of K puts the four values a lane needs for one
//     16-column step (columns 2c, 2c+1, 2c+8, 2c+9) in consecutive bytes, and
//     the eight steps of a lane in 32 consecutive bytes: two 16-byte loads per
//     key row and stage. The slot permutation of V does the same for keys.
//   * The K scale of a key multiplies its scores after the product. The V
//     scale of a key, over the running maximum vm of the item's V scales,
//     multiplies its probability before P V, so that the f16 operand stays in
//     [0, 1]; the accumulator holds O / vm and is rescaled when vm grows, like
//     the softmax maximum (the row sum l takes the unscaled probabilities).
//   * Keys past the item are masked to -inf in S and their V operands are set
//     to zero in registers (stale slots may hold NaN codes).
// Every mbarrier wait is bounded and raises the plan's error flag on timeout.
#include <cuda_fp16.h>
#include <math.h>

#include "common.cuh"
#include "fp8.cuh"
#include "tc.cuh"

namespace fnpu {
namespace {

constexpr int kHkv = 4;
constexpr int kD = 128;
constexpr int kKeys = 16;        // keys per stage = slots per block
constexpr int kStages = 4;        // 64 keys in flight, as many bytes as the bf16 kernel's two stages
constexpr int kWarps = 4;        // compute warps, one per kv head
constexpr int kThreads = 32 * (kWarps + 1);  // + the TMA producer warp
constexpr int kCodeBytes = kKeys * kHkv * kD;   // K or V codes of one block (8 KB)
constexpr int kScaleBytes = kKeys * kHkv * 4;   // K or V scales of one block
constexpr int kBlockBytes = kCodeBytes + kScaleBytes;
constexpr int kStageBytes = 2 * kCodeBytes + 2 * kScaleBytes;  // K codes, V codes, K scales, V scales
constexpr int kStageStride = (kStageBytes + 1023) / 1024 * 1024;  // the swizzled K codes need 1024-byte alignment
constexpr int kBarOff = kStages * kStageStride;
constexpr int kNumBars = 2 * kStages;
constexpr int kSmemBytes = kBarOff + 8 * kNumBars + 32;  // + item ring [4] and the abort flag
static_assert(kCodeBytes % 1024 == 0 && kStageStride % 1024 == 0, "swizzle atoms");

struct Fp8Maps {
    CUtensorMap k;
};

struct DtGeo {
    int t;          // query token
    int bt_row;
    int kb, ke;     // keys [kb, ke)
    int split, ns, part_base, group;
    int b0, b1, b2, b3;  // ids of the item's first four blocks
};

// query fragments (B operand of S^T = K Q^T) in f16: columns 16 kk + 2c,
// 2c + 1 and 16 kk + 2c + 8, 2c + 9 of query head g8 of this kv head
__device__ __forceinline__ void load_q_f16(const AttnParams &p, int t, int head, int g8, int c,
                                           uint32_t (&qb)[kD / 16][2]) {
    const __nv_bfloat16 *qrow = static_cast<const __nv_bfloat16 *>(p.q) +
                                (static_cast<int64_t>(t) * p.num_q_heads + head * p.group) * kD;
#pragma unroll
    for (int kk = 0; kk < kD / 16; ++kk) {
        if (g8 < p.group) {
            qb[kk][0] = bf16x2_to_f16x2(__ldg(reinterpret_cast<const uint32_t *>(qrow + g8 * kD + kk * 16 + 2 * c)));
            qb[kk][1] = bf16x2_to_f16x2(__ldg(reinterpret_cast<const uint32_t *>(qrow + g8 * kD + kk * 16 + 8 + 2 * c)));
        } else {
            qb[kk][0] = qb[kk][1] = 0u;
        }
    }
}

__device__ __forceinline__ int load_blk_lane(const AttnParams &p, const DtGeo &g, int lane) {
    const int b0 = g.kb / kKeys;
    const int nblk = (g.ke - 1) / kKeys - b0 + 1;
    return lane < nblk ? __ldg(p.block_table + static_cast<int64_t>(g.bt_row) * p.bt_stride + b0 + lane) : 0;
}

__global__ void __launch_bounds__(kThreads, 3)
    decode_fp8_kernel(const AttnParams p, const __grid_constant__ Fp8Maps maps) {
    extern __shared__ __align__(1024) uint8_t smem[];
    const uint32_t s_base = smem_u32(smem);
    const uint32_t s_bars = s_base + kBarOff;
    auto FULL = [&](int s) { return s_bars + 8 * s; };
    auto EMPTY = [&](int s) { return s_bars + 8 * (kStages + s); };
    int *ring = reinterpret_cast<int *>(smem + kBarOff + 8 * kNumBars);  // [4]
    volatile int *abort_flag = ring + 4;
    int *sched = p.sched + 2;  // the decode work queue: next item, finished CTAs

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n_items = p.num_ditems;
    pdl_trigger();  // the merge grid may be placed once these CTAs are; it waits for them to finish
    if ((s_base & 1023u) != 0) {  // the swizzled K tiles need 1024-byte alignment
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
    const int G = p.group;
    const int Hq = p.num_q_heads;
    __nv_bfloat16 *out = static_cast<__nv_bfloat16 *>(p.out);
    const uint8_t *k_pool = static_cast<const uint8_t *>(p.k_cache);
    const uint8_t *v_pool = static_cast<const uint8_t *>(p.v_cache);

    // issue stage `j` of item `g` into ring position `gs` (producer warp, whole warp)
    auto issue = [&](const DtGeo &g, int j, int blk_lane, int gs) -> bool {
        const int st = gs % kStages;
        if (gs >= kStages && !wait(EMPTY(st), ((gs / kStages) - 1) & 1)) return false;
        const int key0 = g.kb + j * kKeys;  // a block boundary: items start at multiples of 16
        const int rel = key0 / kKeys - g.kb / kKeys;  // warp-uniform
        int blk;
        if (rel < 4) {  // from the item itself: the lanes' block-id loads may still be in flight
            blk = rel == 0 ? g.b0 : rel == 1 ? g.b1 : rel == 2 ? g.b2 : g.b3;
        } else {
            blk = __shfl_sync(0xffffffffu, blk_lane, rel & 31);
            if (rel >= 32) blk = __ldg(p.block_table + static_cast<int64_t>(g.bt_row) * p.bt_stride + key0 / kKeys);
        }
        // stage: K codes (head-major, swizzled) | V codes and V scales (the
        // block's V half as stored: one contiguous copy) | K scales
        const uint32_t sK = s_base + st * kStageStride, sV = sK + kCodeBytes;
        const int64_t boff = static_cast<int64_t>(blk) * kBlockBytes;
        tc::mbar_arrive_expect_tx_warp(FULL(st), kStageBytes);
        tc::tma_load_4d_warp(sK, &maps.k, FULL(st), 0, 0, 0, blk);
        tc::bulk_load_warp(sV, v_pool + boff, kBlockBytes, FULL(st));
        tc::bulk_load_warp(sV + kBlockBytes, k_pool + boff + kCodeBytes, kScaleBytes, FULL(st));
        return true;
    };

    if (warp == kWarps) {
        // ---------------------------------------------------- TMA producer
        // as in the bf16 kernel: the next item is taken when the current one
        // starts and published before the current item's third stage
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
        uint32_t qb[kD / 16][2];
        load_q_f16(p, cur.t, head, g8, c, qb);
        bool ok = true;
        int g = 0;  // ring position of the current item's first stage
        for (int k = 0; ok; ++k) {
            const int ntiles = (cur.ke - cur.kb + kKeys - 1) / kKeys;
            const int spub = ntiles > 2 ? 2 : ntiles - 1;  // the stage after which the next index is readable
            int idx_n = n_items;
            bool has_next = false;
            DecodeItem nit{};
            DtGeo nxt{};
            uint32_t qn[kD / 16][2];

            float o[kD / 16][4];
#pragma unroll
            for (int mt = 0; mt < kD / 16; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
            float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
            // vm: a power of two at or above every V scale of the item so far;
            // o holds O^T / vm
            float vm = 0.f;
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
                const uint8_t *tK = smem + st * kStageStride, *tV = tK + kCodeBytes;
                const float *vscale = reinterpret_cast<const float *>(tV + kCodeBytes);
                const float *kscale = vscale + kKeys * kHkv;
                const int nv = nkeys - i * kKeys;  // valid keys in this stage (>= 1)
                const bool v0 = g8 < nv, v1 = g8 + 8 < nv;
                // S^T (keys x query heads): rows g8 and g8 + 8 of this head's K codes,
                // 32 bytes each (the eight 16-column steps of lane c)
                uint32_t kw0[8], kw1[8];
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int r0 = head * kKeys + g8, r1 = r0 + 8;  // rows of the head-major box
                    const uint4 x0 = *reinterpret_cast<const uint4 *>(tK + r0 * 128 + (((2 * c + h) ^ (g8 & 7)) << 4));
                    const uint4 x1 = *reinterpret_cast<const uint4 *>(tK + r1 * 128 + (((2 * c + h) ^ ((g8 + 8) & 7)) << 4));
                    kw0[4 * h] = x0.x; kw0[4 * h + 1] = x0.y; kw0[4 * h + 2] = x0.z; kw0[4 * h + 3] = x0.w;
                    kw1[4 * h] = x1.x; kw1[4 * h + 1] = x1.y; kw1[4 * h + 2] = x1.z; kw1[4 * h + 3] = x1.w;
                }
                float s[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
                for (int kk = 0; kk < kD / 16; ++kk) {
                    uint32_t a0, a1, a2, a3;
                    e4m3x4_to_f16x2x2(kw0[kk], a0, a2);
                    e4m3x4_to_f16x2x2(kw1[kk], a1, a3);
                    mma_f16_16816(s, a0, a1, a2, a3, qb[kk][0], qb[kk][1]);
                }
                // V^T operands (keys 2c, 2c + 1, 2c + 8, 2c + 9 of columns 16 mt + g8
                // and + 8): loaded now, converted after the softmax
                uint32_t vw0[kD / 16], vw1[kD / 16];
#pragma unroll
                for (int mt = 0; mt < kD / 16; ++mt) {
                    vw0[mt] = *reinterpret_cast<const uint32_t *>(tV + (head * kD + 16 * mt + g8) * kKeys + 4 * c);
                    vw1[mt] = *reinterpret_cast<const uint32_t *>(tV + (head * kD + 16 * mt + g8 + 8) * kKeys + 4 * c);
                }
                const float ks0 = v0 ? kscale[g8 * kHkv + head] * p.scale_log2 : 0.f;
                const float ks1 = v1 ? kscale[(g8 + 8) * kHkv + head] * p.scale_log2 : 0.f;
                const float vs0 = v0 ? vscale[g8 * kHkv + head] : 0.f;
                const float vs1 = v1 ? vscale[(g8 + 8) * kHkv + head] : 0.f;
                const float x0 = v0 ? s[0] * ks0 : -INFINITY;
                const float x1 = v0 ? s[1] * ks0 : -INFINITY;
                const float x2 = v1 ? s[2] * ks1 : -INFINITY;
                const float x3 = v1 ? s[3] * ks1 : -INFINITY;
                float t0 = fmaxf(x0, x2), t1 = fmaxf(x1, x3), vt = fmaxf(vs0, vs1);
                t0 = warp_max_xor(t0, 4); t1 = warp_max_xor(t1, 4); vt = warp_max_xor(vt, 4);
                t0 = warp_max_xor(t0, 8); t1 = warp_max_xor(t1, 8); vt = warp_max_xor(vt, 8);
                t0 = warp_max_xor(t0, 16); t1 = warp_max_xor(t1, 16); vt = warp_max_xor(vt, 16);
                const float mn0 = fmaxf(m0, t0), mn1 = fmaxf(m1, t1);
                const float b0 = (mn0 == -INFINITY) ? 0.f : mn0;
                const float b1 = (mn1 == -INFINITY) ? 0.f : mn1;
                // probabilities enter P V as p * vs / vm, at most 1, so that f16
                // keeps their precision. vt > 0 (key 0 of a stage is valid, scales
                // are positive) and warp-uniform; vm grows to the power of two at
                // or above it, so 1 / vm and the rescale vm_old / vm_new are exact.
                float rv = 1.f;
                if (vt > vm) {
                    const uint32_t bits = __float_as_uint(vt);
                    const uint32_t up = (bits & 0x7FFFFFu) ? (bits & 0x7F800000u) + 0x800000u : bits;
                    const float vmn = bits < 0x800000u ? 1.17549435e-38f : __uint_as_float(up);  // subnormal: 2^-126
                    rv = vm * __uint_as_float(0x7F000000u - __float_as_uint(vmn));
                    vm = vmn;
                }
                const float ivm = __uint_as_float(0x7F000000u - __float_as_uint(vm));  // 2^-e for vm = 2^e
                const float al0 = fast_exp2(m0 - b0), al1 = fast_exp2(m1 - b1);
                const float ro0 = al0 * rv, ro1 = al1 * rv;
                const float p0 = fast_exp2(x0 - b0), p1 = fast_exp2(x1 - b1);
                const float p2 = fast_exp2(x2 - b0), p3 = fast_exp2(x3 - b1);
                l0 = l0 * al0 + p0 + p2;
                l1 = l1 * al1 + p1 + p3;
                m0 = mn0;
                m1 = mn1;
                if (__any_sync(0xffffffffu, (ro0 != 1.f) | (ro1 != 1.f))) {  // most stages move neither maximum
#pragma unroll
                    for (int mt = 0; mt < kD / 16; ++mt) {
                        o[mt][0] *= ro0; o[mt][1] *= ro1; o[mt][2] *= ro0; o[mt][3] *= ro1;
                    }
                }
                // probabilities times the V scale of their key over vm (0 past the item)
                const float w0 = vs0 * ivm, w1 = vs1 * ivm;
                const uint32_t pb0 = movmatrix_trans(pack_f16x2(p0 * w0, p1 * w0));
                const uint32_t pb1 = movmatrix_trans(pack_f16x2(p2 * w1, p3 * w1));
                if (nv >= kKeys) {
#pragma unroll
                    for (int mt = 0; mt < kD / 16; ++mt) {
                        uint32_t a0, a1, a2, a3;
                        e4m3x4_to_f16x2x2(vw0[mt], a0, a2);
                        e4m3x4_to_f16x2x2(vw1[mt], a1, a3);
                        mma_f16_16816(o[mt], a0, a1, a2, a3, pb0, pb1);
                    }
                } else {  // the item's last, partial block: V of keys past it set to zero
                    const uint32_t lo_keep = (2 * c < nv ? 0x0000FFFFu : 0u) | (2 * c + 1 < nv ? 0xFFFF0000u : 0u);
                    const uint32_t hi_keep = (2 * c + 8 < nv ? 0x0000FFFFu : 0u) | (2 * c + 9 < nv ? 0xFFFF0000u : 0u);
#pragma unroll
                    for (int mt = 0; mt < kD / 16; ++mt) {
                        uint32_t a0, a1, a2, a3;
                        e4m3x4_to_f16x2x2(vw0[mt], a0, a2);
                        e4m3x4_to_f16x2x2(vw1[mt], a1, a3);
                        mma_f16_16816(o[mt], a0 & lo_keep, a1 & lo_keep, a2 & hi_keep, a3 & hi_keep, pb0, pb1);
                    }
                }
                __syncwarp();
                tc::mbar_arrive_warp(EMPTY(st));
                // the next item's query: a stage after its descriptor (at once for
                // a short item)
                if (has_next && i == (spub + 1 < ntiles ? spub + 1 : spub)) {
                    nxt = geo_of(nit);
                    load_q_f16(p, nxt.t, head, g8, c, qn);
                }
            }
            if (!ok) break;
            l0 += __shfl_xor_sync(0xffffffffu, l0, 4);
            l0 += __shfl_xor_sync(0xffffffffu, l0, 8);
            l0 += __shfl_xor_sync(0xffffffffu, l0, 16);
            l1 += __shfl_xor_sync(0xffffffffu, l1, 4);
            l1 += __shfl_xor_sync(0xffffffffu, l1, 8);
            l1 += __shfl_xor_sync(0xffffffffu, l1, 16);
            const float inv0 = vm / l0, inv1 = vm / l1;
            const int h0 = 2 * c, h1 = 2 * c + 1;  // this lane's query heads within the group
            if (cur.ns == 1) {
#pragma unroll
                for (int mt = 0; mt < kD / 16; ++mt) {
                    const int d0 = mt * 16 + g8;
                    if (h0 < G) {
                        __nv_bfloat16 *r = out + (static_cast<int64_t>(cur.t) * Hq + head * G + h0) * kD;
                        r[d0] = __float2bfloat16_rn(o[mt][0] * inv0);
                        r[d0 + 8] = __float2bfloat16_rn(o[mt][2] * inv0);
                    }
                    if (h1 < G) {
                        __nv_bfloat16 *r = out + (static_cast<int64_t>(cur.t) * Hq + head * G + h1) * kD;
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
                for (int mt = 0; mt < kD / 16; ++mt) {
                    const int d0 = mt * 16 + g8;
                    if (h0 < G) {
                        float *r = p.part_o + (part * Hq + head * G + h0) * kD;
                        r[d0] = o[mt][0] * inv0;
                        r[d0 + 8] = o[mt][2] * inv0;
                    }
                    if (h1 < G) {
                        float *r = p.part_o + (part * Hq + head * G + h1) * kD;
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
            for (int kk = 0; kk < kD / 16; ++kk) { qb[kk][0] = qn[kk][0]; qb[kk][1] = qn[kk][1]; }
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

// K codes: bytes [block][slot][head][128] with the slot dimension listed
// before the head dimension, so that a box (128 bytes, 16 slots, 4 heads, 1
// block) lands head-major; 128-byte swizzle keyed by the slot.
bool encode_k_map(CUtensorMap *m, const void *base, int nblocks) {
    EncodeTiledFn enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t dims[4] = {static_cast<cuuint64_t>(kD), kKeys, kHkv, static_cast<cuuint64_t>(nblocks)};
    cuuint64_t strides[3] = {kHkv * kD, kD, kBlockBytes};
    cuuint32_t box[4] = {kD, kKeys, kHkv, 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 4, const_cast<void *>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool decode_fp8_supported(int d_qk, int d_v, int hkv, int group, int block_size) {
    return d_qk == kD && d_v == kD && hkv == kHkv && group <= 8 && block_size == kKeys;
}

int launch_decode_fp8(const AttnParams &p, void *stream, int max_ctas) {
    if (p.num_ditems == 0) return FNPU_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    Fp8Maps maps;
    if (!encode_k_map(&maps.k, p.k_cache, p.num_blocks))
        return cuda_fail(cudaErrorInvalidValue, "cuTensorMapEncodeTiled (fp8 decode)");
    FNPU_CUDA_TRY(cudaFuncSetAttribute(decode_fp8_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes));
    const int grid = p.num_ditems < max_ctas ? p.num_ditems : max_ctas;
    FNPU_CUDA_TRY(launch_ex(decode_fp8_kernel, grid, kThreads, kSmemBytes, st, false, nullptr, p, maps));
    return launch_split_merge(p, stream);
}

}  // namespace fnpu
