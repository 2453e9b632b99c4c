// Decode split-KV attention fed by TMA through an mbarrier pipeline
// (Hkv = 4 kv heads, d = 64 or 128, G <= 8 query heads per kv head, block
// size a multiple of 16).
//
// Decode is bound by KV-cache reads (Sec. 1, Sec. 3.3, Fig. 2), so the kernel
// is organised around keeping HBM busy:
//   * persistent CTAs (two per SM) take items -- a sequence's key range,
//     longest first -- from an atomic queue (the last CTA resets it);
//   * one producer warp streams 16-key stages of K and V for all four kv
//     heads (for Qwen one contiguous 16 KB slot run per stage and tensor) with
//     four TMA boxes per stage into a 3-stage ring. The tensor map lists the
//     slot dimension before the kv-head dimension, so a box lands head-major
//     (16 consecutive slots of one head form 16 rows) and the 128-byte swizzle
//     is keyed by the slot: ldmatrix over eight consecutive slots of one head
//     is conflict-free;
//   * four compute warps, one per kv head, run the GQA-packed mma.sync scheme
//     independently (S^T = K Q^T with 16 keys in M and the G query heads in
//     N; P^T by movmatrix; O^T += V^T P^T) and release a stage with one
//     mbarrier arrival each -- no block-wide barrier per stage;
//   * V rows past the item's keys are zeroed by their warp before the PV
//     product, so stale slots never reach it;
//   * each warp writes its kv head's partial result; the last split of a
//     (sequence, kv head) to finish merges all splits (atomic counter, no
//     waiting).
// Every mbarrier wait is bounded and raises the plan's error flag on timeout.
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "tc.cuh"

namespace fnpu {
namespace {

constexpr int kHkv = 4;
constexpr int kKeys = 16;        // keys per stage
constexpr int kStages = 3;
constexpr int kCompute = 4;      // compute warps = kv heads
constexpr int kThreads = 32 * (kCompute + 1);
constexpr int kHalfBytes = kHkv * kKeys * 128;  // all heads, one 64-column half

template <int D>
struct DtCfg {
    static constexpr int kTileBytes = (D / 64) * kHalfBytes;  // K or V of one stage
    static constexpr int kStageBytes = 2 * kTileBytes;
    static constexpr int kBarOff = kStages * kStageBytes;
    // full[S] empty[S] itemfull[2] itemempty[2]
    static constexpr int kNumBars = 2 * kStages + 4;
    static constexpr int kSmemBytes = 1024 + kBarOff + 8 * kNumBars + 16;
};

struct DtMaps {
    CUtensorMap k, v;
};

// shared-memory offset of (slot, kv head, 16-byte chunk) inside a K or V tile
__device__ __forceinline__ uint32_t dt_off(int slot, int head, int chunk) {
    return static_cast<uint32_t>((chunk >> 3) * kHalfBytes + (head * kKeys + slot) * 128 +
                                 (((chunk & 7) ^ (slot & 7)) << 4));
}

template <int D>
__global__ void __launch_bounds__(kThreads, 2)
    decode_tma_kernel(const AttnParams p, const __grid_constant__ DtMaps maps) {
    using Cfg = DtCfg<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t s_base = smem_u32(smem);
    const uint32_t s_bars = s_base + Cfg::kBarOff;
    auto FULL = [&](int s) { return s_bars + 8 * s; };
    auto EMPTY = [&](int s) { return s_bars + 8 * (kStages + s); };
    auto ITEMFULL = [&](int k) { return s_bars + 8 * (2 * kStages + k); };
    auto ITEMEMPTY = [&](int k) { return s_bars + 8 * (2 * kStages + 2 + k); };
    uint8_t *misc = smem + Cfg::kBarOff + 8 * Cfg::kNumBars;
    volatile int *abort_flag = reinterpret_cast<volatile int *>(misc);
    volatile int *item_slot = reinterpret_cast<volatile int *>(misc + 4);  // [2]
    int *sched = p.sched + 2;  // this kernel's work queue: next item, finished CTAs

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(FULL(s), 1);
            tc::mbar_init(EMPTY(s), kCompute);
        }
        for (int k = 0; k < 2; ++k) {
            tc::mbar_init(ITEMFULL(k), 1);
            tc::mbar_init(ITEMEMPTY(k), kCompute);
        }
        *abort_flag = 0;
        tc::fence_mbar_init();
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

    if (warp == kCompute) {
        // ------------------------------------------------ scheduler + producer
        if (lane == 0) {
            tc::prefetch_tmap(&maps.k);
            tc::prefetch_tmap(&maps.v);
        }
        const int bs = p.block_size;
        int g = 0;  // stages issued so far
        for (int k = 0;; ++k) {
            int idx = 0;
            if (lane == 0) idx = atomicAdd(sched, 1);
            idx = __shfl_sync(0xffffffffu, idx, 0);
            const int slot = k & 1;
            if (k >= 2 && !wait(ITEMEMPTY(slot), ((k >> 1) - 1) & 1)) break;
            if (lane == 0) {
                item_slot[slot] = idx < p.num_ditems ? idx : -1;
                tc::mbar_arrive(ITEMFULL(slot));
            }
            if (idx >= p.num_ditems) break;
            const DecodeItem it = p.ditems[idx];
            const SeqInfo si = p.seqs[it.seq];
            const int32_t *bt = p.block_table + static_cast<int64_t>(si.bt_row) * p.bt_stride;
            const int ntiles = (it.key_end - it.key_begin + kKeys - 1) / kKeys;
            // block id of the next stage, loaded one stage ahead
            int blk_next = __ldg(bt + it.key_begin / bs);
            bool ok = true;
            for (int i = 0; i < ntiles; ++i, ++g) {
                const int st = g % kStages;
                const int key0 = it.key_begin + i * kKeys;
                const int blk = __shfl_sync(0xffffffffu, blk_next, 0);
                if (i + 1 < ntiles) blk_next = __ldg(bt + (key0 + kKeys) / bs);
                if (g >= kStages && !wait(EMPTY(st), ((g / kStages) - 1) & 1)) { ok = false; break; }
                const uint32_t sK = s_base + st * Cfg::kStageBytes, sV = sK + Cfg::kTileBytes;
                const int slot0 = __shfl_sync(0xffffffffu, key0 % bs, 0);
                tc::mbar_arrive_expect_tx_warp(FULL(st), Cfg::kStageBytes);
#pragma unroll
                for (int h = 0; h < D / 64; ++h) {
                    tc::tma_load_4d_warp(sK + h * kHalfBytes, &maps.k, FULL(st), h * 64, slot0, 0, blk);
                    tc::tma_load_4d_warp(sV + h * kHalfBytes, &maps.v, FULL(st), h * 64, slot0, 0, blk);
                }
            }
            if (!ok) break;
        }
    } else {
        // ----------------------------------------- compute warp = one kv head
        const int head = warp;
        const int g8 = lane >> 2, c = lane & 3;
        const int lj = lane >> 3, lr = lane & 7;
        const int G = p.group;
        const int Hq = p.num_q_heads;
        int gs = 0;  // stages consumed so far
        for (int k = 0;; ++k) {
            const int slot = k & 1;
            if (!wait(ITEMFULL(slot), (k >> 1) & 1)) break;
            const int idx = __shfl_sync(0xffffffffu, item_slot[slot], 0);
            if (idx < 0) break;
            const DecodeItem it = p.ditems[idx];
            const SeqInfo si = p.seqs[it.seq];
            const int t = si.q_start;
            const __nv_bfloat16 *qrow = static_cast<const __nv_bfloat16 *>(p.q) +
                                        (static_cast<int64_t>(t) * Hq + head * G) * D;
            uint32_t qb[D / 16][2];
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
                if (g8 < G) {
                    qb[kk][0] = __ldg(reinterpret_cast<const uint32_t *>(qrow + g8 * D + kk * 16 + 2 * c));
                    qb[kk][1] = __ldg(reinterpret_cast<const uint32_t *>(qrow + g8 * D + kk * 16 + 8 + 2 * c));
                } else {
                    qb[kk][0] = qb[kk][1] = 0u;
                }
            }
            const int nkeys = it.key_end - it.key_begin;
            const int ntiles = (nkeys + kKeys - 1) / kKeys;
            float o[D / 16][4];
#pragma unroll
            for (int mt = 0; mt < D / 16; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
            float m0 = -INFINITY, m1 = -INFINITY, l0 = 0.f, l1 = 0.f;
            bool ok = true;
            for (int i = 0; i < ntiles; ++i, ++gs) {
                const int st = gs % kStages;
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
            __nv_bfloat16 *out = static_cast<__nv_bfloat16 *>(p.out);
            if (it.num_splits == 1) {
#pragma unroll
                for (int mt = 0; mt < D / 16; ++mt) {
                    const int d0 = mt * 16 + g8;
                    if (h0 < G) {
                        __nv_bfloat16 *r = out + (static_cast<int64_t>(t) * Hq + head * G + h0) * D;
                        r[d0] = __float2bfloat16_rn(o[mt][0] * inv0);
                        r[d0 + 8] = __float2bfloat16_rn(o[mt][2] * inv0);
                    }
                    if (h1 < G) {
                        __nv_bfloat16 *r = out + (static_cast<int64_t>(t) * Hq + head * G + h1) * D;
                        r[d0] = __float2bfloat16_rn(o[mt][1] * inv1);
                        r[d0 + 8] = __float2bfloat16_rn(o[mt][3] * inv1);
                    }
                }
                if (g8 == 0) {
                    if (h0 < G) p.lse[static_cast<int64_t>(t) * Hq + head * G + h0] = (m0 + log2f(l0)) * kLn2;
                    if (h1 < G) p.lse[static_cast<int64_t>(t) * Hq + head * G + h1] = (m1 + log2f(l1)) * kLn2;
                }
            } else {
                const int64_t part = it.part_base + it.split;
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
                // the last split of this (sequence, kv head) merges all splits
                __threadfence();
                __syncwarp();
                int last = 0;
                if (lane == 0) last = atomicAdd(p.counters + it.group * kHkv + head, 1) == it.num_splits - 1;
                last = __shfl_sync(0xffffffffu, last, 0);
                if (last) {
                    __threadfence();
                    const int ns = it.num_splits;
                    const float4 *po = reinterpret_cast<const float4 *>(p.part_o);
                    for (int hg = 0; hg < G; ++hg) {
                        const int qh = head * G + hg;
                        float M = -INFINITY;
                        for (int sp = lane; sp < ns; sp += 32)
                            M = fmaxf(M, __ldcg(p.part_lse + static_cast<int64_t>(it.part_base + sp) * Hq + qh));
                        for (int o2 = 16; o2 > 0; o2 >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o2));
                        float L = 0.f;
                        for (int sp = lane; sp < ns; sp += 32)
                            L += fast_exp2(__ldcg(p.part_lse + static_cast<int64_t>(it.part_base + sp) * Hq + qh) - M);
                        for (int o2 = 16; o2 > 0; o2 >>= 1) L += __shfl_xor_sync(0xffffffffu, L, o2);
                        if (lane < D / 4) {
                            float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
                            for (int sp = 0; sp < ns; ++sp) {
                                const int64_t pr = it.part_base + sp;
                                const float w = fast_exp2(__ldcg(p.part_lse + pr * Hq + qh) - M);
                                const float4 v = __ldcg(po + (pr * Hq + qh) * (D / 4) + lane);
                                acc.x += w * v.x; acc.y += w * v.y; acc.z += w * v.z; acc.w += w * v.w;
                            }
                            const float il = 1.f / L;
                            uint2 pk;
                            pk.x = pack_bf16x2(acc.x * il, acc.y * il);
                            pk.y = pack_bf16x2(acc.z * il, acc.w * il);
                            *reinterpret_cast<uint2 *>(out + (static_cast<int64_t>(t) * Hq + qh) * D + lane * 4) = pk;
                        }
                        if (lane == 0) p.lse[static_cast<int64_t>(t) * Hq + qh] = (M + log2f(L)) * kLn2;
                    }
                    if (lane == 0) p.counters[it.group * kHkv + head] = 0;  // ready for the next run
                }
            }
            tc::mbar_arrive_warp(ITEMEMPTY(slot));
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
int launch_dt(const AttnParams &p, cudaStream_t st) {
    using Cfg = DtCfg<D>;
    DtMaps maps;
    if (!encode_slot_major_map(&maps.k, p.k_cache, D, p.num_kv_heads, p.block_size, p.num_blocks) ||
        !encode_slot_major_map(&maps.v, p.v_cache, D, p.num_kv_heads, p.block_size, p.num_blocks))
        return cuda_fail(cudaErrorInvalidValue, "cuTensorMapEncodeTiled (decode)");
    FNPU_CUDA_TRY(cudaFuncSetAttribute(decode_tma_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Cfg::kSmemBytes));
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int grid = p.num_ditems < 2 * sms ? p.num_ditems : 2 * sms;
    decode_tma_kernel<D><<<grid, kThreads, Cfg::kSmemBytes, st>>>(p, maps);
    FNPU_CUDA_TRY(cudaGetLastError());
    return FNPU_OK;
}

}  // namespace

bool decode_tma_supported(int d_qk, int d_v, int hkv, int group, int block_size) {
    return d_qk == d_v && (d_qk == 64 || d_qk == 128) && hkv == kHkv && group <= 8 && block_size % kKeys == 0;
}

int launch_decode_tma(const AttnParams &p, void *stream) {
    if (p.num_ditems == 0) return FNPU_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    switch (p.head_dim_qk) {
        case 64: return launch_dt<64>(p, st);
        case 128: return launch_dt<128>(p, st);
        default: return FNPU_EUNSUPPORTED;
    }
}

}  // namespace fnpu
