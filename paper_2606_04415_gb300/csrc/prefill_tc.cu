// Prefill attention on the 5th-generation tensor cores (tcgen05 + TMEM + TMA).
//
// Prefill is the compute-bound phase (Sec. 1, Sec. 3.3, Fig. 1): QK^T and PV
// are dense bf16 contractions, so they run as tcgen05.mma with fp32
// accumulators in tensor memory.
//
// Work item: one kv head and P = floor(128 / G) consecutive query positions of
// a prefill chunk; the 128 MMA rows are (position, query head) pairs of that
// kv head (row = p * G + h), so every K/V byte staged in shared memory serves
// all G heads of the group (GQA packing; 126 of 128 rows busy for G = 7).
//
// Per CTA (192 threads, two CTAs per SM):
//   warps 0-3  one MMA row per thread: Q row into TMEM, online softmax on the
//              S row read from TMEM, P (bf16) written back over S, lazy
//              rescaling of the O row, epilogue;
//   warp 4     TMA producer: 64-key K/V tiles gathered block by block through
//              the block table (one 4-D box per block and 64-column half) into
//              a 3-stage ring; zeroes V rows past the context in the last tile
//              so stale slots never reach the PV product;
//   warp 5     one thread issues the MMAs: S = Q K^T (A = Q from TMEM, B = K
//              K-major) and O += P V (A = P from TMEM, B = V MN-major).
// TMEM (256 columns): Q bf16 at 0, S fp32 / P bf16 at 64, O fp32 at 128.
// Every mbarrier wait is bounded; a timeout raises the plan's error flag and
// the CTA drains, frees its tensor memory and exits.
#include <math.h>

#include <mutex>

#include "common.cuh"
#include "tc.cuh"

namespace fnpu {
namespace {

constexpr int kThreads = 192;
constexpr int kRows = 128;
constexpr int kKeys = 64;
constexpr int kStages = 3;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kColQ = 0, kColS = 64, kColO = 128;
constexpr float kRescaleThreshold = 8.0f;  // log2 units: p <= 2^8 before a rescale

template <int D>
struct TcCfg {
    static constexpr int kTileBytes = kKeys * D * 2;  // one K or V tile
    static constexpr int kStageBytes = 2 * kTileBytes;
    static constexpr int kHalf = kKeys * 128;         // one 64-column half of a tile
    // barriers: kfull[3], vfull[3], kvempty[3], sfull, pfull, pvdone, qready, vzero, drain
    static constexpr int kNumBars = 3 * kStages + 6;
    static constexpr int kSmemBytes = 1024 + kStages * kStageBytes + 8 * kNumBars + 16;
};

struct TcMaps {
    CUtensorMap k, v;
};

template <int D>
__global__ void __launch_bounds__(kThreads, 2)
    prefill_tc_kernel(const AttnParams p, const __grid_constant__ TcMaps maps) {
    using Cfg = TcCfg<D>;
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const uint32_t s_base = smem_u32(smem);
    const uint32_t s_bars = s_base + kStages * Cfg::kStageBytes;
    auto KFULL = [&](int s) { return s_bars + 8 * s; };
    auto VFULL = [&](int s) { return s_bars + 8 * (kStages + s); };
    auto KVEMPTY = [&](int s) { return s_bars + 8 * (2 * kStages + s); };
    const uint32_t SFULL = s_bars + 8 * (3 * kStages), PFULL = SFULL + 8, PVDONE = SFULL + 16,
                   QREADY = SFULL + 24, VZERO = SFULL + 32, DRAIN = SFULL + 40;
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(smem + kStages * Cfg::kStageBytes + 8 * Cfg::kNumBars);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + kStages * Cfg::kStageBytes + 8 * Cfg::kNumBars + 4);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const PrefillItem it = p.pitems[blockIdx.x];
    const SeqInfo si = p.seqs[it.seq];
    const int G = p.group;
    const int kvh = it.head;
    const int prefix = si.ctx_len - si.q_len;
    const int nkeys = prefix + it.row_begin + it.rows;  // keys 0 .. last position
    const int ntiles = (nkeys + kKeys - 1) / kKeys;
    const int ctx = si.ctx_len;
    const bool tail_fix = ntiles * kKeys > ctx;

    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(KFULL(s), 1);
            tc::mbar_init(VFULL(s), 1);
            tc::mbar_init(KVEMPTY(s), 1);
        }
        tc::mbar_init(SFULL, 1);
        tc::mbar_init(PFULL, kRows);
        tc::mbar_init(PVDONE, 1);
        tc::mbar_init(QREADY, kRows);
        tc::mbar_init(VZERO, 1);
        tc::mbar_init(DRAIN, 1);
        *abort_flag = 0;
        tc::fence_mbar_init();
    }
    if (warp == 0) {
        tc::tmem_alloc(smem_u32(const_cast<uint32_t *>(tmem_slot)), kTmemCols);
        tc::tmem_relinquish();
    }
    __syncthreads();
    tc::fence_after_sync();
    const uint32_t tmem = *tmem_slot;

    auto wait = [&](uint32_t bar, uint32_t parity) -> bool {
        if (*abort_flag) return false;
        if (tc::mbar_wait(bar, parity)) return true;
        *abort_flag = 1;
        atomicOr(p.err, 1);
        return false;
    };

    if (warp == 4) {
        // ------------------------------------------------------------ producer
        const int32_t *bt = p.block_table + static_cast<int64_t>(si.bt_row) * p.bt_stride;
        const int bs = p.block_size;
        const int nblk_seq = (ctx + bs - 1) / bs;
        const int per_tile = kKeys / bs;
        if (lane == 0) {
            tc::prefetch_tmap(&maps.k);
            tc::prefetch_tmap(&maps.v);
        }
        for (int i = 0; i < ntiles; ++i) {
            const int st = i % kStages;
            if (i >= kStages && !wait(KVEMPTY(st), ((i / kStages) - 1) & 1)) break;
            const int jb = i * per_tile;
            int nvalid = nblk_seq - jb;
            nvalid = nvalid < 0 ? 0 : (nvalid > per_tile ? per_tile : nvalid);
            const uint32_t sK = s_base + st * Cfg::kStageBytes, sV = sK + Cfg::kTileBytes;
            if (lane == 0) {
                const uint32_t bytes = static_cast<uint32_t>(nvalid) * bs * D * 2;
                tc::mbar_arrive_expect_tx(KFULL(st), bytes);
                for (int b = 0; b < nvalid; ++b) {
                    const int blk = __ldg(bt + jb + b);
#pragma unroll
                    for (int h = 0; h < D / 64; ++h)
                        tc::tma_load_4d(sK + h * Cfg::kHalf + b * bs * 128, &maps.k, KFULL(st), h * 64, kvh, 0, blk);
                }
                tc::mbar_arrive_expect_tx(VFULL(st), bytes);
                for (int b = 0; b < nvalid; ++b) {
                    const int blk = __ldg(bt + jb + b);
#pragma unroll
                    for (int h = 0; h < D / 64; ++h)
                        tc::tma_load_4d(sV + h * Cfg::kHalf + b * bs * 128, &maps.v, VFULL(st), h * 64, kvh, 0, blk);
                }
            }
            __syncwarp();
            if (i == ntiles - 1 && tail_fix) {
                // zero V rows of keys >= ctx (stale slots, unloaded blocks)
                if (!wait(VFULL(st), (i / kStages) & 1)) break;
                const int r0 = ctx - i * kKeys;
                const int nrows = kKeys - r0;
                for (int idx = lane; idx < nrows * 8 * (D / 64); idx += 32) {
                    const int h = idx / (nrows * 8), rem = idx % (nrows * 8);
                    const int row = r0 + rem / 8, ch = rem % 8;
                    *reinterpret_cast<uint4 *>(smem + st * Cfg::kStageBytes + Cfg::kTileBytes + h * Cfg::kHalf +
                                               row * 128 + ch * 16) = make_uint4(0u, 0u, 0u, 0u);
                }
                tc::fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) tc::mbar_arrive(VZERO);
            }
        }
    } else if (warp == 5) {
        // ---------------------------------------------------------- MMA issuer
        if (lane == 0) {
            constexpr uint32_t idS = tc::idesc_bf16(kRows, kKeys, false);
            constexpr uint32_t idO = tc::idesc_bf16(kRows, D, true);
            bool ok = wait(QREADY, 0);
            int issued = 0;
            for (int i = 0; ok && i < ntiles; ++i) {
                const int st = i % kStages;
                const uint32_t ph = (i / kStages) & 1;
                if (!wait(KFULL(st), ph)) { ok = false; break; }
                if (i > 0 && !wait(PVDONE, (i - 1) & 1)) { ok = false; break; }
                tc::fence_after_sync();
                const uint32_t sK = s_base + st * Cfg::kStageBytes, sV = sK + Cfg::kTileBytes;
#pragma unroll
                for (int kk = 0; kk < D / 16; ++kk) {
                    const uint64_t b = tc::sdesc_sw128(sK + (kk / 4) * Cfg::kHalf + (kk % 4) * 32, 16, 1024);
                    tc::mma_ts(tmem + kColS, tmem + kColQ + kk * 8, b, idS, kk > 0);
                }
                tc::commit(SFULL);
                issued = 1;
                if (!wait(PFULL, i & 1)) { ok = false; break; }
                if (i == ntiles - 1 && tail_fix) {
                    if (!wait(VZERO, 0)) { ok = false; break; }
                } else if (!wait(VFULL(st), ph)) {
                    ok = false;
                    break;
                }
                tc::fence_after_sync();
#pragma unroll
                for (int kk = 0; kk < kKeys / 16; ++kk) {
                    const uint64_t b = tc::sdesc_sw128(sV + kk * 2048, Cfg::kHalf, 1024);
                    tc::mma_ts(tmem + kColO, tmem + kColS + kk * 8, b, idO, (i > 0 || kk > 0) ? 1u : 0u);
                }
                tc::commit(KVEMPTY(st));
                tc::commit(PVDONE);
            }
            if (!ok && issued) {  // drain whatever is still in flight
                tc::commit(DRAIN);
                tc::mbar_wait(DRAIN, 0, 200000000ull);
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------- softmax / epilogue rows
        const int r = tid;  // MMA row = TMEM lane
        const int P = kRows / G;
        const int pl = r / G, hl = r % G;
        const bool row_ok = (r < P * G) && (pl < it.rows);
        // rows past the item (padding) keep a position too; their results are
        // never stored, so they need no masking of their own
        const int pos = prefix + it.row_begin + pl;
        const int min_pos = prefix + it.row_begin;
        const int64_t tok = si.q_start + it.row_begin + pl;
        const int head = kvh * G + hl;
        const uint32_t lane_addr = tmem + (static_cast<uint32_t>(warp * 32) << 16);

        {  // Q row -> TMEM (bf16 pairs), zeros for padding rows
            const uint4 *q = reinterpret_cast<const uint4 *>(static_cast<const __nv_bfloat16 *>(p.q) +
                                                             (tok * p.num_q_heads + head) * D);
#pragma unroll
            for (int c = 0; c < D / 64; ++c) {
                uint32_t v[32];
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    uint4 x = row_ok ? __ldg(q + c * 8 + j) : make_uint4(0u, 0u, 0u, 0u);
                    v[4 * j] = x.x; v[4 * j + 1] = x.y; v[4 * j + 2] = x.z; v[4 * j + 3] = x.w;
                }
                tc::tmem_st32(lane_addr + kColQ + 32 * c, v);
            }
            tc::tmem_wait_st();
            tc::fence_before_sync();
            tc::mbar_arrive(QREADY);
        }

        float m_run = -INFINITY;  // reference max (log2 units) of the exponentials
        float l = 0.f;
        bool ok = true;
        for (int i = 0; i < ntiles; ++i) {
            if (!wait(SFULL, i & 1)) { ok = false; break; }
            tc::fence_after_sync();
            uint32_t s[64];
            tc::tmem_ld32(lane_addr + kColS, *reinterpret_cast<uint32_t(*)[32]>(&s[0]));
            tc::tmem_ld32(lane_addr + kColS + 32, *reinterpret_cast<uint32_t(*)[32]>(&s[32]));
            tc::tmem_wait_ld();
            // tiles that reach past the first row's position need the causal
            // mask; all others are fully visible to every row of the item
            const int k0 = i * kKeys;
            const bool masked_tile = k0 + kKeys - 1 > min_pos;
            float mx0 = -INFINITY, mx1 = -INFINITY, mx2 = -INFINITY, mx3 = -INFINITY;
            if (masked_tile) {
#pragma unroll
                for (int j = 0; j < kKeys; j += 4) {
                    float v0 = __uint_as_float(s[j]), v1 = __uint_as_float(s[j + 1]);
                    float v2 = __uint_as_float(s[j + 2]), v3 = __uint_as_float(s[j + 3]);
                    v0 = (k0 + j <= pos) ? v0 : -INFINITY;
                    v1 = (k0 + j + 1 <= pos) ? v1 : -INFINITY;
                    v2 = (k0 + j + 2 <= pos) ? v2 : -INFINITY;
                    v3 = (k0 + j + 3 <= pos) ? v3 : -INFINITY;
                    s[j] = __float_as_uint(v0); s[j + 1] = __float_as_uint(v1);
                    s[j + 2] = __float_as_uint(v2); s[j + 3] = __float_as_uint(v3);
                    mx0 = fmaxf(mx0, v0); mx1 = fmaxf(mx1, v1); mx2 = fmaxf(mx2, v2); mx3 = fmaxf(mx3, v3);
                }
            } else {
#pragma unroll
                for (int j = 0; j < kKeys; j += 4) {
                    mx0 = fmaxf(mx0, __uint_as_float(s[j])); mx1 = fmaxf(mx1, __uint_as_float(s[j + 1]));
                    mx2 = fmaxf(mx2, __uint_as_float(s[j + 2])); mx3 = fmaxf(mx3, __uint_as_float(s[j + 3]));
                }
            }
            // the scale is positive, so the max of scaled scores is the scaled max
            const float tmax = fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)) * p.scale_log2;
            const bool need = (m_run == -INFINITY) ? (tmax != -INFINITY) : (tmax > m_run + kRescaleThreshold);
            if (__any_sync(0xffffffffu, need)) {
                const float m_new = need ? fmaxf(m_run, tmax) : m_run;
                const float alpha = (need && m_run != -INFINITY) ? fast_exp2(m_run - m_new) : 1.f;
                if (i > 0) {  // O of the previous tiles is complete (S(i) was issued after PV(i-1))
#pragma unroll
                    for (int c = 0; c < D / 32; ++c) {
                        uint32_t o[32];
                        tc::tmem_ld32(lane_addr + kColO + 32 * c, o);
                        tc::tmem_wait_ld();
#pragma unroll
                        for (int j = 0; j < 32; ++j) o[j] = __float_as_uint(__uint_as_float(o[j]) * alpha);
                        tc::tmem_st32(lane_addr + kColO + 32 * c, o);
                    }
                }
                l *= alpha;
                m_run = m_new;
            }
            const float nbase = (m_run == -INFINITY) ? 0.f : -m_run;
            const float sc = p.scale_log2;
            float l0 = 0.f, l1 = 0.f;
            uint32_t pk[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                const float p0 = fast_exp2(fmaf(__uint_as_float(s[2 * j]), sc, nbase));
                const float p1 = fast_exp2(fmaf(__uint_as_float(s[2 * j + 1]), sc, nbase));
                if (j & 1) l1 += p0 + p1; else l0 += p0 + p1;
                pk[j] = pack_bf16x2(p0, p1);
            }
            l += l0 + l1;
            tc::tmem_st32(lane_addr + kColS, pk);
            tc::tmem_wait_st();
            tc::fence_before_sync();
            tc::mbar_arrive(PFULL);
        }
        if (ok && wait(PVDONE, (ntiles - 1) & 1)) {
            tc::fence_after_sync();
            const float inv = 1.f / l;
            uint4 *orow = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(p.out) +
                                                    (tok * p.num_q_heads + head) * D);
#pragma unroll
            for (int c = 0; c < D / 32; ++c) {
                uint32_t o[32];
                tc::tmem_ld32(lane_addr + kColO + 32 * c, o);
                tc::tmem_wait_ld();
                if (row_ok) {
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        uint4 w;
                        w.x = pack_bf16x2(__uint_as_float(o[8 * j + 0]) * inv, __uint_as_float(o[8 * j + 1]) * inv);
                        w.y = pack_bf16x2(__uint_as_float(o[8 * j + 2]) * inv, __uint_as_float(o[8 * j + 3]) * inv);
                        w.z = pack_bf16x2(__uint_as_float(o[8 * j + 4]) * inv, __uint_as_float(o[8 * j + 5]) * inv);
                        w.w = pack_bf16x2(__uint_as_float(o[8 * j + 6]) * inv, __uint_as_float(o[8 * j + 7]) * inv);
                        orow[c * 4 + j] = w;
                    }
                }
            }
            if (row_ok) p.lse[tok * p.num_q_heads + head] = (m_run + log2f(l)) * kLn2;
        }
    }

    tc::fence_before_sync();
    __syncthreads();
    if (warp == 0) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, kTmemCols);
    }
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *,
                                  CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                  CUtensorMapFloatOOBfill);

EncodeTiledFn get_encoder() {
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

// 4-D map over a paged cache [num_blocks, bs, Hkv, d]: box = one block of one
// kv head, 64 columns wide, 128-byte swizzle.
bool encode_cache_map(CUtensorMap *m, const void *base, int d, int hkv, int bs, int nblocks) {
    EncodeTiledFn enc = get_encoder();
    if (!enc) return false;
    cuuint64_t dims[4] = {static_cast<cuuint64_t>(d), static_cast<cuuint64_t>(hkv), static_cast<cuuint64_t>(bs),
                          static_cast<cuuint64_t>(nblocks)};
    cuuint64_t strides[3] = {static_cast<cuuint64_t>(d) * 2, static_cast<cuuint64_t>(hkv) * d * 2,
                             static_cast<cuuint64_t>(bs) * hkv * d * 2};
    cuuint32_t box[4] = {64, 1, static_cast<cuuint32_t>(bs), 1};
    cuuint32_t es[4] = {1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void *>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int D>
int launch_tc(const AttnParams &p, cudaStream_t st) {
    using Cfg = TcCfg<D>;
    TcMaps maps;
    if (!encode_cache_map(&maps.k, p.k_cache, D, p.num_kv_heads, p.block_size, p.num_blocks) ||
        !encode_cache_map(&maps.v, p.v_cache, D, p.num_kv_heads, p.block_size, p.num_blocks))
        return FNPU_ECUDA;
    if (cudaFuncSetAttribute(prefill_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg::kSmemBytes) !=
        cudaSuccess)
        return FNPU_ECUDA;
    prefill_tc_kernel<D><<<p.num_pitems, kThreads, Cfg::kSmemBytes, st>>>(p, maps);
    return cudaGetLastError() == cudaSuccess ? FNPU_OK : FNPU_ECUDA;
}

}  // namespace

bool prefill_tc_supported(int d_qk, int d_v, int block_size, int group) {
    return d_qk == d_v && (d_qk == 64 || d_qk == 128) &&
           (block_size == 16 || block_size == 32 || block_size == 64) && group >= 1 && group <= kRows;
}

int prefill_tc_rows_per_item(int group) { return kRows / group; }

int launch_prefill_tc(const AttnParams &p, void *stream) {
    if (p.num_pitems == 0) return FNPU_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    switch (p.head_dim_qk) {
        case 64: return launch_tc<64>(p, st);
        case 128: return launch_tc<128>(p, st);
        default: return FNPU_EUNSUPPORTED;
    }
}

}  // namespace fnpu
