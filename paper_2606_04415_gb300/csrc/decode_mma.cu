// Decode split-KV attention with GQA head packing (split K/V caches, G <= 8).
//
// Decode is bound by KV-cache reads (Sec. 1, Sec. 3.3, Fig. 2), so this path
// is built to stream K/V at HBM speed with as little arithmetic per byte as
// possible:
//   * one CTA per split item (seq, kv head, key range); all G query heads of
//     the kv head share every K/V byte loaded (GQA packing),
//   * 64-key tiles gathered through the block table with 16-byte cp.async
//     into a 3-stage shared-memory ring (XOR-swizzled rows, conflict-free
//     ldmatrix), keys past the range zero-filled so stale slots never leak,
//   * scores as S^T = K Q^T on bf16 mma.sync with the keys in M (16) and the
//     packed heads in N (8): 7 of 8 columns busy for GQA 7:1,
//   * P^T is moved from the accumulator layout into the B-operand layout with
//     movmatrix (no shared-memory round trip), then O^T += V^T P^T,
//   * each warp runs its own online softmax over its 16 keys of every tile;
//     the four warps and then the splits are merged by log-sum-exp. The last
//     split of a group to finish (atomic counter, no waiting) does the merge.
#include <math.h>

#include "common.cuh"

namespace fnpu {
namespace {

constexpr int kThreads = 128;
constexpr int kTileKeys = 64;
constexpr int kStages = 3;

template <int D>
struct DecodeCfg {
    static constexpr int kChunks = D / 8;  // 16-byte chunks per row
    static constexpr int kTileBytes = kTileKeys * D * 2;
    static constexpr int kStageBytes = 2 * kTileBytes;  // K tile then V tile
    static constexpr int kSmemBytes = kStages * kStageBytes;
};

__device__ __forceinline__ uint32_t swz_off(int row, int chunk, int row_bytes) {
    return static_cast<uint32_t>(row * row_bytes + ((chunk ^ (row & 7)) << 4));
}

template <int D>
__global__ void __launch_bounds__(kThreads, 2) decode_mma_kernel(const AttnParams p) {
    using Cfg = DecodeCfg<D>;
    extern __shared__ __align__(128) uint8_t smem[];
    __shared__ int s_last;

    const DecodeItem it = p.ditems[blockIdx.x];
    const SeqInfo si = p.seqs[it.seq];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, c = lane & 3;
    const int G = p.group;
    const int t = si.q_start;
    const __nv_bfloat16 *qrow = static_cast<const __nv_bfloat16 *>(p.q) +
                                (static_cast<int64_t>(t) * p.num_q_heads + it.kvh * G) * D;

    // Q^T as mma B fragments (k = d, n = packed head); heads >= G are zero.
    uint32_t qb[D / 16][2];
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
        if (g < G) {
            qb[kk][0] = *reinterpret_cast<const uint32_t *>(qrow + g * D + kk * 16 + 2 * c);
            qb[kk][1] = *reinterpret_cast<const uint32_t *>(qrow + g * D + kk * 16 + 8 + 2 * c);
        } else {
            qb[kk][0] = qb[kk][1] = 0u;
        }
    }

    const int nkeys = it.key_end - it.key_begin;
    const int ntiles = (nkeys + kTileKeys - 1) / kTileKeys;
    const __nv_bfloat16 *kc = static_cast<const __nv_bfloat16 *>(p.k_cache);
    const __nv_bfloat16 *vc = static_cast<const __nv_bfloat16 *>(p.v_cache);
    const int32_t *bt = p.block_table + static_cast<int64_t>(si.bt_row) * p.bt_stride;
    const int bs = p.block_size;
    const uint32_t smem_base = smem_u32(smem);

    auto load_tile = [&](int tile, int stage) {
        const uint32_t sK = smem_base + stage * Cfg::kStageBytes;
        const uint32_t sV = sK + Cfg::kTileBytes;
        const int kb = it.key_begin + tile * kTileKeys;
#pragma unroll 4
        for (int i = tid; i < kTileKeys * Cfg::kChunks; i += kThreads) {
            const int row = i / Cfg::kChunks, ch = i % Cfg::kChunks;
            const int key = kb + row;
            const bool valid = key < it.key_end;
            int64_t slot = 0;
            if (valid) slot = static_cast<int64_t>(__ldg(bt + key / bs)) * bs + key % bs;
            const uint32_t off = swz_off(row, ch, D * 2);
            cp_async_16(sK + off, kc + slot * p.k_slot_stride + it.kvh * D + ch * 8, valid);
            cp_async_16(sV + off, vc + slot * p.v_slot_stride + it.kvh * D + ch * 8, valid);
        }
    };

    float o[D / 16][4];
#pragma unroll
    for (int mt = 0; mt < D / 16; ++mt) o[mt][0] = o[mt][1] = o[mt][2] = o[mt][3] = 0.f;
    float m0 = -INFINITY, m1 = -INFINITY;  // running max (log2 units), heads 2c and 2c+1
    float l0 = 0.f, l1 = 0.f;              // this thread's share of the running sums

#pragma unroll
    for (int s = 0; s < kStages - 1; ++s) {
        if (s < ntiles) load_tile(s, s);
        cp_async_commit();
    }

    const int lj = lane >> 3, lr = lane & 7;
    for (int tile = 0; tile < ntiles; ++tile) {
        const int pre = tile + kStages - 1;
        if (pre < ntiles) load_tile(pre, pre % kStages);
        cp_async_commit();
        cp_async_wait<kStages - 1>();
        __syncthreads();

        const uint32_t sK = smem_base + (tile % kStages) * Cfg::kStageBytes;
        const uint32_t sV = sK + Cfg::kTileBytes;

        // S^T (16 keys x 8 heads) for this warp's keys [16 warp, 16 warp + 16)
        float s[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
            uint32_t a0, a1, a2, a3;
            const int row = 16 * warp + lr + 8 * (lj & 1);
            ldmatrix_x4(a0, a1, a2, a3, sK + swz_off(row, 2 * kk + (lj >> 1), D * 2));
            mma_bf16_16816(s, a0, a1, a2, a3, qb[kk][0], qb[kk][1]);
        }
        const int kr = tile * kTileKeys + 16 * warp + g;  // key of s[0], s[1]; +8 for s[2], s[3]
        const bool v0 = kr < nkeys, v1 = kr + 8 < nkeys;
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
        // P^T as the B operand (k = key, n = head)
        const uint32_t pb0 = movmatrix_trans(pack_bf16x2(p0, p1));
        const uint32_t pb1 = movmatrix_trans(pack_bf16x2(p2, p3));
#pragma unroll
        for (int mt = 0; mt < D / 16; ++mt) {
            uint32_t a0, a1, a2, a3;
            const int row = 16 * warp + lr + 8 * (lj >> 1);
            ldmatrix_x4_trans(a0, a1, a2, a3, sV + swz_off(row, 2 * mt + (lj & 1), D * 2));
            mma_bf16_16816(o[mt], a0, a1, a2, a3, pb0, pb1);
        }
        __syncthreads();
    }
    cp_async_wait<0>();

    // finish this thread's sums over the 8 key lanes of its column pair
    l0 += __shfl_xor_sync(0xffffffffu, l0, 4);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 8);
    l0 += __shfl_xor_sync(0xffffffffu, l0, 16);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 4);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 8);
    l1 += __shfl_xor_sync(0xffffffffu, l1, 16);

    // merge the four warps through shared memory (the stage ring is free now)
    __syncthreads();
    float *sm_ml = reinterpret_cast<float *>(smem);   // [4][8][2]
    float *sm_o = sm_ml + 4 * 8 * 2;                   // [4][8][D]
    if (g == 0) {
        sm_ml[(warp * 8 + 2 * c) * 2 + 0] = m0;
        sm_ml[(warp * 8 + 2 * c) * 2 + 1] = l0;
        sm_ml[(warp * 8 + 2 * c + 1) * 2 + 0] = m1;
        sm_ml[(warp * 8 + 2 * c + 1) * 2 + 1] = l1;
    }
#pragma unroll
    for (int mt = 0; mt < D / 16; ++mt) {
        float *w0 = sm_o + (warp * 8 + 2 * c) * D + mt * 16 + g;
        float *w1 = sm_o + (warp * 8 + 2 * c + 1) * D + mt * 16 + g;
        w0[0] = o[mt][0];
        w1[0] = o[mt][1];
        w0[8] = o[mt][2];
        w1[8] = o[mt][3];
    }
    __syncthreads();

    const int part = it.part_base + it.split;
    __nv_bfloat16 *out = static_cast<__nv_bfloat16 *>(p.out);
    for (int idx = tid; idx < G * D; idx += kThreads) {
        const int h = idx / D, d = idx % D;
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < 4; ++w) M = fmaxf(M, sm_ml[(w * 8 + h) * 2]);
        float L = 0.f, acc = 0.f;
#pragma unroll
        for (int w = 0; w < 4; ++w) {
            const float mw = sm_ml[(w * 8 + h) * 2];
            const float sc = (mw == -INFINITY) ? 0.f : fast_exp2(mw - M);
            L += sc * sm_ml[(w * 8 + h) * 2 + 1];
            acc += sc * sm_o[(w * 8 + h) * D + d];
        }
        const float val = acc / L;
        const float lse2 = M + log2f(L);
        const int qh = it.kvh * G + h;
        if (it.num_splits == 1) {
            out[(static_cast<int64_t>(t) * p.num_q_heads + qh) * D + d] = __float2bfloat16_rn(val);
            if (d == 0) p.lse[static_cast<int64_t>(t) * p.num_q_heads + qh] = lse2 * kLn2;
        } else {
            p.part_o[(static_cast<int64_t>(part) * G + h) * D + d] = val;
            if (d == 0) p.part_lse[static_cast<int64_t>(part) * G + h] = lse2;
        }
    }
    if (it.num_splits == 1) return;

    // the last split of this (seq, kv head) merges all splits
    __threadfence();
    __syncthreads();
    if (tid == 0) s_last = (atomicAdd(p.counters + it.group, 1) == it.num_splits - 1);
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    for (int idx = tid; idx < G * D; idx += kThreads) {
        const int h = idx / D, d = idx % D;
        float M = -INFINITY;
        for (int sp = 0; sp < it.num_splits; ++sp)
            M = fmaxf(M, __ldcg(p.part_lse + static_cast<int64_t>(it.part_base + sp) * G + h));
        float L = 0.f, acc = 0.f;
        for (int sp = 0; sp < it.num_splits; ++sp) {
            const int64_t pr = it.part_base + sp;
            const float w = fast_exp2(__ldcg(p.part_lse + pr * G + h) - M);
            L += w;
            acc += w * __ldcg(p.part_o + (pr * G + h) * D + d);
        }
        const int qh = it.kvh * G + h;
        out[(static_cast<int64_t>(t) * p.num_q_heads + qh) * D + d] = __float2bfloat16_rn(acc / L);
        if (d == 0) p.lse[static_cast<int64_t>(t) * p.num_q_heads + qh] = (M + log2f(L)) * kLn2;
    }
    if (tid == 0) p.counters[it.group] = 0;  // ready for the next run of the plan
}

template <int D>
int launch_d(const AttnParams &p, cudaStream_t st) {
    using Cfg = DecodeCfg<D>;
    static bool attr_set = false;  // per process; the attribute is per device function
    if (!attr_set) {
        if (cudaFuncSetAttribute(decode_mma_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 Cfg::kSmemBytes) != cudaSuccess)
            return FNPU_ECUDA;
        attr_set = true;
    }
    decode_mma_kernel<D><<<p.num_ditems, kThreads, Cfg::kSmemBytes, st>>>(p);
    return cudaGetLastError() == cudaSuccess ? FNPU_OK : FNPU_ECUDA;
}

}  // namespace

int launch_decode_mma(const AttnParams &p, void *stream) {
    if (p.num_ditems == 0) return FNPU_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    switch (p.head_dim_qk) {
        case 64: return launch_d<64>(p, st);
        case 128: return launch_d<128>(p, st);
        default: return FNPU_EUNSUPPORTED;
    }
}

}  // namespace fnpu
