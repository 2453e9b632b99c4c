// Absorbed multi-head latent attention (MLA, the DeepSeek-R1 shape): every
// query head reads one shared latent cache row of d_qk = 576 values per key,
// and V is the first d_v = 512 of them (Eq. 1 with K = latent, V = latent[:,
// :512]). Prefill rows and decode rows of a step go through the same kernel:
// with 128 heads on one latent, a 64-row tile is 64 heads of one query token
// in either phase, so the phase only changes how many keys the row sees.
//
// One CTA takes one work item: 64 heads of one token over a key range (a
// split of its keys, merged by log-sum-exp when a token needs several). Eight
// warps in pairs: the pair owns 16 heads; for each 32-key tile of the latent
// cache (gathered through the block table with cp.async into a two-stage
// ring), warp h of the pair computes S = Q K^T for keys 16h..16h+15 of the
// tile (m16n8k16, 36 steps over d_qk) and the pair agrees on the row maxima
// through shared memory; each warp writes its half of P (bf16) to shared
// memory and then accumulates O for its half of d_v (256 columns) over all
// 32 keys. No product is computed twice, and the 16 x 256 fp32 accumulator of
// a warp fits its registers.
//
// The legacy mma.sync tensor path is used here; a tcgen05 version of this
// shape needs the 512-column fp32 accumulator of a 128-row tile, which is all
// of tensor memory, and is left for later.
#include <math.h>

#include "common.cuh"

namespace fnpu {
namespace {

constexpr int kDq = 576, kDv = 512;
constexpr int kHeads = 64;            // query heads (rows) per CTA
constexpr int kKeysT = 32;            // keys per tile
constexpr int kThreads = 256;
constexpr int kRowB = kDq * 2;        // bytes of one latent row
constexpr int kChunks = kDq / 8;      // 16-byte chunks per row
constexpr int kQBytes = kHeads * kRowB;
constexpr int kTileBytes = kKeysT * kRowB;
constexpr int kPBytes = kHeads * kKeysT * 2;
constexpr int kOffKV = kQBytes;
constexpr int kOffP = kOffKV + 2 * kTileBytes;
constexpr int kOffX = kOffP + kPBytes;  // float xmax[2][64], xsum[2][64], merge M[64], L[64]
constexpr int kSmemBytes = kOffX + 6 * 64 * 4 + 16;

// a 1152-byte latent row (Q or K/V tile): chunk j of row r at chunk j ^ (r % 8)
__device__ __forceinline__ uint32_t swz(int row, int chunk) {
    return static_cast<uint32_t>(row * kRowB + ((chunk ^ (row & 7)) << 4));
}
// a 64-byte P row: chunk j of row r at chunk j ^ ((r / 2) % 4)
__device__ __forceinline__ uint32_t swzp(int row, int chunk) {
    return static_cast<uint32_t>(row * 64 + ((chunk ^ ((row >> 1) & 3)) << 4));
}
__device__ __forceinline__ void pair_sync(int pair) {
    asm volatile("bar.sync %0, 64;\n" ::"r"(pair + 1) : "memory");
}

__global__ void __launch_bounds__(kThreads, 1) mla_mma_kernel(const AttnParams p) {
    extern __shared__ __align__(128) uint8_t smem[];
    const MlaItem it = p.mitems[blockIdx.x];
    const SeqInfo si = p.seqs[it.seq];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, c = lane & 3;
    const int lj = lane >> 3, lr = lane & 7;
    const int pair = warp >> 1, h = warp & 1;  // rows 16 pair .. +15; keys / d_v half h
    const int Hq = p.num_q_heads;
    const int64_t tok = si.q_start + it.row;
    const int kb = it.key_begin, ke = it.key_end;
    const int ntiles = (ke - kb + kKeysT - 1) / kKeysT;
    const int bs = p.block_size;

    const __nv_bfloat16 *q = static_cast<const __nv_bfloat16 *>(p.q);
    const __nv_bfloat16 *kc = static_cast<const __nv_bfloat16 *>(p.k_cache);
    const int32_t *bt = p.block_table + static_cast<int64_t>(si.bt_row) * p.bt_stride;
    const uint32_t sQ = smem_u32(smem);
    const uint32_t sKV = sQ + kOffKV;
    const uint32_t sP = sQ + kOffP;
    float *xmax = reinterpret_cast<float *>(smem + kOffX);  // [2][64]
    float *xsum = xmax + 128;                                // [2][64]
    float *mM = xsum + 128, *mL = mM + 64;                   // merge
    int *flag = reinterpret_cast<int *>(mL + 64);

    const __nv_bfloat16 *qrow0 = q + (tok * Hq + static_cast<int64_t>(it.hb) * kHeads) * kDq;
    for (int i = tid; i < kHeads * kChunks; i += kThreads) {
        const int row = i / kChunks, ch = i % kChunks;
        cp_async_16(sQ + swz(row, ch), qrow0 + static_cast<int64_t>(row) * kDq + ch * 8, true);
    }
    auto load_kv = [&](int tile, int stage) {
        const uint32_t sT = sKV + stage * kTileBytes;
#pragma unroll 3
        for (int i = tid; i < kKeysT * kChunks; i += kThreads) {
            const int row = i / kChunks, ch = i % kChunks;
            const int key = kb + tile * kKeysT + row;
            const bool valid = key < ke;
            int64_t slot = 0;
            if (valid) slot = static_cast<int64_t>(__ldg(bt + key / bs)) * bs + key % bs;
            cp_async_16(sT + swz(row, ch), kc + slot * kDq + ch * 8, valid);
        }
    };
    load_kv(0, 0);
    cp_async_commit();

    float o[32][4];
#pragma unroll
    for (int nt = 0; nt < 32; ++nt) o[nt][0] = o[nt][1] = o[nt][2] = o[nt][3] = 0.f;
    float mrow[2] = {-INFINITY, -INFINITY};
    float lown[2] = {0.f, 0.f};  // sum of this warp's keys only; the pair's sum at the end
    const int rbase = 16 * pair;

    for (int tile = 0; tile < ntiles; ++tile) {
        if (tile + 1 < ntiles) load_kv(tile + 1, (tile + 1) & 1);
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        const uint32_t sT = sKV + (tile & 1) * kTileBytes;

        // S for rows rbase.. +15, keys 16h .. 16h+15 of the tile
        float s[2][4] = {{0.f, 0.f, 0.f, 0.f}, {0.f, 0.f, 0.f, 0.f}};
#pragma unroll 4
        for (int kk = 0; kk < kDq / 16; ++kk) {
            uint32_t a0, a1, a2, a3, b0, b1, b2, b3;
            ldmatrix_x4(a0, a1, a2, a3, sQ + swz(rbase + lr + 8 * (lj & 1), 2 * kk + (lj >> 1)));
            ldmatrix_x4(b0, b1, b2, b3, sT + swz(16 * h + lr + 8 * (lj >> 1), 2 * kk + (lj & 1)));
            mma_bf16_16816(s[0], a0, a1, a2, a3, b0, b1);
            mma_bf16_16816(s[1], a0, a1, a2, a3, b2, b3);
        }
        // mask keys past the item, scale into log2 units, row maxima of the pair
        float tmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
        for (int nt = 0; nt < 2; ++nt)
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int key = kb + tile * kKeysT + 16 * h + 8 * nt + 2 * c + (e & 1);
                const float x = key < ke ? s[nt][e] * p.scale_log2 : -INFINITY;
                s[nt][e] = x;
                tmax[e >> 1] = fmaxf(tmax[e >> 1], x);
            }
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            tmax[r] = warp_max_xor(tmax[r], 1);
            tmax[r] = warp_max_xor(tmax[r], 2);
        }
        if (c == 0) {
            xmax[h * 64 + rbase + g] = tmax[0];
            xmax[h * 64 + rbase + g + 8] = tmax[1];
        }
        pair_sync(pair);
        float base[2];
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            const float t = fmaxf(tmax[r], xmax[(h ^ 1) * 64 + rbase + g + 8 * r]);
            const float mn = fmaxf(mrow[r], t);  // finite: key kb + 32 tile is always visible
            const float alpha = fast_exp2(mrow[r] - mn);
            base[r] = mn;
            mrow[r] = mn;
            lown[r] *= alpha;
#pragma unroll
            for (int nt = 0; nt < 32; ++nt) {
                o[nt][2 * r] *= alpha;
                o[nt][2 * r + 1] *= alpha;
            }
        }
#pragma unroll
        for (int nt = 0; nt < 2; ++nt) {
            const float p0 = fast_exp2(s[nt][0] - base[0]), p1 = fast_exp2(s[nt][1] - base[0]);
            const float p2 = fast_exp2(s[nt][2] - base[1]), p3 = fast_exp2(s[nt][3] - base[1]);
            lown[0] += p0 + p1;
            lown[1] += p2 + p3;
            const int key = 16 * h + 8 * nt + 2 * c;  // within the tile
            *reinterpret_cast<uint32_t *>(smem + kOffP + swzp(rbase + g, key >> 3) + (key & 7) * 2) =
                pack_bf16x2(p0, p1);
            *reinterpret_cast<uint32_t *>(smem + kOffP + swzp(rbase + g + 8, key >> 3) + (key & 7) * 2) =
                pack_bf16x2(p2, p3);
        }
        pair_sync(pair);
        // O[:, 256h .. 256h+255] += P (16 x 32) V (32 x 256)
#pragma unroll
        for (int kk2 = 0; kk2 < 2; ++kk2) {
            uint32_t a0, a1, a2, a3;
            ldmatrix_x4(a0, a1, a2, a3, sP + swzp(rbase + lr + 8 * (lj & 1), 2 * kk2 + (lj >> 1)));
#pragma unroll
            for (int dp = 0; dp < 16; ++dp) {
                uint32_t b0, b1, b2, b3;
                ldmatrix_x4_trans(b0, b1, b2, b3, sT + swz(16 * kk2 + lr + 8 * (lj & 1), 32 * h + 2 * dp + (lj >> 1)));
                mma_bf16_16816(o[2 * dp], a0, a1, a2, a3, b0, b1);
                mma_bf16_16816(o[2 * dp + 1], a0, a1, a2, a3, b2, b3);
            }
        }
        __syncthreads();
    }
    cp_async_wait<0>();

    // the pair's row sums
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        lown[r] += __shfl_xor_sync(0xffffffffu, lown[r], 1);
        lown[r] += __shfl_xor_sync(0xffffffffu, lown[r], 2);
    }
    if (c == 0) {
        xsum[h * 64 + rbase + g] = lown[0];
        xsum[h * 64 + rbase + g + 8] = lown[1];
    }
    pair_sync(pair);
    float l[2];
#pragma unroll
    for (int r = 0; r < 2; ++r) l[r] = lown[r] + xsum[(h ^ 1) * 64 + rbase + g + 8 * r];

    __nv_bfloat16 *out = static_cast<__nv_bfloat16 *>(p.out);
    const int64_t head0 = static_cast<int64_t>(it.hb) * kHeads;
    if (it.num_splits == 1) {
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            const int row = rbase + g + 8 * r;
            const float inv = 1.f / l[r];
            __nv_bfloat16 *orow = out + (tok * Hq + head0 + row) * kDv + 256 * h;
#pragma unroll
            for (int nt = 0; nt < 32; ++nt)
                *reinterpret_cast<uint32_t *>(orow + nt * 8 + 2 * c) =
                    pack_bf16x2(o[nt][2 * r] * inv, o[nt][2 * r + 1] * inv);
            if (h == 0 && c == 0) p.lse[tok * Hq + head0 + row] = (mrow[r] + log2f(l[r])) * kLn2;
        }
        return;
    }
    // a key split: partial O / l and m + log2 l, then the last split merges
    const int64_t part = it.part_base + it.split;
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        const int row = rbase + g + 8 * r;
        const float inv = 1.f / l[r];
        float *prow = p.part_o + (part * kHeads + row) * kDv + 256 * h;
#pragma unroll
        for (int nt = 0; nt < 32; ++nt)
            *reinterpret_cast<float2 *>(prow + nt * 8 + 2 * c) = make_float2(o[nt][2 * r] * inv, o[nt][2 * r + 1] * inv);
        if (h == 0 && c == 0) p.part_lse[part * kHeads + row] = mrow[r] + log2f(l[r]);
    }
    __threadfence();
    __syncthreads();
    if (tid == 0) *flag = atomicAdd(p.counters + it.group, 1) == it.num_splits - 1;
    __syncthreads();
    if (!*flag) return;
    __threadfence();
    const int ns = it.num_splits;
    if (tid < kHeads) {
        float M = -INFINITY;
        for (int sp = 0; sp < ns; ++sp) M = fmaxf(M, __ldcg(p.part_lse + (static_cast<int64_t>(it.part_base + sp)) * kHeads + tid));
        float L = 0.f;
        for (int sp = 0; sp < ns; ++sp) L += fast_exp2(__ldcg(p.part_lse + (static_cast<int64_t>(it.part_base + sp)) * kHeads + tid) - M);
        mM[tid] = M;
        mL[tid] = L;
        p.lse[tok * Hq + head0 + tid] = (M + log2f(L)) * kLn2;
    }
    __syncthreads();
    const float4 *po = reinterpret_cast<const float4 *>(p.part_o);
    for (int e = tid; e < kHeads * (kDv / 4); e += kThreads) {
        const int row = e / (kDv / 4), q4 = e % (kDv / 4);
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int sp = 0; sp < ns; ++sp) {
            const int64_t pr = static_cast<int64_t>(it.part_base + sp) * kHeads + row;
            const float w = fast_exp2(__ldcg(p.part_lse + pr) - mM[row]);
            const float4 v = __ldcg(po + pr * (kDv / 4) + q4);
            acc.x += w * v.x; acc.y += w * v.y; acc.z += w * v.z; acc.w += w * v.w;
        }
        const float il = 1.f / mL[row];
        uint2 pk;
        pk.x = pack_bf16x2(acc.x * il, acc.y * il);
        pk.y = pack_bf16x2(acc.z * il, acc.w * il);
        *reinterpret_cast<uint2 *>(out + (tok * Hq + head0 + row) * kDv + q4 * 4) = pk;
    }
    if (tid == 0) p.counters[it.group] = 0;  // ready for the next run
}

}  // namespace

bool mla_supported(int d_qk, int d_v, int hq, int hkv) {
    return d_qk == kDq && d_v == kDv && hkv == 1 && hq % kHeads == 0;
}

int mla_heads_per_item() { return kHeads; }

int launch_mla(const AttnParams &p, void *stream) {
    if (p.num_mitems == 0) return FNPU_OK;
    FNPU_CUDA_TRY(cudaFuncSetAttribute(mla_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes));
    mla_mma_kernel<<<p.num_mitems, kThreads, kSmemBytes, static_cast<cudaStream_t>(stream)>>>(p);
    FNPU_CUDA_TRY(cudaGetLastError());
    return FNPU_OK;
}

}  // namespace fnpu
