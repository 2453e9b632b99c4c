// Prefill attention on bf16 mma.sync (the legacy tensor path).
//
// A causal chunk of q query tokens on top of a cached prefix of ctx - q
// tokens: row i of the chunk sits at absolute position ctx - q + i and sees
// keys 0..pos. Query and key rows have DQ columns, value and output rows DV
// (equal except for the decompressed latent cache: 192 and 128). One CTA
// computes 64 query rows of one query head; four warps
// own 16 rows each. K/V tiles of 64 keys are gathered through the block table
// with cp.async into a double-buffered shared ring; S = Q K^T and O += P V run
// on m16n8k16 with fp32 accumulation, the online softmax in fp32 registers,
// and P is fed to the second product straight from the accumulator layout.
//
// This path serves as the comparison baseline for the tcgen05 prefill kernel
// and as the prefill path for shapes that kernel does not cover.
#include <math.h>

#include "common.cuh"

namespace fnpu {
namespace {

constexpr int kThreads = 128;
constexpr int kRows = 64;
constexpr int kKeys = 64;

// DQ: width of the query and key rows; DV: width of the value and output rows
template <int DQ, int DV>
struct PrefillCfg {
    static constexpr int kQChunks = DQ / 8, kVChunks = DV / 8;  // 16-byte chunks of a row
    static constexpr int kKBytes = kKeys * DQ * 2;
    static constexpr int kVBytes = kKeys * DV * 2;
    static constexpr int kQBytes = kRows * DQ * 2;
    static constexpr int kStageBytes = kKBytes + kVBytes;
    static constexpr int kSmemBytes = kQBytes + 2 * kStageBytes;  // Q + 2 x (K, V)
};

__device__ __forceinline__ uint32_t swz_off(int row, int chunk, int row_bytes) {
    return static_cast<uint32_t>(row * row_bytes + ((chunk ^ (row & 7)) << 4));
}

template <int DQ, int DV>
__global__ void __launch_bounds__(kThreads, 2) prefill_mma_kernel(const AttnParams p) {
    using Cfg = PrefillCfg<DQ, DV>;
    extern __shared__ __align__(128) uint8_t smem[];
    const PrefillItem it = p.pitems[blockIdx.x];
    const SeqInfo si = p.seqs[it.seq];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, c = lane & 3;
    const int lj = lane >> 3, lr = lane & 7;
    const int h = it.head, kvh = h / p.group;
    const int prefix = si.ctx_len - si.q_len;
    const int pos_first = prefix + it.row_begin;
    const int nkeys = pos_first + it.rows;  // keys 0 .. pos_last
    const int ntiles = (nkeys + kKeys - 1) / kKeys;

    const __nv_bfloat16 *q = static_cast<const __nv_bfloat16 *>(p.q);
    const __nv_bfloat16 *kc = static_cast<const __nv_bfloat16 *>(p.k_cache);
    const __nv_bfloat16 *vc = static_cast<const __nv_bfloat16 *>(p.v_cache);
    const int32_t *bt = p.block_table + static_cast<int64_t>(si.bt_row) * p.bt_stride;
    const int bs = p.block_size;
    const uint32_t sQ = smem_u32(smem);
    const uint32_t sKV = sQ + Cfg::kQBytes;

    for (int i = tid; i < kRows * Cfg::kQChunks; i += kThreads) {
        const int row = i / Cfg::kQChunks, ch = i % Cfg::kQChunks;
        const bool valid = row < it.rows;
        const int64_t tok = si.q_start + it.row_begin + (valid ? row : 0);
        cp_async_16(sQ + swz_off(row, ch, DQ * 2), q + (tok * p.num_q_heads + h) * DQ + ch * 8, valid);
    }
    auto load_kv = [&](int tile, int stage) {
        const uint32_t sK = sKV + stage * Cfg::kStageBytes;
        const uint32_t sV = sK + Cfg::kKBytes;
        if constexpr (DQ == DV) {  // one slot lookup for a K and a V chunk
            static_assert(Cfg::kQChunks == Cfg::kVChunks, "equal row widths");
#pragma unroll 4
            for (int i = tid; i < kKeys * Cfg::kQChunks; i += kThreads) {
                const int row = i / Cfg::kQChunks, ch = i % Cfg::kQChunks;
                const int key = tile * kKeys + row;
                const bool valid = key < nkeys;
                int64_t slot = 0;
                if (valid) slot = static_cast<int64_t>(__ldg(bt + key / bs)) * bs + key % bs;
                const uint32_t off = swz_off(row, ch, DQ * 2);
                cp_async_16(sK + off, kc + slot * p.k_slot_stride + kvh * DQ + ch * 8, valid);
                cp_async_16(sV + off, vc + slot * p.v_slot_stride + kvh * DV + ch * 8, valid);
            }
        } else {  // K rows of DQ and V rows of DV columns: the chunks of a key in one range
            constexpr int kC = Cfg::kQChunks + Cfg::kVChunks;
#pragma unroll 4
            for (int i = tid; i < kKeys * kC; i += kThreads) {
                const int row = i / kC, ch = i % kC;
                const int key = tile * kKeys + row;
                const bool valid = key < nkeys;
                int64_t slot = 0;
                if (valid) slot = static_cast<int64_t>(__ldg(bt + key / bs)) * bs + key % bs;
                if (ch < Cfg::kQChunks)
                    cp_async_16(sK + swz_off(row, ch, DQ * 2), kc + slot * p.k_slot_stride + kvh * DQ + ch * 8, valid);
                else
                    cp_async_16(sV + swz_off(row, ch - Cfg::kQChunks, DV * 2),
                                vc + slot * p.v_slot_stride + kvh * DV + (ch - Cfg::kQChunks) * 8, valid);
            }
        }
    };
    load_kv(0, 0);
    cp_async_commit();

    float o[DV / 8][4];
#pragma unroll
    for (int nt = 0; nt < DV / 8; ++nt) o[nt][0] = o[nt][1] = o[nt][2] = o[nt][3] = 0.f;
    float mrow[2] = {-INFINITY, -INFINITY};
    float lrow[2] = {0.f, 0.f};
    const int pr0 = pos_first + 16 * warp + g;  // position of row g; row g + 8 is pr0 + 8
    uint32_t qa[DQ / 16][4];

    for (int tile = 0; tile < ntiles; ++tile) {
        if (tile + 1 < ntiles) load_kv(tile + 1, (tile + 1) & 1);
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        if (tile == 0) {
#pragma unroll
            for (int kk = 0; kk < DQ / 16; ++kk) {
                const int row = 16 * warp + lr + 8 * (lj & 1);
                ldmatrix_x4(qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3],
                            sQ + swz_off(row, 2 * kk + (lj >> 1), DQ * 2));
            }
        }
        const uint32_t sK = sKV + (tile & 1) * Cfg::kStageBytes;
        const uint32_t sV = sK + Cfg::kKBytes;

        float s[8][4];
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
#pragma unroll
        for (int kk = 0; kk < DQ / 16; ++kk) {
#pragma unroll
            for (int np = 0; np < 4; ++np) {
                uint32_t b0, b1, b2, b3;
                const int row = 16 * np + lr + 8 * (lj >> 1);
                ldmatrix_x4(b0, b1, b2, b3, sK + swz_off(row, 2 * kk + (lj & 1), DQ * 2));
                mma_bf16_16816(s[2 * np], qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], b0, b1);
                mma_bf16_16816(s[2 * np + 1], qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], b2, b3);
            }
        }
        // causal mask at absolute positions, scale into log2 units, online softmax
        float tmax[2] = {-INFINITY, -INFINITY};
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int key = tile * kKeys + nt * 8 + 2 * c + (e & 1);
                const int pr = pr0 + 8 * (e >> 1);
                const float x = (key <= pr) ? s[nt][e] * p.scale_log2 : -INFINITY;
                s[nt][e] = x;
                tmax[e >> 1] = fmaxf(tmax[e >> 1], x);
            }
        }
        float alpha[2], base[2];
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            tmax[r] = warp_max_xor(tmax[r], 1);
            tmax[r] = warp_max_xor(tmax[r], 2);
            const float mn = fmaxf(mrow[r], tmax[r]);
            base[r] = (mn == -INFINITY) ? 0.f : mn;
            alpha[r] = fast_exp2(mrow[r] - base[r]);
            mrow[r] = mn;
            lrow[r] *= alpha[r];
        }
#pragma unroll
        for (int nt = 0; nt < DV / 8; ++nt) {
            o[nt][0] *= alpha[0]; o[nt][1] *= alpha[0];
            o[nt][2] *= alpha[1]; o[nt][3] *= alpha[1];
        }
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float pv = fast_exp2(s[nt][e] - base[e >> 1]);
                s[nt][e] = pv;
                lrow[e >> 1] += pv;
            }
        }
        // O += P V, P straight from the accumulator layout
#pragma unroll
        for (int kk2 = 0; kk2 < 4; ++kk2) {
            const uint32_t a0 = pack_bf16x2(s[2 * kk2][0], s[2 * kk2][1]);
            const uint32_t a1 = pack_bf16x2(s[2 * kk2][2], s[2 * kk2][3]);
            const uint32_t a2 = pack_bf16x2(s[2 * kk2 + 1][0], s[2 * kk2 + 1][1]);
            const uint32_t a3 = pack_bf16x2(s[2 * kk2 + 1][2], s[2 * kk2 + 1][3]);
#pragma unroll
            for (int dp = 0; dp < DV / 16; ++dp) {
                uint32_t b0, b1, b2, b3;
                const int row = 16 * kk2 + lr + 8 * (lj & 1);
                ldmatrix_x4_trans(b0, b1, b2, b3, sV + swz_off(row, 2 * dp + (lj >> 1), DV * 2));
                mma_bf16_16816(o[2 * dp], a0, a1, a2, a3, b0, b1);
                mma_bf16_16816(o[2 * dp + 1], a0, a1, a2, a3, b2, b3);
            }
        }
        __syncthreads();
    }
    cp_async_wait<0>();

#pragma unroll
    for (int r = 0; r < 2; ++r) {
        lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 1);
        lrow[r] += __shfl_xor_sync(0xffffffffu, lrow[r], 2);
    }
    __nv_bfloat16 *out = static_cast<__nv_bfloat16 *>(p.out);
#pragma unroll
    for (int r = 0; r < 2; ++r) {
        const int row = 16 * warp + g + 8 * r;
        if (row >= it.rows) continue;
        const int64_t tok = si.q_start + it.row_begin + row;
        const float inv = 1.f / lrow[r];
        __nv_bfloat16 *orow = out + (tok * p.num_q_heads + h) * DV;
#pragma unroll
        for (int nt = 0; nt < DV / 8; ++nt) {
            *reinterpret_cast<uint32_t *>(orow + nt * 8 + 2 * c) =
                pack_bf16x2(o[nt][2 * r] * inv, o[nt][2 * r + 1] * inv);
        }
        if (c == 0) p.lse[tok * p.num_q_heads + h] = (mrow[r] + log2f(lrow[r])) * kLn2;
    }
}

template <int DQ, int DV>
int launch_p(const AttnParams &p, cudaStream_t st) {
    using Cfg = PrefillCfg<DQ, DV>;
    if (cudaFuncSetAttribute(prefill_mma_kernel<DQ, DV>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             Cfg::kSmemBytes) != cudaSuccess)
        return FNPU_ECUDA;
    prefill_mma_kernel<DQ, DV><<<p.num_pitems, kThreads, Cfg::kSmemBytes, st>>>(p);
    return cudaGetLastError() == cudaSuccess ? FNPU_OK : FNPU_ECUDA;
}

}  // namespace

int launch_prefill_mma(const AttnParams &p, void *stream) {
    if (p.num_pitems == 0) return FNPU_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (p.head_dim_qk == 64 && p.head_dim_v == 64) return launch_p<64, 64>(p, st);
    if (p.head_dim_qk == 128 && p.head_dim_v == 128) return launch_p<128, 128>(p, st);
    // the per-head keys and values of a decompressed latent cache (MLA without absorption)
    if (p.head_dim_qk == 192 && p.head_dim_v == 128) return launch_p<192, 128>(p, st);
    return FNPU_EUNSUPPORTED;
}

}  // namespace fnpu
