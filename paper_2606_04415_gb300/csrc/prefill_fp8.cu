// Prefill over the FP8 (e4m3) KV cache.
//
// Two ways. By default the plan stages an f16 copy of its prefill sequences'
// blocks (fp8_stage_kernel: code value x row scale, rounded once to f16)
// and of the queries, and the tcgen05 prefill kernel runs on those with f16
// operands. With FNPU_PLAN_NO_TCGEN05, prefill_fp8_kernel below reads the
// codes directly on f16 mma.sync.
//
// prefill_fp8_kernel: the chunk rows of a mixed step whose cache is stored in the library's FP8
// format (include/fnpu.h; Hkv = 4, d = 128, 16-slot blocks). The structure is
// the mma.sync prefill kernel's: one CTA computes 64 query rows of one query
// head, four warps own 16 rows each, 64-key tiles (four blocks) are staged
// with cp.async into a double-buffered ring, the online softmax runs in fp32
// registers. What differs:
//   * A stage holds the codes as stored: the head's 64 K rows (128 bytes each,
//     16-byte chunks swizzled by the row), its four V blocks ([128 columns][16
//     slots] each) and the blocks' K and V scale areas.
//   * The products run in f16 (e4m3 values are exact in f16; the query is
//     converted once). The column permutation of a stored K row puts the four
//     values a lane needs for one 16-column step of S = Q K^T (columns 2c,
//     2c+1, 2c+8, 2c+9 of key g) in four consecutive bytes, so a lane reads
//     its operands for a key with two 16-byte loads; the slot permutation of
//     a stored V column does the same for the keys of O += P V (one 4-byte
//     load per column and 16 keys). Four codes become two f16x2 operands with
//     two cvt instructions.
//   * The K scale of a key multiplies its scores after the product. The V
//     scale of a key, over vm (a power of two at or above every V scale seen
//     so far, rescaled exactly when it grows), multiplies its probability
//     before P V, so that the f16 operand stays at most 1.
//   * Keys past the sequence (the tail of its last block) have their V
//     operands set to zero in registers: stale slots may hold NaN codes.
#include <math.h>

#include "common.cuh"
#include "fp8.cuh"

namespace fnpu {
namespace {

constexpr int kThreads = 128;
constexpr int kRows = 64;
constexpr int kKeys = 64;  // four blocks of 16 slots
constexpr int kHkv = 4, kD = 128, kBs = 16;
constexpr int kCodeBytes = kBs * kHkv * kD;           // K or V codes of one block
constexpr int kBlockBytes = kCodeBytes + kBs * kHkv * 4;
constexpr int kQBytes = kRows * kD * 2;               // bf16 queries
constexpr int kKBytes = kKeys * kD;                   // the head's 64 K rows
constexpr int kVBytes = (kKeys / kBs) * kD * kBs;     // the head's four V blocks
constexpr int kSBytes = (kKeys / kBs) * kBs * kHkv * 4;  // four scale areas
constexpr int kStageBytes = kKBytes + kVBytes + 2 * kSBytes;
constexpr int kSmemBytes = kQBytes + 2 * kStageBytes;

__device__ __forceinline__ uint32_t swz_q(int row, int chunk) {
    return static_cast<uint32_t>(row * kD * 2 + ((chunk ^ (row & 7)) << 4));
}

__global__ void __launch_bounds__(kThreads, 2) prefill_fp8_kernel(const AttnParams p) {
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
    const uint8_t *kp = static_cast<const uint8_t *>(p.k_cache);
    const uint8_t *vp = static_cast<const uint8_t *>(p.v_cache);
    const int32_t *bt = p.block_table + static_cast<int64_t>(si.bt_row) * p.bt_stride;
    const uint32_t sQ = smem_u32(smem);

    for (int i = tid; i < kRows * (kD / 8); i += kThreads) {
        const int row = i / (kD / 8), ch = i % (kD / 8);
        const bool valid = row < it.rows;
        const int64_t tok = si.q_start + it.row_begin + (valid ? row : 0);
        cp_async_16(sQ + swz_q(row, ch), q + (tok * p.num_q_heads + h) * kD + ch * 8, valid);
    }
    // stage: K rows [64][128] (chunk ^ row & 7) | V blocks [4][128][16] | K scale areas [4][16][4] | V scale areas
    auto load_kv = [&](int tile, int stage) {
        const uint32_t sK = sQ + kQBytes + stage * kStageBytes;
        const uint32_t sV = sK + kKBytes, sKS = sV + kVBytes, sVS = sKS + kSBytes;
        for (int i = tid; i < kKeys * 8 + (kKeys / kBs) * (kD * kBs / 16) + 2 * (kKeys / kBs) * 16; i += kThreads) {
            int b, blk_i;
            if (i < kKeys * 8) {  // K: row (key) i / 8, chunk i % 8
                const int row = i >> 3, ch = i & 7;
                b = row >> 4;
                const int key0 = tile * kKeys + b * kBs;
                const bool valid = key0 < nkeys;
                blk_i = valid ? __ldg(bt + key0 / kBs) : 0;
                cp_async_16(sK + row * kD + ((ch ^ (row & 7)) << 4),
                            kp + static_cast<int64_t>(blk_i) * kBlockBytes + ((row & 15) * kHkv + kvh) * kD + ch * 16,
                            valid);
            } else if (i < kKeys * 8 + (kKeys / kBs) * (kD * kBs / 16)) {  // V: block, 16-byte chunk of the head's codes
                const int j = i - kKeys * 8;
                b = j >> 7;
                const int ch = j & 127;
                const int key0 = tile * kKeys + b * kBs;
                const bool valid = key0 < nkeys;
                blk_i = valid ? __ldg(bt + key0 / kBs) : 0;
                cp_async_16(sV + b * (kD * kBs) + ch * 16,
                            vp + static_cast<int64_t>(blk_i) * kBlockBytes + kvh * (kD * kBs) + ch * 16, valid);
            } else {  // scale areas: 16 chunks each, K then V
                const int j = i - kKeys * 8 - (kKeys / kBs) * (kD * kBs / 16);
                const int kv = j >> 6, jj = j & 63;
                b = jj >> 4;
                const int ch = jj & 15;
                const int key0 = tile * kKeys + b * kBs;
                const bool valid = key0 < nkeys;
                blk_i = valid ? __ldg(bt + key0 / kBs) : 0;
                cp_async_16((kv ? sVS : sKS) + b * 256 + ch * 16,
                            (kv ? vp : kp) + static_cast<int64_t>(blk_i) * kBlockBytes + kCodeBytes + ch * 16, valid);
            }
        }
    };
    load_kv(0, 0);
    cp_async_commit();

    float o[kD / 8][4];
#pragma unroll
    for (int nt = 0; nt < kD / 8; ++nt) o[nt][0] = o[nt][1] = o[nt][2] = o[nt][3] = 0.f;
    float mrow[2] = {-INFINITY, -INFINITY};
    float lrow[2] = {0.f, 0.f};
    float vm = 0.f;  // power of two at or above every V scale so far: o holds O / vm
    const int pr0 = pos_first + 16 * warp + g;  // position of row g; row g + 8 is pr0 + 8
    uint32_t qa[kD / 16][4];

    for (int tile = 0; tile < ntiles; ++tile) {
        if (tile + 1 < ntiles) load_kv(tile + 1, (tile + 1) & 1);
        cp_async_commit();
        cp_async_wait<1>();
        __syncthreads();
        if (tile == 0) {
#pragma unroll
            for (int kk = 0; kk < kD / 16; ++kk) {
                const int row = 16 * warp + lr + 8 * (lj & 1);
                ldmatrix_x4(qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], sQ + swz_q(row, 2 * kk + (lj >> 1)));
#pragma unroll
                for (int r = 0; r < 4; ++r) qa[kk][r] = bf16x2_to_f16x2(qa[kk][r]);
            }
        }
        const uint8_t *tK = smem + kQBytes + (tile & 1) * kStageBytes;
        const uint8_t *tV = tK + kKBytes;
        const float *ks = reinterpret_cast<const float *>(tV + kVBytes);  // [4 blocks][16 slots][4 heads]
        const float *vs = ks + (kKeys / kBs) * kBs * kHkv;
        const int kvalid = nkeys - tile * kKeys;  // keys of this tile inside the sequence (>= 1)

        // S = Q K^T: key group nt, key 8 nt + g of the B operand from its stored row
        float s[8][4];
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
            s[nt][0] = s[nt][1] = s[nt][2] = s[nt][3] = 0.f;
            const int row = 8 * nt + g;
            const uint4 x0 = *reinterpret_cast<const uint4 *>(tK + row * kD + (((2 * c) ^ (row & 7)) << 4));
            const uint4 x1 = *reinterpret_cast<const uint4 *>(tK + row * kD + (((2 * c + 1) ^ (row & 7)) << 4));
            const uint32_t kw[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
#pragma unroll
            for (int kk = 0; kk < kD / 16; ++kk) {
                uint32_t b0, b1;
                e4m3x4_to_f16x2x2(kw[kk], b0, b1);
                mma_f16_16816(s[nt], qa[kk][0], qa[kk][1], qa[kk][2], qa[kk][3], b0, b1);
            }
        }
        // K scales, causal mask at absolute positions, log2 units; the tile's V scales
        float tmax[2] = {-INFINITY, -INFINITY};
        float w[8][2];  // V scale of keys 8 nt + 2c, + 1 (0 past the sequence)
        float vt = 0.f;
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
            for (int e2 = 0; e2 < 2; ++e2) {
                const int key = nt * 8 + 2 * c + e2;
                const float ksc = ks[((key >> 4) * kBs + (key & 15)) * kHkv + kvh] * p.scale_log2;
                const float vsc = key < kvalid ? vs[((key >> 4) * kBs + (key & 15)) * kHkv + kvh] : 0.f;
                w[nt][e2] = vsc;
                vt = fmaxf(vt, vsc);
#pragma unroll
                for (int r = 0; r < 2; ++r) {
                    const int kabs = tile * kKeys + key;
                    const float x = (kabs <= pr0 + 8 * r) ? s[nt][2 * r + e2] * ksc : -INFINITY;
                    s[nt][2 * r + e2] = x;
                    tmax[r] = fmaxf(tmax[r], x);
                }
            }
        }
        vt = fmaxf(vt, __shfl_xor_sync(0xffffffffu, vt, 1));
        vt = fmaxf(vt, __shfl_xor_sync(0xffffffffu, vt, 2));  // every lane: the max over the tile's keys
        float rv = 1.f;
        if (vt > vm) {  // > 0: key 0 of a tile is inside the sequence and scales are positive
            const float vmn = pow2_ceil(vt);
            rv = vm * pow2_inverse(vmn);
            vm = vmn;
        }
        const float ivm = pow2_inverse(vm);
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
        const float ro0 = alpha[0] * rv, ro1 = alpha[1] * rv;
#pragma unroll
        for (int nt = 0; nt < kD / 8; ++nt) {
            o[nt][0] *= ro0; o[nt][1] *= ro0;
            o[nt][2] *= ro1; o[nt][3] *= ro1;
        }
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const float pv = fast_exp2(s[nt][e] - base[e >> 1]);
                lrow[e >> 1] += pv;
                s[nt][e] = pv * w[nt][e & 1] * ivm;  // the P V operand: p * vs / vm
            }
        }
        // O += P V over the tile's four 16-key blocks; V operands of keys
        // past the sequence zeroed (the last tile only)
#pragma unroll
        for (int kk2 = 0; kk2 < 4; ++kk2) {
            const uint32_t a0 = pack_f16x2(s[2 * kk2][0], s[2 * kk2][1]);
            const uint32_t a1 = pack_f16x2(s[2 * kk2][2], s[2 * kk2][3]);
            const uint32_t a2 = pack_f16x2(s[2 * kk2 + 1][0], s[2 * kk2 + 1][1]);
            const uint32_t a3 = pack_f16x2(s[2 * kk2 + 1][2], s[2 * kk2 + 1][3]);
            const int nv = kvalid - 16 * kk2;  // valid keys of this block (may be <= 0)
            const uint32_t lo_keep = (2 * c < nv ? 0x0000FFFFu : 0u) | (2 * c + 1 < nv ? 0xFFFF0000u : 0u);
            const uint32_t hi_keep = (2 * c + 8 < nv ? 0x0000FFFFu : 0u) | (2 * c + 9 < nv ? 0xFFFF0000u : 0u);
            const uint8_t *vb = tV + kk2 * (kD * kBs);
#pragma unroll
            for (int nt = 0; nt < kD / 8; ++nt) {
                uint32_t b0, b1;
                e4m3x4_to_f16x2x2(*reinterpret_cast<const uint32_t *>(vb + (8 * nt + g) * kBs + 4 * c), b0, b1);
                mma_f16_16816(o[nt], a0, a1, a2, a3, b0 & lo_keep, b1 & hi_keep);
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
        const float inv = vm / lrow[r];
        __nv_bfloat16 *orow = out + (tok * p.num_q_heads + h) * kD;
#pragma unroll
        for (int nt = 0; nt < kD / 8; ++nt)
            *reinterpret_cast<uint32_t *>(orow + nt * 8 + 2 * c) = pack_bf16x2(o[nt][2 * r] * inv, o[nt][2 * r + 1] * inv);
        if (c == 0) p.lse[tok * p.num_q_heads + h] = (mrow[r] + log2f(lrow[r])) * kLn2;
    }
}

// One staged block (a CTA): the 16 slots x 4 heads x 128 columns of K and of
// V of a source block, dequantised (code value x row scale, rounded to f16)
// into the plain cache layout [slot][head][column]; slots past `valid` are
// zero. K rows: a thread writes 16 columns from the four words that hold them
// (column 16 k + j at byte 32 c + 4 k + r); V: a thread reads one stored
// column (16 slots, 16 bytes; a warp reads 512 contiguous bytes) and writes
// its 16 values into their rows (a warp writes 64 contiguous bytes a row).
__device__ __forceinline__ void fp8_dequant_block(const uint8_t *__restrict__ kp, const uint8_t *__restrict__ vp,
                                                  const Fp8StageJob jb, uint4 *__restrict__ kd,
                                                  uint4 *__restrict__ vd) {
    const uint8_t *kb = kp + static_cast<int64_t>(jb.src) * kBlockBytes;
    const uint8_t *vb = vp + static_cast<int64_t>(jb.src) * kBlockBytes;
    const float *ksc = reinterpret_cast<const float *>(kb + kCodeBytes);
    const float *vsc = reinterpret_cast<const float *>(vb + kCodeBytes);
    uint4 *ko = kd + static_cast<int64_t>(jb.dst) * (kBs * kHkv * kD / 8);
    uint4 *vo = vd + static_cast<int64_t>(jb.dst) * (kBs * kHkv * kD / 8);
    auto scaled = [](uint32_t h2, float sc) {  // f16x2 * sc, rounded to f16x2
        const float2 f = __half22float2(*reinterpret_cast<const __half2 *>(&h2));
        return pack_f16x2(f.x * sc, f.y * sc);
    };
    for (int task = threadIdx.x; task < kBs * kHkv * 8; task += 128) {  // K: row (slot, head) x 16 columns
        const int row = task >> 3, cg = task & 7;
        uint4 a = make_uint4(0u, 0u, 0u, 0u), b = a;
        if ((row >> 2) < jb.valid) {
            const float sc = ksc[row];
            uint32_t lo[4], hi[4];
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                e4m3x4_to_f16x2x2(__ldg(reinterpret_cast<const uint32_t *>(kb + row * kD + 32 * c + 4 * cg)), lo[c], hi[c]);
                lo[c] = scaled(lo[c], sc);
                hi[c] = scaled(hi[c], sc);
            }
            a = make_uint4(lo[0], lo[1], lo[2], lo[3]);
            b = make_uint4(hi[0], hi[1], hi[2], hi[3]);
        }
        ko[row * (kD / 8) + 2 * cg] = a;
        ko[row * (kD / 8) + 2 * cg + 1] = b;
    }
    __half *vh = reinterpret_cast<__half *>(vo);
    for (int task = threadIdx.x; task < kHkv * kD; task += 128) {  // V: one stored column (head, d), 16 slots
        const int head = task >> 7, d = task & (kD - 1);
        const uint4 w = __ldg(reinterpret_cast<const uint4 *>(vb + head * (kD * kBs) + d * kBs));
        const uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int c = 0; c < 4; ++c) {  // word c: slots 2c, 2c + 1 (lo) and 2c + 8, 2c + 9 (hi)
            uint32_t lo, hi;
            e4m3x4_to_f16x2x2(ws[c], lo, hi);
            const float2 fl = __half22float2(*reinterpret_cast<const __half2 *>(&lo));
            const float2 fh = __half22float2(*reinterpret_cast<const __half2 *>(&hi));
            const int sl[4] = {2 * c, 2 * c + 1, 2 * c + 8, 2 * c + 9};
            const float f[4] = {fl.x, fl.y, fh.x, fh.y};
#pragma unroll
            for (int e = 0; e < 4; ++e) {
                const int o = sl[e];
                vh[(o * kHkv + head) * kD + d] =
                    __float2half_rn(o < jb.valid ? f[e] * vsc[o * kHkv + head] : 0.f);
            }
        }
    }
}

// The staging in one launch: CTAs below num_jobs dequantise one block each,
// the others convert the queries bf16 -> f16 (8 values per thread and step).
__global__ void __launch_bounds__(128) fp8_stage_kernel(const uint8_t *__restrict__ kp, const uint8_t *__restrict__ vp,
                                                        const Fp8StageJob *__restrict__ jobs, int32_t num_jobs,
                                                        uint4 *__restrict__ kd, uint4 *__restrict__ vd,
                                                        const uint4 *__restrict__ qin, uint4 *__restrict__ qout,
                                                        int64_t n8) {
    if (static_cast<int32_t>(blockIdx.x) < num_jobs) {
        fp8_dequant_block(kp, vp, jobs[blockIdx.x], kd, vd);
        return;
    }
    const int64_t nq = static_cast<int64_t>(gridDim.x) - num_jobs;
    for (int64_t i = (static_cast<int64_t>(blockIdx.x) - num_jobs) * blockDim.x + threadIdx.x; i < n8;
         i += nq * blockDim.x) {
        const uint4 v = __ldg(qin + i);
        qout[i] = make_uint4(bf16x2_to_f16x2(v.x), bf16x2_to_f16x2(v.y), bf16x2_to_f16x2(v.z), bf16x2_to_f16x2(v.w));
    }
}

}  // namespace

int launch_fp8_stage(const void *k_pool, const void *v_pool, const Fp8StageJob *jobs, int32_t num_jobs, void *k_f16,
                     void *v_f16, const void *q_bf16, void *q_f16, int64_t q_values, void *stream) {
    const int64_t n8 = q_values / 8;
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t want = (n8 + 127) / 128;
    const int64_t qctas = want < 4LL * sms ? want : 4LL * sms;
    if (num_jobs + qctas == 0) return FNPU_OK;
    fp8_stage_kernel<<<static_cast<int>(num_jobs + qctas), 128, 0, static_cast<cudaStream_t>(stream)>>>(
        static_cast<const uint8_t *>(k_pool), static_cast<const uint8_t *>(v_pool), jobs, num_jobs,
        static_cast<uint4 *>(k_f16), static_cast<uint4 *>(v_f16), static_cast<const uint4 *>(q_bf16),
        static_cast<uint4 *>(q_f16), n8);
    FNPU_CUDA_TRY(cudaGetLastError());
    return FNPU_OK;
}

int launch_prefill_fp8(const AttnParams &p, void *stream) {
    if (p.num_pitems == 0) return FNPU_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    FNPU_CUDA_TRY(cudaFuncSetAttribute(prefill_fp8_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes));
    prefill_fp8_kernel<<<p.num_pitems, kThreads, kSmemBytes, st>>>(p);
    FNPU_CUDA_TRY(cudaGetLastError());
    return FNPU_OK;
}

}  // namespace fnpu
