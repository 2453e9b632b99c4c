// Absorbed multi-head latent attention (MLA, the DeepSeek-R1 shape) on the
// fifth-generation tensor cores: every query head reads one shared latent
// cache row of d_qk = 576 values per key, and V is its first d_v = 512 values
// (Eq. 1 with K = latent, V = latent[:, :512]). Prefill and decode rows share
// the kernel: the 128 heads of one query token are the 128 rows of a tile, so
// the phase only changes how many keys a token sees.
//
// The fp32 accumulator of 128 rows x 512 columns would fill all of tensor
// memory, so one work item is (token, half of d_v, key range) and two CTAs
// take the two halves of a token; both compute the same S = Q K^T (the
// product is 1.5x the minimum, against none of the accumulator fitting
// otherwise) and each keeps O for its 256 columns. Both halves read the same
// latent tiles at about the same time (they are neighbours in the work list),
// so the second read is served by L2.
//
// Tensor memory (512 columns): O half [0, 256), S [256, 320) with P (bf16)
// written over its first 32 columns, and Q columns 192..575 as packed bf16
// pairs [320, 512), the A operand of 24 of the 36 k-steps of S. Q columns
// 0..191 sit in shared memory for the other 12 steps, beside a two-stage ring
// of 64-key latent tiles (nine 64-column chunks, 128-byte swizzle), which
// also serve as the V operand of P V (chunks 4h..4h+3 for half h).
//
// Warps 0-3: softmax and epilogue, one row each (TMEM lane = head). Warp 4:
// TMA producer. Warp 5: MMA issuer, which issues P V of tile j - 1 before S
// of tile j, so the in-order tensor pipe never overwrites P before it is
// read and the lazy O rescale (only when the row maximum grows by more than
// 2^8) happens while no product is writing O.
#include <math.h>

#include "common.cuh"
#include "tc.cuh"

namespace fnpu {
namespace {

constexpr int kDq = 576, kDv = 512, kDvHalf = 256;
constexpr int kRows = 128;                    // heads of one token = TMEM lanes
constexpr int kKeysT = 64;                    // keys per latent tile
constexpr int kNChunk = kDq / 64;             // 64-column chunks per latent row
constexpr int kQsChunks = 3;                  // Q chunks in shared memory (columns 0..191)
constexpr int kQsSteps = kQsChunks * 4;       // k-steps of 16 columns with A in shared memory
constexpr int kSteps = kDq / 16;              // 36
constexpr int kThreads = 192;
constexpr int kStages = 2;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kColO = 0, kColS = 256, kColQ = 320;
constexpr float kRescaleThreshold = 8.0f;     // log2 units

constexpr int kChunkBytes = kKeysT * 128;             // 8 KB
constexpr int kTileBytes = kNChunk * kChunkBytes;      // 72 KB
constexpr int kQChunkBytes = kRows * 128;             // 16 KB
constexpr int kOffQ = 0;
constexpr int kOffKV = kQsChunks * kQChunkBytes;
constexpr int kOffBar = kOffKV + kStages * kTileBytes;
// full[2] empty[2] sfull pready odone qfull qready drain
constexpr int kNumBars = 2 * kStages + 6;
constexpr int kSmemBytes = kOffBar + 8 * kNumBars + 16;
static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
static_assert(kColQ + (kDq - 64 * kQsChunks) / 2 == kTmemCols, "tensor memory budget");

struct MlaMaps {
    CUtensorMap kv, q;
};

__global__ void __launch_bounds__(kThreads, 1) mla_tc_kernel(const AttnParams p, const __grid_constant__ MlaMaps maps) {
    extern __shared__ __align__(1024) uint8_t smem[];
    const uint32_t s_base = smem_u32(smem);
    const uint32_t bars = s_base + kOffBar;
    auto FULL = [&](int s) { return bars + 8 * s; };
    auto EMPTY = [&](int s) { return bars + 8 * (kStages + s); };
    const uint32_t SFULL = bars + 8 * (2 * kStages);
    const uint32_t PREADY = SFULL + 8, ODONE = SFULL + 16, QFULL = SFULL + 24, QREADY = SFULL + 32,
                   DRAIN = SFULL + 40;
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(smem + kOffBar + 8 * kNumBars);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(smem + kOffBar + 8 * kNumBars + 4);

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const MlaItem it = p.mitems[blockIdx.x];
    const SeqInfo si = p.seqs[it.seq];
    const int half = it.hb;  // d_v columns 256 half .. 256 half + 255
    const int64_t tok = si.q_start + it.row;
    const int kb = it.key_begin, ke = it.key_end;  // kb is a multiple of 64
    const int n = (ke - kb + kKeysT - 1) / kKeysT;
    if ((s_base & 1023u) != 0) {  // the swizzled tiles need 1024-byte alignment
        if (tid == 0) atomicOr(p.err, 2);
        return;
    }
    // Q columns 192..575 of this head (softmax warps), loaded before the
    // set-up so that their memory latency overlaps it: all 48 16-byte loads
    // in flight at once
    constexpr int kQtLoads = (kTmemCols - kColQ) * 4 / 16;  // 48
    uint4 qv[kQtLoads];
    if (warp < 4) {
        const uint4 *qrow = reinterpret_cast<const uint4 *>(static_cast<const __nv_bfloat16 *>(p.q) +
                                                            (tok * kRows + tid) * kDq + 64 * kQsChunks);
#pragma unroll
        for (int u = 0; u < kQtLoads; ++u) qv[u] = __ldg(qrow + u);
    }
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            tc::mbar_init(FULL(s), 1);
            tc::mbar_init(EMPTY(s), 1);
        }
        tc::mbar_init(SFULL, 1);
        tc::mbar_init(PREADY, kRows);
        tc::mbar_init(ODONE, 1);
        tc::mbar_init(QFULL, 1);
        tc::mbar_init(QREADY, kRows);
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
        if (tc::mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if (tc::mbar_wait(bar, parity)) return true;
        *abort_flag = 1;
        atomicOr(p.err, 1);
        return false;
    };

    if (warp == 4) {
        // ------------------------------------------------------ TMA producer
        if (lane == 0) {
            tc::prefetch_tmap(&maps.kv);
            tc::prefetch_tmap(&maps.q);
        }
        tc::mbar_arrive_expect_tx_warp(QFULL, kQsChunks * kQChunkBytes);
#pragma unroll
        for (int c = 0; c < kQsChunks; ++c)
            tc::tma_load_3d_warp(s_base + kOffQ + c * kQChunkBytes, &maps.q, QFULL, 64 * c, 0, static_cast<int>(tok));
        const int bs = p.block_size;
        const int per_tile = kKeysT / bs;  // blocks per tile (1, 2 or 4)
        const int32_t *bt = p.block_table + static_cast<int64_t>(si.bt_row) * p.bt_stride;
        const int nblk_seq = (si.ctx_len + bs - 1) / bs;
        int j = 0;
        for (; j < n; ++j) {
            const int st = j % kStages;
            if (j >= kStages && !wait(EMPTY(st), ((j / kStages) - 1) & 1)) break;
            const int b0 = (kb + j * kKeysT) / bs;
            int nvalid = nblk_seq - b0;
            nvalid = nvalid > per_tile ? per_tile : nvalid;
            const int blk_lane = lane < nvalid ? __ldg(bt + b0 + lane) : 0;
            tc::mbar_arrive_expect_tx_warp(FULL(st), static_cast<uint32_t>(nvalid * bs * 128 * kNChunk));
            for (int b = 0; b < nvalid; ++b) {
                const int blk = __shfl_sync(0xffffffffu, blk_lane, b);
#pragma unroll
                for (int c = 0; c < kNChunk; ++c)
                    tc::tma_load_3d_warp(s_base + kOffKV + st * kTileBytes + c * kChunkBytes + b * bs * 128, &maps.kv,
                                         FULL(st), 64 * c, 0, blk);
            }
        }
        if (j < n) {
            // gave up: let the copies already issued land before the CTA
            // leaves (bounded), so that none writes into a later CTA
            for (int jj = (j - kStages > 0 ? j - kStages : 0); jj < j; ++jj)
                tc::mbar_wait(FULL(jj % kStages), (jj / kStages) & 1, 200000000ull);
        }
    } else if (warp == 5) {
        // -------------------------------------------------------- MMA issuer
        constexpr uint32_t idS = tc::idesc_bf16(kRows, kKeysT, false);
        constexpr uint32_t idO = tc::idesc_bf16(kRows, kDvHalf, true);
        const uint32_t utmem = __shfl_sync(0xffffffffu, tmem, 0);
        const uint32_t us = __shfl_sync(0xffffffffu, s_base, 0);
        const uint32_t tS = utmem + kColS, tO = utmem + kColO, tQ = utmem + kColQ;
        const uint64_t qd = tc::sdesc_sw128(us + kOffQ, 16, 1024);
        bool ok = wait(QFULL, 0) && wait(QREADY, 0);
        bool issued = false;
        for (int j = 0; ok && j <= n; ++j) {
            if (j > 0) {
                // O += P(j - 1) V(j - 1)
                if (!wait(PREADY, (j - 1) & 1)) { ok = false; break; }
                tc::fence_after_sync();
                const int st = (j - 1) % kStages;
                const uint64_t vd =
                    tc::sdesc_sw128(us + kOffKV + st * kTileBytes + half * 4 * kChunkBytes, kChunkBytes, 1024);
#pragma unroll
                for (int kk = 0; kk < kKeysT / 16; ++kk)
                    tc::mma_ts_warp(tO, tS + kk * 8, vd + (kk * 2048) / 16, idO, (j > 1 || kk > 0) ? 1u : 0u);
                tc::commit_warp(EMPTY(st));
                if (j == n) {
                    tc::commit_warp(ODONE);
                    break;
                }
            }
            // S(j) = Q K(j)^T over the 36 k-steps of d_qk
            const int st = j % kStages;
            if (!wait(FULL(st), (j / kStages) & 1)) { ok = false; break; }
            tc::fence_after_sync();
            const uint64_t kd = tc::sdesc_sw128(us + kOffKV + st * kTileBytes, 16, 1024);
#pragma unroll
            for (int kk = 0; kk < kQsSteps; ++kk)
                tc::mma_ss_warp(tS, qd + ((kk / 4) * kQChunkBytes + (kk % 4) * 32) / 16,
                                kd + ((kk / 4) * kChunkBytes + (kk % 4) * 32) / 16, idS, kk > 0 ? 1u : 0u);
#pragma unroll
            for (int kk = kQsSteps; kk < kSteps; ++kk)
                tc::mma_ts_warp(tS, tQ + (kk - kQsSteps) * 8, kd + ((kk / 4) * kChunkBytes + (kk % 4) * 32) / 16, idS,
                                1u);
            tc::commit_warp(SFULL);
            issued = true;
        }
        if (!ok && issued) {  // drain whatever is still in flight
            tc::commit_warp(DRAIN);
            tc::mbar_wait(DRAIN, 0, 200000000ull);
        }
    } else {
        // ------------------------------------------- softmax / epilogue rows
        const int r = tid;  // head = TMEM lane
        const uint32_t lane_addr = tmem + (static_cast<uint32_t>(warp * 32) << 16);
        const float sc = p.scale_log2;
        // Q columns 192..575 of this head, packed in bf16 pairs, into tensor
        // memory (the A operand of the TS steps of S)
        {
#pragma unroll
            for (int c = 0; c < (kTmemCols - kColQ) / 32; ++c) {
                uint32_t v[32];
#pragma unroll
                for (int u = 0; u < 8; ++u) {
                    const uint4 x = qv[c * 8 + u];
                    v[4 * u] = x.x; v[4 * u + 1] = x.y; v[4 * u + 2] = x.z; v[4 * u + 3] = x.w;
                }
                tc::tmem_st32(lane_addr + kColQ + 32 * c, v);
            }
            tc::tmem_wait_st();
            tc::fence_before_sync();
            tc::mbar_arrive(QREADY);
        }
        float m_run = -INFINITY, l = 0.f;
        bool ok = true;
        for (int j = 0; j < n; ++j) {
            if (!wait(SFULL, j & 1)) { ok = false; break; }
            tc::fence_after_sync();
            uint32_t s[kKeysT];
            tc::tmem_ld32(lane_addr + kColS, *reinterpret_cast<uint32_t(*)[32]>(&s[0]));
            tc::tmem_ld32(lane_addr + kColS + 32, *reinterpret_cast<uint32_t(*)[32]>(&s[32]));
            tc::tmem_wait_ld();
            const int nv = ke - (kb + j * kKeysT);  // keys of this tile inside the item (>= 1)
            if (nv < kKeysT) {
#pragma unroll
                for (int x = 0; x < kKeysT; ++x)
                    if (x >= nv) s[x] = __float_as_uint(-INFINITY);
            }
            float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
            for (int x = 0; x < kKeysT; x += 4) {
                mx0 = fmax3(mx0, __uint_as_float(s[x]), __uint_as_float(s[x + 1]));
                mx1 = fmax3(mx1, __uint_as_float(s[x + 2]), __uint_as_float(s[x + 3]));
            }
            const float tmax = fmaxf(mx0, mx1) * sc;  // finite: the tile has a visible key
            const bool need = m_run == -INFINITY || tmax > m_run + kRescaleThreshold;
            // tensor-memory loads and stores are warp-wide: the warp rescales
            // together, lanes that need none with alpha = 1
            if (__any_sync(0xffffffffu, need)) {
                const float m_new = need ? fmaxf(m_run, tmax) : m_run;
                if (j > 0) {
                    // P V(j - 1) is complete: S(j) was issued after it
                    const float alpha = need ? fast_exp2(m_run - m_new) : 1.f;
#pragma unroll 1
                    for (int c = 0; c < kDvHalf / 32; ++c) {
                        uint32_t o[32];
                        tc::tmem_ld32(lane_addr + kColO + 32 * c, o);
                        tc::tmem_wait_ld();
#pragma unroll
                        for (int x = 0; x < 32; ++x) o[x] = __float_as_uint(__uint_as_float(o[x]) * alpha);
                        tc::tmem_st32(lane_addr + kColO + 32 * c, o);
                    }
                    l *= alpha;
                }
                m_run = m_new;
            }
            const uint64_t sc2 = f2_pack(sc, sc), nb2 = f2_pack(-m_run, -m_run);
            uint64_t lacc0 = f2_pack(0.f, 0.f), lacc1 = lacc0;
#pragma unroll
            for (int q4 = 0; q4 < kKeysT / 32; ++q4) {
                uint32_t pk[16];
#pragma unroll
                for (int x = 0; x < 16; ++x) {
                    const uint64_t x2 = f2_fma(
                        f2_pack(__uint_as_float(s[32 * q4 + 2 * x]), __uint_as_float(s[32 * q4 + 2 * x + 1])), sc2, nb2);
                    float x0, x1;
                    f2_unpack(x2, x0, x1);
                    const float p0 = fast_exp2(x0), p1 = fast_exp2(x1);
                    if (x & 1) lacc1 = f2_add(lacc1, f2_pack(p0, p1));
                    else lacc0 = f2_add(lacc0, f2_pack(p0, p1));
                    pk[x] = pack_bf16x2(p0, p1);
                }
                tc::tmem_st16(lane_addr + kColS + 16 * q4, pk);
            }
            {
                float a0, a1;
                f2_unpack(f2_add(lacc0, lacc1), a0, a1);
                l += a0 + a1;
            }
            if (nv < kKeysT) {
                // rows past the item hold keys of the next piece or stale slots:
                // zero this half's V columns there (their P is 0, but 0 * NaN is not)
                uint8_t *vt = smem + kOffKV + (j % kStages) * kTileBytes + half * 4 * kChunkBytes;
                for (int e = r; e < (kKeysT - nv) * 4 * 8; e += kRows) {
                    const int row = nv + e / 32, rem = e % 32;
                    *reinterpret_cast<uint4 *>(vt + (rem / 8) * kChunkBytes + row * 128 + (rem % 8) * 16) =
                        make_uint4(0u, 0u, 0u, 0u);
                }
                tc::fence_proxy_async_smem();
            }
            tc::tmem_wait_st();
            tc::fence_before_sync();
            tc::mbar_arrive(PREADY);
        }
        if (ok && wait(ODONE, 0)) {
            tc::fence_after_sync();
            const float inv = 1.f / l;
            const int ns = it.num_splits;
            if (ns == 1) {
                uint4 *orow = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(p.out) +
                                                        (tok * kRows + r) * kDv + kDvHalf * half);
#pragma unroll 1
                for (int c = 0; c < kDvHalf / 32; ++c) {
                    uint32_t o[32];
                    tc::tmem_ld32(lane_addr + kColO + 32 * c, o);
                    tc::tmem_wait_ld();
#pragma unroll
                    for (int x = 0; x < 2; ++x) {  // 32-byte stores: whole sectors of this row
                        uint32_t v[8];
#pragma unroll
                        for (int y = 0; y < 8; ++y)
                            v[y] = pack_bf16x2(__uint_as_float(o[16 * x + 2 * y]) * inv,
                                               __uint_as_float(o[16 * x + 2 * y + 1]) * inv);
                        st_global_v8(orow + c * 4 + 2 * x, v[0], v[1], v[2], v[3], v[4], v[5], v[6], v[7]);
                    }
                }
                if (half == 0) p.lse[tok * kRows + r] = (m_run + log2f(l)) * kLn2;
            } else {
                // a key split: O / l over its keys and m + log2 l (the partial
                // of Eq. 1), merged by the split-merge kernel
                const int64_t prow = static_cast<int64_t>(it.part_base + it.split) * kRows + r;
                float4 *po = reinterpret_cast<float4 *>(p.part_o + prow * kDv + kDvHalf * half);
#pragma unroll 1
                for (int c = 0; c < kDvHalf / 32; ++c) {
                    uint32_t o[32];
                    tc::tmem_ld32(lane_addr + kColO + 32 * c, o);
                    tc::tmem_wait_ld();
#pragma unroll
                    for (int x = 0; x < 8; ++x)
                        po[c * 8 + x] = make_float4(__uint_as_float(o[4 * x]) * inv, __uint_as_float(o[4 * x + 1]) * inv,
                                                    __uint_as_float(o[4 * x + 2]) * inv, __uint_as_float(o[4 * x + 3]) * inv);
                }
                if (half == 0) p.part_lse[prow] = m_run + log2f(l);
            }
        }
    }

    tc::fence_before_sync();
    __syncthreads();
    if (warp == 0) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, kTmemCols);
    }
}

// 3-D map, 64 columns by `rows` rows by 1, 128-byte swizzle: over the latent
// cache [blocks, bs, 576] (box = one block) or over Q [T, 128, 576] (box = one
// token's 128 heads).
bool encode_rows_map(CUtensorMap *m, const void *base, int64_t row_stride_elems, int rows, int64_t outer) {
    EncodeTiledFn enc = tensor_map_encoder();
    if (!enc) return false;
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(kDq), static_cast<cuuint64_t>(rows), static_cast<cuuint64_t>(outer)};
    cuuint64_t strides[2] = {static_cast<cuuint64_t>(row_stride_elems) * 2,
                             static_cast<cuuint64_t>(row_stride_elems) * 2 * rows};
    cuuint32_t box[3] = {64, static_cast<cuuint32_t>(rows), 1};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(base), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

bool mla_tc_supported(int d_qk, int d_v, int hq, int hkv, int block_size) {
    return d_qk == kDq && d_v == kDv && hkv == 1 && hq == kRows &&
           (block_size == 16 || block_size == 32 || block_size == 64);
}

int mla_tc_keys_per_tile() { return kKeysT; }

int launch_mla_tc(const AttnParams &p, void *stream) {
    if (p.num_mitems == 0) return FNPU_OK;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (p.k_slot_stride % 8 != 0) return FNPU_EUNSUPPORTED;  // TMA strides are multiples of 16 bytes
    MlaMaps maps;
    if (!encode_rows_map(&maps.kv, p.k_cache, p.k_slot_stride, p.block_size, p.num_blocks) ||
        !encode_rows_map(&maps.q, p.q, kDq, kRows, p.num_tokens))
        return cuda_fail(cudaErrorInvalidValue, "cuTensorMapEncodeTiled (latent)");
    FNPU_CUDA_TRY(cudaFuncSetAttribute(mla_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes));
    FNPU_CUDA_TRY(launch_ex(mla_tc_kernel, p.num_mitems, kThreads, kSmemBytes, st, false, nullptr, p, maps));
    return launch_split_merge(p, stream);
}

}  // namespace fnpu
