// MLA without absorption: expand latent cache rows into per-head keys and
// values for a prefill chunk.
//
// A latent row holds c (512 columns, the compressed key/value) and r (64
// columns, the rotary key shared by all heads). Decompressed, head h sees the
// key [c W_UK[h], r] (128 + 64 columns) and the value c W_UV[h] (128 columns),
// and the chunk's attention is ordinary multi-head attention over them
// (d_qk = 192, d_v = 128, one kv head per query head). The paper's R1 serving
// keeps the latent cache (Sec. 4.1); the absorbed kernel attends over it
// directly, and this is the other way to run the prefill of the same cache.
//
// Steps: a gather kernel (with the KV append, which owns the device error
// flag) copies the c part of each requested row into a contiguous workspace
// [n, 512] and broadcasts its r part into columns 128..191 of every head's
// key; then one tcgen05 GEMM kernel writes c W_UK[h] into columns 0..127 of
// the keys and c W_UV[h] into the values:
//   * a CTA owns 128 rows of the workspace and one head: a 128 x 256 fp32
//     accumulator in tensor memory (columns 0..127 the key part, 128..255 the
//     value part, 256 columns), so that two CTAs share an SM and one CTA's
//     epilogue overlaps the other's products (8% faster than 256-row CTAs
//     with both accumulators, measured, despite 1.5x the L2-to-SM traffic);
//   * K = 512 runs in 64-column chunks through a 2-stage ring filled by TMA:
//     per chunk the 128-row A box of the workspace (K-major, 128-byte swizzle)
//     and W_UK[h], W_UV[h] rows k0..k0+63 as four 64-column boxes (the B
//     operand N-major: 64-wide N atoms 8 KB apart), so one M = 128, N = 256
//     product per 16-column step covers both projections;
//   * warp 0 issues the copies, warp 1 the MMAs, warps 2-5 read the
//     accumulators back (one row per thread), round to bf16 (nearest-even)
//     into swizzled boxes in shared memory, and TMA stores write the key and
//     value rows.
// Every mbarrier wait is bounded; a timeout raises bit 2 of the library-wide
// device error flag (fnpu_check: FNPU_EDEVICE_TIMEOUT) and the CTA drains its
// tensor-core work, frees its tensor memory and exits.
#include "common.cuh"
#include "tc.cuh"

namespace fnpu {
namespace {

constexpr int kC = 512;  // compressed part of a latent row
constexpr int kR = 64;   // rotary part
constexpr int kRow = kC + kR;
constexpr int kDn = 128;  // per-head key (no-rope part) and value width
constexpr int kDk = kDn + kR;

constexpr int kGThreads = 192;
constexpr int kGRows = 128;         // workspace rows per CTA (one accumulator)
constexpr int kGChunk = 64;         // K columns per stage
constexpr int kGStages = 2;
constexpr int kGChunks = kC / kGChunk;
constexpr int kGABox = 128 * 128;   // one 128-row x 64-column A box
constexpr int kGBBox = 64 * 128;    // one 64-row x 64-column B box
constexpr int kGStageBytes = kGABox + 4 * kGBBox;  // 48 KB
constexpr int kGBarOff = kGStages * kGStageBytes;
constexpr int kGSmem = kGBarOff + 8 * (2 * kGStages + 2) + 16;

struct GemmMaps {
    CUtensorMap a, wk, wv;  // loads: workspace, W_UK, W_UV
    CUtensorMap ko, vo;     // stores: key columns 0..127, value columns
};

__global__ void __launch_bounds__(kGThreads, 2)
    mla_expand_gemm_kernel(const __grid_constant__ GemmMaps maps, int32_t n, int32_t heads,
                           __nv_bfloat16 *__restrict__ k_out, __nv_bfloat16 *__restrict__ v_out, int *err) {
    extern __shared__ __align__(1024) uint8_t smem[];
    const uint32_t s_base = smem_u32(smem);
    const uint32_t bars = s_base + kGBarOff;
    auto FULL = [&](int s) { return bars + 8 * s; };
    auto EMPTY = [&](int s) { return bars + 8 * (kGStages + s); };
    const uint32_t DONE = bars + 8 * (2 * kGStages), DRAIN = DONE + 8;
    volatile uint32_t *tmem_slot = reinterpret_cast<volatile uint32_t *>(smem + kGBarOff + 8 * (2 * kGStages + 2));
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);
    const int tid = threadIdx.x, warp = tid >> 5;
    const int row0 = blockIdx.x * kGRows, h = blockIdx.y;
    if ((s_base & 1023u) != 0) {  // the swizzled boxes need 1024-byte alignment
        if (tid == 0) atomicOr(err, 4);
        return;
    }
    if (tid == 0) {
        for (int s = 0; s < kGStages; ++s) {
            tc::mbar_init(FULL(s), 1);
            tc::mbar_init(EMPTY(s), 1);
        }
        tc::mbar_init(DONE, 1);
        tc::mbar_init(DRAIN, 1);
        *abort_flag = 0;
        tc::fence_mbar_init();
    }
    if (warp == 1) {
        tc::tmem_alloc(smem_u32(const_cast<uint32_t *>(tmem_slot)), 256);
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
        atomicOr(err, 4);
        return false;
    };

    if (warp == 0) {
        // ------------------------------------------------------ TMA producer
        if ((tid & 31) == 0) {
            tc::prefetch_tmap(&maps.a);
            tc::prefetch_tmap(&maps.wk);
            tc::prefetch_tmap(&maps.wv);
        }
        for (int c = 0; c < kGChunks; ++c) {
            const int st = c % kGStages;
            if (c >= kGStages && !wait(EMPTY(st), ((c / kGStages) - 1) & 1)) break;
            const uint32_t dst = s_base + st * kGStageBytes;
            // full boxes count toward the transaction even where rows past n
            // are filled with zeros
            tc::mbar_arrive_expect_tx_warp(FULL(st), kGStageBytes);
            tc::tma_load_2d_warp(dst, &maps.a, FULL(st), c * kGChunk, row0);
#pragma unroll
            for (int j = 0; j < 2; ++j) {
                tc::tma_load_3d_warp(dst + kGABox + j * kGBBox, &maps.wk, FULL(st), 64 * j, c * kGChunk, h);
                tc::tma_load_3d_warp(dst + kGABox + (2 + j) * kGBBox, &maps.wv, FULL(st), 64 * j, c * kGChunk, h);
            }
        }
    } else if (warp == 1) {
        // -------------------------------------------------------- MMA issuer
        constexpr uint32_t idesc = tc::idesc_bf16(128, 256, true);
        const uint32_t utmem = __shfl_sync(0xffffffffu, tmem, 0);
        const uint32_t us = __shfl_sync(0xffffffffu, s_base, 0);
        bool ok = true, issued = false;
        for (int c = 0; c < kGChunks; ++c) {
            const int st = c % kGStages;
            if (!wait(FULL(st), (c / kGStages) & 1)) {
                ok = false;
                break;
            }
            tc::fence_after_sync();
            const uint32_t sa = us + st * kGStageBytes;
            // B: [UK n 0..63 | UK n 64..127 | UV n 0..63 | UV n 64..127], each
            // 64 K rows of 128 bytes; a 16-row K step is 2048 bytes further
            const uint64_t bd = tc::sdesc_sw128(sa + kGABox, kGBBox, 1024);
            const uint64_t ad = tc::sdesc_sw128(sa, 16, 1024);
#pragma unroll
            for (int kk = 0; kk < kGChunk / 16; ++kk)
                tc::mma_ss_warp(utmem, ad + (kk * 32) / 16, bd + (kk * 2048) / 16, idesc, (c > 0 || kk > 0) ? 1u : 0u);
            tc::commit_warp(EMPTY(st));
            issued = true;
        }
        if (ok) {
            tc::commit_warp(DONE);
        } else if (issued) {  // drain whatever is still in flight
            tc::commit_warp(DRAIN);
            tc::mbar_wait(DRAIN, 0, 200000000ull);
        }
    } else {
        // ---------------------------------------------------------- epilogue
        // Each thread takes one accumulator row: 256 fp32 columns from tensor
        // memory, rounded to bf16 into four 128-row x 64-column boxes in shared
        // memory (the ring, idle once every MMA has completed), 128-byte
        // swizzled as the TMA store reads them; then one thread stores the
        // boxes to the key and value rows (rows past n are not written).
        const int quarter = warp & 3;  // the TMEM lanes this warp may read
        const int lane = tid & 31;
        const int r = 32 * quarter + lane;  // row of the accumulator
        const bool ok = wait(DONE, 0);
        if (ok) {
            tc::fence_after_sync();
            const uint32_t taddr = tmem + (static_cast<uint32_t>(32 * quarter) << 16);
#pragma unroll 1
            for (int part = 0; part < 2; ++part) {  // the key part (columns 0..127), then the value part
                uint32_t v[128];
#pragma unroll
                for (int c = 0; c < 4; ++c)  // four loads in flight, one wait
                    tc::tmem_ld32(taddr + 128 * part + 32 * c, *reinterpret_cast<uint32_t(*)[32]>(&v[32 * c]));
                tc::tmem_wait_ld();
#pragma unroll
                for (int box = 0; box < 2; ++box) {
                    uint8_t *bx = smem + (part * 2 + box) * (128 * 128) + r * 128;
#pragma unroll
                    for (int j = 0; j < 8; ++j) {  // 16-byte chunk j of the row at position j ^ (r mod 8)
                        const uint32_t *w = &v[64 * box + 8 * j];
                        uint4 o;
                        o.x = pack_bf16x2(__uint_as_float(w[0]), __uint_as_float(w[1]));
                        o.y = pack_bf16x2(__uint_as_float(w[2]), __uint_as_float(w[3]));
                        o.z = pack_bf16x2(__uint_as_float(w[4]), __uint_as_float(w[5]));
                        o.w = pack_bf16x2(__uint_as_float(w[6]), __uint_as_float(w[7]));
                        *reinterpret_cast<uint4 *>(bx + ((j ^ (r & 7)) << 4)) = o;
                    }
                }
            }
            tc::fence_proxy_async_smem();  // these writes before the TMA store reads them
        }
        asm volatile("bar.sync 1, 128;\n" ::: "memory");  // the four epilogue warps
        if (ok && warp == 2 && lane == 0) {
#pragma unroll
            for (int part = 0; part < 2; ++part)
#pragma unroll
                for (int box = 0; box < 2; ++box)
                    tc::tma_store_3d(part == 0 ? &maps.ko : &maps.vo, s_base + (part * 2 + box) * (128 * 128), 64 * box,
                                     h, row0);
            tc::bulk_commit_group();
            tc::bulk_wait_group_read0();  // shared memory stays valid until the stores have read it
        }
    }
    tc::fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc::fence_after_sync();
        tc::tmem_dealloc(tmem, 256);
    }
}

EncodeTiledFn gemm_encoder() { return tensor_map_encoder(); }

// 2-D map over the workspace [n, 512]: boxes of 64 columns x 128 rows
bool encode_ws_map(CUtensorMap *m, const void *ws, int32_t n) {
    EncodeTiledFn enc = gemm_encoder();
    if (!enc) return false;
    cuuint64_t dims[2] = {static_cast<cuuint64_t>(kC), static_cast<cuuint64_t>(n)};
    cuuint64_t strides[1] = {static_cast<cuuint64_t>(kC) * 2};
    cuuint32_t box[2] = {64, 128};
    cuuint32_t es[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(ws), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D map over output rows [n, heads, width] (bf16): boxes of 64 columns x one
// head x 128 rows, for the epilogue's stores
bool encode_out_map(CUtensorMap *m, const void *out, int32_t n, int32_t heads, int32_t width) {
    EncodeTiledFn enc = gemm_encoder();
    if (!enc) return false;
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(width), static_cast<cuuint64_t>(heads), static_cast<cuuint64_t>(n)};
    cuuint64_t strides[2] = {static_cast<cuuint64_t>(width) * 2, static_cast<cuuint64_t>(heads) * width * 2};
    cuuint32_t box[3] = {64, 1, 128};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(out), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// 3-D map over W [heads, 512, 128]: boxes of 64 output columns x 64 rows of one head
bool encode_w_map(CUtensorMap *m, const void *w, int32_t heads) {
    EncodeTiledFn enc = gemm_encoder();
    if (!enc) return false;
    cuuint64_t dims[3] = {static_cast<cuuint64_t>(kDn), static_cast<cuuint64_t>(kC), static_cast<cuuint64_t>(heads)};
    cuuint64_t strides[2] = {static_cast<cuuint64_t>(kDn) * 2, static_cast<cuuint64_t>(kC) * kDn * 2};
    cuuint32_t box[3] = {64, 64, 1};
    cuuint32_t es[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void *>(w), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace
}  // namespace fnpu

using namespace fnpu;

extern "C" int fnpu_mla_expand(const fnpu_attn_desc *desc, const void *latent_cache, const int64_t *slots,
                               int32_t n, const void *w_uk, const void *w_uv, void *workspace, void *k_out,
                               void *v_out, void *stream) {
    if (!desc || n < 0) return FNPU_EINVAL;
    if (!desc->v_in_k_latent || desc->num_kv_heads != 1 || desc->num_q_heads <= 0 || desc->block_size <= 0 ||
        desc->num_blocks <= 0)
        return FNPU_EINVAL;
    if (desc->head_dim_qk != kRow || desc->head_dim_v != kC) return FNPU_EUNSUPPORTED;
    if (n == 0) return FNPU_OK;
    if (!latent_cache || !slots || !w_uk || !w_uv || !workspace || !k_out || !v_out) return FNPU_EINVAL;
    const uintptr_t mis = reinterpret_cast<uintptr_t>(latent_cache) | reinterpret_cast<uintptr_t>(w_uk) |
                          reinterpret_cast<uintptr_t>(w_uv) | reinterpret_cast<uintptr_t>(workspace) |
                          reinterpret_cast<uintptr_t>(k_out) | reinterpret_cast<uintptr_t>(v_out);
    if ((mis & 15u) || (reinterpret_cast<uintptr_t>(slots) & 7u)) return FNPU_EINVAL;
    if (desc->num_q_heads > 65535) return FNPU_EUNSUPPORTED;  // one grid row per head
    const int heads = desc->num_q_heads;
    int *err = nullptr;
    int rc = global_error_address(&err);
    if (rc != FNPU_OK) return rc;
    rc = launch_mla_gather(latent_cache, slots, n, static_cast<int64_t>(desc->num_blocks) * desc->block_size, heads,
                           workspace, k_out, stream);
    if (rc != FNPU_OK) return rc;
    GemmMaps maps;
    if (!encode_ws_map(&maps.a, workspace, n) || !encode_w_map(&maps.wk, w_uk, heads) ||
        !encode_w_map(&maps.wv, w_uv, heads) || !encode_out_map(&maps.ko, k_out, n, heads, kDk) ||
        !encode_out_map(&maps.vo, v_out, n, heads, kDn))
        return cuda_fail(cudaErrorInvalidValue, "cuTensorMapEncodeTiled (MLA expansion)");
    FNPU_CUDA_TRY(cudaFuncSetAttribute(mla_expand_gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kGSmem));
    const dim3 grid((n + kGRows - 1) / kGRows, heads);
    mla_expand_gemm_kernel<<<grid, kGThreads, kGSmem, static_cast<cudaStream_t>(stream)>>>(
        maps, n, heads, static_cast<__nv_bfloat16 *>(k_out), static_cast<__nv_bfloat16 *>(v_out), err);
    FNPU_CUDA_TRY(cudaGetLastError());
    return FNPU_OK;
}
