// KV append: scatter the step's new K/V rows into their paged slots.
//
// The new tokens of a step must be in the cache before the step's attention
// reads it (prefill and decode share one KV pool, Sec. 3.4). A slot row is
// contiguous (Hkv*d bf16 values, or d_qk for the latent cache), so each
// thread moves one 16-byte chunk and consecutive threads cover consecutive
// chunks of the same row: fully coalesced 16-B loads and stores. Pure copy,
// bit-exact.
#include <cuda_fp8.h>

#include <mutex>

#include "common.cuh"

namespace fnpu {

// Library-wide device error flag, one per device that loads the library;
// read and cleared by fnpu_check(). Bit 0: an append met an out-of-range
// slot; bit 1: the allocation-free decode met a context length or a block
// id out of range.
__device__ int g_device_error = 0;

__global__ void __launch_bounds__(256) kv_append_kernel(
    const uint4 *__restrict__ k_new, const uint4 *__restrict__ v_new,
    const int64_t *__restrict__ slots, int32_t num_tokens, int32_t k_chunks, int32_t v_chunks,
    uint4 *__restrict__ k_cache, uint4 *__restrict__ v_cache, int64_t num_slots) {
    pdl_trigger();  // a dependent launch after this one may start its set-up now
    const int32_t per_tok = k_chunks + v_chunks;
    const int64_t total = static_cast<int64_t>(num_tokens) * per_tok;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        int64_t t;
        int32_t c;
        if (total < (1LL << 31)) {  // 32-bit division at step sizes
            const uint32_t t32 = static_cast<uint32_t>(i) / static_cast<uint32_t>(per_tok);
            t = t32;
            c = static_cast<int32_t>(static_cast<uint32_t>(i) - t32 * static_cast<uint32_t>(per_tok));
        } else {
            t = i / per_tok;
            c = static_cast<int32_t>(i - t * per_tok);
        }
        // the new row and its slot are independent loads: both in flight at once
        const bool is_k = c < k_chunks;
        const int32_t cv = c - k_chunks;
        const uint4 v = is_k ? __ldg(k_new + t * k_chunks + c) : __ldg(v_new + t * v_chunks + cv);
        const int64_t s = __ldg(slots + t);
        if (s < 0) continue;
        if (s >= num_slots) {
            if (c == 0) atomicOr(&g_device_error, 1);
            continue;
        }
        if (is_k) k_cache[s * k_chunks + c] = v;
        else v_cache[s * v_chunks + cv] = v;
    }
}

namespace {

// byte position of column `col` of a stored fp8 K row, and of slot `o` of a
// stored fp8 V column (the four operands of one lane of a 16x8x16 product
// in four consecutive bytes)
__device__ __forceinline__ int fp8_kpos(int col) {
    const int k = col >> 4, j = col & 15;
    return 32 * ((j & 7) >> 1) + 4 * k + (j & 1) + 2 * (j >> 3);
}
__device__ __forceinline__ int fp8_vpos(int o) { return 4 * ((o & 7) >> 1) + (o & 1) + 2 * (o >> 3); }

// two e4m3 codes (low byte first) of two fp32 values, nearest with ties to
// even, saturating at 448; a zero code is stored positive
__device__ __forceinline__ uint32_t e4m3x2(float lo, float hi) {
    uint32_t c = __nv_cvt_float2_to_fp8x2(make_float2(lo, hi), __NV_SATFINITE, __NV_E4M3);
    if ((c & 0x7Fu) == 0) c &= 0xFF00u;
    if ((c & 0x7F00u) == 0) c &= 0x00FFu;
    return c;
}

constexpr int kF8Hkv = 4, kF8D = 128, kF8Bs = 16;
constexpr int kF8Codes = kF8Bs * kF8Hkv * kF8D;       // codes of one block (K or V)
constexpr int kF8Block = kF8Codes + kF8Bs * kF8Hkv * 4;  // + fp32 scales [bs][Hkv]

}  // namespace

// FP8 (e4m3) append, one warp per (token, K or V, kv head) row of 128 values:
// the row's absolute maximum sets its scale (amax / 448, 1 for a zero row),
// each value is stored as the code of value / scale. K rows keep the slot-major
// layout with permuted columns; V rows are scattered into the transposed
// [head][column][slot] layout. Bit-exact with IEEE fp32 division.
__global__ void __launch_bounds__(256) kv_append_fp8_kernel(
    const uint2 *__restrict__ k_new, const uint2 *__restrict__ v_new, const int64_t *__restrict__ slots,
    int32_t num_tokens, uint8_t *__restrict__ k_pool, uint8_t *__restrict__ v_pool, int64_t num_slots) {
    const int lane = threadIdx.x & 31;
    const int64_t nrows = static_cast<int64_t>(num_tokens) * 2 * kF8Hkv;
    const int64_t step = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
    for (int64_t r = (blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x) >> 5; r < nrows; r += step) {
        const int64_t t = r / (2 * kF8Hkv);
        const int kv = static_cast<int>(r / kF8Hkv) & 1, h = static_cast<int>(r % kF8Hkv);
        const uint2 raw = __ldg((kv ? v_new : k_new) + (t * kF8Hkv + h) * (kF8D / 4) + lane);
        const int64_t s = __ldg(slots + t);
        if (s < 0) continue;  // warp-uniform: one row per warp
        if (s >= num_slots) {
            if (lane == 0 && r % (2 * kF8Hkv) == 0) atomicOr(&g_device_error, 1);
            continue;
        }
        const float x0 = __uint_as_float(raw.x << 16), x1 = __uint_as_float(raw.x & 0xFFFF0000u);
        const float x2 = __uint_as_float(raw.y << 16), x3 = __uint_as_float(raw.y & 0xFFFF0000u);
        float a = fmaxf(fmaxf(fabsf(x0), fabsf(x1)), fmaxf(fabsf(x2), fabsf(x3)));
#pragma unroll
        for (int m = 16; m > 0; m >>= 1) a = fmaxf(a, __shfl_xor_sync(0xffffffffu, a, m));
        const float scale = a > 0.f ? a / 448.f : 1.f;
        const uint32_t c01 = e4m3x2(x0 / scale, x1 / scale), c23 = e4m3x2(x2 / scale, x3 / scale);
        const int o = static_cast<int>(s % kF8Bs);
        uint8_t *blk = (kv ? v_pool : k_pool) + (s / kF8Bs) * kF8Block;
        if (kv == 0) {  // columns 4 lane .. 4 lane + 3: two pairs of adjacent bytes
            uint8_t *row = blk + (o * kF8Hkv + h) * kF8D;
            *reinterpret_cast<uint16_t *>(row + fp8_kpos(4 * lane)) = static_cast<uint16_t>(c01);
            *reinterpret_cast<uint16_t *>(row + fp8_kpos(4 * lane + 2)) = static_cast<uint16_t>(c23);
        } else {
            uint8_t *col = blk + (h * kF8D + 4 * lane) * kF8Bs + fp8_vpos(o);
            col[0] = static_cast<uint8_t>(c01);
            col[kF8Bs] = static_cast<uint8_t>(c01 >> 8);
            col[2 * kF8Bs] = static_cast<uint8_t>(c23);
            col[3 * kF8Bs] = static_cast<uint8_t>(c23 >> 8);
        }
        if (lane == 0) *reinterpret_cast<float *>(blk + kF8Codes + (o * kF8Hkv + h) * 4) = scale;
    }
}

int launch_kv_append_fp8(const fnpu_attn_desc *d, const void *k_new, const void *v_new, const int64_t *slots,
                         int32_t num_tokens, void *k_cache, void *v_cache, void *stream) {
    if (num_tokens == 0) return FNPU_OK;
    const int64_t warps = static_cast<int64_t>(num_tokens) * 2 * kF8Hkv;
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t want = (warps + 7) / 8;
    const int grid = static_cast<int>(want < 32LL * sms ? want : 32LL * sms);
    kv_append_fp8_kernel<<<grid, 256, 0, static_cast<cudaStream_t>(stream)>>>(
        static_cast<const uint2 *>(k_new), static_cast<const uint2 *>(v_new), slots, num_tokens,
        static_cast<uint8_t *>(k_cache), static_cast<uint8_t *>(v_cache),
        static_cast<int64_t>(d->num_blocks) * kF8Bs);
    return cudaGetLastError() == cudaSuccess ? FNPU_OK : FNPU_ECUDA;
}

int launch_kv_append(const fnpu_attn_desc *d, const void *k_new, const void *v_new,
                     const int64_t *slots, int32_t num_tokens, void *k_cache, void *v_cache,
                     void *stream) {
    if (num_tokens == 0) return FNPU_OK;
    const bool latent = d->v_in_k_latent != 0;
    const int64_t k_row = static_cast<int64_t>(latent ? 1 : d->num_kv_heads) * d->head_dim_qk * 2;
    const int64_t v_row = latent ? 0 : static_cast<int64_t>(d->num_kv_heads) * d->head_dim_v * 2;
    const int32_t kc = static_cast<int32_t>(k_row / 16), vc = static_cast<int32_t>(v_row / 16);
    const int64_t total = static_cast<int64_t>(num_tokens) * (kc + vc);
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    // one pass over all chunks when it fits 32 blocks per SM: the copy is
    // latency-bound at step sizes, so every chunk should be in flight at once
    const int64_t want = (total + 255) / 256;
    const int grid = static_cast<int>(want < 32LL * sms ? want : 32LL * sms);
    kv_append_kernel<<<grid, 256, 0, static_cast<cudaStream_t>(stream)>>>(
        static_cast<const uint4 *>(k_new), static_cast<const uint4 *>(v_new), slots, num_tokens,
        kc, vc, static_cast<uint4 *>(k_cache), static_cast<uint4 *>(v_cache),
        static_cast<int64_t>(d->num_blocks) * d->block_size);
    return cudaGetLastError() == cudaSuccess ? FNPU_OK : FNPU_ECUDA;
}

// The append of listed tokens only (the decode rows of a step whose prefill
// grid appends the prefill rows itself): chunk i belongs to token
// tokens[i / (k_chunks + v_chunks)].
__global__ void __launch_bounds__(256) kv_append_list_kernel(
    const uint4 *__restrict__ k_new, const uint4 *__restrict__ v_new, const int64_t *__restrict__ slots,
    const int32_t *__restrict__ tokens, int32_t n, int32_t k_chunks, int32_t v_chunks, uint4 *__restrict__ k_cache,
    uint4 *__restrict__ v_cache, int64_t num_slots) {
    const int32_t per_tok = k_chunks + v_chunks;
    const int64_t total = static_cast<int64_t>(n) * per_tok;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int32_t ti = static_cast<int32_t>(i / per_tok);
        const int32_t c = static_cast<int32_t>(i - static_cast<int64_t>(ti) * per_tok);
        const int64_t t = __ldg(tokens + ti);
        const uint4 v = c < k_chunks ? __ldg(k_new + t * k_chunks + c) : __ldg(v_new + t * v_chunks + (c - k_chunks));
        const int64_t s = __ldg(slots + t);
        if (s < 0) continue;
        if (s >= num_slots) {
            if (c == 0) atomicOr(&g_device_error, 1);
            continue;
        }
        if (c < k_chunks) k_cache[s * k_chunks + c] = v;
        else v_cache[s * v_chunks + (c - k_chunks)] = v;
    }
}

int launch_kv_append_list(const fnpu_attn_desc *d, const void *k_new, const void *v_new, const int64_t *slots,
                          const int32_t *tokens, int32_t n, void *k_cache, void *v_cache, void *stream) {
    if (n == 0) return FNPU_OK;
    const int32_t kc = static_cast<int32_t>(static_cast<int64_t>(d->num_kv_heads) * d->head_dim_qk * 2 / 16);
    const int32_t vc = static_cast<int32_t>(static_cast<int64_t>(d->num_kv_heads) * d->head_dim_v * 2 / 16);
    const int64_t want = (static_cast<int64_t>(n) * (kc + vc) + 255) / 256;
    const int grid = static_cast<int>(want < 4096 ? want : 4096);
    kv_append_list_kernel<<<grid, 256, 0, static_cast<cudaStream_t>(stream)>>>(
        static_cast<const uint4 *>(k_new), static_cast<const uint4 *>(v_new), slots, tokens, n, kc, vc,
        static_cast<uint4 *>(k_cache), static_cast<uint4 *>(v_cache),
        static_cast<int64_t>(d->num_blocks) * d->block_size);
    return cudaGetLastError() == cudaSuccess ? FNPU_OK : FNPU_ECUDA;
}

// One warp per row: the 64 16-byte chunks of c into the workspace (two per
// lane), then the 8 chunks of r into every head's key (lane e writes chunk
// e mod 8 of heads e / 8, e / 8 + 4, ...). A negative slot gives a zero row;
// a slot past the pool gives a zero row and raises the device error flag.
// MLA expansion gather (latent rows of 512 + 64 columns; see mla_expand.cu).
__global__ void __launch_bounds__(256) mla_gather_kernel(const uint4 *__restrict__ latent,
                                                         const int64_t *__restrict__ slots, int32_t n,
                                                         int64_t num_slots, int32_t heads,
                                                         uint4 *__restrict__ ws, uint4 *__restrict__ k_out) {
    const int lane = threadIdx.x & 31;
    const int64_t step = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
    for (int64_t i = (blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x) >> 5; i < n; i += step) {
        int64_t s = __ldg(slots + i);
        if (s >= num_slots) {
            if (lane == 0) atomicOr(&g_device_error, 1);
            s = -1;
        }
        const uint4 zero = make_uint4(0u, 0u, 0u, 0u);
        const uint4 *row = latent + (s < 0 ? 0 : s) * (576 / 8);
        uint4 *w = ws + i * (512 / 8);
        w[lane] = s < 0 ? zero : __ldg(row + lane);
        w[lane + 32] = s < 0 ? zero : __ldg(row + lane + 32);
        const uint4 r = (lane < 64 / 8 && s >= 0) ? __ldg(row + 512 / 8 + lane) : zero;
        uint4 rr;  // chunk lane mod 8 of r
        rr.x = __shfl_sync(0xffffffffu, r.x, lane & 7);
        rr.y = __shfl_sync(0xffffffffu, r.y, lane & 7);
        rr.z = __shfl_sync(0xffffffffu, r.z, lane & 7);
        rr.w = __shfl_sync(0xffffffffu, r.w, lane & 7);
        uint4 *krow = k_out + i * heads * (192 / 8);
        for (int e = lane; e < heads * (64 / 8); e += 32) krow[(e >> 3) * (192 / 8) + 128 / 8 + (e & 7)] = rr;
    }
}

int launch_mla_gather(const void *latent, const int64_t *slots, int32_t n, int64_t num_slots, int32_t heads,
                      void *ws, void *k_out, void *stream) {
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int64_t want = (static_cast<int64_t>(n) + 7) / 8;  // 8 rows (warps) per block
    const int grid = static_cast<int>(want < 16LL * sms ? want : 16LL * sms);
    mla_gather_kernel<<<grid, 256, 0, static_cast<cudaStream_t>(stream)>>>(
        static_cast<const uint4 *>(latent), slots, n, num_slots, heads, static_cast<uint4 *>(ws),
        static_cast<uint4 *>(k_out));
    return cudaGetLastError() == cudaSuccess ? FNPU_OK : FNPU_ECUDA;
}

int global_error_address(int **out) {
    constexpr int kMaxDevices = 64;
    static std::mutex mu;
    static int *addr[kMaxDevices] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return FNPU_ECUDA;
    if (dev < 0 || dev >= kMaxDevices) return FNPU_EUNSUPPORTED;
    std::lock_guard<std::mutex> lk(mu);
    if (!addr[dev]) {
        void *ptr = nullptr;
        if (cudaGetSymbolAddress(&ptr, g_device_error) != cudaSuccess || !ptr) {
            cudaGetLastError();
            return FNPU_ECUDA;
        }
        addr[dev] = static_cast<int *>(ptr);
    }
    *out = addr[dev];
    return FNPU_OK;
}

int read_and_clear_global_error(void *stream, int *flag) {
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (cudaStreamSynchronize(s) != cudaSuccess) return FNPU_ECUDA;
    int v = 0, zero = 0;
    if (cudaMemcpyFromSymbol(&v, g_device_error, sizeof(int)) != cudaSuccess) return FNPU_ECUDA;
    if (v != 0 && cudaMemcpyToSymbol(g_device_error, &zero, sizeof(int)) != cudaSuccess)
        return FNPU_ECUDA;
    *flag = v;
    return FNPU_OK;
}

}  // namespace fnpu
