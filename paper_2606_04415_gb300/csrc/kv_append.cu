// KV append: scatter the step's new K/V rows into their paged slots.
//
// The new tokens of a step must be in the cache before the step's attention
// reads it (prefill and decode share one KV pool, Sec. 3.4). A slot row is
// contiguous (Hkv*d bf16 values, or d_qk for the latent cache), so each
// thread moves one 16-byte chunk and consecutive threads cover consecutive
// chunks of the same row: fully coalesced 16-B loads and stores. Pure copy,
// bit-exact.
#include "common.cuh"

namespace fnpu {

// Library-wide device error flag (bit 0: out-of-range slot), one per device
// that loads the library; read and cleared by fnpu_check().
__device__ int g_device_error = 0;

__global__ void __launch_bounds__(256) kv_append_kernel(
    const uint4 *__restrict__ k_new, const uint4 *__restrict__ v_new,
    const int64_t *__restrict__ slots, int32_t num_tokens, int32_t k_chunks, int32_t v_chunks,
    uint4 *__restrict__ k_cache, uint4 *__restrict__ v_cache, int64_t num_slots) {
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
