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
// flag) copies the c part of each requested row into a
// contiguous workspace [n, 512] and broadcasts its r part into columns
// 128..191 of every head's key; then two strided-batched cuBLAS GEMMs (one
// batch entry per head, bf16 in, fp32 accumulation, bf16 out) write c W_UK[h]
// into columns 0..127 of the keys and c W_UV[h] into the values. The GEMMs
// are plain library GEMMs; the attention that follows runs in this library's
// kernels.
#include <cublas_v2.h>

#include <mutex>

#include "common.cuh"

namespace fnpu {
namespace {

constexpr int kC = 512;  // compressed part of a latent row
constexpr int kR = 64;   // rotary part
constexpr int kRow = kC + kR;
constexpr int kDn = 128;  // per-head key (no-rope part) and value width
constexpr int kDk = kDn + kR;

struct CublasHandles {
    std::mutex mu;
    cublasHandle_t h[64] = {};
};
CublasHandles &handles() {
    static CublasHandles hs;
    return hs;
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
    const int heads = desc->num_q_heads;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return FNPU_ECUDA;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    const int rc = launch_mla_gather(latent_cache, slots, n, static_cast<int64_t>(desc->num_blocks) * desc->block_size,
                                     heads, workspace, k_out, stream);
    if (rc != FNPU_OK) return rc;

    // per head h (column-major view of the row-major arrays):
    //   C_h (128 x n, ld = heads * width) = W_h^T view (128 x 512, ld 128) * ws view (512 x n, ld 512)
    CublasHandles &hs = handles();
    std::lock_guard<std::mutex> lock(hs.mu);
    if (!hs.h[dev] && cublasCreate(&hs.h[dev]) != CUBLAS_STATUS_SUCCESS) {
        hs.h[dev] = nullptr;
        return cuda_fail(cudaErrorUnknown, "cublasCreate");
    }
    cublasHandle_t h = hs.h[dev];
    if (cublasSetStream(h, st) != CUBLAS_STATUS_SUCCESS) return cuda_fail(cudaErrorUnknown, "cublasSetStream");
    const float one = 1.f, zero = 0.f;
    const __nv_bfloat16 *wsb = static_cast<const __nv_bfloat16 *>(workspace);
    cublasStatus_t r = cublasGemmStridedBatchedEx(
        h, CUBLAS_OP_N, CUBLAS_OP_N, kDn, n, kC, &one, w_uk, CUDA_R_16BF, kDn, static_cast<long long>(kC) * kDn, wsb,
        CUDA_R_16BF, kC, 0LL, &zero, k_out, CUDA_R_16BF, heads * kDk, static_cast<long long>(kDk), heads,
        CUBLAS_COMPUTE_32F, CUBLAS_GEMM_DEFAULT);
    if (r != CUBLAS_STATUS_SUCCESS) return cuda_fail(cudaErrorUnknown, "cublasGemmStridedBatchedEx (keys)");
    r = cublasGemmStridedBatchedEx(h, CUBLAS_OP_N, CUBLAS_OP_N, kDn, n, kC, &one, w_uv, CUDA_R_16BF, kDn,
                                   static_cast<long long>(kC) * kDn, wsb, CUDA_R_16BF, kC, 0LL, &zero, v_out,
                                   CUDA_R_16BF, heads * kDn, static_cast<long long>(kDn), heads, CUBLAS_COMPUTE_32F,
                                   CUBLAS_GEMM_DEFAULT);
    if (r != CUBLAS_STATUS_SUCCESS) return cuda_fail(cudaErrorUnknown, "cublasGemmStridedBatchedEx (values)");
    return FNPU_OK;
}
