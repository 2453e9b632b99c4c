// Helpers of the FP8 (e4m3) cache kernels: code conversion to f16 operands
// and the f16 m16n8k16 product.
#pragma once

#include <cuda_fp16.h>

#include "common.cuh"

namespace fnpu {

// four e4m3 codes (bytes 0..3 of w) -> two f16x2: lo = (byte 0, byte 1),
// hi = (byte 2, byte 3), the lower byte in the lower half
__device__ __forceinline__ void e4m3x4_to_f16x2x2(uint32_t w, uint32_t &lo, uint32_t &hi) {
    asm("{\n .reg .b16 l, h;\n mov.b32 {l, h}, %2;\n cvt.rn.f16x2.e4m3x2 %0, l;\n"
        " cvt.rn.f16x2.e4m3x2 %1, h;\n}\n"
        : "=r"(lo), "=r"(hi)
        : "r"(w));
}

__device__ __forceinline__ uint32_t bf16x2_to_f16x2(uint32_t b) {
    const float lo = __uint_as_float(b << 16), hi = __uint_as_float(b & 0xFFFF0000u);
    const __half2 h = __floats2half2_rn(lo, hi);
    return *reinterpret_cast<const uint32_t *>(&h);
}

__device__ __forceinline__ uint32_t pack_f16x2(float lo, float hi) {
    const __half2 h = __floats2half2_rn(lo, hi);
    return *reinterpret_cast<const uint32_t *>(&h);
}

// D += A(16x16, row) * B(16x8, col), f16 inputs, fp32 accumulation.
__device__ __forceinline__ void mma_f16_16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                              uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};\n"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// 2^-e for a power of two 2^e in the normal range (exact)
__device__ __forceinline__ float pow2_inverse(float pow2) { return __uint_as_float(0x7F000000u - __float_as_uint(pow2)); }

// the power of two at or above x > 0 (2^-126 for subnormal x)
__device__ __forceinline__ float pow2_ceil(float x) {
    const uint32_t bits = __float_as_uint(x);
    if (bits < 0x800000u) return 1.17549435e-38f;
    return __uint_as_float((bits & 0x7FFFFFu) ? (bits & 0x7F800000u) + 0x800000u : bits);
}

}  // namespace fnpu
