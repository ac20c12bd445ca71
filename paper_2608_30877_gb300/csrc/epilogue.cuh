// Element math of the fused epilogue (operator fusion of what follows a
// linear layer, Sec. 5): z = acc + bias; SwiGLU h = silu(z_gate) * z_up with
// silu(t) = t / (1 + e^-t); GELU h = z * Phi(z) = z/2 (1 + erf(z / sqrt 2));
// out = h + residual.  fp32 throughout, one bf16 rounding at the store.
#pragma once

#include <cstdint>

namespace w4a16 {

enum : int { kActNone = 0, kActSwiGLU = 1, kActGELU = 2 };

__device__ __forceinline__ float bf16_to_f32(uint16_t h) {
    return __uint_as_float(static_cast<uint32_t>(h) << 16);
}

__device__ __forceinline__ float silu_f32(float t) { return t / (1.0f + expf(-t)); }

__device__ __forceinline__ float gelu_f32(float t) {
    return 0.5f * t * (1.0f + erff(t * 0.70710678118654752f));
}

__device__ __forceinline__ uint16_t f32_to_bf16_rn(float f) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %1;" : "=r"(r) : "f"(f));
    return static_cast<uint16_t>(r & 0xFFFFu);
}

}  // namespace w4a16
