// Element-wise kernels: the exported dequant (bit-exact test hook) and the
// weight quantiser (weight preparation).  Both are HBM-bound streams.
#include "dequant.cuh"
#include "internal.h"

#include <cuda_bf16.h>

namespace w4a16 {

// One thread per packed 32-bit word: 8 codes of one row -> 16 bytes of bf16.
__global__ void __launch_bounds__(256) dequant_kernel(const uint32_t* __restrict__ w,
                                                      const uint16_t* __restrict__ scales,
                                                      uint4* __restrict__ wd, int64_t N,
                                                      int64_t K, int64_t g) {
    const int64_t words_per_row = K / 8;
    const int64_t total = N * words_per_row;
    const int64_t KG = K / g;
    for (int64_t i = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; i < total;
         i += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        const int64_t n = i / words_per_row;
        const int64_t k0 = (i - n * words_per_row) * 8;
        const uint16_t s = __ldg(scales + n * KG + k0 / g);
        uint32_t v[4];
        dequant_word(__ldg(w + i), splat_bf16(s), v);
        wd[i] = make_uint4(v[0], v[1], v[2], v[3]);
    }
}

cudaError_t launch_dequant(const uint8_t* w, const uint16_t* scales, uint16_t* wd, int64_t N,
                           int64_t K, int64_t g, cudaStream_t stream) {
    const int64_t total = N * (K / 8);
    int64_t blocks = (total + 255) / 256;
    if (blocks > 152 * 64) blocks = 152 * 64;
    dequant_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(
        reinterpret_cast<const uint32_t*>(w), scales, reinterpret_cast<uint4*>(wd), N, K, g);
    return cudaGetLastError();
}

// One warp per (row, group).  Lane l owns the g/32 consecutive elements
// starting at l*g/32 (an even count, so whole bytes).
__global__ void __launch_bounds__(256) quantize_kernel(const float* __restrict__ w,
                                                       uint8_t* __restrict__ packed,
                                                       uint16_t* __restrict__ scales, int64_t N,
                                                       int64_t K, int64_t g) {
    const int64_t KG = K / g;
    const int64_t groups = N * KG;
    const int lane = threadIdx.x & 31;
    const int per_lane = static_cast<int>(g / 32);
    const int64_t warps_total = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
    for (int64_t gi = (blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x) >> 5;
         gi < groups; gi += warps_total) {
        const int64_t n = gi / KG;
        const int64_t j = gi - n * KG;
        const float* src = w + n * K + j * g + static_cast<int64_t>(lane) * per_lane;
        float amax = 0.0f;
        for (int e = 0; e < per_lane; ++e) amax = fmaxf(amax, fabsf(src[e]));
#pragma unroll
        for (int off = 16; off > 0; off >>= 1)
            amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, off));
        const __nv_bfloat16 sb = __float2bfloat16_rn(__fdiv_rn(amax, 7.0f));
        const float s = __bfloat162float(sb);
        if (lane == 0) scales[gi] = __bfloat16_as_ushort(sb);
        uint8_t* dst = packed + n * (K / 2) + (j * g + static_cast<int64_t>(lane) * per_lane) / 2;
        for (int e = 0; e < per_lane; e += 2) {
            int c[2];
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                if (s == 0.0f) {
                    c[h] = 8;
                } else {
                    float r = rintf(__fdiv_rn(src[e + h], s));
                    r = fminf(fmaxf(r, -8.0f), 7.0f);
                    c[h] = static_cast<int>(r) + 8;
                }
            }
            dst[e / 2] = static_cast<uint8_t>(c[0] | (c[1] << 4));
        }
    }
}

cudaError_t launch_quantize(const float* w, uint8_t* packed, uint16_t* scales, int64_t N,
                            int64_t K, int64_t g, cudaStream_t stream) {
    const int64_t groups = N * (K / g);
    int64_t blocks = (groups * 32 + 255) / 256;
    if (blocks > 152 * 64) blocks = 152 * 64;
    quantize_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(w, packed, scales, N, K,
                                                                       g);
    return cudaGetLastError();
}

}  // namespace w4a16
