// Register-level int4 -> bf16 dequantisation shared by every kernel of the
// library (the exported dequant, the GEMM and the small-M path), so that the
// GEMM's weights are bit-identical to w4a16_dequant's output.
//
// A packed 32-bit word holds eight consecutive codes q_0..q_7 of one row
// (q_i in bits 4i..4i+3: byte j carries the even k in its low nibble and the
// odd k in its high nibble).  For each pair (q_2j, q_2j+1) the word is turned
// into a bf16x2 without any int->float conversion:
//   - PRMT puts byte j of w in byte 0 and byte j of (w >> 4) in byte 2;
//   - masking to bits 0..3 / 16..19 and OR-ing 0x4300 into each half gives
//     the bf16 pattern 0x430q, whose value is 128 + q (bf16 spacing on
//     [128, 256) is exactly 1);
//   - a bf16x2 subtraction of 136 gives q - 8 exactly (|q - 8| <= 8);
//   - a bf16x2 multiply by the scale rounds the exact product once, to
//     nearest even -- the definition wd = RNE_bf16((q - 8) * s).
#pragma once

#include <cstdint>

namespace w4a16 {

__device__ __forceinline__ uint32_t prmt_b32(uint32_t a, uint32_t b, uint32_t sel) {
    uint32_t r;
    asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(a), "r"(b), "r"(sel));
    return r;
}

__device__ __forceinline__ uint32_t bf16x2_sub(uint32_t a, uint32_t b) {
    uint32_t r;
    asm("sub.rn.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
}

__device__ __forceinline__ uint32_t bf16x2_mul(uint32_t a, uint32_t b) {
    uint32_t r;
    asm("mul.rn.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
    return r;
}

// 8 codes -> 4 bf16x2 words; out[j] = (wd(k=2j) low half, wd(k=2j+1) high half).
// s2 holds the row's bf16 scale in both halves.
__device__ __forceinline__ void dequant_word(uint32_t w, uint32_t s2, uint32_t* out) {
    const uint32_t w4 = w >> 4;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        uint32_t t = prmt_b32(w, w4, static_cast<uint32_t>(j | ((4 + j) << 8)));
        t = (t & 0x000F000Fu) | 0x43004300u;               // (128 + q_2j, 128 + q_2j+1)
        out[j] = bf16x2_mul(bf16x2_sub(t, 0x43084308u), s2);  // (q - 8) * s, one rounding
    }
}

// Puts the 8 bf16 of a 16-byte chunk (x0..x7) in the pair order
// (x0,x4),(x1,x5),(x2,x6),(x3,x7): the order in which one packed word yields
// its codes when each pair is masked out of a shifted copy of the word.
__device__ __forceinline__ uint4 interleave_chunk(uint4 c) {
    uint4 r;
    r.x = prmt_b32(c.x, c.z, 0x5410u);
    r.y = prmt_b32(c.x, c.z, 0x7632u);
    r.z = prmt_b32(c.y, c.w, 0x5410u);
    r.w = prmt_b32(c.y, c.w, 0x7632u);
    return r;
}

__device__ __forceinline__ uint32_t splat_bf16(uint16_t s) {
    return static_cast<uint32_t>(s) | (static_cast<uint32_t>(s) << 16);
}

// (w >> n) & 0x000F000F | 0x43004300 as one shift and one three-input logic
// op; written out so that the mask and the bias merge into a single LOP3.
template <int n>
__device__ __forceinline__ uint32_t nibble_pair_biased(uint32_t w) {
    uint32_t r;
    if constexpr (n == 0) {
        asm("lop3.b32 %0, %1, 0x000F000F, 0x43004300, 0xEA;" : "=r"(r) : "r"(w));
    } else {
        asm("{\n\t.reg .b32 t;\n\t"
            "shr.b32 t, %1, %2;\n\t"
            "lop3.b32 %0, t, 0x000F000F, 0x43004300, 0xEA;\n\t}"
            : "=r"(r)
            : "r"(w), "n"(n));
    }
    return r;
}

// Codes minus the zero point, q - 8, as exact bf16 pairs (k = j, k = j + 4)
// of one packed word: nibbles j and j + 4 sit 16 bits apart, so the mask of
// the word shifted by 4j gives (128 + q_j, 128 + q_j+4), and subtracting 136
// (all exact in bf16) the signed codes.
__device__ __forceinline__ void codes_signed(uint32_t w, uint32_t* out) {
    out[0] = bf16x2_sub(nibble_pair_biased<0>(w), 0x43084308u);
    out[1] = bf16x2_sub(nibble_pair_biased<4>(w), 0x43084308u);
    out[2] = bf16x2_sub(nibble_pair_biased<8>(w), 0x43084308u);
    out[3] = bf16x2_sub(nibble_pair_biased<12>(w), 0x43084308u);
}

// Shared-memory loads by 32-bit address (volatile: they stay after the
// barrier waits that guard them).
__device__ __forceinline__ uint2 lds64(uint32_t addr) {
    uint2 v;
    asm volatile("ld.shared.v2.u32 {%0, %1}, [%2];" : "=r"(v.x), "=r"(v.y) : "r"(addr));
    return v;
}

__device__ __forceinline__ uint4 lds128(uint32_t addr) {
    uint4 v;
    asm volatile("ld.shared.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "r"(addr));
    return v;
}

__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

}  // namespace w4a16
