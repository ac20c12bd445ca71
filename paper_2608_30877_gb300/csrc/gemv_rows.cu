// Small-M (M <= 32) int4-dequant + matmul for sm_103a: the bandwidth-bound
// regime where the whole packed weight matrix streams from HBM once per call.
//
// Design, GB300-first:
//   - persistent grid, one CTA per SM; CTA c owns a contiguous range of RB
//     weight rows (RB even, at most 352), so every SM streams the same number
//     of bytes -- no tile-count quantisation;
//   - one shared-memory stage covers 128 k = one scale group (g = 128): two
//     TMA boxes of RB/2 rows x 64 B of packed weights (64-byte swizzle) and
//     two 128-byte-swizzled boxes of x (T = 8, 16 or 32 token rows; rows >= M
//     are TMA zero fill); warp 0 keeps S stages in flight;
//   - warp 1 reorders each staged x chunk once, in place, into the pair order
//     the weight codes come out in (below), for all compute warps;
//   - one compute warp per 32 weight rows (two m16 tiles).  Its threads
//     unpack codes straight into the A fragments of mma.sync.m16n8k16 (bf16
//     in, fp32 out): nothing is staged in shared or tensor memory and there
//     is no hand-off between warps inside the K loop.  With 8-32 token
//     columns an MMA carries little work, and the fine-grained tcgen05
//     hand-offs (TMEM stores, commits, barrier round trips) would cost more
//     than the math;
//   - each 8-code word is unpacked as the pairs (k, k+4): a mask of the word
//     shifted by 4j gives the exact bf16 pair 128 + q, one bf16x2 subtraction
//     of 136 the exact q - 8 -- two integer-pipe instructions and one
//     half-precision one per pair.  Per group the MMA sums d = sum x (q - 8)
//     in fp32 and acc += s * d applies the scale;
//   - stages move in rounds of U (2 or 4): the TMA loads of a stage signal
//     its own barrier, but warp 1 releases, and the compute warps wait for and
//     give back, a whole round at a time, so the unrolled round body has no
//     barrier inside it and every shared-memory address in it is a per-thread
//     base plus an immediate.  A chunk's stage count is padded to a multiple of
//     U with empty stages that only cycle the barriers;
//   - scales are fetched U groups at a time (one vector load per row) a round
//     before use;
//   - each CTA walks K from its own starting group, so the CTAs do not all
//     read the same x slice from L2 at the same moment.
// Fragment k mapping: within a 128-k stage, thread quad index c owns k in
// [16c, 16c+16) and [64+16c, 64+16c+16); with the 128-byte swizzle of x this
// keeps every 16-byte shared-memory read of a quarter warp on distinct banks.
// Every wait is bounded (ptx.cuh): on a timeout the kernel records
// W4A16_ERR_TIMEOUT, drains its copies and returns.
#include "dequant.cuh"
#include "epilogue.cuh"
#include "internal.h"
#include "ptx.cuh"

#include <cuda_bf16.h>

// Stage slots and unroll (scale block) per token-tile count.
#ifndef W4A16_GEMV_S1
#define W4A16_GEMV_S1 8
#endif
#ifndef W4A16_GEMV_U1
#define W4A16_GEMV_U1 4
#endif
#ifndef W4A16_GEMV_S2
#define W4A16_GEMV_S2 8
#endif
#ifndef W4A16_GEMV_U2
#define W4A16_GEMV_U2 4
#endif
#ifndef W4A16_GEMV_S4
#define W4A16_GEMV_S4 6
#endif
#ifndef W4A16_GEMV_U4
#define W4A16_GEMV_U4 2
#endif

namespace w4a16 {

namespace {

constexpr int kRowsMax = 352;  // 11 compute warps of 32 rows
constexpr int kBKS = 128;      // k per shared-memory stage = one scale group
constexpr int kRowsPerWarp = 32;
constexpr int kFirstComputeWarp = 2;
constexpr int kMaxThreads = 32 * (kFirstComputeWarp + kRowsMax / kRowsPerWarp);

template <int NT, int S>
struct GLayout {
    static_assert(S >= 2, "stage slots");
    static constexpr int T = 8 * NT;                            // token rows staged
    static constexpr int X_BOX = T * 128;                       // one 64-k box of x
    static constexpr int X_BYTES = 2 * X_BOX;
    static constexpr int W_HALF = (kRowsMax / 2) * (kBKS / 2);  // 11 KB per box
    static constexpr int W_BYTES = 2 * W_HALF;
    static constexpr int X_OFF = 0;
    static constexpr int W_OFF = S * X_BYTES;
    static constexpr int BAR_OFF = W_OFF + S * W_BYTES;
    // full: one per stage slot (TMA landed); ready (x reordered) and empty:
    // one per round of stage slots
    static constexpr int NBARS = S + 2 * (S / 2);
    static constexpr int MISC_OFF = BAR_OFF + NBARS * 8;
    static constexpr int SMEM_BYTES = MISC_OFF + 16 + 1024;
    static_assert(X_BOX % 1024 == 0, "x boxes keep the 128-byte swizzle phase");
    static_assert(W_HALF % 1024 == 0, "weight boxes keep the 64-byte swizzle phase");
    static_assert(SMEM_BYTES <= 227 * 1024, "shared memory");
};

// d += A * B: m16n8k16, bf16 inputs, fp32 accumulators.
__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1,
                                               uint32_t a2, uint32_t a3, uint32_t b0,
                                               uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// d = A * B: a zero C operand starts a fresh accumulator without clearing it.
__device__ __forceinline__ void mma_bf16_16816_first(float (&d)[4], uint32_t a0, uint32_t a1,
                                                     uint32_t a2, uint32_t a3, uint32_t b0,
                                                     uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%10, %10, %10, %10};"
        : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1), "f"(0.0f));
}

// Scale e of a block held as bf16 pairs, as fp32: a low half by an integer
// multiply by 2^16 (FMA pipe), a high half by a mask.
// (e is a constant once the stage loop is unrolled.)
template <int W>
__device__ __forceinline__ float scale_at(const uint32_t (&blk)[W], int e) {
    const uint32_t w = blk[e >> 1];
    if ((e & 1) == 0) {
        uint32_t r;
        asm("mul.lo.u32 %0, %1, 65536;" : "=r"(r) : "r"(w));
        return __uint_as_float(r);
    } else {
        return __uint_as_float(w & 0xFFFF0000u);
    }
}

// NT: 8-token MMA column tiles (T = 8 NT staged token rows); S: stage slots;
// U: stages per unrolled round of the K loop, and scale groups per load (a
// divisor of S); FUSED: the fused epilogue (bias, activation, residual).
template <int NT, int S, int U, bool FUSED>
__global__ void __launch_bounds__(kMaxThreads, 1)
    w4a16_gemv_kernel(const __grid_constant__ CUtensorMap tmap_x,
                      const __grid_constant__ CUtensorMap tmap_w, const GemvParams p) {
    using L = GLayout<NT, S>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;
    uint8_t* smem = smem_raw + (sbase - raw);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int RB = p.rows_per_cta;
    const int NW = (RB + kRowsPerWarp - 1) / kRowsPerWarp;  // compute warps

    const uint32_t bars = sbase + L::BAR_OFF;
    static_assert(S % U == 0 && (U == 2 || U == 4), "rounds tile the stage slots");
    constexpr int RS = S / U;  // round slots: rounds in flight
    auto full = [&](int s) { return bars + 8u * s; };
    auto ready = [&](int rs) { return bars + 8u * (S + rs); };
    auto empty = [&](int rs) { return bars + 8u * (S + RS + rs); };
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::MISC_OFF);

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) mbar_init(full(s), 1);
        for (int rs = 0; rs < RS; ++rs) {
            mbar_init(ready(rs), 1);
            mbar_init(empty(rs), NW);  // every compute warp has read the round
        }
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tmap_x);
        prefetch_tmap(&tmap_w);
    }
    __syncthreads();

    const int KS = p.K / kBKS;        // scale groups = real stages per chunk
    const int R = (KS + U - 1) / U;   // rounds per chunk
    // Scales are read U groups at a time, as one vector load per row when
    // every block is aligned (KS a multiple of U).
    const bool vec_scales = KS % U == 0;
    // Each CTA walks K from its own starting group (a multiple of U when the
    // scale loads are vectors): the CTAs then read different x slices at any
    // moment instead of all hitting the same L2 lines.
    const int rot = vec_scales
                        ? static_cast<int>(static_cast<int64_t>(blockIdx.x) * (KS / U) /
                                           gridDim.x) * U
                        : static_cast<int>(static_cast<int64_t>(blockIdx.x) * KS / gridDim.x);

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint32_t tx = L::X_BYTES + static_cast<uint32_t>(RB) * (kBKS / 2);
            uint32_t it = 0;  // stage slot = it % S, phase = (it / S) & 1
            bool ok = true;
            for (int chunk = blockIdx.x; ok && chunk < p.num_chunks; chunk += gridDim.x) {
                const int row0 = chunk * RB;
                int kk = rot;  // group of stage ks, rotated
                for (int ks = 0; ks < R * U; ++ks, ++it) {
                    const int s = it % S;
                    // a round's slots are refilled once every compute warp has left it
                    if (s % U == 0 &&
                        !wait_one(empty(s / U), ((it / S) & 1u) ^ 1u, abort_flag, p.status, p.wait_ns)) {
                        ok = false;
                        break;
                    }
                    if (ks >= KS) {  // padding stage: cycles the barrier only
                        mbar_arrive(full(s));
                        continue;
                    }
                    mbar_arrive_expect_tx(full(s), tx);
                    const uint32_t xs = sbase + L::X_OFF + s * L::X_BYTES;
                    const uint32_t ws = sbase + L::W_OFF + s * L::W_BYTES;
                    const uint32_t wbox = static_cast<uint32_t>(RB / 2) * (kBKS / 2);
                    if (dbg_check(tma_box_ok(xs, L::X_BOX, 1024, sbase, sbase + L::W_OFF,
                                             kk * kBKS, 2) &&
                                      tma_box_ok(xs + L::X_BOX, L::X_BOX, 1024, sbase,
                                                 sbase + L::W_OFF, kk * kBKS + 64, 2) &&
                                      wbox <= L::W_HALF &&
                                      tma_box_ok(ws, wbox, 1024, sbase + L::W_OFF,
                                                 sbase + L::BAR_OFF, kk * (kBKS / 2), 1) &&
                                      tma_box_ok(ws + L::W_HALF, wbox, 1024, sbase + L::W_OFF,
                                                 sbase + L::BAR_OFF, kk * (kBKS / 2), 1),
                                  p.status)) {
                        tma_load_2d(xs, &tmap_x, full(s), kk * kBKS, 0);
                        tma_load_2d(xs + L::X_BOX, &tmap_x, full(s), kk * kBKS + 64, 0);
                        tma_load_2d(ws, &tmap_w, full(s), kk * (kBKS / 2), row0);
                        tma_load_2d(ws + L::W_HALF, &tmap_w, full(s), kk * (kBKS / 2),
                                    row0 + RB / 2);
                    }
                    if (++kk == KS) kk = 0;
                }
            }
            // every load this thread issued has landed before exit
            const uint32_t last = it < static_cast<uint32_t>(S) ? it : S;
            for (uint32_t i = it - last; i < it; ++i) settle(full(i % S), (i / S) & 1u);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ x reorder
        // Every 16-byte chunk (x0..x7) of the stage's x boxes becomes
        // (x0,x4),(x1,x5),(x2,x6),(x3,x7): the pair order of codes_signed.
        constexpr int kChunks = L::X_BYTES / 16;
        static_assert(kChunks % 32 == 0, "whole chunks per lane");
        uint32_t round = 0;  // global round: slots U (round % RS) .., phase (round / RS) & 1
        bool ok = true;
        for (int chunk = blockIdx.x; ok && chunk < p.num_chunks; chunk += gridDim.x) {
            for (int r = 0; ok && r < R; ++r, ++round) {
                const int s0 = static_cast<int>(round % RS) * U;
                const uint32_t ph = (round / RS) & 1u;
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int s = s0 + u;
                    if (!wait_warp(full(s), ph, abort_flag, p.status, p.wait_ns)) {
                        ok = false;
                        break;
                    }
                    if (r * U + u < KS) {
                        uint4* xs = reinterpret_cast<uint4*>(smem + L::X_OFF + s * L::X_BYTES);
#pragma unroll
                        for (int i = 0; i < kChunks / 32; ++i)
                            xs[lane + 32 * i] = interleave_chunk(xs[lane + 32 * i]);
                    }
                }
                if (!ok) break;
                // these generic writes precede the next TMA writes of the slots
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(ready(s0 / U));
            }
        }
    } else if (warp - kFirstComputeWarp < NW) {
        // ------------------------------------------------------------ compute warps
        // Warp cw owns local rows [32cw, 32cw+32): m16 tiles tt = 0, 1.
        // Thread (g, c): fragment rows g and g + 8 of tiles tt = 0, 1; k quad
        // c owns k in [16c, 16c+16) and [64+16c, 64+16c+16) of each 128-k
        // stage.  Fragment row g holds weight row 32cw + 16tt + gr (+8), with
        // gr = g with bits 1 and 2 swapped: the four rows a half warp reads
        // in one 8-byte load are then 0, 1, 4, 5 (or 2, 3, 6, 7) of an 8-row
        // group, which the 64-byte swizzle puts on distinct banks.
        const int cw = warp - kFirstComputeWarp;
        const int g = lane >> 2;
        const int c = lane & 3;
        const int gr = (g & 1) | ((g & 2) << 1) | ((g & 4) >> 1);
        auto w_off = [&](int r, int piece) {
            // rows >= RB read row 0; their results are never stored
            const int rs = r < RB ? r : 0;
            const int b = rs >= RB / 2 ? 1 : 0;
            const int rr = rs - b * (RB / 2);
            const int j = 2 * piece + (c >> 1);
            return L::W_OFF + b * L::W_HALF + rr * (kBKS / 2) + 16 * (j ^ ((rr >> 1) & 3)) +
                   8 * (c & 1);
        };
        int row[4];  // rows of (tt, upper/lower half): index 2*tt + hh
        uint32_t wp[4][2];  // shared-memory addresses in stage slot 0
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            row[q] = cw * kRowsPerWarp + (q >> 1) * 16 + (q & 1) * 8 + gr;
            wp[q][0] = sbase + w_off(row[q], 0);
            wp[q][1] = sbase + w_off(row[q], 1);
        }
        // x chunk of word i (k 64*(i>>1) + 16c + 8*(i&1) .. +8): chunk
        // 2c + (i&1) of box i>>1, 128-byte swizzle by row g
        uint32_t xp[4];
#pragma unroll
        for (int i = 0; i < 4; ++i)
            xp[i] = sbase + L::X_OFF + g * 128 + (i >> 1) * L::X_BOX + 16 * ((2 * c + (i & 1)) ^ g);

        uint32_t round = 0;
        bool ok = true;
        for (int chunk = blockIdx.x; ok && chunk < p.num_chunks; chunk += gridDim.x) {
            int n[4];
            bool v[4];
            const uint16_t* srow[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                n[q] = chunk * RB + row[q];
                v[q] = row[q] < RB && n[q] < p.N;
                srow[q] = p.scales + static_cast<int64_t>(v[q] ? n[q] : 0) * KS;
            }
            float acc[2][NT][4];
#pragma unroll
            for (int tt = 0; tt < 2; ++tt)
#pragma unroll
                for (int nn = 0; nn < NT; ++nn)
#pragma unroll
                    for (int e = 0; e < 4; ++e) acc[tt][nn][e] = 0.0f;
            // Scales as bf16 pairs: the current block of U groups and the
            // next one, loaded U stages before use.
            uint32_t scb[4][U / 2], scn[4][U / 2];

            int kb = rot;  // first group of the next block
            auto load_block = [&]() {
                if (vec_scales) {
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        if constexpr (U == 4) {
                            const uint2 t = __ldg(reinterpret_cast<const uint2*>(srow[q] + kb));
                            scn[q][0] = t.x;
                            scn[q][1] = t.y;
                        } else {
                            scn[q][0] = __ldg(reinterpret_cast<const uint32_t*>(srow[q] + kb));
                        }
                    }
                    kb += U;
                    if (kb == KS) kb = 0;
                } else {
#pragma unroll
                    for (int e = 0; e < U; ++e) {
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const uint32_t h = __ldg(srow[q] + kb);
                            scn[q][e >> 1] = (e & 1) ? (scn[q][e >> 1] | (h << 16)) : h;
                        }
                        if (++kb == KS) kb = 0;
                    }
                }
            };
            load_block();

            for (int r = 0; ok && r < R; ++r, ++round) {
                const int s0 = static_cast<int>(round % RS) * U;
                const uint32_t ph = (round / RS) & 1u;
                // ready completes after warp 1 has seen every full(s) of the
                // round complete, so the stages' TMA data is visible here too
                if (!wait_warp(ready(s0 / U), ph, abort_flag, p.status, p.wait_ns)) {
                    ok = false;
                    break;
                }
#pragma unroll
                for (int u = 0; u < U; ++u) {
                    const int s = s0 + u;
                    if (r * U + u < KS) {
                        if (u == 0) {
#pragma unroll
                            for (int q = 0; q < 4; ++q)
#pragma unroll
                                for (int e = 0; e < U / 2; ++e) scb[q][e] = scn[q][e];
                            load_block();
                        }

                        const int wso = s * L::W_BYTES;
                        uint32_t wq[4][4];
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const uint2 p0 = lds64(wp[q][0] + wso);
                            const uint2 p1 = lds64(wp[q][1] + wso);
                            wq[q][0] = p0.x;
                            wq[q][1] = p0.y;
                            wq[q][2] = p1.x;
                            wq[q][3] = p1.y;
                        }
                        float d[2][NT][4];
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            uint4 xb[NT];
#pragma unroll
                            for (int nn = 0; nn < NT; ++nn)
                                xb[nn] = lds128(xp[i] + s * L::X_BYTES + nn * 8 * 128);
                            uint32_t A[4][4];
#pragma unroll
                            for (int q = 0; q < 4; ++q) codes_signed(wq[q][i], A[q]);
#pragma unroll
                            for (int h = 0; h < 2; ++h)
#pragma unroll
                                for (int tt = 0; tt < 2; ++tt)
#pragma unroll
                                    for (int nn = 0; nn < NT; ++nn) {
                                        const uint32_t b0 = h ? xb[nn].z : xb[nn].x;
                                        const uint32_t b1 = h ? xb[nn].w : xb[nn].y;
                                        if (i == 0 && h == 0)
                                            mma_bf16_16816_first(d[tt][nn], A[2 * tt][0],
                                                                 A[2 * tt + 1][0], A[2 * tt][1],
                                                                 A[2 * tt + 1][1], b0, b1);
                                        else
                                            mma_bf16_16816(d[tt][nn], A[2 * tt][2 * h],
                                                           A[2 * tt + 1][2 * h],
                                                           A[2 * tt][2 * h + 1],
                                                           A[2 * tt + 1][2 * h + 1], b0, b1);
                                    }
                        }
                        // acc += s * d: d0, d1 belong to the upper row, d2, d3 to the lower
#pragma unroll
                        for (int tt = 0; tt < 2; ++tt) {
                            const float su = scale_at(scb[2 * tt], u);
                            const float sl = scale_at(scb[2 * tt + 1], u);
#pragma unroll
                            for (int nn = 0; nn < NT; ++nn) {
                                acc[tt][nn][0] = fmaf(su, d[tt][nn][0], acc[tt][nn][0]);
                                acc[tt][nn][1] = fmaf(su, d[tt][nn][1], acc[tt][nn][1]);
                                acc[tt][nn][2] = fmaf(sl, d[tt][nn][2], acc[tt][nn][2]);
                                acc[tt][nn][3] = fmaf(sl, d[tt][nn][3], acc[tt][nn][3]);
                            }
                        }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(empty(s0 / U));
            }
            if (!ok) break;
            // epilogue: d0, d1 -> (upper row, tokens 2c, 2c+1); d2, d3 -> lower row
            const Epilogue& ep = p.epi;
            if constexpr (!FUSED) {
#pragma unroll
                for (int tt = 0; tt < 2; ++tt)
#pragma unroll
                    for (int nn = 0; nn < NT; ++nn)
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const int q = 2 * tt + (e >> 1);
                            const int m = nn * 8 + 2 * c + (e & 1);
                            if (v[q] && m < p.M)
                                p.out[static_cast<int64_t>(m) * p.N + n[q]] =
                                    __bfloat16_as_ushort(__float2bfloat16_rn(acc[tt][nn][e]));
                        }
            } else {
                // Fused epilogue.  A row's parity is that of g (the row remap
                // keeps bit 0), so SwiGLU's partner row n ^ 1 is held by lane
                // ^ 4 with the same tokens; the gate (even-row) lane finishes.
                float bq[4];
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    bq[q] = (ep.bias != nullptr && v[q]) ? bf16_to_f32(ep.bias[n[q]]) : 0.0f;
#pragma unroll
                for (int tt = 0; tt < 2; ++tt)
#pragma unroll
                    for (int nn = 0; nn < NT; ++nn)
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const int q = 2 * tt + (e >> 1);
                            const int m = nn * 8 + 2 * c + (e & 1);
                            const float z = acc[tt][nn][e] + bq[q];
                            if (ep.act == kActSwiGLU) {
                                const float up = __shfl_xor_sync(0xffffffffu, z, 4);
                                if ((g & 1) == 0 && v[q] && m < p.M) {
                                    const int64_t o = static_cast<int64_t>(m) * ep.n_out + (n[q] >> 1);
                                    float h = silu_f32(z) * up;
                                    if (ep.residual != nullptr) h += bf16_to_f32(ep.residual[o]);
                                    p.out[o] = f32_to_bf16_rn(h);
                                }
                            } else if (v[q] && m < p.M) {
                                const int64_t o = static_cast<int64_t>(m) * ep.n_out + n[q];
                                float h = ep.act == kActGELU ? gelu_f32(z) : z;
                                if (ep.residual != nullptr) h += bf16_to_f32(ep.residual[o]);
                                p.out[o] = f32_to_bf16_rn(h);
                            }
                        }
            }
        }
    }
    __syncthreads();
}

template <int NT, int S, int U>
cudaError_t launch_gemv_variant(const CUtensorMap* tx, const CUtensorMap* tw,
                                const GemvParams& p, int grid, cudaStream_t stream) {
    using L = GLayout<NT, S>;
    // the plain variant keeps the fused epilogue's registers out of the K loop
    const bool fused =
        p.epi.bias != nullptr || p.epi.residual != nullptr || p.epi.act != kActNone;
    auto kern = fused ? w4a16_gemv_kernel<NT, S, U, true> : w4a16_gemv_kernel<NT, S, U, false>;
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    const int threads =
        32 * (kFirstComputeWarp + (p.rows_per_cta + kRowsPerWarp - 1) / kRowsPerWarp);
    kern<<<grid, threads, L::SMEM_BYTES, stream>>>(*tx, *tw, p);
    return cudaGetLastError();
}

}  // namespace

int gemv_rows_per_cta(int64_t N, int sm_count) {
    // even (SwiGLU pairs rows 2j, 2j+1 within a CTA); the compute warps mask
    // the rows of their last tile past RB, so RB need not fill whole tiles and
    // every SM gets a range (12288 x 49152: 324 rows on 152 SMs, not 336 on 147)
    int64_t per = (N + sm_count - 1) / sm_count;
    per = (per + 1) / 2 * 2;
    if (per > kRowsMax) per = kRowsMax;
    if (per < 16) per = 16;
    return static_cast<int>(per);
}

int gemv_tokens_per_tile(int64_t M) { return M <= 8 ? 8 : M <= 16 ? 16 : 32; }

cudaError_t gemv_launch(const CUtensorMap* tx, const CUtensorMap* tw, const GemvParams& p,
                        int sm_count, cudaStream_t stream) {
    const int grid = p.num_chunks < sm_count ? p.num_chunks : sm_count;
    if (p.M <= 8)
        return launch_gemv_variant<1, W4A16_GEMV_S1, W4A16_GEMV_U1>(tx, tw, p, grid, stream);
    if (p.M <= 16)
        return launch_gemv_variant<2, W4A16_GEMV_S2, W4A16_GEMV_U2>(tx, tw, p, grid, stream);
    return launch_gemv_variant<4, W4A16_GEMV_S4, W4A16_GEMV_U4>(tx, tw, p, grid, stream);
}

}  // namespace w4a16
