// Small-M (M <= 16) int4-dequant + matmul for sm_103a: the bandwidth-bound
// regime where the whole packed weight matrix streams from HBM once per call.
//
// Design, GB300-first:
//   - persistent grid, one CTA per SM; CTA c owns a contiguous range of RB
//     weight rows (RB a multiple of 16, at most 352), so every SM streams the
//     same number of bytes -- no tile-count quantisation;
//   - one shared-memory stage covers 128 k = one scale group (g = 128): two
//     TMA boxes of RB/2 rows x 64 B of packed weights (64-byte swizzle) and
//     two 128-byte-swizzled boxes of x (T = 8 or 16 token rows; rows >= M
//     are TMA zero fill); warp 0 keeps S stages in flight;
//   - one compute warp per 32 weight rows (two m16 tiles).  Its threads
//     unpack codes straight into the A fragments of mma.sync.m16n8k16 (bf16
//     in, fp32 out): nothing is staged in shared or tensor memory and there
//     is no hand-off between warps inside the K loop.  With 8-16 token
//     columns an MMA carries little work, and the fine-grained tcgen05
//     hand-offs (TMEM stores, commits, barrier round trips) would cost more
//     than the math;
//   - each 8-code word is unpacked as the pairs (k, k+4) into the exact bf16
//     128 + q: one integer-pipe op per pair, the shifts as multiply-high on
//     the FMA pipe, no per-weight arithmetic.  The thread puts its x chunks
//     in the same pair order in registers.  Per group the MMA sums
//     d = sum x * (128 + q); one more MMA per k step with the constant A =
//     -136 (exact in bf16) sums db = -136 * sum x, already in the layout of
//     d, and acc += s * (d + db) applies zero point and scale in fp32;
//   - reading an MMA accumulator waits for every MMA the warp still has in
//     flight, so G consecutive groups accumulate into G separate register
//     sets and are folded together: one drain per G groups;
//   - each CTA walks K from its own starting group, so the CTAs do not all
//     read the same x slice from L2 at the same moment.
// Fragment k mapping: within a 128-k stage, thread quad index c owns k in
// [16c, 16c+16) and [64+16c, 64+16c+16); with the 128-byte swizzle of x this
// keeps every 16-byte shared-memory read of a quarter warp on distinct banks.
// Every wait is bounded (ptx.cuh): on a timeout the kernel records
// W4A16_ERR_TIMEOUT, drains its copies and returns.
#include "dequant.cuh"
#include "internal.h"
#include "ptx.cuh"

#include <cuda_bf16.h>

#ifndef W4A16_GEMV_G1
#define W4A16_GEMV_G1 1
#endif
#ifndef W4A16_GEMV_G2
#define W4A16_GEMV_G2 1
#endif
#ifndef W4A16_GEMV_TPW
#define W4A16_GEMV_TPW 2
#endif

namespace w4a16 {

namespace {

constexpr int kRowsMax = 352;  // 11 compute warps of 32 rows
constexpr int kBKS = 128;      // k per shared-memory stage = one scale group

template <int NT, int S>
struct GLayout {
    static constexpr int T = 8 * NT;                            // token rows staged
    static constexpr int X_BOX = T * 128;                       // one 64-k box of x
    static constexpr int X_BYTES = 2 * X_BOX;
    static constexpr int W_HALF = (kRowsMax / 2) * (kBKS / 2);  // 11 KB per box
    static constexpr int W_BYTES = 2 * W_HALF;
    static constexpr int X_OFF = 0;
    static constexpr int W_OFF = S * X_BYTES;
    static constexpr int BAR_OFF = W_OFF + S * W_BYTES;
    static constexpr int NBARS = 2 * S;  // full_tma, empty_smem
    static constexpr int MISC_OFF = BAR_OFF + NBARS * 8;
    static constexpr int SMEM_BYTES = MISC_OFF + 16 + 1024;
    static_assert(X_BOX % 1024 == 0, "x boxes keep the 128-byte swizzle phase");
    static_assert(W_HALF % 1024 == 0, "weight boxes keep the 64-byte swizzle phase");
};

__device__ __forceinline__ void mma_bf16_16816(float (&d)[4], uint32_t a0, uint32_t a1,
                                               uint32_t a2, uint32_t a3, uint32_t b0,
                                               uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 "
        "{%0, %1, %2, %3}, {%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// Biased codes (128 + q) as exact bf16 pairs (k = j, k = j + 4) of one packed
// word (the shifts are multiply-high by run-time 2^28, 2^24, 2^20).
__device__ __forceinline__ void codes_biased(uint32_t w, uint32_t m4, uint32_t m8, uint32_t m12,
                                             uint32_t* out) {
    out[0] = (w & 0x000F000Fu) | 0x43004300u;
    out[1] = (mulhi_u32(w, m4) & 0x000F000Fu) | 0x43004300u;
    out[2] = (mulhi_u32(w, m8) & 0x000F000Fu) | 0x43004300u;
    out[3] = (mulhi_u32(w, m12) & 0x000F000Fu) | 0x43004300u;
}

__device__ __forceinline__ float bf16_bits_to_float(uint32_t h) {
    return __uint_as_float(h << 16);
}

// 12 warps at most with two tiles per warp (384 threads, up to 144
// registers), 23 with one (736 threads, up to 80).
template <int NT, int S, int G, int TPW>
__global__ void __launch_bounds__(TPW == 2 ? 384 : 736, 1)
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
    constexpr int RPW = 16 * TPW;    // weight rows per compute warp
    const int NW = (RB + RPW - 1) / RPW;  // compute warps
    constexpr int CW0 = 1;           // first compute warp

    const uint32_t bars = sbase + L::BAR_OFF;
    auto full_tma = [&](int s) { return bars + 8u * s; };
    auto empty_smem = [&](int s) { return bars + 8u * (S + s); };
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::MISC_OFF);

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(full_tma(s), 1);
            mbar_init(empty_smem(s), NW);  // every compute warp has read the stage
        }
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tmap_x);
        prefetch_tmap(&tmap_w);
    }
    __syncthreads();

    const int KS = p.K / kBKS;  // stages per chunk = scale groups
    // Each CTA walks K from its own starting group (a multiple of the fold
    // batch G, so that batches never wrap): the CTAs then read different x
    // slices at any moment instead of all hitting the same L2 lines.
    const int rot = KS % G == 0 ? (static_cast<int>(blockIdx.x) * (KS / G) / static_cast<int>(gridDim.x)) * G : 0;
    auto kgroup = [&](int j) { return j + rot < KS ? j + rot : j + rot - KS; };

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint32_t tx = L::X_BYTES + static_cast<uint32_t>(RB) * (kBKS / 2);
            uint32_t it = 0;
            bool ok = true;
            for (int chunk = blockIdx.x; ok && chunk < p.num_chunks; chunk += gridDim.x) {
                const int row0 = chunk * RB;
                for (int ks = 0; ks < KS; ++ks, ++it) {
                    const int s = it % S;
                    if (!wait_one(empty_smem(s), ((it / S) & 1u) ^ 1u, abort_flag, p.status)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(full_tma(s), tx);
                    const int kk = kgroup(ks);
                    const uint32_t xs = sbase + L::X_OFF + s * L::X_BYTES;
                    tma_load_2d(xs, &tmap_x, full_tma(s), kk * kBKS, 0);
                    tma_load_2d(xs + L::X_BOX, &tmap_x, full_tma(s), kk * kBKS + 64, 0);
                    const uint32_t ws = sbase + L::W_OFF + s * L::W_BYTES;
                    tma_load_2d(ws, &tmap_w, full_tma(s), kk * (kBKS / 2), row0);
                    tma_load_2d(ws + L::W_HALF, &tmap_w, full_tma(s), kk * (kBKS / 2),
                                row0 + RB / 2);
                }
            }
            // every load this thread issued has landed before exit
            const uint32_t last = it < static_cast<uint32_t>(S) ? it : S;
            for (uint32_t i = it - last; i < it; ++i) {
                const uint64_t t0 = global_timer_ns();
                while (!mbar_try_wait(full_tma(i % S), (i / S) & 1u)) {
                    if (global_timer_ns() - t0 > kWaitLimitNs) break;
                }
            }
        }
    } else if (warp - CW0 < NW) {
        // ------------------------------------------------------------ compute warps
        // Warp cw owns local rows [32cw, 32cw+32): m16 tiles tt = 0, 1.
        // Thread (g, c): rows 32cw + 16tt + g (+8); k quad c owns k in
        // [16c, 16c+16) and [64+16c, 64+16c+16) of each 128-k stage.
        const int cw = warp - CW0;
        const int g = lane >> 2;
        const int c = lane & 3;
        const uint32_t m4 = p.m4, m8 = p.m8, m12 = p.m12;
        auto w_off = [&](int r, int piece) {
            // rows >= RB read row 0; their results are never stored
            const int rs = r < RB ? r : 0;
            const int b = rs >= RB / 2 ? 1 : 0;
            const int rr = rs - b * (RB / 2);
            const int j = 2 * piece + (c >> 1);
            return L::W_OFF + b * L::W_HALF + rr * (kBKS / 2) + 16 * (j ^ ((rr >> 1) & 3)) +
                   8 * (c & 1);
        };
        int row[2 * TPW];  // rows of (tt, upper/lower half): index 2*tt + hh
        int woff[2 * TPW][2];
#pragma unroll
        for (int q = 0; q < 2 * TPW; ++q) {
            row[q] = cw * RPW + (q >> 1) * 16 + (q & 1) * 8 + g;
            woff[q][0] = w_off(row[q], 0);
            woff[q][1] = w_off(row[q], 1);
        }
        uint32_t it = 0;
        bool ok = true;
        for (int chunk = blockIdx.x; ok && chunk < p.num_chunks; chunk += gridDim.x) {
            int n[2 * TPW];
            bool v[2 * TPW];
            const uint16_t* srow[2 * TPW];
#pragma unroll
            for (int q = 0; q < 2 * TPW; ++q) {
                n[q] = chunk * RB + row[q];
                v[q] = row[q] < RB && n[q] < p.N;
                srow[q] = p.scales + static_cast<int64_t>(v[q] ? n[q] : 0) * KS;
            }
            float acc[TPW][NT][4];
            float d[G][TPW][NT][4];
            float db[G][NT][4];  // -136 * sum x per token (same for every row)
            uint32_t sc[2 * TPW][G];   // bf16 bits of the batch's scales, per row
            uint32_t scn[2 * TPW][G];  // the next batch's, loaded one batch ahead
#pragma unroll
            for (int tt = 0; tt < TPW; ++tt)
#pragma unroll
                for (int nn = 0; nn < NT; ++nn)
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        acc[tt][nn][e] = 0.0f;
#pragma unroll
                        for (int u = 0; u < G; ++u) d[u][tt][nn][e] = 0.0f;
                    }
#pragma unroll
            for (int u = 0; u < G; ++u)
#pragma unroll
                for (int nn = 0; nn < NT; ++nn)
#pragma unroll
                    for (int e = 0; e < 4; ++e) db[u][nn][e] = 0.0f;

            // one 128-k stage (scale group) into accumulator set u
            auto stage = [&](int u) -> bool {
                const int s = it % S;
                if (!wait_warp(full_tma(s), (it / S) & 1u, abort_flag, p.status)) return false;
                const uint8_t* ws = smem + s * L::W_BYTES;
                uint32_t wq[2 * TPW][4];
#pragma unroll
                for (int q = 0; q < 2 * TPW; ++q) {
                    const uint2 p0 = *reinterpret_cast<const uint2*>(ws + woff[q][0]);
                    const uint2 p1 = *reinterpret_cast<const uint2*>(ws + woff[q][1]);
                    wq[q][0] = p0.x;
                    wq[q][1] = p0.y;
                    wq[q][2] = p1.x;
                    wq[q][3] = p1.y;
                }
                const uint8_t* xst = smem + L::X_OFF + s * L::X_BYTES + g * 128;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    // word i: k 64*(i>>1) + 16c + 8*(i&1) .. +8 = x chunk
                    // 2c + (i&1) of box i>>1; it feeds two k16 steps
                    uint4 xb[NT];
#pragma unroll
                    for (int nn = 0; nn < NT; ++nn)
                        xb[nn] = interleave_chunk(*reinterpret_cast<const uint4*>(
                            xst + (i >> 1) * L::X_BOX + nn * 8 * 128 +
                            16 * ((2 * c + (i & 1)) ^ g)));
                    uint32_t A[2 * TPW][4];
#pragma unroll
                    for (int q = 0; q < 2 * TPW; ++q) codes_biased(wq[q][i], m4, m8, m12, A[q]);
#pragma unroll
                    for (int h = 0; h < 2; ++h)
#pragma unroll
                        for (int tt = 0; tt < TPW; ++tt)
#pragma unroll
                            for (int nn = 0; nn < NT; ++nn)
                                mma_bf16_16816(d[u][tt][nn], A[2 * tt][2 * h],
                                               A[2 * tt + 1][2 * h], A[2 * tt][2 * h + 1],
                                               A[2 * tt + 1][2 * h + 1],
                                               h ? xb[nn].z : xb[nn].x,
                                               h ? xb[nn].w : xb[nn].y);
                    // zero point and bias: -136 * sum x for every token
                    constexpr uint32_t kMinus136 = 0xC308C308u;
#pragma unroll
                    for (int h = 0; h < 2; ++h)
#pragma unroll
                        for (int nn = 0; nn < NT; ++nn)
                            mma_bf16_16816(db[u][nn], kMinus136, kMinus136, kMinus136, kMinus136,
                                           h ? xb[nn].z : xb[nn].x, h ? xb[nn].w : xb[nn].y);
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(empty_smem(s));
                ++it;
                return true;
            };
            // acc += s * (d - 136 * xsum) for the first `count` sets
            auto fold = [&](int count) {
#pragma unroll
                for (int u = 0; u < G; ++u) {
                    if (u >= count) break;
#pragma unroll
                    for (int tt = 0; tt < TPW; ++tt)
#pragma unroll
                        for (int nn = 0; nn < NT; ++nn)
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                const float corr = d[u][tt][nn][e] + db[u][nn][e];
                                acc[tt][nn][e] = fmaf(bf16_bits_to_float(sc[2 * tt + (e >> 1)][u]),
                                                      corr, acc[tt][nn][e]);
                                d[u][tt][nn][e] = 0.0f;
                            }
#pragma unroll
                    for (int nn = 0; nn < NT; ++nn)
#pragma unroll
                        for (int e = 0; e < 4; ++e) db[u][nn][e] = 0.0f;
                }
            };
            auto load_scales = [&](int g0) {
#pragma unroll
                for (int q = 0; q < 2 * TPW; ++q)
#pragma unroll
                    for (int u = 0; u < G; ++u)
                        scn[q][u] = (v[q] && g0 + u < KS)
                                       ? static_cast<uint32_t>(__ldg(srow[q] + kgroup(g0 + u)))
                                       : 0u;
            };
            auto take_scales = [&]() {
#pragma unroll
                for (int q = 0; q < 2 * TPW; ++q)
#pragma unroll
                    for (int u = 0; u < G; ++u) sc[q][u] = scn[q][u];
            };
            int ks = 0;
            load_scales(0);
            for (; ok && ks + G <= KS; ks += G) {
                take_scales();
                load_scales(ks + G);  // the next batch's, two batches before use
#pragma unroll
                for (int u = 0; u < G; ++u)
                    if (!stage(u)) { ok = false; break; }
                if (ok) fold(G);
            }
            if (ok && ks < KS) load_scales(ks);
            for (; ok && ks < KS; ++ks) {  // remainder, one group at a time
                take_scales();
                if (ks + 1 < KS) load_scales(ks + 1);
                if (!stage(0)) { ok = false; break; }
                fold(1);
            }
            if (!ok) break;
            // epilogue: d0, d1 -> (upper row, tokens 2c, 2c+1); d2, d3 -> lower row
#pragma unroll
            for (int tt = 0; tt < TPW; ++tt)
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
        }
    }
    __syncthreads();
}

template <int NT, int S, int G, int TPW>
cudaError_t launch_gemv_variant(const CUtensorMap* tx, const CUtensorMap* tw,
                                const GemvParams& p, int grid, cudaStream_t stream) {
    using L = GLayout<NT, S>;
    auto kern = w4a16_gemv_kernel<NT, S, G, TPW>;
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    const int threads = 32 * (1 + (p.rows_per_cta + 16 * TPW - 1) / (16 * TPW));
    kern<<<grid, threads, L::SMEM_BYTES, stream>>>(*tx, *tw, p);
    return cudaGetLastError();
}

}  // namespace

int gemv_rows_per_cta(int64_t N, int sm_count) {
    int64_t per = (N + sm_count - 1) / sm_count;
    per = (per + 15) / 16 * 16;
    if (per > kRowsMax) per = kRowsMax;
    if (per < 16) per = 16;
    return static_cast<int>(per);
}

int gemv_tokens_per_tile(int64_t M) { return M <= 8 ? 8 : M <= 16 ? 16 : 32; }

cudaError_t gemv_launch(const CUtensorMap* tx, const CUtensorMap* tw, const GemvParams& p,
                        int sm_count, cudaStream_t stream) {
    const int grid = p.num_chunks < sm_count ? p.num_chunks : sm_count;
    if (p.M <= 8)
        return launch_gemv_variant<1, 6, W4A16_GEMV_G1, W4A16_GEMV_TPW>(tx, tw, p, grid, stream);
    return launch_gemv_variant<2, 6, W4A16_GEMV_G2, W4A16_GEMV_TPW>(tx, tw, p, grid, stream);
}

}  // namespace w4a16
