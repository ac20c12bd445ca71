// Fused int4-dequant + tcgen05 GEMM for sm_103a.
//
// out[m, n] = sum_k x[m, k] * wd[n, k], wd = RNE_bf16((code - 8) * scale).
//
// Mapping onto the 5th-generation tensor core.  The MMA computes
// D[128 x T] = A[128 x 16] * B[T x 16]^T per instruction with
//   A = 128 dequantised weight rows, held in TENSOR MEMORY,
//   B = T tokens of x, K-major in shared memory (TMA, 128-byte swizzle),
//   D = fp32 accumulator in tensor memory: lane = weight row, column = token.
// Putting the weights in A lets the dequantising warps write bf16 pairs
// straight from registers into tensor memory (tcgen05.st) -- the 4x larger
// bf16 weight tile never touches shared memory, which keeps shared-memory
// bandwidth for the x tiles the MMA reads.
//
// Warp roles (32 * (2 + 4*DQ + 4*EP) threads):
//   warp 0      TMA producer: x tile [T x 64] and packed weight tile [128 x 32 B]
//               per stage into a ring of S_SMEM shared-memory stages;
//   warp 1      allocates tensor memory, one thread issues the MMAs;
//   next 4*DQ   dequantisers, DQ groups of four warps taking stages in turn:
//               thread = one weight row (its TMEM lane), 32 packed bytes ->
//               64 bf16 -> 32 TMEM columns per stage, into a ring of S_TMEM
//               tensor-memory A stages;
//   last 4*EP   epilogue, EP groups of four warps splitting the tile's
//               32-token chunks: tcgen05.ld of the accumulator, the fused
//               epilogue if any (bias, activation, residual), fp32 -> bf16,
//               stores to out.  The next tile's MMAs wait until the
//               accumulator is drained, so two groups halve that wait.
// A warp may only touch the 32 TMEM lanes of its sub-partition (warp % 4), so
// each group of four warps covers all 128 lanes.
//
// Large M runs in thread-block clusters of two CTAs that take the same token
// tile and neighbouring weight tiles in lockstep: each CTA loads half of every
// x stage and multicasts it to both (x crosses from L2 to the SMs once per
// two weight tiles), and a stage slot is refilled only when the MMAs of both
// CTAs are done with it.  Under the GPU's power cap the lower on-chip traffic
// buys clock.
//
// Every wait is bounded (see ptx.cuh); on a timeout the kernel records
// W4A16_ERR_TIMEOUT, drains its own copies and MMAs, frees tensor memory and
// returns.
#include "dequant.cuh"
#include "epilogue.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace w4a16 {

namespace {

constexpr int kRows = 128;  // weight rows per tile (MMA M)
#ifndef W4A16_EPI_SLEEP_NS
#define W4A16_EPI_SLEEP_NS 256
#endif
constexpr uint32_t kEpilogueSleepNs = W4A16_EPI_SLEEP_NS;
constexpr int kBK = 64;     // k per stage (one 128-byte swizzle row of bf16)

template <int T, int S_SMEM, int S_TMEM>
struct Layout {
    static constexpr int X_BYTES = T * kBK * 2;
    static constexpr int W_BYTES = kRows * kBK / 2;
    static constexpr int X_OFF = 0;
    static constexpr int W_OFF = S_SMEM * X_BYTES;
    static constexpr int BAR_OFF = W_OFF + S_SMEM * W_BYTES;
    // full_tma[S_SMEM], empty_smem[S_SMEM], full_a[S_TMEM], empty_a[S_TMEM],
    // d_full, d_empty, drain
    static constexpr int NBARS = 2 * S_SMEM + 2 * S_TMEM + 3;
    static constexpr int MISC_OFF = BAR_OFF + NBARS * 8;
    static constexpr int SMEM_BYTES = MISC_OFF + 16 + 1024;  // + slack for 1024-B alignment
    static constexpr int D_COL = 0;
    static constexpr int A_COL = T;
    static constexpr int COLS_USED = T + S_TMEM * (kBK / 2);
    static constexpr int TMEM_COLS = COLS_USED <= 32    ? 32
                                     : COLS_USED <= 64  ? 64
                                     : COLS_USED <= 128 ? 128
                                     : COLS_USED <= 256 ? 256
                                                        : 512;
    static_assert(COLS_USED <= 512, "tensor memory holds 512 columns");
    static_assert(X_BYTES % 1024 == 0, "x stages must keep 1024-byte alignment");
    static_assert(T % 32 == 0 && T >= 32 && T <= 256, "tokens per tile");
};

// Unit -> (token tile, weight unit): units are rastered in groups of group_t
// token tiles, token tiles fastest; a weight unit is CL consecutive weight
// tiles (one per CTA of a cluster).
__device__ __forceinline__ void unit_coords(int tile, const TsParams& p, int nwu, int& tt, int& wt) {
    const int per_group = p.group_t * nwu;
    const int grp = tile / per_group;
    const int first_t = grp * p.group_t;
    const int rest = p.num_t_tiles - first_t;
    const int gsize = rest < p.group_t ? rest : p.group_t;
    const int local = tile - grp * per_group;
    tt = first_t + local % gsize;
    wt = local / gsize;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// Fused epilogue of one tile for the epilogue thread that owns weight row n
// (TMEM lane `lane` of its sub-partition): the 32-token chunks c0, c0 + cs,
// ... of the T tokens from TMEM column d_col.  Residuals of a chunk are read
// before any of its outputs is written (the residual may be the output).
// SwiGLU pairs rows (n, n ^ 1) = (gate, up) of output column n / 2 across
// neighbouring lanes: the even lane finishes the even tokens, the odd lane
// the odd ones.  Otherwise neighbouring lanes swap values so that each store
// writes the outputs (n, n+1) of one token as a 32-bit word (even n_out).
// The units of a CTA: unit_first, + unit_stride, ... below unit_count (a
// unit is one tile, or with clusters one token tile x CL weight tiles).
// These read the special registers and parameters where they are used,
// which keeps the loops' register use as low as with plain tile indices.
template <int CL>
__device__ __forceinline__ unsigned unit_first() { return blockIdx.x / CL; }
template <int CL>
__device__ __forceinline__ unsigned unit_stride() { return gridDim.x / CL; }
template <int CL>
__device__ __forceinline__ int weight_units(const TsParams& p) {
    return CL == 1 ? p.num_w_tiles : (p.num_w_tiles + CL - 1) / CL;
}
template <int CL>
__device__ __forceinline__ int unit_count(const TsParams& p) {
    return CL == 1 ? p.num_tiles : p.num_t_tiles * weight_units<CL>(p);
}

// (token tile, weight tile) of rank `rank` of a cluster of CL in a unit; a
// weight tile past N (odd tile count, second CTA) loads zeros and stores
// nothing.
template <int CL>
__device__ __forceinline__ void unit_tile(int unit, const TsParams& p, int rank, int& tt, int& wt) {
    if constexpr (CL == 1) {
        unit_coords(unit, p, p.num_w_tiles, tt, wt);
    } else {
        int wu;
        unit_coords(unit, p, weight_units<CL>(p), tt, wu);
        wt = wu * CL + rank;
    }
}

template <int T>
__device__ __forceinline__ void fused_epilogue_tile(const TsParams& p, uint32_t d_col, int m0,
                                                    int n, int lane, int c0, int cs) {
    const Epilogue& e = p.epi;
    const bool n_ok = n < p.N;
    const bool has_res = e.residual != nullptr;
    const float b = (e.bias != nullptr && n_ok) ? bf16_to_f32(e.bias[n]) : 0.0f;
    const bool odd = (lane & 1) != 0;
#pragma unroll 1
    for (int c = c0; c < T / 32; c += cs) {
        uint32_t v[32];
        tmem_ld_32x32b_x32(d_col + c * 32, v);
        tmem_ld_wait(v);
        const int mbase = m0 + c * 32;
        if (e.act == kActSwiGLU) {
            const int col = n >> 1;
            float r[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                const int m = mbase + 2 * j + (odd ? 1 : 0);
                r[j] = (has_res && m < p.M && n_ok)
                           ? bf16_to_f32(e.residual[static_cast<int64_t>(m) * e.n_out + col])
                           : 0.0f;
            }
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                const float z0 = __uint_as_float(v[2 * j]) + b;
                const float z1 = __uint_as_float(v[2 * j + 1]) + b;
                const float other = __shfl_xor_sync(0xffffffffu, odd ? z0 : z1, 1);
                const int m = mbase + 2 * j + (odd ? 1 : 0);
                const float h = (odd ? silu_f32(other) * z1 : silu_f32(z0) * other) + r[j];
                if (m < p.M && n_ok) p.out[static_cast<int64_t>(m) * e.n_out + col] = f32_to_bf16_rn(h);
            }
        } else if ((e.n_out & 1) == 0) {
            // even lane: token 2j, columns (n, n+1); odd lane: token 2j+1, (n-1, n)
            const int col = odd ? n - 1 : n;
            uint32_t rw[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                const int m = mbase + 2 * j + (odd ? 1 : 0);
                rw[j] = (has_res && m < p.M && n_ok)
                            ? *reinterpret_cast<const uint32_t*>(
                                  e.residual + static_cast<int64_t>(m) * e.n_out + col)
                            : 0u;
            }
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                float h0 = __uint_as_float(v[2 * j]) + b, h1 = __uint_as_float(v[2 * j + 1]) + b;
                if (e.act == kActGELU) {
                    h0 = gelu_f32(h0);
                    h1 = gelu_f32(h1);
                }
                const float other = __shfl_xor_sync(0xffffffffu, odd ? h0 : h1, 1);
                const int m = mbase + 2 * j + (odd ? 1 : 0);
                // (lo, hi) = outputs (col, col + 1) of token m
                float lo = odd ? other : h0, hi = odd ? h1 : other;
                lo += __uint_as_float(rw[j] << 16);
                hi += __uint_as_float(rw[j] & 0xFFFF0000u);
                if (m < p.M && n_ok)
                    *reinterpret_cast<uint32_t*>(p.out + static_cast<int64_t>(m) * e.n_out + col) =
                        pack_bf16x2(lo, hi);
            }
        } else {
            float r[32];
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                const int m = mbase + j;
                r[j] = (has_res && m < p.M && n_ok)
                           ? bf16_to_f32(e.residual[static_cast<int64_t>(m) * e.n_out + n])
                           : 0.0f;
            }
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                const int m = mbase + j;
                const float z = __uint_as_float(v[j]) + b;
                const float h = (e.act == kActGELU ? gelu_f32(z) : z) + r[j];
                if (m < p.M && n_ok) p.out[static_cast<int64_t>(m) * e.n_out + n] = f32_to_bf16_rn(h);
            }
        }
    }
}

// Plain epilogue of one tile: bf16 stores of the accumulators; for even N
// neighbouring lanes pair up so that each store writes two adjacent outputs
// (n, n+1) of one token as a 32-bit word.
template <int T>
__device__ __forceinline__ void plain_epilogue_tile(const TsParams& p, uint32_t d_col, int m0,
                                                    int n, int lane, bool n_even, int c0, int cs) {
#pragma unroll 1
    for (int c = c0; c < T / 32; c += cs) {
        uint32_t v[32];
        tmem_ld_32x32b_x32(d_col + c * 32, v);
        tmem_ld_wait(v);
        const int mbase = m0 + c * 32;
        if (n_even) {
            // Pair neighbouring lanes so that each store writes two
            // adjacent outputs (n, n+1) of one token as a 32-bit word.
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                const float f0 = __uint_as_float(v[2 * j]);
                const float f1 = __uint_as_float(v[2 * j + 1]);
                const float send = (lane & 1) ? f0 : f1;
                const float other = __shfl_xor_sync(0xffffffffu, send, 1);
                int m, col;
                uint32_t word;
                if ((lane & 1) == 0) {
                    m = mbase + 2 * j;
                    col = n;
                    word = pack_bf16x2(f0, other);
                } else {
                    m = mbase + 2 * j + 1;
                    col = n - 1;
                    word = pack_bf16x2(other, f1);
                }
                if (m < p.M && col < p.N)
                    *reinterpret_cast<uint32_t*>(p.out + static_cast<int64_t>(m) * p.N +
                                                 col) = word;
            }
        } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) {
                const int m = mbase + j;
                if (m < p.M && n < p.N) {
                    const uint32_t word = pack_bf16x2(__uint_as_float(v[j]), 0.0f);
                    p.out[static_cast<int64_t>(m) * p.N + n] =
                        static_cast<uint16_t>(word & 0xFFFFu);
                }
            }
        }
    }
}

template <int DQ, int EP>
constexpr int threads_for() {
    return 32 * (2 + 4 * DQ + 4 * EP);
}

// CL: CTAs per thread-block cluster.  With CL = 2 the two CTAs of a cluster
// take the same token tile and neighbouring weight tiles in lockstep; each
// loads half of every x stage and multicasts it to both, so x crosses from
// L2 once per pair of weight tiles, and a stage slot is refilled only when
// the MMAs of both CTAs are done with it (each CTA's MMA completion arrives
// on the empty barrier of both).
template <int T, int S_SMEM, int S_TMEM, int DQ, int EP, int MIN_BLOCKS, bool FUSED, int CL>
__global__ void __launch_bounds__(threads_for<DQ, EP>(), MIN_BLOCKS)
    w4a16_ts_kernel(const __grid_constant__ CUtensorMap tmap_x,
                    const __grid_constant__ CUtensorMap tmap_w, const TsParams p) {
    using L = Layout<T, S_SMEM, S_TMEM>;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;
    uint8_t* smem = smem_raw + (sbase - raw);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    static_assert(CL == 1 || CL == 2, "cluster size");
    constexpr uint16_t kClusterMask = (1u << CL) - 1u;
    const int rank = static_cast<int>(blockIdx.x % CL);  // rank in the cluster

    const uint32_t bars = sbase + L::BAR_OFF;
    auto full_tma = [&](int s) { return bars + 8u * s; };
    auto empty_smem = [&](int s) { return bars + 8u * (S_SMEM + s); };
    auto full_a = [&](int s) { return bars + 8u * (2 * S_SMEM + s); };
    auto empty_a = [&](int s) { return bars + 8u * (2 * S_SMEM + S_TMEM + s); };
    const uint32_t d_full = bars + 8u * (2 * S_SMEM + 2 * S_TMEM);
    const uint32_t d_empty = d_full + 8u;
    const uint32_t drain = d_full + 16u;
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::MISC_OFF);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::MISC_OFF + 4);

    if (threadIdx.x == 0) {
        for (int s = 0; s < S_SMEM; ++s) {
            mbar_init(full_tma(s), 1);
            mbar_init(empty_smem(s), CL);  // the MMA completion of every CTA of the cluster
        }
        for (int s = 0; s < S_TMEM; ++s) {
            mbar_init(full_a(s), 4);  // one arrival per dequant warp of the stage's group
            mbar_init(empty_a(s), 1);
        }
        mbar_init(d_full, 1);
        mbar_init(d_empty, 4 * EP);  // one arrival per epilogue warp
        mbar_init(drain, 1);
        *abort_flag = 0;
        fence_mbar_init();
        prefetch_tmap(&tmap_x);
        prefetch_tmap(&tmap_w);
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), L::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    if constexpr (CL > 1)
        cluster_sync();  // barriers initialised before any peer signals them
    else
        __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    const int KT = p.K / kBK;
    const int KG = p.K / p.g;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            uint32_t it = 0;
            bool ok = true;
            for (int unit = unit_first<CL>(); ok && unit < unit_count<CL>(p); unit += unit_stride<CL>()) {
                int tt, wt;
                unit_tile<CL>(unit, p, rank, tt, wt);
                const int t0 = tt * T, n0 = wt * kRows;
                for (int kt = 0; kt < KT; ++kt, ++it) {
                    const int s = it % S_SMEM;
                    const uint32_t ph = (it / S_SMEM) & 1u;
                    if (!wait_one(empty_smem(s), ph ^ 1u, abort_flag, p.status)) {
                        ok = false;
                        break;
                    }
                    // x: all of it from this CTA, or this CTA's half multicast to both
                    mbar_arrive_expect_tx(full_tma(s), L::X_BYTES + L::W_BYTES);
                    if constexpr (CL == 1)
                        tma_load_2d(sbase + L::X_OFF + s * L::X_BYTES, &tmap_x, full_tma(s),
                                    kt * kBK, t0);
                    else
                        tma_load_2d_multicast(
                            sbase + L::X_OFF + s * L::X_BYTES + rank * (L::X_BYTES / CL), &tmap_x,
                            full_tma(s), kt * kBK, t0 + rank * (T / CL), kClusterMask);
                    tma_load_2d(sbase + L::W_OFF + s * L::W_BYTES, &tmap_w, full_tma(s),
                                kt * (kBK / 2), n0);
                }
            }
            // Drain: every load this thread issued has landed before exit.
            const uint32_t last = it < static_cast<uint32_t>(S_SMEM) ? it : S_SMEM;
            for (uint32_t i = it - last; i < it; ++i) {
                uint64_t t0 = global_timer_ns();
                while (!mbar_try_wait(full_tma(i % S_SMEM), (i / S_SMEM) & 1u)) {
                    if (global_timer_ns() - t0 > kWaitLimitNs) break;
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t idesc = idesc_bf16_f32(kRows, T);
            uint32_t it = 0, tcount = 0;
            bool ok = true;
            bool issued = false;
            for (int unit = unit_first<CL>(); ok && unit < unit_count<CL>(p); unit += unit_stride<CL>(), ++tcount) {
                if (!wait_one(d_empty, (tcount & 1u) ^ 1u, abort_flag, p.status)) break;
                tc_fence_after();
                for (int kt = 0; kt < KT; ++kt, ++it) {
                    const int s = it % S_SMEM;
                    const int sa = it % S_TMEM;
                    if (!wait_one(full_tma(s), (it / S_SMEM) & 1u, abort_flag, p.status) ||
                        !wait_one(full_a(sa), (it / S_TMEM) & 1u, abort_flag, p.status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t xs = sbase + L::X_OFF + s * L::X_BYTES;
#pragma unroll
                    for (int ks = 0; ks < kBK / 16; ++ks) {
                        const uint32_t a = tmem + L::A_COL + sa * (kBK / 2) + ks * 8;
                        const uint64_t b = sdesc_kmajor_sw128(xs + ks * 32);
                        tc_mma_ts(tmem + L::D_COL, a, b, idesc, (kt | ks) != 0);
                    }
                    issued = true;
                    if constexpr (CL == 1)
                        tc_commit(empty_smem(s));
                    else
                        tc_commit_multicast(empty_smem(s), kClusterMask);
                    tc_commit(empty_a(sa));
                }
                if (!ok) break;
                tc_commit(d_full);
            }
            if (issued) {
                // Drain: all MMAs issued by this thread have completed.
                tc_commit(drain);
                uint64_t t0 = global_timer_ns();
                while (!mbar_try_wait(drain, 0)) {
                    if (global_timer_ns() - t0 > kWaitLimitNs) break;
                }
            }
            if constexpr (CL > 1) {
                // and every CTA's completion arrivals on this CTA's empty
                // barriers have landed (none is in flight at exit)
                const uint32_t last = it < static_cast<uint32_t>(S_SMEM) ? it : S_SMEM;
                for (uint32_t i = it - last; i < it; ++i) {
                    const uint64_t t1 = global_timer_ns();
                    while (!mbar_try_wait(empty_smem(i % S_SMEM), (i / S_SMEM) & 1u)) {
                        if (global_timer_ns() - t1 > kWaitLimitNs) break;
                    }
                }
            }
        }
    } else if (warp < 2 + 4 * DQ) {
        // ------------------------------------------------------------ dequantisers
        const int dgrp = (warp - 2) >> 2;  // which group of four warps
        const int sub = warp & 3;
        const int r = sub * 32 + lane;
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(sub * 32) << 16);
        // stages per scale group; a shift when that is a power of two
        const int spg = p.g / kBK;
        const int spg_shift = (spg & (spg - 1)) == 0 ? __ffs(spg) - 1 : -1;
        auto grp_of = [&](int kt) { return spg_shift >= 0 ? (kt >> spg_shift) : kt / spg; };
        // scale row of the tile processed at per-CTA tile index j (nullptr: none)
        auto scale_row = [&](int j) -> const uint16_t* {
            const int unit = unit_first<CL>() + j * unit_stride<CL>();
            if (unit >= unit_count<CL>(p)) return nullptr;
            int tt, wt;
            unit_tile<CL>(unit, p, rank, tt, wt);
            const int n = wt * kRows + r;
            return n < p.N ? p.scales + static_cast<int64_t>(n) * KG : nullptr;
        };
        // one-stage lookahead: the scale for this warp's next stage is loaded
        // while the current one is dequantised
        auto load_scale = [&](uint32_t i) -> uint16_t {
            const int j = static_cast<int>(i / static_cast<uint32_t>(KT));
            const int kt = static_cast<int>(i - static_cast<uint32_t>(j) * KT);
            const uint16_t* row = scale_row(j);
            return row ? __ldg(row + grp_of(kt)) : static_cast<uint16_t>(0);
        };
        uint32_t it = 0;
        bool ok = true;
        uint16_t s_next = load_scale(static_cast<uint32_t>(dgrp));
        for (int j = 0, unit = unit_first<CL>(); ok && unit < unit_count<CL>(p); ++j, unit += unit_stride<CL>()) {
            const uint16_t* srow = scale_row(j);
            for (int kt = 0; kt < KT; ++kt, ++it) {
                if (static_cast<int>(it % DQ) != dgrp) continue;
                const uint16_t s_cur = s_next;
                const int kt2 = kt + DQ;
                if (kt2 < KT)
                    s_next = srow ? __ldg(srow + grp_of(kt2)) : static_cast<uint16_t>(0);
                else
                    s_next = load_scale(it + DQ);
                const int s = it % S_SMEM;
                const int sa = it % S_TMEM;
                if (!wait_warp(full_tma(s), (it / S_SMEM) & 1u, abort_flag, p.status) ||
                    !wait_warp(empty_a(sa), ((it / S_TMEM) & 1u) ^ 1u, abort_flag, p.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint4* wrow =
                    reinterpret_cast<const uint4*>(smem + L::W_OFF + s * L::W_BYTES + r * 32);
                const uint4 w0 = wrow[0];
                const uint4 w1 = wrow[1];
                const uint32_t s2 = splat_bf16(s_cur);
                uint32_t v[32];
                dequant_word(w0.x, s2, v + 0);
                dequant_word(w0.y, s2, v + 4);
                dequant_word(w0.z, s2, v + 8);
                dequant_word(w0.w, s2, v + 12);
                dequant_word(w1.x, s2, v + 16);
                dequant_word(w1.y, s2, v + 20);
                dequant_word(w1.z, s2, v + 24);
                dequant_word(w1.w, s2, v + 28);
                tmem_st_32x32b_x32(lane_base + L::A_COL + sa * (kBK / 2), v);
                tmem_st_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(full_a(sa));
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue
        // EP groups of four warps; group eg takes the 32-token chunks eg, eg + EP, ...
        const int sub = warp & 3;
        const int eg = (warp - (2 + 4 * DQ)) >> 2;
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(sub * 32) << 16);
        const bool n_even = (p.N & 1) == 0;
        uint32_t tcount = 0;
        for (int unit = unit_first<CL>(); unit < unit_count<CL>(p); unit += unit_stride<CL>(), ++tcount) {
            int tt, wt;
            unit_tile<CL>(unit, p, rank, tt, wt);
            if (!wait_warp_sleep(d_full, tcount & 1u, abort_flag, p.status, kEpilogueSleepNs))
                break;
            tc_fence_after();
            const int n = wt * kRows + sub * 32 + lane;
            if constexpr (FUSED)
                fused_epilogue_tile<T>(p, lane_base + L::D_COL, tt * T, n, lane, eg, EP);
            else
                plain_epilogue_tile<T>(p, lane_base + L::D_COL, tt * T, n, lane, n_even, eg, EP);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(d_empty);
        }
    }

    tc_fence_before();
    if constexpr (CL > 1)
        cluster_sync();  // no CTA leaves while a peer may still signal it
    else
        __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, L::TMEM_COLS);
}

template <int T, int S_SMEM, int S_TMEM, int DQ, int EP, int MIN_BLOCKS, int CL>
cudaError_t launch_variant(const CUtensorMap* tx, const CUtensorMap* tw, const TsParams& p,
                           int grid, cudaStream_t stream) {
    using L = Layout<T, S_SMEM, S_TMEM>;
    // the plain variant carries none of the fused epilogue's code or registers
    const bool fused =
        p.epi.bias != nullptr || p.epi.residual != nullptr || p.epi.act != kActNone;
    auto kern = fused ? w4a16_ts_kernel<T, S_SMEM, S_TMEM, DQ, EP, MIN_BLOCKS, true, CL>
                      : w4a16_ts_kernel<T, S_SMEM, S_TMEM, DQ, EP, MIN_BLOCKS, false, CL>;
    // Idempotent; cheap enough to repeat per launch and per device.
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    if constexpr (CL == 1) {
        kern<<<grid, threads_for<DQ, EP>(), L::SMEM_BYTES, stream>>>(*tx, *tw, p);
    } else {
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = CL;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.gridDim = dim3(static_cast<unsigned>(grid));
        cfg.blockDim = dim3(threads_for<DQ, EP>());
        cfg.dynamicSmemBytes = L::SMEM_BYTES;
        cfg.stream = stream;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        e = cudaLaunchKernelEx(&cfg, kern, *tx, *tw, p);
        if (e != cudaSuccess) return e;
    }
    return cudaGetLastError();
}

// Large M: 256 tokens per tile, 6 stages of (32 KB x + 4 KB packed weights),
// tensor memory = 256 accumulator columns + 6 x 32 A columns.
#ifndef W4A16_GEMM_DQ
#define W4A16_GEMM_DQ 2
#endif
#ifndef W4A16_GEMM_SS
#define W4A16_GEMM_SS 6
#endif
#ifndef W4A16_GEMM_EP
#define W4A16_GEMM_EP 2
#endif
constexpr int kGemmT = 256, kGemmSS = W4A16_GEMM_SS, kGemmST = 6, kGemmDQ = W4A16_GEMM_DQ,
              kGemmEP = W4A16_GEMM_EP;
// Small M: 32 tokens per tile, 8 shared-memory stages of 8 KB, 3 A stages;
// 128 tensor-memory columns so that three CTAs share an SM.
constexpr int kGemvT = 32, kGemvSS = 8, kGemvST = 3, kGemvDQ = 1, kGemvEP = 1;

}  // namespace

int ts_tokens_per_tile(TsVariant v) { return v == TsVariant::kGemm256 ? kGemmT : kGemvT; }

// Clusters of CL that can be resident at once (SMs left over in a GPC cannot
// take one); cached per device and cluster size.
template <int CL>
int gemm_cluster_slots(int sm_count) {
    constexpr int kMaxDev = 64;
    static int cache[kMaxDev] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return sm_count / CL;
    if (cache[dev] > 0) return cache[dev];
    using L = Layout<kGemmT, kGemmSS, kGemmST>;
    auto kern = w4a16_ts_kernel<kGemmT, kGemmSS, kGemmST, kGemmDQ, kGemmEP, 1, false, CL>;
    int n = 0;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM_BYTES) ==
        cudaSuccess) {
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = CL;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.gridDim = dim3(static_cast<unsigned>(sm_count / CL * CL));
        cfg.blockDim = dim3(threads_for<kGemmDQ, kGemmEP>());
        cfg.dynamicSmemBytes = L::SMEM_BYTES;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) n = 0;
    }
    cudaGetLastError();  // a failed query leaves no sticky error for the next launch
    if (n <= 0) n = sm_count / CL;
    cache[dev] = n;
    return n;
}

int ts_grid(TsVariant v, const TsParams& p, int sm_count) {
    if (v == TsVariant::kGemm256) {
        if (p.cluster == 2) {
            const int units = p.num_t_tiles * ((p.num_w_tiles + 1) / 2);
            const int slots = gemm_cluster_slots<2>(sm_count);
            return 2 * (units < slots ? units : slots);
        }
        return p.num_tiles < sm_count ? p.num_tiles : sm_count;
    }
    return p.num_tiles;
}

cudaError_t ts_launch(TsVariant v, const CUtensorMap* tx, const CUtensorMap* tw,
                      const TsParams& p, int grid, cudaStream_t stream) {
    if (v == TsVariant::kGemm256) {
        if (p.cluster == 2)
            return launch_variant<kGemmT, kGemmSS, kGemmST, kGemmDQ, kGemmEP, 1, 2>(tx, tw, p,
                                                                                   grid, stream);
        return launch_variant<kGemmT, kGemmSS, kGemmST, kGemmDQ, kGemmEP, 1, 1>(tx, tw, p, grid,
                                                                               stream);
    }
    return launch_variant<kGemvT, kGemvSS, kGemvST, kGemvDQ, kGemvEP, 3, 1>(tx, tw, p, grid,
                                                                           stream);
}

}  // namespace w4a16
