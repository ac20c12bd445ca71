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

// PAIR: a CTA pair (cta_group::2) computes 2 x 128 weight rows x T tokens;
// each CTA stages T/2 tokens of x and its own 128 weight rows.  NB: the tile's
// tokens form NB accumulator blocks of T/NB columns, one MMA each per k step,
// all reading the same A stage (so one dequantised stage serves T tokens).
template <int T, int S_SMEM, int S_TMEM, bool PAIR, int NB = 1>
struct Layout {
    static constexpr int XT = PAIR ? T / 2 : T;  // tokens of x staged per CTA
    static constexpr int XB = XT / NB;           // token rows per x box (one per block)
    static constexpr int X_BOX = XB * kBK * 2;
    static constexpr int X_BYTES = NB * X_BOX;
    static constexpr int W_BYTES = kRows * kBK / 2;
    static constexpr int X_OFF = 0;
    static constexpr int W_OFF = S_SMEM * X_BYTES;
    static constexpr int BAR_OFF = W_OFF + S_SMEM * W_BYTES;
    // full_tma[S_SMEM], empty_smem[S_SMEM], full_a[S_TMEM], empty_a[S_TMEM],
    // d_full, d_empty, drain
    static constexpr int NBARS = 2 * S_SMEM + 2 * S_TMEM + 3;
    // misc: tensor-memory base, abort flag, and (pairs) the stages and tiles
    // whose completion the MMA thread committed, handed to both CTAs at exit
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
    static_assert(X_BOX % 1024 == 0, "x boxes must keep 1024-byte alignment");
    static_assert(T % 32 == 0 && T >= 32 && T / NB <= 256 && T % NB == 0, "tokens per tile");
};

// Unit -> (token tile, weight unit): units are rastered in groups of group_t
// token tiles, token tiles fastest, so that the CTAs running at the same time
// share x and weight tiles in L2.  A weight unit is CW consecutive weight
// tiles: one per CTA (CW = 1), or the two tiles of a CTA pair (CW = 2).
__device__ __forceinline__ void unit_coords(int unit, const TsParams& p, int nwu, int& tt, int& wu) {
    const int per_group = p.group_t * nwu;
    const int grp = unit / per_group;
    const int first_t = grp * p.group_t;
    const int rest = p.num_t_tiles - first_t;
    const int gsize = rest < p.group_t ? rest : p.group_t;
    const int local = unit - grp * per_group;
    tt = first_t + local % gsize;
    wu = local / gsize;
}

// The units of a CTA: unit_first, + unit_stride, ... below unit_count.  The
// two CTAs of a pair walk the same units.  These read the special registers
// and parameters where they are used, which keeps the loops' register use as
// low as with plain tile indices.
template <int CW>
__device__ __forceinline__ int unit_first() { return static_cast<int>(blockIdx.x) / CW; }
template <int CW>
__device__ __forceinline__ int unit_stride() { return static_cast<int>(gridDim.x) / CW; }
template <int CW>
__device__ __forceinline__ int weight_units(const TsParams& p) {
    return CW == 1 ? p.num_w_tiles : (p.num_w_tiles + CW - 1) / CW;
}
template <int CW>
__device__ __forceinline__ int unit_count(const TsParams& p) {
    return CW == 1 ? p.num_tiles : p.num_t_tiles * weight_units<CW>(p);
}

// (token tile, weight tile) of the CTA of rank `rank` in its pair; a weight
// tile past N (odd tile count, second CTA) loads zeros and stores nothing.
template <int CW>
__device__ __forceinline__ void unit_tile(int unit, const TsParams& p, int rank, int& tt, int& wt) {
    int wu;
    unit_coords(unit, p, weight_units<CW>(p), tt, wu);
    wt = wu * CW + rank;
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
                if (m < p.M && col < p.N &&
                    dbg_check((col & 1) == 0 && col + 1 < p.N && m >= 0 && col >= 0, p.status))
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

// PAIR = false: one CTA per tile, D[128 x T] per tcgen05.mma.cta_group::1.
// PAIR = true: a thread-block cluster of two CTAs computes 256 weight rows x T
// tokens with tcgen05.mma.cta_group::2 (M = 256), issued by one thread of
// the even CTA.  Each CTA stages its own T/2 tokens of x and its own 128
// weight rows, dequantises them into its own tensor memory (A) and holds its
// 128 rows x T of the accumulator; the MMA reads B from both CTAs' shared
// memory, so x crosses from L2 to the SMs once per two weight tiles and each
// SM's shared memory supplies half of the B operand.  Hand-offs between the
// CTAs: the odd CTA's dequant and epilogue warps arrive on the even CTA's
// full_a and d_empty barriers (remote arrivals without release: they hand
// over tensor-memory reads and writes that tcgen05.wait has completed); the
// even CTA's commits
// arrive on the empty_smem / empty_a / d_full barriers of both CTAs.  Each
// CTA's TMA loads complete on its own full_tma barrier, which its dequant
// warps wait on before they arrive on full_a: the MMA's wait on full_a
// covers both CTAs' x and weight stages.
template <int T, int S_SMEM, int S_TMEM, int DQ, int EP, int MIN_BLOCKS, bool FUSED, bool PAIR,
          int NB>
__global__ void __launch_bounds__(threads_for<DQ, EP>(), MIN_BLOCKS)
    w4a16_ts_kernel(const __grid_constant__ CUtensorMap tmap_x,
                    const __grid_constant__ CUtensorMap tmap_w, const TsParams p) {
    using L = Layout<T, S_SMEM, S_TMEM, PAIR, NB>;
    constexpr int CW = PAIR ? 2 : 1;
    // Pairs run one ring: a stage's shared-memory slot and tensor-memory A
    // slot are released together by one commit per CTA (two commits per
    // stage instead of four; 1463 -> 1607 TFLOP/s on the QKV prefill).
    constexpr bool kUnified = PAIR && S_SMEM == S_TMEM;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;
    uint8_t* smem = smem_raw + (sbase - raw);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int rank = PAIR ? static_cast<int>(cluster_ctarank()) : 0;
    const bool leader = rank == 0;  // issues the MMAs (always, without pairs)

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
    volatile uint32_t* handoff = reinterpret_cast<volatile uint32_t*>(smem + L::MISC_OFF + 8);
    // arrivals for the MMA thread go to the even CTA's barriers
    auto at_leader = [&](uint32_t a) { return PAIR ? mapa_shared(a, 0) : a; };

    if (threadIdx.x == 0) {
        for (int s = 0; s < S_SMEM; ++s) {
            mbar_init(full_tma(s), 1);
            mbar_init(empty_smem(s), 1);
        }
        for (int s = 0; s < S_TMEM; ++s) {
            mbar_init(full_a(s), 4 * CW);  // one arrival per dequant warp of the stage's group, per CTA
            mbar_init(empty_a(s), 1);
        }
        mbar_init(d_full, 1);
        mbar_init(d_empty, 4 * EP * CW);  // one arrival per epilogue warp, per CTA
        mbar_init(drain, 1);
        *abort_flag = 0;
        handoff[0] = 0u;
        handoff[1] = 0u;
        fence_mbar_init();
        prefetch_tmap(&tmap_x);
        prefetch_tmap(&tmap_w);
    }
    if (warp == 1) {
        if constexpr (PAIR) {
            tmem_alloc_pair(smem_u32(tmem_slot), L::TMEM_COLS);
            tmem_relinquish_pair();
        } else {
            tmem_alloc(smem_u32(tmem_slot), L::TMEM_COLS);
            tmem_relinquish();
        }
    }
    tc_fence_before();
    if constexpr (PAIR)
        cluster_sync();  // both CTAs' barriers and tensor memory exist before any hand-off
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
            for (int unit = unit_first<CW>(); ok && unit < unit_count<CW>(p); unit += unit_stride<CW>()) {
                int tt, wt;
                unit_tile<CW>(unit, p, rank, tt, wt);
                // block nb of the tile: tokens tt T + nb T/NB .., this CTA's XB of them
                const int t0 = tt * T + rank * L::XB, n0 = wt * kRows;
                for (int kt = 0; kt < KT; ++kt, ++it) {
                    const int s = it % S_SMEM;
                    const uint32_t ph = (it / S_SMEM) & 1u;
                    if (!wait_one<PAIR>(empty_smem(s), ph ^ 1u, abort_flag, p.status, p.wait_ns)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(full_tma(s), L::X_BYTES + L::W_BYTES);
                    const uint32_t xd = sbase + L::X_OFF + s * L::X_BYTES;
                    const uint32_t wd = sbase + L::W_OFF + s * L::W_BYTES;
#pragma unroll
                    for (int nb = 0; nb < NB; ++nb) {
                        if (dbg_check(tma_box_ok(xd + nb * L::X_BOX, L::X_BOX, 1024, sbase,
                                                 sbase + L::W_OFF, kt * kBK, 2) && t0 >= 0,
                                      p.status))
                            tma_load_2d(xd + nb * L::X_BOX, &tmap_x, full_tma(s), kt * kBK,
                                        t0 + nb * (T / NB));
                    }
                    if (dbg_check(tma_box_ok(wd, L::W_BYTES, 256, sbase + L::W_OFF,
                                             sbase + L::BAR_OFF, kt * (kBK / 2), 1) && n0 >= 0,
                                  p.status))
                        tma_load_2d(wd, &tmap_w, full_tma(s), kt * (kBK / 2), n0);
                }
            }
            // Drain: every load this thread issued has landed before exit.
            const uint32_t last = it < static_cast<uint32_t>(S_SMEM) ? it : S_SMEM;
            for (uint32_t i = it - last; i < it; ++i) settle(full_tma(i % S_SMEM), (i / S_SMEM) & 1u);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0 && leader) {
            constexpr uint32_t idesc = idesc_bf16_f32(kRows * CW, T / NB);
            uint32_t it = 0, tcount = 0, tiles_done = 0;
            bool ok = true;
            bool issued = false;
            // every commit arrives on this CTA's barrier and, for a pair, on
            // the same barrier of the odd CTA
            auto commit = [&](uint32_t bar) {
                if constexpr (PAIR) {
                    tc_commit_pair(bar);
                    tc_commit_pair(mapa_shared(bar, 1));
                } else {
                    tc_commit(bar);
                }
            };
            for (int unit = unit_first<CW>(); ok && unit < unit_count<CW>(p); unit += unit_stride<CW>(), ++tcount) {
                if (!wait_one<PAIR>(d_empty, (tcount & 1u) ^ 1u, abort_flag, p.status, p.wait_ns)) break;
                tc_fence_after();
                for (int kt = 0; kt < KT; ++kt, ++it) {
                    const int s = it % S_SMEM;
                    const int sa = it % S_TMEM;
                    if (!wait_one(full_tma(s), (it / S_SMEM) & 1u, abort_flag, p.status, p.wait_ns) ||
                        !wait_one<PAIR>(full_a(sa), (it / S_TMEM) & 1u, abort_flag, p.status, p.wait_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t xs = sbase + L::X_OFF + s * L::X_BYTES;
                    if (!dbg_check(L::A_COL + (sa + 1) * (kBK / 2) <= L::TMEM_COLS &&
                                       L::D_COL + T <= L::A_COL,
                                   p.status))
                        continue;
#pragma unroll
                    for (int ks = 0; ks < kBK / 16; ++ks) {
                        const uint32_t a = tmem + L::A_COL + sa * (kBK / 2) + ks * 8;
#pragma unroll
                        for (int nb = 0; nb < NB; ++nb) {
                            const uint32_t d = tmem + L::D_COL + nb * (T / NB);
                            const uint64_t b = sdesc_kmajor_sw128(xs + nb * L::X_BOX + ks * 32);
                            if constexpr (PAIR)
                                tc_mma_ts_pair(d, a, b, idesc, (kt | ks) != 0);
                            else
                                tc_mma_ts(d, a, b, idesc, (kt | ks) != 0);
                        }
                    }
                    issued = true;
                    commit(empty_smem(s));
                    if constexpr (!kUnified) commit(empty_a(sa));
                }
                if (!ok) break;
                commit(d_full);
                ++tiles_done;
            }
            if (issued) {
                // Drain: all MMAs issued by this thread have completed.
                if constexpr (PAIR)
                    tc_commit_pair(drain);
                else
                    tc_commit(drain);
                settle(drain, 0);
            }
            if constexpr (PAIR) {
                // what both CTAs must see land on their barriers before exit
                handoff[0] = it;
                handoff[1] = tiles_done;
                const uint32_t h = smem_u32(const_cast<uint32_t*>(handoff));
                st_shared_cluster_u32(mapa_shared(h, 1), it);
                st_shared_cluster_u32(mapa_shared(h + 4, 1), tiles_done);
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
        // scale row of the tile processed at per-CTA unit index j (nullptr: none)
        auto scale_row = [&](int j) -> const uint16_t* {
            const int unit = unit_first<CW>() + j * unit_stride<CW>();
            if (unit >= unit_count<CW>(p)) return nullptr;
            int tt, wt;
            unit_tile<CW>(unit, p, rank, tt, wt);
            const int n = wt * kRows + r;
            return n < p.N ? p.scales + static_cast<int64_t>(n) * KG : nullptr;
        };
        // one-stage lookahead: the scale for this warp's next stage is loaded
        // while the current one is dequantised
        auto load_scale = [&](uint32_t i) -> uint16_t {
            const int j = static_cast<int>(i / static_cast<uint32_t>(KT));
            const int kt = static_cast<int>(i - static_cast<uint32_t>(j) * KT);
            const uint16_t* row = scale_row(j);
            return row && dbg_check(grp_of(kt) < KG, p.status) ? __ldg(row + grp_of(kt))
                                                              : static_cast<uint16_t>(0);
        };
        uint32_t it = 0;
        bool ok = true;
        uint16_t s_next = load_scale(static_cast<uint32_t>(dgrp));
        for (int j = 0, unit = unit_first<CW>(); ok && unit < unit_count<CW>(p); ++j, unit += unit_stride<CW>()) {
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
                if (!wait_warp(full_tma(s), (it / S_SMEM) & 1u, abort_flag, p.status, p.wait_ns) ||
                    !wait_warp<PAIR>(kUnified ? empty_smem(s) : empty_a(sa),
                                     ((it / S_TMEM) & 1u) ^ 1u, abort_flag, p.status, p.wait_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                // the weight box comes with the 32-byte swizzle: the two 16-byte
                // halves of rows 4-7 of every 8 are swapped, so the 8 lanes of a
                // load phase read 8 distinct bank groups
                const uint8_t* wrow = smem + L::W_OFF + s * L::W_BYTES + r * 32;
                const uint32_t swz = static_cast<uint32_t>((r >> 2) & 1) * 16u;
                const uint4 w0 = *reinterpret_cast<const uint4*>(wrow + swz);
                const uint4 w1 = *reinterpret_cast<const uint4*>(wrow + (16u ^ swz));
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
                if (dbg_check(L::A_COL + (sa + 1) * (kBK / 2) <= L::TMEM_COLS, p.status))
                    tmem_st_32x32b_x32(lane_base + L::A_COL + sa * (kBK / 2), v);
                tmem_st_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    // the odd CTA signals its A stage across the pair; its
                    // tensor-memory stores are complete (wait::st above)
                    if (PAIR && !leader)
                        mbar_arrive_cluster_relaxed(at_leader(full_a(sa)));
                    else
                        mbar_arrive(full_a(sa));
                }
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
        for (int unit = unit_first<CW>(); unit < unit_count<CW>(p); unit += unit_stride<CW>(), ++tcount) {
            int tt, wt;
            unit_tile<CW>(unit, p, rank, tt, wt);
            if (!wait_warp_sleep<PAIR>(d_full, tcount & 1u, abort_flag, p.status, p.wait_ns, kEpilogueSleepNs))
                break;
            tc_fence_after();
            const int n = wt * kRows + sub * 32 + lane;
            if constexpr (FUSED)
                fused_epilogue_tile<T>(p, lane_base + L::D_COL, tt * T, n, lane, eg, EP);
            else
                plain_epilogue_tile<T>(p, lane_base + L::D_COL, tt * T, n, lane, n_even, eg, EP);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                // the odd CTA's accumulator reads are complete (wait::ld in
                // the tile's epilogue)
                if (PAIR && !leader)
                    mbar_arrive_cluster_relaxed(at_leader(d_empty));
                else
                    mbar_arrive(d_empty);
            }
        }
    }

    __syncwarp();
    tc_fence_before();
    if constexpr (PAIR) {
        // Both CTAs have left their loops: no thread arrives on the other CTA
        // any more, the MMAs have completed (drained above) and the MMA
        // thread has handed over what it committed.  Before a CTA frees its
        // tensor memory and exits, the commits' arrivals on its own barriers
        // (the last stages, the last tile) must have landed.
        cluster_sync();
        tc_fence_after();
        if (warp == 1) {
            if (lane == 0) {
                const uint32_t it = handoff[0], tiles = handoff[1];
                const uint32_t ls = it < static_cast<uint32_t>(S_SMEM) ? it : S_SMEM;
                for (uint32_t i = it - ls; i < it; ++i)
                    settle<true>(empty_smem(i % S_SMEM), (i / S_SMEM) & 1u);
                const uint32_t la = it < static_cast<uint32_t>(S_TMEM) ? it : S_TMEM;
                if (!kUnified)
                    for (uint32_t i = it - la; i < it; ++i)
                        settle<true>(empty_a(i % S_TMEM), (i / S_TMEM) & 1u);
                if (tiles > 0) settle<true>(d_full, (tiles - 1) & 1u);
            }
            __syncwarp();
            tmem_dealloc_pair(tmem, L::TMEM_COLS);
        }
    } else {
        __syncthreads();
        tc_fence_after();
        if (warp == 1) tmem_dealloc(tmem, L::TMEM_COLS);
    }
}

template <int T, int S_SMEM, int S_TMEM, int DQ, int EP, int MIN_BLOCKS, bool PAIR, int NB = 1>
cudaError_t launch_variant(const CUtensorMap* tx, const CUtensorMap* tw, const TsParams& p,
                           int grid, cudaStream_t stream) {
    using L = Layout<T, S_SMEM, S_TMEM, PAIR, NB>;
    // the plain variant carries none of the fused epilogue's code or registers
    const bool fused =
        p.epi.bias != nullptr || p.epi.residual != nullptr || p.epi.act != kActNone;
    auto kern = fused ? w4a16_ts_kernel<T, S_SMEM, S_TMEM, DQ, EP, MIN_BLOCKS, true, PAIR, NB>
                      : w4a16_ts_kernel<T, S_SMEM, S_TMEM, DQ, EP, MIN_BLOCKS, false, PAIR, NB>;
    // Idempotent; cheap enough to repeat per launch and per device.
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    if constexpr (!PAIR) {
        kern<<<grid, threads_for<DQ, EP>(), L::SMEM_BYTES, stream>>>(*tx, *tw, p);
    } else {
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = 2;
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
// CTA pairs: 256 tokens per tile, each CTA a ring of 8 stages of (16 KB x +
// 4 KB packed weights) and 8 tensor-memory A stages: 256 accumulator + 8 x 32
// A columns fill the 512 columns.
#ifndef W4A16_PAIR_STAGES
#define W4A16_PAIR_STAGES 8
#endif
constexpr int kPairSS = W4A16_PAIR_STAGES, kPairST = W4A16_PAIR_STAGES;
// Wide CTA pairs: 384 tokens per tile as two accumulators of 192 columns, so
// one dequantised A stage serves 384 tokens; tensor memory = 384 accumulator
// + 4 x 32 A columns.  Shared memory per stage: 24 KB x + 4 KB weights.
#ifndef W4A16_WIDE_SS
#define W4A16_WIDE_SS 4
#endif
constexpr int kWideT = 384, kWideSS = W4A16_WIDE_SS, kWideST = 4;
// Small M: 32 tokens per tile, 8 shared-memory stages of 8 KB, 3 A stages;
// 128 tensor-memory columns so that three CTAs share an SM.
constexpr int kGemvT = 32, kGemvSS = 8, kGemvST = 3, kGemvDQ = 1, kGemvEP = 1;

// CTA pairs that can be resident at once (SMs left over in a GPC cannot
// take one); cached per device.
int pair_slots(int sm_count) {
    constexpr int kMaxDev = 64;
    static int cache[kMaxDev] = {};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDev) return sm_count / 2;
    if (cache[dev] > 0) return cache[dev];
    using L = Layout<kGemmT, kPairSS, kPairST, true>;
    auto kern = w4a16_ts_kernel<kGemmT, kPairSS, kPairST, kGemmDQ, kGemmEP, 1, false, true, 1>;
    int n = 0;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM_BYTES) ==
        cudaSuccess) {
        cudaLaunchConfig_t cfg = {};
        cudaLaunchAttribute attr[1];
        attr[0].id = cudaLaunchAttributeClusterDimension;
        attr[0].val.clusterDim.x = 2;
        attr[0].val.clusterDim.y = 1;
        attr[0].val.clusterDim.z = 1;
        cfg.gridDim = dim3(static_cast<unsigned>(sm_count / 2 * 2));
        cfg.blockDim = dim3(threads_for<kGemmDQ, kGemmEP>());
        cfg.dynamicSmemBytes = L::SMEM_BYTES;
        cfg.attrs = attr;
        cfg.numAttrs = 1;
        if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) n = 0;
    }
    cudaGetLastError();  // a failed query leaves no sticky error for the next launch
    if (n <= 0) n = sm_count / 2;
    cache[dev] = n;
    return n;
}

}  // namespace

int ts_tokens_per_tile(TsVariant v) {
    return v == TsVariant::kGemv32 ? kGemvT : v == TsVariant::kGemmPairWide ? kWideT : kGemmT;
}

int ts_x_box_tokens(TsVariant v) {
    if (v == TsVariant::kGemmPair) return kGemmT / 2;
    if (v == TsVariant::kGemmPairWide) return kWideT / 4;  // two blocks, half per CTA
    return ts_tokens_per_tile(v);
}

bool ts_prefer_wide(int64_t M, int64_t N, int sm_count) {
    // Each CTA pair walks ceil(units / pairs) units of (token tile, 256 weight
    // rows); a unit of the 384-token tiles costs ~1.37 of a 256-token one
    // (measured: 1.35-1.37 on the 4096- and 8192-token projections, 1.39 for
    // one tile of each).  The tiles that give the fewer unit-costs per pair win.
    const int64_t pairs = pair_slots(sm_count);
    const int64_t per_tile = (N + 255) / 256;
    const int64_t w256 = ((M + kGemmT - 1) / kGemmT * per_tile + pairs - 1) / pairs;
    const int64_t w384 = ((M + kWideT - 1) / kWideT * per_tile + pairs - 1) / pairs;
    return w384 * 137 < w256 * 100;
}

int ts_grid(TsVariant v, const TsParams& p, int sm_count) {
    if (v == TsVariant::kGemm256) return p.num_tiles < sm_count ? p.num_tiles : sm_count;
    if (v == TsVariant::kGemmPair || v == TsVariant::kGemmPairWide) {
        const int units = p.num_t_tiles * ((p.num_w_tiles + 1) / 2);
        const int slots = pair_slots(sm_count);
        return 2 * (units < slots ? units : slots);
    }
    return p.num_tiles;
}

cudaError_t ts_launch(TsVariant v, const CUtensorMap* tx, const CUtensorMap* tw,
                      const TsParams& p, int grid, cudaStream_t stream) {
    if (v == TsVariant::kGemm256)
        return launch_variant<kGemmT, kGemmSS, kGemmST, kGemmDQ, kGemmEP, 1, false>(tx, tw, p,
                                                                                   grid, stream);
    if (v == TsVariant::kGemmPair)
        return launch_variant<kGemmT, kPairSS, kPairST, kGemmDQ, kGemmEP, 1, true>(tx, tw, p,
                                                                                  grid, stream);
    if (v == TsVariant::kGemmPairWide)
        return launch_variant<kWideT, kWideSS, kWideST, kGemmDQ, kGemmEP, 1, true, 2>(
            tx, tw, p, grid, stream);
    return launch_variant<kGemvT, kGemvSS, kGemvST, kGemvDQ, kGemvEP, 3, false>(tx, tw, p, grid,
                                                                               stream);
}

}  // namespace w4a16
