// Small-M (M <= 128, g = 128) int4-dequant + matmul on the 5th-generation
// tensor core: the regime where the whole packed weight matrix streams from
// HBM once per call (the GEMM's 256-token tiles would leave most of their
// columns empty and split the weight rows unevenly over the SMs).
//
// out[m, n] = sum_k x[m, k] * wd[n, k],   wd = RNE_bf16((q[n, k] - 8) * s[n, k / g])
//
// (the same weights as w4a16_dequant and the large-M GEMM: the result differs
// from theirs only in the fp32 summation order).
//
// Why the tensor core here: at M = 16-32 tokens the matmul is 19-39 GFLOP per
// call, and warp-level mma.sync runs at ~610 TFLOP/s on this GPU -- 32-64 us,
// more than the ~46 us the weights take to stream.  tcgen05.mma runs
// asynchronously, leaving the SM's integer and half-precision pipes to the
// dequantisation.
//
// Per CTA (persistent, one per SM): a contiguous range of RB <= 384 weight
// rows (RB = N / #SMs rounded up to even), as three MMA tiles of 128 rows,
// each with ONE fp32 accumulator of NTOK = 16, 32, 64 or 128 token columns in
// tensor memory for the whole K walk.
// Per scale group of 128 k:
//   warp 0      TMA: two 64-k boxes of x (NTOK token rows, 128-byte swizzle,
//               rows >= M zero-filled) and two boxes of RB/2 rows x 64 B of
//               packed weights (64-byte swizzle) into a ring of S stages;
//   warp 2      reorders each staged x chunk in place into the (k, k+4) pair
//               order in which the codes come out of a packed word;
//   warps 4-15  dequant: thread = one weight row of one tile (its TMEM lane);
//               per scale group, 16 words -> bf16 pairs (q - 8) * s (shift,
//               three-input LOP3, one bf16x2 subtraction and one bf16x2
//               multiply per pair) -> tcgen05.st into a ring of SA A stages
//               (one per group);
//               after the last group, the epilogue: tcgen05.ld of the row's
//               NTOK accumulators in slices of up to 32, each slice's (fused)
//               epilogue from registers;
//   warps 1, 3, 16  one thread each, one per tile, issues
//               D_t[128 x NTOK] += A_t[128 x 16] x B[NTOK x 16]^T (A from
//               tensor memory, B = x in shared memory), 8 MMAs per group,
//               accumulating into its tile's accumulator.
// With the scale applied in the dequant there is no per-group accumulator to
// fold: nothing waits on the MMAs inside the K walk except the A ring.  A
// single thread issues these small MMAs at ~130 SM clocks each, slower than
// the tensor pipe runs them, hence one issuing thread (and one A ring and
// accumulator hand-off) per tile.
//
// Every wait is bounded (ptx.cuh); on a timeout the kernel records
// W4A16_ERR_TIMEOUT, drains its copies and MMAs, frees tensor memory and
// returns.
#include "dequant.cuh"
#include "epilogue.cuh"
#include "internal.h"
#include "ptx.cuh"

namespace w4a16 {

namespace {

constexpr int kTilesMax = 3;              // MMA tiles of 128 rows per CTA, at most
constexpr int kGroupK = 128;              // k per TMA stage = one scale group
constexpr int kFirstRowWarp = 4;          // warps 4..15 (warp % 4 = TMEM sub-partition)
constexpr int kRowWarps = 4 * kTilesMax;  // dequant + epilogue warps
constexpr int kLastIssuerWarp = kFirstRowWarp + kRowWarps;  // warp 16: tile 2's MMAs
constexpr int kThreads = 32 * (kLastIssuerWarp + 1);

// MMA-issuing warp of tile t: 1, 3, 16.
__device__ __forceinline__ int issuer_tile(int warp) {
    return warp == 1 ? 0 : warp == 3 ? 1 : warp == kLastIssuerWarp ? 2 : -1;
}

// 32 lanes x 16 columns of 32 bits (see tmem_st_32x32b_x32).
__device__ __forceinline__ void tmem_st_32x32b_x16(uint32_t taddr, const uint32_t* v) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
        "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
        "r"(v[15])
        : "memory");
}

template <int NTOK>
struct TLayout {
    static_assert(NTOK == 16 || NTOK == 32 || NTOK == 64 || NTOK == 128, "MMA N for M = 128");
    // MMA tiles of 128 rows per CTA (with 128 tokens, two tiles and 256 rows
    // per CTA would leave room for more A stages but need a second wave of
    // chunks at N = 49152: 207 against 141 us)
    static constexpr int TILES = kTilesMax;
    static constexpr int ROWS_MAX = 128 * TILES;                     // rows per CTA chunk
    static constexpr int S = NTOK == 128 ? 3 : NTOK == 64 ? 5 : NTOK == 32 ? 6 : 7;  // TMA slots
    // k per tensor-memory A stage: a whole scale group; half of one where the
    // 64-token accumulators leave room for three half-group slots only; a
    // quarter where the 128-token accumulators leave room for two
    static constexpr int AK = NTOK == 128 ? 32 : NTOK == 64 ? 64 : 128;
    static constexpr int CHUNKS = AK / 32;  // 16-byte chunks (32 codes) per row and A stage
    // A stage slots: as many as fit next to the accumulators
    static constexpr int SA = NTOK == 64 ? 3 : 2;
    static constexpr int X_BOX = NTOK * 128;                         // 64 k x NTOK tokens
    static constexpr int X_BYTES = 2 * X_BOX;
    static constexpr int W_HALF = (ROWS_MAX / 2) * (kGroupK / 2);    // ROWS_MAX / 2 rows x 64 B
    static constexpr int W_BYTES = 2 * W_HALF;
    static constexpr int STAGE = X_BYTES + W_BYTES;                  // x, then the weights
    // full_tma[S], empty_smem[S], x_ready[S], then per tile: full_a[SA],
    // empty_a[SA], d_full, d_empty, drain
    static constexpr int BAR_OFF = S * STAGE;
    static constexpr int TILE_BARS = 2 * SA + 3;
    static constexpr int NBARS = 3 * S + TILES * TILE_BARS;
    static constexpr int MISC_OFF = BAR_OFF + NBARS * 8;
    static constexpr int SMEM_BYTES = MISC_OFF + 16 + 1024;          // + 1024-B alignment slack
    // tensor memory: the accumulators (TILES x NTOK columns) at column 0,
    // then from column A_COL SA A stages (TILES x AK / 2 columns each: AK k
    // of bf16 pairs).  A stages of a whole group (two slots) measured ~3%
    // faster than half-group stages (four slots): half the hand-offs.
    static constexpr int D_COLS = TILES * NTOK;
    static constexpr int A_COL = NTOK == 128 ? 384 : NTOK == 64 ? 192 : 128;
    static constexpr int A_COLS = TILES * (AK / 2);
    static constexpr int TMEM_COLS = 512;
    static_assert(D_COLS <= A_COL && A_COL + SA * A_COLS <= TMEM_COLS,
                  "tensor memory holds 512 columns");
    static_assert(X_BOX % 1024 == 0 && W_HALF % 1024 == 0 && STAGE % 1024 == 0,
                  "swizzled boxes keep 1024-byte alignment");
    static_assert(SMEM_BYTES <= 227 * 1024, "shared memory");
};

template <int NTOK, bool FUSED>
__global__ void __launch_bounds__(kThreads, 1)
    w4a16_gemv_tc_kernel(const __grid_constant__ CUtensorMap tmap_x,
                         const __grid_constant__ CUtensorMap tmap_w, const GemvParams p) {
    using L = TLayout<NTOK>;
    constexpr int S = L::S, SA = L::SA;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;
    uint8_t* smem = smem_raw + (sbase - raw);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int RB = p.rows_per_cta;

    const uint32_t bars = sbase + L::BAR_OFF;
    auto full_tma = [&](int s) { return bars + 8u * s; };
    auto empty_smem = [&](int s) { return bars + 8u * (S + s); };
    auto x_ready = [&](int s) { return bars + 8u * (2 * S + s); };
    auto tile_bar = [&](int t, int i) { return bars + 8u * (3 * S + t * L::TILE_BARS + i); };
    auto full_a = [&](int t, int a) { return tile_bar(t, a); };
    auto empty_a = [&](int t, int a) { return tile_bar(t, SA + a); };
    auto d_full = [&](int t) { return tile_bar(t, 2 * SA); };
    auto d_empty = [&](int t) { return tile_bar(t, 2 * SA + 1); };
    auto drain = [&](int t) { return tile_bar(t, 2 * SA + 2); };
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::MISC_OFF);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::MISC_OFF + 4);

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(full_tma(s), 1);
            // every row warp of the p.nt tiles in use has read W, and every
            // such tile's MMAs have read x
            mbar_init(empty_smem(s), 5 * p.nt);
            mbar_init(x_ready(s), 1);
        }
        for (int t = 0; t < L::TILES; ++t) {
            for (int a = 0; a < SA; ++a) {
                mbar_init(full_a(t, a), 4);  // the tile's four row warps
                mbar_init(empty_a(t, a), 1);
            }
            mbar_init(d_full(t), 1);
            mbar_init(d_empty(t), 4);
            mbar_init(drain(t), 1);
        }
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
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;

    const int KS = p.K / kGroupK;  // scale groups = stages per chunk
    // Each CTA walks K from its own starting group, so that the CTAs read
    // different x slices from L2 at any moment.
    const int rot = static_cast<int>(static_cast<int64_t>(blockIdx.x) * KS / gridDim.x);

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint32_t tx = L::X_BYTES + static_cast<uint32_t>(RB) * (kGroupK / 2);
            uint32_t it = 0;
            bool ok = true;
            for (int chunk = blockIdx.x; ok && chunk < p.num_chunks; chunk += gridDim.x) {
                const int row0 = chunk * RB;
                int kk = rot;
                for (int g = 0; g < KS; ++g, ++it) {
                    const int s = it % S;
                    if (!wait_one(empty_smem(s), ((it / S) & 1u) ^ 1u, abort_flag, p.status,
                                  p.wait_ns)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(full_tma(s), tx);
                    const uint32_t st = sbase + s * L::STAGE;
                    const uint32_t end = sbase + L::BAR_OFF;
                    if (dbg_check(tma_box_ok(st, L::X_BOX, 1024, sbase, end, kk * kGroupK, 2) &&
                                      tma_box_ok(st + L::X_BOX, L::X_BOX, 1024, sbase, end,
                                                 kk * kGroupK + 64, 2),
                                  p.status)) {
                        tma_load_2d(st, &tmap_x, full_tma(s), kk * kGroupK, 0);
                        tma_load_2d(st + L::X_BOX, &tmap_x, full_tma(s), kk * kGroupK + 64, 0);
                    }
                    const uint32_t wbox = static_cast<uint32_t>(RB / 2) * (kGroupK / 2);
                    if (dbg_check(wbox <= L::W_HALF &&
                                      tma_box_ok(st + L::X_BYTES, wbox, 1024, sbase, end,
                                                 kk * (kGroupK / 2), 1) &&
                                      tma_box_ok(st + L::X_BYTES + L::W_HALF, wbox, 1024, sbase,
                                                 end, kk * (kGroupK / 2), 1),
                                  p.status)) {
                        tma_load_2d(st + L::X_BYTES, &tmap_w, full_tma(s), kk * (kGroupK / 2),
                                    row0);
                        tma_load_2d(st + L::X_BYTES + L::W_HALF, &tmap_w, full_tma(s),
                                    kk * (kGroupK / 2), row0 + RB / 2);
                    }
                    if (++kk == KS) kk = 0;
                }
            }
            // every load this thread issued has landed before exit
            const uint32_t last = it < static_cast<uint32_t>(S) ? it : S;
            for (uint32_t i = it - last; i < it; ++i) settle(full_tma(i % S), (i / S) & 1u);
        }
    } else if (issuer_tile(warp) >= 0) {
        // ------------------------------------------------------------ MMA issuers
        // (tiles past the chunk's rows, t >= p.nt, are not computed)
        const int t = issuer_tile(warp);
        if (lane == 0 && t < p.nt && t < L::TILES) {
            constexpr uint32_t idesc = idesc_bf16_f32(128, NTOK);
            uint32_t it = 0, ia = 0, nchunk = 0;
            bool ok = true, issued = false;
            for (int chunk = blockIdx.x; ok && chunk < p.num_chunks;
                 chunk += gridDim.x, ++nchunk) {
                // the epilogue has read the previous chunk's accumulators
                if (nchunk > 0 &&
                    !wait_one(d_empty(t), (nchunk - 1u) & 1u, abort_flag, p.status, p.wait_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                for (int g = 0; ok && g < KS; ++g, ++it) {
                    const int s = it % S;
                    if (!wait_one(x_ready(s), (it / S) & 1u, abort_flag, p.status, p.wait_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t bdesc = sdesc_kmajor_sw128(sbase + s * L::STAGE);
                    for (int h = 0; h < kGroupK / L::AK; ++h, ++ia) {
                        const int a = ia % SA;
                        if (!wait_one(full_a(t, a), (ia / SA) & 1u, abort_flag, p.status,
                                      p.wait_ns)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
#pragma unroll
                        for (int ks = 0; ks < L::AK / 16; ++ks) {
                            // k offset in the group -> x box (64 k) and 32-byte step
                            // in it; the descriptor's start address is in 16-byte units
                            const int kg = h * L::AK + ks * 16;
                            tc_mma_ts(tmem + t * NTOK,
                                      tmem + L::A_COL + a * L::A_COLS + t * (L::AK / 2) + ks * 8,
                                      bdesc + static_cast<uint64_t>(
                                                  ((kg >> 6) * L::X_BOX + (kg & 63) * 2) >> 4),
                                      idesc, (g | h | ks) != 0);
                        }
                        issued = true;
                        tc_commit(empty_a(t, a));
                    }
                    if (!ok) break;
                    tc_commit(empty_smem(s));
                }
                if (!ok) break;
                tc_commit(d_full(t));  // the chunk's accumulators of tile t are final
            }
            if (issued) {
                // every MMA issued has completed before tensor memory is freed
                tc_commit(drain(t));
                settle(drain(t), 0);
            }
        }
    } else if (warp == 2) {
        // ------------------------------------------------------------ x reorder
        // Every 16-byte chunk (x0..x7) of the stage's x boxes becomes
        // (x0,x4),(x1,x5),(x2,x6),(x3,x7): the pair order of codes_signed.
        constexpr int kChunks = L::X_BYTES / 16;
        static_assert(kChunks % 32 == 0, "whole chunks per lane");
        uint32_t it = 0;
        bool ok = true;
        for (int chunk = blockIdx.x; ok && chunk < p.num_chunks; chunk += gridDim.x) {
            for (int g = 0; g < KS; ++g, ++it) {
                const int s = it % S;
                if (!wait_warp(full_tma(s), (it / S) & 1u, abort_flag, p.status, p.wait_ns)) {
                    ok = false;
                    break;
                }
                uint4* xs = reinterpret_cast<uint4*>(smem + s * L::STAGE);
#pragma unroll
                for (int i = 0; i < kChunks / 32; ++i)
                    xs[lane + 32 * i] = interleave_chunk(xs[lane + 32 * i]);
                // these generic writes precede the MMAs' async-proxy reads
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(x_ready(s));
            }
        }
    } else if (warp >= kFirstRowWarp && warp < kLastIssuerWarp &&
               (warp - kFirstRowWarp) / 4 < p.nt && (warp - kFirstRowWarp) / 4 < L::TILES) {
        // ------------------------------------------------------------ dequant + epilogue
        const int t = (warp - kFirstRowWarp) >> 2;  // MMA tile
        const int sub = warp & 3;                   // TMEM sub-partition
        const int r = t * 128 + sub * 32 + lane;    // local row
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(sub * 32) << 16);
        // the row's four 16-byte chunks in a stage (64-byte swizzle)
        const bool in_range = r < RB;
        const int bx = r >= RB / 2 ? 1 : 0;
        const int rr = in_range ? r - bx * (RB / 2) : 0;
        const uint32_t row_off = L::X_BYTES + bx * L::W_HALF + rr * (kGroupK / 2);
        const uint32_t swz = static_cast<uint32_t>((rr >> 1) & 3);
        uint32_t it = 0, ia = 0, nchunk = 0;
        bool ok = true;
        for (int chunk = blockIdx.x; ok && chunk < p.num_chunks; chunk += gridDim.x, ++nchunk) {
            const int n = chunk * RB + r;
            const bool valid = in_range && n < p.N;
            // the row's scales in the rotated group order, one group ahead
            const uint16_t* srow = p.scales + static_cast<int64_t>(valid ? n : 0) * KS;
            int kk = rot;
            uint16_t s_next = __ldg(srow + kk);
            for (int g = 0; ok && g < KS; ++g, ++it) {
                const int s = it % S;
                const uint32_t s2 = valid ? splat_bf16(s_next) : 0u;
                if (++kk == KS) kk = 0;
                if (g + 1 < KS) s_next = __ldg(srow + kk);
                if (!wait_warp(full_tma(s), (it / S) & 1u, abort_flag, p.status, p.wait_ns)) {
                    ok = false;
                    break;
                }
                const uint32_t wrow = sbase + s * L::STAGE + row_off;
                for (int h = 0; h < kGroupK / L::AK; ++h, ++ia) {
                    const int a = ia % SA;
                    // code 8 everywhere: rows past the range are zero
                    uint4 c[L::CHUNKS];
#pragma unroll
                    for (int i = 0; i < L::CHUNKS; ++i) {
                        c[i] = make_uint4(0x88888888u, 0x88888888u, 0x88888888u, 0x88888888u);
                        if (valid)
                            c[i] = lds128(wrow + 16u * (static_cast<uint32_t>(L::CHUNKS * h + i) ^ swz));
                    }
                    if (!wait_warp(empty_a(t, a), ((ia / SA) & 1u) ^ 1u, abort_flag, p.status,
                                   p.wait_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    // per 32 codes: exact q - 8 pairs, then wd = RNE_bf16((q - 8) * s)
                    // (one rounding), stored as 32 x 16 bf16 pairs of the row's lane
                    const bool st_ok =
                        dbg_check(L::A_COL + a * L::A_COLS + (t + 1) * (L::AK / 2) <= L::TMEM_COLS,
                                  p.status);
                    if constexpr (L::CHUNKS == 1) {
                        uint32_t v[16];
                        codes_signed(c[0].x, v + 0);
                        codes_signed(c[0].y, v + 4);
                        codes_signed(c[0].z, v + 8);
                        codes_signed(c[0].w, v + 12);
#pragma unroll
                        for (int j = 0; j < 16; ++j) v[j] = bf16x2_mul(v[j], s2);
                        if (st_ok)
                            tmem_st_32x32b_x16(lane_base + L::A_COL + a * L::A_COLS + t * (L::AK / 2),
                                               v);
                    } else {
#pragma unroll
                        for (int i = 0; i < L::CHUNKS; i += 2) {
                            uint32_t v[32];
                            codes_signed(c[i].x, v + 0);
                            codes_signed(c[i].y, v + 4);
                            codes_signed(c[i].z, v + 8);
                            codes_signed(c[i].w, v + 12);
                            codes_signed(c[i + 1].x, v + 16);
                            codes_signed(c[i + 1].y, v + 20);
                            codes_signed(c[i + 1].z, v + 24);
                            codes_signed(c[i + 1].w, v + 28);
#pragma unroll
                            for (int j = 0; j < 32; ++j) v[j] = bf16x2_mul(v[j], s2);
                            if (st_ok)
                                tmem_st_32x32b_x32(lane_base + L::A_COL + a * L::A_COLS +
                                                       t * (L::AK / 2) + i * 16,
                                                   v);
                        }
                    }
                    tmem_st_wait();
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(full_a(t, a));
                }
                if (!ok) break;
                __syncwarp();
                if (lane == 0) mbar_arrive(empty_smem(s));  // this warp's weight reads are done
            }
            if (!ok) break;
            // ---- epilogue: the row's NTOK accumulators, tokens 0 .. M - 1
            if (!wait_warp(d_full(t), nchunk & 1u, abort_flag, p.status, p.wait_ns)) {
                ok = false;
                break;
            }
            tc_fence_after();
            // the row's accumulators in slices of EC tokens (registers), then
            // the (fused) epilogue of each slice
            constexpr int EC = NTOK < 32 ? NTOK : 32;
            const Epilogue& ep = p.epi;
            // SwiGLU pairs rows (n, n ^ 1) = (gate, up): RB is even, so n has
            // the parity of its lane and the partner is lane ^ 1
            const float bias =
                (FUSED && ep.bias != nullptr && valid) ? bf16_to_f32(ep.bias[n]) : 0.0f;
#pragma unroll 1
            for (int m0 = 0; m0 < NTOK; m0 += EC) {
                float acc[EC];
#pragma unroll
                for (int half = 0; half < EC / 16; ++half) {
                    uint32_t d[16];
                    tmem_ld_32x32b_x16(lane_base + t * NTOK + m0 + half * 16, d);
                    tmem_ld_wait_x16(d);
#pragma unroll
                    for (int j = 0; j < 16; ++j) acc[half * 16 + j] = __uint_as_float(d[j]);
                }
                if constexpr (!FUSED) {
#pragma unroll
                    for (int j = 0; j < EC; ++j) {
                        const int m = m0 + j;
                        if (valid && m < p.M)
                            p.out[static_cast<int64_t>(m) * p.N + n] = f32_to_bf16_rn(acc[j]);
                    }
                } else {
#pragma unroll
                    for (int j = 0; j < EC; ++j) {
                        const int m = m0 + j;
                        const float z = acc[j] + bias;
                        if (ep.act == kActSwiGLU) {
                            const float up = __shfl_xor_sync(0xffffffffu, z, 1);
                            if ((lane & 1) == 0 && valid && m < p.M) {
                                const int64_t o = static_cast<int64_t>(m) * ep.n_out + (n >> 1);
                                float h = silu_f32(z) * up;
                                if (ep.residual != nullptr) h += bf16_to_f32(ep.residual[o]);
                                p.out[o] = f32_to_bf16_rn(h);
                            }
                        } else if (valid && m < p.M) {
                            const int64_t o = static_cast<int64_t>(m) * ep.n_out + n;
                            float h = ep.act == kActGELU ? gelu_f32(z) : z;
                            if (ep.residual != nullptr) h += bf16_to_f32(ep.residual[o]);
                            p.out[o] = f32_to_bf16_rn(h);
                        }
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(d_empty(t));  // the next chunk's MMAs may overwrite D
        }
    }

    __syncwarp();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, L::TMEM_COLS);
}

template <int NTOK>
cudaError_t launch_tc_variant(const CUtensorMap* tx, const CUtensorMap* tw, const GemvParams& p,
                              int grid, cudaStream_t stream) {
    using L = TLayout<NTOK>;
    const bool fused =
        p.epi.bias != nullptr || p.epi.residual != nullptr || p.epi.act != kActNone;
    auto kern = fused ? w4a16_gemv_tc_kernel<NTOK, true> : w4a16_gemv_tc_kernel<NTOK, false>;
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, L::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    kern<<<grid, kThreads, L::SMEM_BYTES, stream>>>(*tx, *tw, p);
    return cudaGetLastError();
}

}  // namespace

int gemv_tc_rows_per_cta(int64_t N, int sm_count) {
    int64_t per = (N + sm_count - 1) / sm_count;
    per = (per + 1) / 2 * 2;
    if (per > 128 * kTilesMax) per = 128 * kTilesMax;
    if (per < 2) per = 2;
    return static_cast<int>(per);
}

int gemv_tc_tokens(int64_t M) { return M <= 16 ? 16 : M <= 32 ? 32 : M <= 64 ? 64 : 128; }

cudaError_t gemv_tc_launch(const CUtensorMap* tx, const CUtensorMap* tw, const GemvParams& p,
                           int sm_count, cudaStream_t stream) {
    const int grid = p.num_chunks < sm_count ? p.num_chunks : sm_count;
    if (p.M <= 16) return launch_tc_variant<16>(tx, tw, p, grid, stream);
    if (p.M <= 32) return launch_tc_variant<32>(tx, tw, p, grid, stream);
    if (p.M <= 64) return launch_tc_variant<64>(tx, tw, p, grid, stream);
    return launch_tc_variant<128>(tx, tw, p, grid, stream);
}

}  // namespace w4a16
