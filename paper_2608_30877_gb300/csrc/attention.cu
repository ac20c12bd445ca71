// Attention prefill over packed sequences for sm_103a: the decoder's
// attention between the QKV and output projections, causal within each
// protein-ligand pair's sequence and limited to a sliding window (the
// model's 32K window, Sec. 2.1).
//
//   o[i, h, :] = sum_j softmax_j(q_i . k_j / sqrt(d)) v_j,
//   j in the sequence of i, i - W < j <= i;  d = 128.
//
// A job is one (128-query block, head), flash-attention style on the
// 5th-generation tensor core, over blocks of 64 keys:
//   S  = Q K^T   tcgen05.mma kind::f16, A = Q and B = K from shared memory
//                (TMA, 128-byte swizzle, K-major), S fp32 in tensor memory,
//                two S buffers that blocks alternate between;
//   softmax      four warps, thread = query row: tcgen05.ld of its S row into
//                registers, causal/window mask per 32-key chunk, running max
//                and sum in fp32 (exp2 with the scale folded in), P as bf16
//                pairs written over S with tcgen05.st; O rescaled in tensor
//                memory when the running max grows (lazily, by more than 2^8);
//   O += P V     tcgen05.mma with A = P from tensor memory and B = V from
//                shared memory as an MN-major operand (V is stored token-
//                major, d contiguous -- exactly the layout the TMA box has);
//   epilogue     O / l, bf16, staged through shared memory for coalesced
//                stores.
// S runs two blocks ahead of PV, so the S product of the next block is
// ready when the softmax of the current one ends.  The kernel is persistent
// with two CTAs per SM (256 tensor-memory columns and 104 KB of shared memory
// each), every CTA taking every grid-th job, heads fastest; one CTA's softmax
// and epilogue overlap the other's MMAs.  Within a CTA the roles are one TMA
// warp, one MMA warp and the four softmax warps, linked by mbarriers whose
// phases run on across jobs: Q and K of the next job load during the current
// job's last blocks, and its first S products run during the epilogue.
// Every wait is bounded (ptx.cuh); on a timeout the kernel records
// W4A16_ERR_TIMEOUT, waits for its own copies and MMAs and frees tensor memory.
#include "internal.h"
#include "ptx.cuh"

#include <cuda_bf16.h>

namespace w4a16 {

namespace {

constexpr int kD = 128;        // head dimension
constexpr int kBQ = 128;       // queries per job (MMA M)
constexpr int kBKV = 64;       // keys per block (MMA N of S, K of PV)
constexpr int kPvWarp = 2;
constexpr int kFirstSoftmaxWarp = 3;  // warps 3..10: two per TMEM sub-partition (warp % 4)
constexpr int kSoftmaxWarps = 8;
constexpr int kThreads = (kFirstSoftmaxWarp + kSoftmaxWarps) * 32;  // + TMA, S-MMA, PV-MMA warps

struct AttnLayout {
    static constexpr int QBOX = kBQ * 128;    // one [128 rows x 64 cols] bf16 box: 16 KB
    static constexpr int KBOX = kBKV * 128;   // one [64 rows x 64 cols] bf16 box: 8 KB
    static constexpr int Q_TILE = 2 * QBOX;   // [128 x 128]: 32 KB
    static constexpr int KV_TILE = 2 * KBOX;  // [64 x 128]: 16 KB
    static constexpr int Q_OFF = 0;
    static constexpr int K_OFF = Q_OFF + Q_TILE;       // two stages
    static constexpr int V_OFF = K_OFF + 2 * KV_TILE;  // two stages
    // epilogue staging: per softmax warp 16 rows x 32 columns of bf16 output
    static constexpr int STAGE_OFF = V_OFF + 2 * KV_TILE;
    static constexpr int STAGE_WARP = 16 * 64;
    static constexpr int BAR_OFF = STAGE_OFF + kSoftmaxWarps * STAGE_WARP;
    // q_full, q_empty, k_full[2], k_empty[2], v_full[2], v_empty[2],
    // s_full[2], p_full[2], o_ready[2], drain[2]
    static constexpr int NBARS = 18;
    static constexpr int MISC_OFF = BAR_OFF + NBARS * 8;
    static constexpr int SMEM_BYTES = MISC_OFF + 32 + 1024;
    // tensor memory columns: two S buffers (blocks alternate; P of a block is
    // written over the first half of its S) and O
    static constexpr int S_COL = 0, O_COL = 2 * kBKV, TMEM_COLS = 256;
    static_assert(O_COL + kD <= TMEM_COLS, "tensor memory");
    // two CTAs per SM: 228 KB per SM, 1 KB of it reserved per CTA
    static_assert(2 * (SMEM_BYTES + 1024) <= 228 * 1024, "shared memory");
};

// SS MMA: D[tmem] (+)= A[smem] * B[smem]^T, kind::f16.
__device__ __forceinline__ void tc_mma_ss(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc,
                                          uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
        : "memory");
}

// Shared-memory descriptor of an MN-major operand with the 128-byte swizzle:
// 128-byte rows of 64 MN-contiguous elements, one row per K index, 8-row
// (1024-byte) swizzle atoms; the next 8 K rows are `sbo` bytes on, the next
// 64 MN elements `lbo` bytes on.
__device__ __forceinline__ uint64_t sdesc_mnmajor_sw128(uint32_t saddr, uint32_t lbo,
                                                        uint32_t sbo) {
    uint64_t d = 0;
    d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);
    d |= static_cast<uint64_t>((lbo & 0x3FFFFu) >> 4) << 16;
    d |= static_cast<uint64_t>((sbo & 0x3FFFFu) >> 4) << 32;
    d |= static_cast<uint64_t>(1) << 46;
    d |= static_cast<uint64_t>(2) << 61;
    return d;
}

// 32 lanes x 16 columns of 32 bits (see tmem_st_32x32b_x32).
__device__ __forceinline__ void tmem_st_32x32b_x16(uint32_t taddr, const uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
        "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
        "r"(v[15])
        : "memory");
}

// 16-lane tensor-memory shapes (the warp covers 16 lanes from the address's
// lane; thread t = 4 g + c).  16x256b.xN: register 4j + {0, 1} holds lane g,
// columns 8j + 2c + {0, 1}; 4j + {2, 3} the same columns of lane g + 8.
// 16x128b.xN: register 2j holds lane g, column 4j + c; 2j + 1 lane g + 8.
__device__ __forceinline__ void tmem_ld_16x256b_x8(uint32_t taddr, uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.16x256b.x8.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, "
        "[%32];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
          "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]),
          "=r"(v[13]), "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]),
          "=r"(v[19]), "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]),
          "=r"(v[25]), "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]),
          "=r"(v[31])
        : "r"(taddr)
        : "memory");
}

__device__ __forceinline__ void tmem_ld_16x256b_x4(uint32_t taddr, uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.16x256b.x4.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
        : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
          "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]),
          "=r"(v[13]), "=r"(v[14]), "=r"(v[15])
        : "r"(taddr)
        : "memory");
}

__device__ __forceinline__ void tmem_st_16x256b_x4(uint32_t taddr, const uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.16x256b.x4.b32 [%0], "
        "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
        "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
        "r"(v[15])
        : "memory");
}

__device__ __forceinline__ void tmem_st_16x128b_x8(uint32_t taddr, const uint32_t (&v)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.16x128b.x8.b32 [%0], "
        "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
        "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
        "r"(v[15])
        : "memory");
}

// the tcgen05.ld above complete (registers tied so that no use moves above)
template <int N>
__device__ __forceinline__ void tmem_ld_wait_n(uint32_t (&v)[N]) {
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < N; ++i) asm volatile("" : "+r"(v[i]));
}

__device__ __forceinline__ float ex2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// max of three (a single instruction on sm_100 and later)
__device__ __forceinline__ float fmax3(float a, float b, float c) {
    float d;
    asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
    return d;
}

// (a.x b + c, a.y b + c) as one paired fp32 FMA, round to nearest
__device__ __forceinline__ float2 ffma2(float2 a, float b, float c) {
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\t"
        "mov.b64 rb, {%4, %4};\n\t"
        "mov.b64 rc, {%5, %5};\n\t"
        "fma.rn.f32x2 rd, ra, rb, rc;\n\t"
        "mov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b), "f"(c));
    return d;
}

// paired fp32 add, round to nearest
__device__ __forceinline__ float2 fadd2(float2 a, float2 b) {
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\t"
        "mov.b64 rb, {%4, %5};\n\t"
        "add.rn.f32x2 rd, ra, rb;\n\t"
        "mov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
    return d;
}

__device__ __forceinline__ uint32_t pack_bf16x2_rn(float lo, float hi) {
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// Initial running max: finite, so 2^(s - m) of a masked (-inf) score is 0, never NaN.
constexpr float kMaskedScore = -1.0e30f;

// One unit of work: query block [q0, q0 + 128) of the sequence [ss, se),
// for head h.
struct AttnJob {
    int ss, se, q0, h;
    bool valid;
};

// Resumable warp-collective search for the x-th query block over the
// sequences (blocks of a sequence numbered from its last, the heaviest under
// the causal mask, down).  x never decreases between calls of one warp, so
// the search resumes at the 32-sequence group where the last one ended.
struct JobCursor {
    int s0 = 0;    // first sequence of the current group
    int base = 0;  // query blocks of the sequences before s0
};

__device__ __forceinline__ bool find_block(const AttnParams& p, int x, int lane, JobCursor& cur,
                                           int& ss, int& se, int& q0) {
    for (; cur.s0 < p.nseq; cur.s0 += 32) {
        const int s = cur.s0 + lane;
        int a = 0, b = 0, nqb = 0;
        if (s < p.nseq) {
            a = p.seq_start[s];
            b = p.seq_start[s + 1];
            nqb = b > a ? (b - a + kBQ - 1) / kBQ : 0;
        }
        int incl = nqb;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int t = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += t;
        }
        const int excl = incl - nqb;
        const bool mine = s < p.nseq && x >= cur.base + excl && x < cur.base + incl;
        const unsigned who = __ballot_sync(0xffffffffu, mine);
        if (who) {
            const int src = __ffs(who) - 1;
            const int e = __shfl_sync(0xffffffffu, excl, src);
            const int n = __shfl_sync(0xffffffffu, nqb, src);
            ss = __shfl_sync(0xffffffffu, a, src);
            se = __shfl_sync(0xffffffffu, b, src);
            q0 = ss + (n - 1 - (x - cur.base - e)) * kBQ;
            return true;
        }
        cur.base += __shfl_sync(0xffffffffu, incl, 31);
    }
    return false;
}

// Job t of the CTA's sequence t = blockIdx.x, blockIdx.x + gridDim.x, ...:
// heads vary fastest, so the CTAs running at one time share the K/V of a
// few sequences in L2.
__device__ __forceinline__ AttnJob job_at(const AttnParams& p, int64_t t, int lane, JobCursor& cur) {
    AttnJob j{};
    const int x = static_cast<int>(t / p.H);
    j.h = static_cast<int>(t % p.H);
    j.valid = find_block(p, x, lane, cur, j.ss, j.se, j.q0);
    return j;
}

// key blocks of the sequence that some query of the block can see
__device__ __forceinline__ void key_range(const AttnJob& jb, int W, int& b_first, int& nblk) {
    const int q_last = (jb.q0 + kBQ - 1 < jb.se - 1 ? jb.q0 + kBQ - 1 : jb.se - 1);
    const int k_first = jb.q0 - W + 1 > jb.ss ? jb.q0 - W + 1 : jb.ss;
    b_first = (k_first - jb.ss) / kBKV;
    nblk = (q_last - jb.ss) / kBKV - b_first + 1;
}

// Walks the CTA's key blocks in order across its jobs; warp-collective (the
// job search uses the whole warp).
struct BlockWalk {
    JobCursor cur;
    int64_t t = 0;
    AttnJob jb{};
    int b_first = 0, nblk = 0, j = 0;
    uint32_t jn = 0;  // jobs of the CTA before this one
    bool valid = false;
};

__device__ __forceinline__ void walk_job(const AttnParams& p, int64_t njobs, int lane, BlockWalk& w) {
    w.valid = false;
    if (w.t < njobs) {
        w.jb = job_at(p, w.t, lane, w.cur);
        if (w.jb.valid) {
            key_range(w.jb, p.window, w.b_first, w.nblk);
            w.j = 0;
            w.valid = true;
        }
    }
}

__device__ __forceinline__ void walk_next(const AttnParams& p, int64_t njobs, int64_t step,
                                          int lane, BlockWalk& w) {
    if (++w.j < w.nblk) return;
    w.t += step;
    ++w.jn;
    walk_job(p, njobs, lane, w);
}

__global__ void __launch_bounds__(kThreads, 2)
    attention_prefill_kernel(const __grid_constant__ CUtensorMap tmap_q,
                             const __grid_constant__ CUtensorMap tmap_kv, const AttnParams p,
                             int64_t njobs) {
    using L = AttnLayout;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t sbase = (raw + 1023u) & ~1023u;
    uint8_t* smem = smem_raw + (sbase - raw);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    const uint32_t bars = sbase + L::BAR_OFF;
    const uint32_t q_full = bars, q_empty = bars + 8u;
    auto k_full = [&](uint32_t s) { return bars + 16u + 8u * s; };
    auto k_empty = [&](uint32_t s) { return bars + 32u + 8u * s; };
    auto v_full = [&](uint32_t s) { return bars + 48u + 8u * s; };
    auto v_empty = [&](uint32_t s) { return bars + 64u + 8u * s; };
    auto s_full = [&](uint32_t b) { return bars + 80u + 8u * b; };
    // The barriers of block g are those of index g & 1 and complete once per
    // two blocks.  A parity wait is unambiguous only while its barrier is at
    // most one completion ahead or behind the awaited one; with S two blocks
    // ahead of PV, the softmax may finish P of block g + 1 before the MMA
    // warp takes P of block g (hence two p_full), and the softmax waits for
    // PV products only now and then (hence two o_ready).
    auto p_full = [&](uint32_t b) { return bars + 96u + 8u * b; };
    auto o_ready = [&](uint32_t b) { return bars + 112u + 8u * b; };
    auto drain = [&](uint32_t i) { return bars + 128u + 8u * i; };
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + L::MISC_OFF);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + L::MISC_OFF + 4);
    int* bad_flag = reinterpret_cast<int*>(smem + L::MISC_OFF + 8);

    if (warp == 0) {
        // the sequence boundaries must be non-decreasing within [0, M]
        int bad = 0;
        for (int s = lane; s < p.nseq; s += 32) {
            const int a = p.seq_start[s], b = p.seq_start[s + 1];
            if (a < 0 || b < a || b > p.M) bad = 1;
        }
        bad = __any_sync(0xffffffffu, bad);
        if (lane == 0) {
            if (bad) record_status(p.status, 1 /* W4A16_ERR_INVALID_ARG */);
            *bad_flag = bad;
            mbar_init(q_full, 1);
            mbar_init(q_empty, 1);
            for (uint32_t i = 0; i < 2; ++i) {
                mbar_init(k_full(i), 1);
                mbar_init(k_empty(i), 1);
                mbar_init(v_full(i), 1);
                mbar_init(v_empty(i), 1);
                mbar_init(s_full(i), 1);
                mbar_init(p_full(i), kSoftmaxWarps);  // one arrival per softmax warp
                mbar_init(o_ready(i), 1);
            }
            mbar_init(drain(0), 1);
            mbar_init(drain(1), 1);
            *abort_flag = 0;
            fence_mbar_init();
            prefetch_tmap(&tmap_q);
            prefetch_tmap(&tmap_kv);
        }
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), L::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const int Hd = p.H * kD;
    const int W = p.window;
    const int64_t t_first = blockIdx.x, t_step = gridDim.x;
    const bool run = *bad_flag == 0;

    // Global block g of the CTA (counted across its jobs) uses K/V stage and
    // S buffer g & 1; each of those barriers completes once per two blocks.
    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        // Q of a job loads once the last S product of the previous job is
        // done; K of block g once the S product of block g - 2 is, V once its
        // PV product is.
        bool ok = run;
        JobCursor cur;
        uint32_t g = 0, jn = 0, nq = 0, nk = 0, nv = 0;
        for (int64_t t = t_first; ok && t < njobs; t += t_step) {
            const AttnJob jb = job_at(p, t, lane, cur);
            if (!jb.valid) break;
            int b_first, nblk;
            key_range(jb, W, b_first, nblk);
            if (lane == 0) {
                if (!wait_one(q_empty, (jn & 1u) ^ 1u, abort_flag, p.status, p.wait_ns)) ok = false;
                if (ok) {
                    mbar_arrive_expect_tx(q_full, L::Q_TILE);
                    if (dbg_check(tma_box_ok(sbase + L::Q_OFF, L::QBOX, 1024, sbase,
                                             sbase + L::K_OFF, jb.h * kD, 2) &&
                                      tma_box_ok(sbase + L::Q_OFF + L::QBOX, L::QBOX, 1024, sbase,
                                                 sbase + L::K_OFF, jb.h * kD + 64, 2) &&
                                      jb.q0 >= 0 && jb.q0 < p.M,
                                  p.status)) {
                        tma_load_2d(sbase + L::Q_OFF, &tmap_q, q_full, jb.h * kD, jb.q0);
                        tma_load_2d(sbase + L::Q_OFF + L::QBOX, &tmap_q, q_full, jb.h * kD + 64,
                                    jb.q0);
                    }
                    ++nq;
                }
                for (int j = 0; ok && j < nblk; ++j, ++g) {
                    const uint32_t s = g & 1u, par = ((g >> 1) & 1u) ^ 1u;
                    const int row = jb.ss + (b_first + j) * kBKV;
                    const uint32_t ks = sbase + L::K_OFF + s * L::KV_TILE;
                    const uint32_t vs = sbase + L::V_OFF + s * L::KV_TILE;
                    if (!wait_one(k_empty(s), par, abort_flag, p.status, p.wait_ns)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(k_full(s), L::KV_TILE);
                    // key rows of the block start inside the job's sequence
                    if (dbg_check(tma_box_ok(ks, L::KV_TILE, 1024, sbase + L::K_OFF,
                                             sbase + L::V_OFF, Hd + jb.h * kD, 2) &&
                                      row >= jb.ss && row < jb.se,
                                  p.status)) {
                        tma_load_2d(ks, &tmap_kv, k_full(s), Hd + jb.h * kD, row);
                        tma_load_2d(ks + L::KBOX, &tmap_kv, k_full(s), Hd + jb.h * kD + 64, row);
                    }
                    ++nk;
                    if (!wait_one(v_empty(s), par, abort_flag, p.status, p.wait_ns)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(v_full(s), L::KV_TILE);
                    if (dbg_check(tma_box_ok(vs, L::KV_TILE, 1024, sbase + L::V_OFF,
                                             sbase + L::STAGE_OFF, 2 * Hd + jb.h * kD, 2),
                                  p.status)) {
                        tma_load_2d(vs, &tmap_kv, v_full(s), 2 * Hd + jb.h * kD, row);
                        tma_load_2d(vs + L::KBOX, &tmap_kv, v_full(s), 2 * Hd + jb.h * kD + 64,
                                    row);
                    }
                    ++nv;
                }
            }
            ok = __shfl_sync(0xffffffffu, ok, 0);
            ++jn;
        }
        if (lane == 0) {
            // every load issued has landed before exit (the Q loads are the
            // jobs' first nq, one per job, so load i is phase i of q_full)
            if (nq > 0) settle(q_full, (nq - 1) & 1u);
            for (uint32_t i = nk > 2 ? nk - 2 : 0; i < nk; ++i) settle(k_full(i & 1u), (i >> 1) & 1u);
            for (uint32_t i = nv > 2 ? nv - 2 : 0; i < nv; ++i) settle(v_full(i & 1u), (i >> 1) & 1u);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuers
        // Two threads: this warp's issues the S products, warp 6's the PV
        // products, each waiting only on what its own products need and
        // committing its own barriers, so neither's waits hold up the other's
        // MMAs.  S runs two blocks ahead of PV: S of block g + 2 goes into S
        // buffer g & 1 as soon as the PV product of block g has read P from
        // it, so it overlaps the softmax of block g + 1.
        constexpr uint32_t idesc_s = idesc_bf16_f32(kBQ, kBKV);
        bool ok = run;
        BlockWalk ws;  // the next block to take its S product
        if (ok) {
            ws.t = t_first;
            walk_job(p, njobs, lane, ws);
        }
        uint32_t gs = 0;
        while (ok && ws.valid) {
            const uint32_t b = gs & 1u;
            if (lane == 0) {
                // the buffer's previous block (gs - 2) has had its PV product
                ok = gs < 2 || wait_one(o_ready(b), ((gs - 2) >> 1) & 1u, abort_flag, p.status,
                                        p.wait_ns);
                if (ok && ws.j == 0)
                    ok = wait_one(q_full, ws.jn & 1u, abort_flag, p.status, p.wait_ns);
                if (ok) ok = wait_one(k_full(b), (gs >> 1) & 1u, abort_flag, p.status, p.wait_ns);
                if (ok) {
                    tc_fence_after();
                    const uint32_t qs = sbase + L::Q_OFF, ks = sbase + L::K_OFF + b * L::KV_TILE;
#pragma unroll
                    for (int kk = 0; kk < kD / 16; ++kk) {
                        tc_mma_ss(tmem + L::S_COL + b * kBKV,
                                  sdesc_kmajor_sw128(qs + (kk >> 2) * L::QBOX + (kk & 3) * 32),
                                  sdesc_kmajor_sw128(ks + (kk >> 2) * L::KBOX + (kk & 3) * 32),
                                  idesc_s, kk > 0 ? 1u : 0u);
                    }
                    tc_commit(s_full(b));
                    tc_commit(k_empty(b));
                    if (ws.j == ws.nblk - 1) tc_commit(q_empty);  // the job's last S frees Q
                }
            }
            ok = __shfl_sync(0xffffffffu, ok, 0);
            ++gs;
            walk_next(p, njobs, t_step, lane, ws);
        }
        if (lane == 0) {
            tc_commit(drain(0));  // every MMA issued has completed before tensor memory is freed
            settle(drain(0), 0);
        }
    } else if (warp == kPvWarp) {
        // ------------------------------------------------------------ PV issuer
        constexpr uint32_t idesc_o = idesc_bf16_f32(kBQ, kD) | (1u << 16);  // B MN-major
        bool ok = run;
        BlockWalk wp;  // the next block to take its PV product
        if (ok) {
            wp.t = t_first;
            walk_job(p, njobs, lane, wp);
        }
        uint32_t g = 0;
        while (ok && wp.valid) {
            const uint32_t b = g & 1u;
            if (lane == 0) {
                // O += P V once the softmax warps have written P of block g (for
                // a job's first block, after they read out the previous job's O)
                ok = wait_one(p_full(b), (g >> 1) & 1u, abort_flag, p.status, p.wait_ns) &&
                     wait_one(v_full(b), (g >> 1) & 1u, abort_flag, p.status, p.wait_ns);
                if (ok) {
                    tc_fence_after();
                    const uint32_t vs = sbase + L::V_OFF + b * L::KV_TILE;
#pragma unroll
                    for (int kk = 0; kk < kBKV / 16; ++kk) {
                        // keys 16 kk .. 16 kk + 15: rows of the V tile; P columns 8 kk ..
                        tc_mma_ts(tmem + L::O_COL, tmem + L::S_COL + b * kBKV + kk * 8,
                                  sdesc_mnmajor_sw128(vs + kk * 16 * 128, L::KBOX, 1024), idesc_o,
                                  (wp.j > 0 || kk > 0) ? 1u : 0u);
                    }
                    tc_commit(o_ready(b));
                    tc_commit(v_empty(b));
                }
            }
            ok = __shfl_sync(0xffffffffu, ok, 0);
            ++g;
            walk_next(p, njobs, t_step, lane, wp);
        }
        if (lane == 0) {
            tc_commit(drain(1));
            settle(drain(1), 0);
        }
    } else {
        // ------------------------------------------------------------ softmax + epilogue
        // Two warps per TMEM sub-partition: warp (sub, hh) takes the 16 rows
        // 32 sub + 16 hh .. + 15 of the block.  Thread (g, c) = (lane / 4,
        // lane % 4) holds rows g and g + 8 of them at keys 8 j + 2 c and
        // 8 j + 2 c + 1 (16x256b loads), so a row's max and sum combine over
        // the four threads of a quad with two shuffles; its P pairs (key
        // pair 4 j + c) go back with one 16x128b store.
        const int sw = warp - kFirstSoftmaxWarp;
        const int sub = warp & 3;
        const int rb = sub * 32 + (sw >> 2) * 16;  // first row of the warp within the block
        const int g = lane >> 2, c = lane & 3;
        const uint32_t lane_base = tmem + (static_cast<uint32_t>(rb) << 16);
        const float cs = 1.4426950408889634f * p.scale;  // log2(e) / sqrt(d)
        bool ok = run;
        JobCursor cur;
        uint32_t gb = 0;
        for (int64_t t = t_first; ok && t < njobs; t += t_step) {
            const AttnJob jb = job_at(p, t, lane, cur);
            if (!jb.valid) break;
            int b_first, nblk;
            key_range(jb, W, b_first, nblk);
            const int i0 = jb.q0 + rb + g;  // query tokens of rows g and g + 8
            // Running max m (log2 units, scale folded in) and this thread's
            // part of the sum l, per row.  The max is raised lazily: only when
            // a block's max exceeds it by more than 8 (p <= 2^8 otherwise), so
            // O is rescaled rarely; O and l always use the same m, so the
            // final O / l is exact either way.
            float m0 = kMaskedScore, m1 = kMaskedScore, l0 = 0.0f, l1 = 0.0f;
            for (int j = 0; ok && j < nblk; ++j, ++gb) {
                const uint32_t b = gb & 1u;
                if (!wait_warp(s_full(b), (gb >> 1) & 1u, abort_flag, p.status, p.wait_ns)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const int kbase = jb.ss + (b_first + j) * kBKV;
                // every key of the block allowed for every query of the block
                const bool interior = kbase + kBKV - 1 <= jb.q0 && kbase > jb.q0 + kBQ - 1 - W;
                const uint32_t s_tm = lane_base + L::S_COL + b * kBKV;
                uint32_t v[32];
                tmem_ld_16x256b_x8(s_tm, v);
                tmem_ld_wait_n(v);
                if (!interior) {
                    // allowed key offsets for the two rows: lo .. hi (masked
                    // keys become -inf, so their p = 2^(-inf) is exactly 0)
                    const int hi0 = i0 - kbase, lo0 = hi0 - W + 1;
#pragma unroll
                    for (int jj = 0; jj < 8; ++jj)
#pragma unroll
                        for (int e = 0; e < 2; ++e) {
                            const int k = 8 * jj + 2 * c + e;
                            if (k > hi0 || k < lo0) v[4 * jj + e] = 0xFF800000u;
                            if (k > hi0 + 8 || k < lo0 + 8) v[4 * jj + 2 + e] = 0xFF800000u;
                        }
                }
                float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
                for (int jj = 0; jj < 8; ++jj) {
                    mx0 = fmax3(mx0, __uint_as_float(v[4 * jj]), __uint_as_float(v[4 * jj + 1]));
                    mx1 = fmax3(mx1, __uint_as_float(v[4 * jj + 2]), __uint_as_float(v[4 * jj + 3]));
                }
                mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
                mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
                mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
                mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
                const float mb0 = mx0 * cs, mb1 = mx1 * cs;  // cs > 0
                const bool raise0 = mb0 > m0 + 8.0f, raise1 = mb1 > m1 + 8.0f;
                const float mn0 = raise0 ? mb0 : m0, mn1 = raise1 ? mb1 : m1;
                const float alpha0 = ex2(m0 - mn0), alpha1 = ex2(m1 - mn1);
                float2 sum0 = make_float2(0.0f, 0.0f), sum1 = make_float2(0.0f, 0.0f);
                uint32_t pk[16];
#pragma unroll
                for (int jj = 0; jj < 8; ++jj) {
                    // p = 2^(s c - m) for a key pair of each row: a paired FMA, two ex2
                    float2 e0 = ffma2(make_float2(__uint_as_float(v[4 * jj]),
                                                  __uint_as_float(v[4 * jj + 1])), cs, -mn0);
                    float2 e1 = ffma2(make_float2(__uint_as_float(v[4 * jj + 2]),
                                                  __uint_as_float(v[4 * jj + 3])), cs, -mn1);
                    e0.x = ex2(e0.x);
                    e0.y = ex2(e0.y);
                    e1.x = ex2(e1.x);
                    e1.y = ex2(e1.y);
                    sum0 = fadd2(sum0, e0);
                    sum1 = fadd2(sum1, e1);
                    pk[2 * jj] = pack_bf16x2_rn(e0.x, e0.y);
                    pk[2 * jj + 1] = pack_bf16x2_rn(e1.x, e1.y);
                }
                tmem_st_16x128b_x8(s_tm, pk);  // P of block gb over the first half of its S
                // rescale O (the sum over the job's blocks before j) to the new
                // max, once the PV product of block gb - 1 has completed
                if (j > 0 && __any_sync(0xffffffffu, raise0 || raise1)) {
                    if (!wait_warp(o_ready((gb - 1) & 1u), ((gb - 1) >> 1) & 1u, abort_flag,
                                   p.status, p.wait_ns)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
#pragma unroll 1
                    for (int ch = 0; ch < kD / 32; ++ch) {
                        uint32_t o[16];
                        tmem_ld_16x256b_x4(lane_base + L::O_COL + ch * 32, o);
                        tmem_ld_wait_n(o);
#pragma unroll
                        for (int jj = 0; jj < 4; ++jj) {
                            o[4 * jj] = __float_as_uint(__uint_as_float(o[4 * jj]) * alpha0);
                            o[4 * jj + 1] = __float_as_uint(__uint_as_float(o[4 * jj + 1]) * alpha0);
                            o[4 * jj + 2] = __float_as_uint(__uint_as_float(o[4 * jj + 2]) * alpha1);
                            o[4 * jj + 3] = __float_as_uint(__uint_as_float(o[4 * jj + 3]) * alpha1);
                        }
                        tmem_st_16x256b_x4(lane_base + L::O_COL + ch * 32, o);
                    }
                }
                l0 = l0 * alpha0 + (sum0.x + sum0.y);
                l1 = l1 * alpha1 + (sum1.x + sum1.y);
                m0 = mn0;
                m1 = mn1;
                tmem_st_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(p_full(b));  // P of block gb written over its S
            }
            // ---- epilogue: O / l -> bf16.  The next job's first PV product,
            // which overwrites O, waits for P of that job, which these warps
            // write only after this epilogue has read O.
            if (!ok || !wait_warp(o_ready((gb - 1) & 1u), ((gb - 1) >> 1) & 1u, abort_flag, p.status, p.wait_ns)) {
                ok = false;
                break;
            }
            tc_fence_after();
            // the rows' sums over the quad's four parts
            l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
            l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
            l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
            l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
            const float inv0 = l0 > 0.0f ? 1.0f / l0 : 0.0f;
            const float inv1 = l1 > 0.0f ? 1.0f / l1 : 0.0f;
            // Each 32-column chunk of the warp's 16 rows goes through its
            // staging buffer (16 rows x 64 bytes), so that a store instruction
            // writes 8 rows x 64 contiguous bytes: 16-byte unit u of row q sits
            // at unit u ^ ((q >> 1) & 3), which puts the 32 four-byte writes of
            // a staging store on distinct banks.
            uint8_t* stage = smem + L::STAGE_OFF + sw * L::STAGE_WARP;
            uint32_t* stage32 = reinterpret_cast<uint32_t*>(stage);
            const int rows_left = jb.se - (jb.q0 + rb);  // rows of this warp to store
            __nv_bfloat16* obase = reinterpret_cast<__nv_bfloat16*>(p.out) +
                                   static_cast<int64_t>(jb.q0 + rb) * Hd + jb.h * kD;
            const int sw0 = (g >> 1) & 3;  // rows g and g + 8 share the swizzle
#pragma unroll 1
            for (int ch = 0; ch < kD / 32; ++ch) {
                uint32_t o[16];
                tmem_ld_16x256b_x4(lane_base + L::O_COL + ch * 32, o);
                tmem_ld_wait_n(o);
#pragma unroll
                for (int jj = 0; jj < 4; ++jj) {
                    // columns 8 jj + 2 c, + 1: word 4 jj + c of the row, in unit jj
                    const int word = 4 * (jj ^ sw0) + c;
                    stage32[g * 16 + word] = pack_bf16x2_rn(__uint_as_float(o[4 * jj]) * inv0,
                                                            __uint_as_float(o[4 * jj + 1]) * inv0);
                    stage32[(g + 8) * 16 + word] =
                        pack_bf16x2_rn(__uint_as_float(o[4 * jj + 2]) * inv1,
                                       __uint_as_float(o[4 * jj + 3]) * inv1);
                }
                __syncwarp();
#pragma unroll
                for (int it = 0; it < 2; ++it) {
                    const int q = it * 8 + (lane >> 2), u = lane & 3;
                    const uint4 w = *reinterpret_cast<const uint4*>(stage + q * 64 +
                                                                    ((u ^ ((q >> 1) & 3)) << 4));
                    if (q < rows_left &&
                        dbg_check(jb.q0 + rb + q < jb.se && jb.q0 + rb + q >= jb.ss, p.status))
                        *reinterpret_cast<uint4*>(obase + static_cast<int64_t>(q) * Hd + ch * 32 + u * 8) = w;
                }
                __syncwarp();
            }
        }
        // a softmax warp that gave up may have tensor-memory stores in flight
        tmem_st_wait();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, L::TMEM_COLS);
}

}  // namespace

cudaError_t launch_attention_prefill(const CUtensorMap* tmap_q, const CUtensorMap* tmap_kv,
                                     const AttnParams& p, cudaStream_t stream) {
    using L = AttnLayout;
    cudaError_t e = cudaFuncSetAttribute(attention_prefill_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         L::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    // upper bound on the query blocks: sum over sequences of ceil(len / 128)
    const int64_t qblocks = (static_cast<int64_t>(p.M) + kBQ - 1) / kBQ + p.nseq;
    const int64_t njobs = qblocks * p.H;
    // persistent: two CTAs per SM, each taking every grid-th job
    int dev = 0, sms = 0;
    e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
    const int64_t grid = njobs < 2 * static_cast<int64_t>(sms) ? njobs : 2 * static_cast<int64_t>(sms);
    attention_prefill_kernel<<<static_cast<unsigned>(grid), kThreads, L::SMEM_BYTES, stream>>>(
        *tmap_q, *tmap_kv, p, njobs);
    return cudaGetLastError();
}

int attention_head_dim() { return kD; }
int attention_key_block() { return kBKV; }

}  // namespace w4a16
