/*
 * CPU oracle for the group-wise int4 weight-only (W4A16) linear layer.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call, link or
 * load this file: it is used by tests/, by __graft_entry__.smoke() and by
 * the cpu_baseline / --impl reference legs of bench.py.  It shares no code,
 * header, table or constant with the CUDA library.
 *
 * What it computes.  The paper runs its 175B decoder "4-bit pre-quantized"
 * with "mixed-precision quantization" (Sec. 3.1, Sec. 4.1) and gives no
 * format.  The format used here is the one fixed for this library:
 *   - symmetric int4 per group of g consecutive k, zero point 8,
 *     stored code q in 0..15;
 *   - two codes per byte, the even k in bits 0..3, the odd k in bits 4..7;
 *   - one bf16 scale per (row n, group k/g);
 *   - dequantised weight wd = RNE_bf16( (q - 8) * s ), one rounding of the
 *     exact fp32 product;
 *   - out[m,n] = sum_k x[m,k] * wd[n,k], accumulated here in fp64 with k
 *     ascending (the reference value that the GPU result is measured against).
 * The quantiser (data generation): s = RNE_bf16(amax / 7) with an fp32
 * division, q = clamp(round_half_even(w / s), -8, 7) + 8, all-zero group ->
 * s = 0 and q = 8.
 *
 * Every function is a direct transcription of that definition: no blocking,
 * no fusion, no reordering.  The bf16 rounding is written out from the IEEE
 * binary32 bit pattern (round to nearest, ties to even) rather than taken from
 * any library.
 */
#include <stdint.h>
#include <string.h>
#include <math.h>

#ifdef _OPENMP
#include <omp.h>
#endif

/* ---- bf16 <-> fp32 ----------------------------------------------------- */

/* bf16 is the top 16 bits of an IEEE binary32.  Widening is exact. */
float oracle_bf16_to_f32(uint16_t h) {
    uint32_t u = ((uint32_t)h) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

/* Round a binary32 to the nearest bf16, ties to even.  Dropping the low 16
 * bits is a truncation toward zero of the magnitude; adding 0x7FFF plus the
 * lowest kept bit before truncating moves every value that lies more than
 * halfway (or exactly halfway with an odd kept part) up to the next bf16.
 * A carry out of the mantissa correctly bumps the exponent (and overflows to
 * infinity).  NaN inputs stay NaN (quiet bit forced, sign kept). */
uint16_t oracle_bf16_rne(float f) {
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu) != 0u)
        return (uint16_t)((u >> 16) | 0x0040u);
    uint32_t kept_lsb = (u >> 16) & 1u;
    u += 0x7FFFu + kept_lsb;
    return (uint16_t)(u >> 16);
}

/* ---- packing ------------------------------------------------------------ */

/* q[n*K + k] = code of weight (n, k), 0..15. */
void oracle_unpack(const uint8_t* packed, int64_t N, int64_t K, uint8_t* q) {
    for (int64_t n = 0; n < N; ++n)
        for (int64_t k = 0; k < K; ++k) {
            uint8_t b = packed[n * (K / 2) + k / 2];
            q[n * K + k] = (k % 2 == 0) ? (uint8_t)(b & 0x0F) : (uint8_t)(b >> 4);
        }
}

void oracle_pack(const uint8_t* q, int64_t N, int64_t K, uint8_t* packed) {
    for (int64_t n = 0; n < N; ++n)
        for (int64_t j = 0; j < K / 2; ++j) {
            uint8_t lo = q[n * K + 2 * j] & 0x0F;
            uint8_t hi = q[n * K + 2 * j + 1] & 0x0F;
            packed[n * (K / 2) + j] = (uint8_t)(lo | (hi << 4));
        }
}

/* ---- quantiser (input generation) --------------------------------------- */

/* w: fp32 [N, K] row-major.  packed: [N, K/2].  scales: bf16 bits [N, K/g].
 * Returns 0, or -1 if the shape is not one the format admits. */
int oracle_quantize(const float* w, int64_t N, int64_t K, int64_t g,
                    uint8_t* packed, uint16_t* scales) {
    if (N < 0 || K <= 0 || g <= 0 || K % g != 0 || K % 2 != 0) return -1;
    int64_t KG = K / g;
    for (int64_t n = 0; n < N; ++n) {
        for (int64_t j = 0; j < KG; ++j) {
            const float* grp = w + n * K + j * g;
            float amax = 0.0f;
            for (int64_t t = 0; t < g; ++t) {
                float a = fabsf(grp[t]);
                if (a > amax) amax = a;
            }
            volatile float seven = 7.0f;           /* keep the division in fp32 */
            float s_exact = amax / seven;
            uint16_t s_bits = oracle_bf16_rne(s_exact);
            float s = oracle_bf16_to_f32(s_bits);
            scales[n * KG + j] = s_bits;
            for (int64_t t = 0; t < g; ++t) {
                int64_t k = j * g + t;
                int code;
                if (s == 0.0f) {
                    code = 8;
                } else {
                    float r = nearbyintf(grp[t] / s);  /* current mode: nearest-even */
                    if (r < -8.0f) r = -8.0f;
                    if (r > 7.0f) r = 7.0f;
                    code = (int)r + 8;
                }
                uint8_t* byte = &packed[n * (K / 2) + k / 2];
                if (k % 2 == 0) *byte = (uint8_t)((*byte & 0xF0) | code);
                else            *byte = (uint8_t)((*byte & 0x0F) | (code << 4));
            }
        }
    }
    return 0;
}

/* ---- dequantisation ----------------------------------------------------- */

/* wd[n*K + k] = RNE_bf16( (q - 8) * s[n, k/g] ), as bf16 bits. */
void oracle_dequant(const uint8_t* packed, const uint16_t* scales,
                    int64_t N, int64_t K, int64_t g, uint16_t* wd) {
    int64_t KG = K / g;
    for (int64_t n = 0; n < N; ++n)
        for (int64_t k = 0; k < K; ++k) {
            uint8_t b = packed[n * (K / 2) + k / 2];
            int q = (k % 2 == 0) ? (b & 0x0F) : (b >> 4);
            float s = oracle_bf16_to_f32(scales[n * KG + k / g]);
            float prod = (float)(q - 8) * s;  /* exact: 4-bit times 8-bit significand */
            wd[n * K + k] = oracle_bf16_rne(prod);
        }
}

/* ---- linear -------------------------------------------------------------- */

/* One output row: out_row[n] = sum_k x[m,k] * wd[n,k] in fp64, k ascending. */
static void linear_one_n(const uint16_t* xrow, const uint8_t* packed,
                         const uint16_t* scales, int64_t n, int64_t K,
                         int64_t g, double* acc_out) {
    int64_t KG = K / g;
    double acc = 0.0;
    for (int64_t k = 0; k < K; ++k) {
        uint8_t b = packed[n * (K / 2) + k / 2];
        int q = (k % 2 == 0) ? (b & 0x0F) : (b >> 4);
        float s = oracle_bf16_to_f32(scales[n * KG + k / g]);
        float wd = oracle_bf16_to_f32(oracle_bf16_rne((float)(q - 8) * s));
        acc += (double)oracle_bf16_to_f32(xrow[k]) * (double)wd;
    }
    *acc_out = acc;
}

/* x: bf16 bits [M, K]; out: fp64 [nrows, N] for the listed rows of x.
 * nthreads > 1 splits the n loop across OpenMP threads (same arithmetic). */
void oracle_linear_rows(const uint16_t* x, const uint8_t* packed,
                        const uint16_t* scales, int64_t M, int64_t N, int64_t K,
                        int64_t g, const int64_t* rows, int64_t nrows,
                        double* out, int nthreads) {
    (void)M;
    for (int64_t r = 0; r < nrows; ++r) {
        const uint16_t* xrow = x + rows[r] * K;
#ifdef _OPENMP
        #pragma omp parallel for num_threads(nthreads > 0 ? nthreads : 1) schedule(static)
#endif
        for (int64_t n = 0; n < N; ++n)
            linear_one_n(xrow, packed, scales, n, K, g, &out[r * N + n]);
    }
    (void)nthreads;
}

/* Sampled points: out[i] = ref[mi[i], ni[i]]. */
void oracle_linear_points(const uint16_t* x, const uint8_t* packed,
                          const uint16_t* scales, int64_t M, int64_t N, int64_t K,
                          int64_t g, const int64_t* mi, const int64_t* ni,
                          int64_t npts, double* out, int nthreads) {
    (void)M; (void)N;
#ifdef _OPENMP
    #pragma omp parallel for num_threads(nthreads > 0 ? nthreads : 1) schedule(static)
#endif
    for (int64_t i = 0; i < npts; ++i)
        linear_one_n(x + mi[i] * K, packed, scales, ni[i], K, g, &out[i]);
    (void)nthreads;
}

/* ---- fused epilogue --------------------------------------------------------
 *
 * Operator fusion of what follows a linear layer into its output stage -- the
 * optimisation the paper names as future work (Sec. 5).  The paper names no
 * activation; the readings fixed for this library are the usual decoder ones:
 *   z[n]   = y[n] + bias[n]                       (bias optional, bf16 [N])
 *   act 0: h[n] = z[n]                            (N_out = N)
 *   act 1: SwiGLU over interleaved rows: h[j] = silu(z[2j]) * z[2j+1],
 *          silu(t) = t / (1 + exp(-t))            (N_out = N / 2)
 *   act 2: GELU, h[n] = z[n] * Phi(z[n]) = z/2 * (1 + erf(z / sqrt 2))
 *   out[j] = h[j] + residual[m, j]                (residual optional, bf16
 *                                                  [M, N_out])
 * all in fp64.  y: fp64 [nrows, N] for the rows `rows` of the batch. */
static double silu_d(double t) { return t / (1.0 + exp(-t)); }
static double gelu_d(double t) { return 0.5 * t * (1.0 + erf(t / sqrt(2.0))); }

void oracle_epilogue_rows(const double* y, int64_t nrows, int64_t N, const uint16_t* bias,
                          const uint16_t* residual, const int64_t* rows, int act,
                          double* out) {
    int64_t n_out = act == 1 ? N / 2 : N;
    for (int64_t r = 0; r < nrows; ++r) {
        const double* yr = y + r * N;
        for (int64_t j = 0; j < n_out; ++j) {
            double h;
            if (act == 1) {
                double gate = yr[2 * j] + (bias ? (double)oracle_bf16_to_f32(bias[2 * j]) : 0.0);
                double up = yr[2 * j + 1] + (bias ? (double)oracle_bf16_to_f32(bias[2 * j + 1]) : 0.0);
                h = silu_d(gate) * up;
            } else {
                double z = yr[j] + (bias ? (double)oracle_bf16_to_f32(bias[j]) : 0.0);
                h = act == 2 ? gelu_d(z) : z;
            }
            if (residual) h += (double)oracle_bf16_to_f32(residual[rows[r] * n_out + j]);
            out[r * n_out + j] = h;
        }
    }
}

/* ---- scoring readout: gather and top-k ------------------------------------
 *
 * The pipeline's last modules (Sec. 3.3): the affinity head reads one hidden
 * state per pair (rows of the packed batch picked by index), and the
 * predicted affinities are sorted for export.  Readings fixed for this
 * library: affinities are binding free energies in kcal/mol, so the best
 * candidates are the k smallest; scores are ordered by the IEEE 754
 * totalOrder predicate on non-NaN values (-0 before +0), every NaN after
 * every number, and equal scores by ascending index. */

/* dst[p, :] = src[idx[p], :]; an index outside [0, src_rows) gives a zero row
 * and a nonzero return. */
int oracle_gather_rows(const uint16_t* src, int64_t src_rows, int64_t D, const int32_t* idx,
                       int64_t P, uint16_t* dst) {
    int bad = 0;
    for (int64_t p = 0; p < P; ++p) {
        if (idx[p] < 0 || idx[p] >= src_rows) {
            for (int64_t d = 0; d < D; ++d) dst[p * D + d] = 0;
            bad = 1;
            continue;
        }
        for (int64_t d = 0; d < D; ++d) dst[p * D + d] = src[(int64_t)idx[p] * D + d];
    }
    return bad;
}

/* -1, 0, 1 as (a, ia) orders before, equal to, after (b, ib). */
static int score_order(float a, int64_t ia, float b, int64_t ib) {
    int na = isnan(a) != 0, nb = isnan(b) != 0;
    if (na != nb) return na ? 1 : -1;          /* NaN after every number */
    if (!na) {
        if (a < b) return -1;
        if (a > b) return 1;
        if (a == 0.0f) {                        /* equal zeros: -0 before +0 */
            int sa = signbit(a) != 0, sb = signbit(b) != 0;
            if (sa != sb) return sa ? -1 : 1;
        }
    }
    return ia < ib ? -1 : (ia > ib ? 1 : 0);   /* ties by index */
}

/* The k smallest scores in order: out_idx[j], out_val[j] for j < k, by
 * repeated selection of the least remaining element (O(n k), plain). */
void oracle_topk_smallest(const float* scores, int64_t n, int64_t k, int32_t* out_idx,
                          float* out_val, unsigned char* taken) {
    memset(taken, 0, (size_t)n);
    for (int64_t j = 0; j < k; ++j) {
        int64_t best = -1;
        for (int64_t i = 0; i < n; ++i) {
            if (taken[i]) continue;
            if (best < 0 || score_order(scores[i], i, scores[best], best) < 0) best = i;
        }
        taken[best] = 1;
        out_idx[j] = (int32_t)best;
        out_val[j] = scores[best];
    }
}

/* ---- attention prefill over packed sequences --------------------------------
 *
 * The decoder's attention between the QKV and output projections: causal
 * within each protein-ligand pair's packed token sequence, limited to a
 * sliding window of W tokens (the model's 32K window, Sec. 2.1).  Readings:
 * standard multi-head scaled dot-product attention; qkv is the fused QKV
 * projection output [M, 3 H d] (bf16) with q of head h in columns h d ..,
 * k at H d + h d, v at 2 H d + h d; sequence s holds tokens
 * [seq_start[s], seq_start[s+1]); query i attends to keys j of its own
 * sequence with i - W < j <= i:
 *   o[i, h, :] = sum_j softmax_j(q_i . k_j / sqrt(d)) v_j     (fp64)
 * out: fp64 [M, H d] for the listed query tokens (rows). */
void oracle_attention_rows(const uint16_t* qkv, int64_t M, int64_t H, int64_t d,
                           const int64_t* seq_start, int64_t nseq, int64_t window,
                           const int64_t* rows, int64_t nrows, double* out, double* scratch) {
    (void)M;
    const int64_t ld = 3 * H * d;
    const double scale = 1.0 / sqrt((double)d);
    for (int64_t r = 0; r < nrows; ++r) {
        const int64_t i = rows[r];
        int64_t s = 0;
        while (s + 1 < nseq && seq_start[s + 1] <= i) ++s;
        const int64_t lo0 = seq_start[s];
        const int64_t lo = i - window + 1 > lo0 ? i - window + 1 : lo0;
        for (int64_t h = 0; h < H; ++h) {
            const uint16_t* q = qkv + i * ld + h * d;
            double mx = -INFINITY;
            for (int64_t j = lo; j <= i; ++j) {
                const uint16_t* k = qkv + j * ld + H * d + h * d;
                double dot = 0.0;
                for (int64_t t = 0; t < d; ++t)
                    dot += (double)oracle_bf16_to_f32(q[t]) * (double)oracle_bf16_to_f32(k[t]);
                scratch[j - lo] = dot * scale;
                if (scratch[j - lo] > mx) mx = scratch[j - lo];
            }
            double den = 0.0;
            for (int64_t j = lo; j <= i; ++j) {
                scratch[j - lo] = exp(scratch[j - lo] - mx);
                den += scratch[j - lo];
            }
            for (int64_t t = 0; t < d; ++t) {
                double acc = 0.0;
                for (int64_t j = lo; j <= i; ++j)
                    acc += scratch[j - lo] * (double)oracle_bf16_to_f32(qkv[j * ld + 2 * H * d + h * d + t]);
                out[r * H * d + h * d + t] = acc / den;
            }
        }
    }
}

int oracle_max_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
