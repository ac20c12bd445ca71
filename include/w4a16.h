/*
 * w4a16.h -- C ABI of the GB300 (sm_103a) group-wise int4 weight-only linear
 * layer library.
 *
 * The operation.  The paper scores protein-ligand pairs with a 175B-class
 * decoder whose weights are quantised to 4 bits ahead of time, with mixed
 * precision (Sec. 3.1, Sec. 4.1), run in batches through its prediction module
 * (Sec. 3.3).  On the prefill path the linear layers (fused QKV, attention
 * output, MLP up, MLP down) are y = x W^T with W held at 4 bits.  The paper
 * gives no format; this library fixes one:
 *
 *   w_packed  uint8 [N, K/2]   byte (n, j) holds the code of k = 2j in bits
 *                              0..3 and of k = 2j+1 in bits 4..7; codes are
 *                              0..15 with zero point 8 (symmetric int4)
 *   scales    bf16  [N, K/g]   one scale per row n and group of g consecutive k
 *   dequant   wd[n,k] = RNE_bf16((code - 8) * scales[n, k/g])
 *   x         bf16  [M, K]     activations (M = packed tokens of the batch)
 *   out       bf16  [M, N]     out[m,n] = RNE_bf16( sum_k x[m,k] * wd[n,k] ),
 *                              the sum accumulated in fp32 in an unspecified
 *                              order
 *
 * All matrices are row-major with the last dimension contiguous and no
 * padding between rows.
 *
 * Conventions shared by every entry point:
 *   - Every buffer is owned by the caller and lives in device memory unless
 *     stated otherwise.  The library allocates nothing per call, frees
 *     nothing and does not synchronise: work is enqueued on `stream` and the
 *     call returns.  `stream` is a cudaStream_t passed as void* (0 = the
 *     legacy default stream).  `out` must not overlap any input.
 *   - Arguments are validated before anything is launched; a rejected call
 *     launches nothing and leaves every buffer untouched.
 *   - Device pointers must be 16-byte aligned (W4A16_ERR_ALIGNMENT).
 *   - Supported shapes: M, N >= 1; K >= g; g a multiple of 64; K a multiple
 *     of g; M, N, K < 2^31 (W4A16_ERR_INVALID_ARG / W4A16_ERR_UNSUPPORTED).
 *     g = 128 is the tuned case.
 *   - A launch failure returns W4A16_ERR_CUDA (the CUDA error is left for
 *     cudaGetLastError to report).
 *   - The kernels bound every internal wait.  If a wait runs out (it never
 *     should) the kernel records W4A16_ERR_TIMEOUT in a device status word
 *     and finishes early; w4a16_get_device_error reports it.  Kernels that
 *     check device-side data (sequence tables, gather indices) record
 *     W4A16_ERR_INVALID_ARG there.  The word keeps the first error recorded
 *     until it is read.
 *   - Results are deterministic: the same inputs give the same bits.
 *   - Thread safety: calls from several host threads are safe; per-device
 *     state (SM count, driver entry point) is initialised once.
 *   - Debug build: compiled with -DW4A16_DEBUG (libw4a16_debug.so), the
 *     kernels check every TMA coordinate and destination, tensor-memory column
 *     range and global store index they compute; a failed check records
 *     W4A16_ERR_INDEX in the device status word and skips the access (no
 *     trap).  The release build carries none of these checks.
 */
#ifndef W4A16_H
#define W4A16_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    W4A16_OK = 0,
    W4A16_ERR_INVALID_ARG = 1,   /* null pointer, non-positive or inconsistent size */
    W4A16_ERR_UNSUPPORTED = 2,   /* valid request outside the supported shapes */
    W4A16_ERR_ALIGNMENT = 3,     /* a pointer is not 16-byte aligned */
    W4A16_ERR_CUDA = 4,          /* a CUDA runtime/driver call or launch failed */
    W4A16_ERR_TIMEOUT = 5,       /* a kernel gave up on a bounded wait */
    W4A16_ERR_INDEX = 6          /* an index check of a W4A16_DEBUG build failed */
} w4a16_status;

/*
 * out = x * dequant(w_packed, scales)^T.
 * The hot path of the paper's scoring workflow (Sec. 3.3: batched encoding and
 * affinity prediction) for one int4 linear layer (Sec. 3.1, Sec. 4.1).
 *   x_bf16       [M, K]   bf16, device
 *   w_packed_u8  [N, K/2] uint8, device, layout above
 *   scales_bf16  [N, K/g] bf16, device
 *   out_bf16     [M, N]   bf16, device, written in full
 * Dispatch: M > 128 runs the fused dequant + tcgen05 GEMM; M <= 128 with
 * g = 128 runs a row-range streaming kernel that reads the weights once
 * (warp-level MMAs for M <= 16, tcgen05 for M = 17..128); M <= 32 with
 * g != 128 runs the tcgen05 GEMM with 32-token tiles, other M with g != 128
 * the GEMM.  The tcgen05 kernels multiply x by
 * the dequantised weights wd defined above, so they differ from each other
 * only in the fp32 summation order.  The warp-level streaming kernel factors
 * the scale out of each group instead: it sums x * (code - 8) over the group
 * exactly in fp32 (the codes are small integers) and adds scale * that sum,
 * so it never rounds (code - 8) * scale to bf16.  Both stay within the same
 * error bound of the exact product x * wd^T (fp32 accumulation followed by
 * one bf16 rounding of the output); they are not bit-identical to each
 * other.
 */
int w4a16_linear(const void* x_bf16, const void* w_packed_u8, const void* scales_bf16,
                 void* out_bf16, int64_t M, int64_t N, int64_t K, int64_t g,
                 void* stream);

/* Activation of the fused epilogue (w4a16_linear_fused). */
typedef enum {
    W4A16_ACT_NONE = 0,
    /* SwiGLU over interleaved rows: rows 2j and 2j+1 of the weights are the
     * gate and up projections of output column j; h[m,j] = silu(z[m,2j]) *
     * z[m,2j+1] with silu(t) = t / (1 + e^-t).  N must be even; the output
     * has N/2 columns. */
    W4A16_ACT_SWIGLU = 1,
    /* GELU, exact form: h = z * Phi(z) = z/2 * (1 + erf(z / sqrt 2)). */
    W4A16_ACT_GELU = 2
} w4a16_activation;

/*
 * out = act(x * dequant(w_packed, scales)^T + bias) + residual: the linear
 * layer with what follows it fused into its output stage -- the operator
 * fusion the paper names as the next optimisation (Sec. 5).  The paper names
 * no activation; SwiGLU and GELU are the usual decoder ones.
 *   x, w_packed, scales, M, N, K, g   as in w4a16_linear
 *   bias_bf16      [N] bf16, device, added to every row before the
 *                  activation; NULL for none
 *   residual_bf16  [M, N_out] bf16, device, added after the activation; NULL
 *                  for none.  It may be out itself (in-place residual add);
 *                  otherwise it must not overlap out.
 *   out_bf16       [M, N_out] bf16, device: N_out = N/2 for SwiGLU, else N
 *   activation     a w4a16_activation (else W4A16_ERR_INVALID_ARG; SwiGLU
 *                  with odd N is W4A16_ERR_INVALID_ARG)
 * Everything after the fp32 accumulation is computed in fp32 with one bf16
 * rounding at the store.  Pointers follow the 16-byte rule.  With
 * activation NONE and both pointers NULL this is w4a16_linear.
 */
int w4a16_linear_fused(const void* x_bf16, const void* w_packed_u8, const void* scales_bf16,
                       const void* bias_bf16, const void* residual_bf16, void* out_bf16,
                       int64_t M, int64_t N, int64_t K, int64_t g, int activation,
                       void* stream);

/* One int4 linear layer of a stack.  The caller owns every pointer. */
typedef struct {
    const void* x;          /* bf16 [M, K] */
    const void* w_packed;   /* uint8 [N, K/2] */
    const void* scales;     /* bf16 [N, K/g] */
    void* out;              /* bf16 [M, N] */
    int64_t N;
    int64_t K;
} w4a16_layer;

/*
 * Runs n_layers linear layers in order on `stream`, all with the same M
 * (packed tokens of the scored batch) and group size g: the per-pass layer
 * loop of the paper's prediction module (Sec. 3.3) over the quantised
 * decoder (Sec. 4.1).  `layers` is a HOST array the call reads before it
 * returns.  Every layer is validated before the first launch; layer i may read
 * the output of layer i-1 (chaining) because launches are stream-ordered.
 */
int w4a16_linear_stack(const w4a16_layer* layers, int64_t n_layers,
                       int64_t M, int64_t g, void* stream);

/*
 * A layer stack captured once as a CUDA graph and replayed per batch: the
 * continuous-batching loop of the paper's pipeline (Sec. 3.3) runs the same
 * stack over batch after batch, with each batch's inputs copied into the same
 * buffers.  Replaying the graph removes the per-layer host launch work.
 *
 * w4a16_stack_graph_create validates every layer (as w4a16_linear_stack) and
 * captures the stack's launches -- the pointers in `layers` are baked in --
 * into *out.  Unlike the per-call entry points it allocates: the graph and
 * its host handle, released by w4a16_stack_graph_destroy.
 * w4a16_stack_graph_launch enqueues one pass on `stream` (the current device
 * must be the one the graph was created on, else W4A16_ERR_INVALID_ARG) and
 * allocates nothing.  Results are bit-identical to w4a16_linear_stack.
 */
typedef struct w4a16_stack_graph w4a16_stack_graph;
int w4a16_stack_graph_create(const w4a16_layer* layers, int64_t n_layers, int64_t M, int64_t g,
                             w4a16_stack_graph** out);
int w4a16_stack_graph_launch(w4a16_stack_graph* graph, void* stream);
int w4a16_stack_graph_destroy(w4a16_stack_graph* graph);

/*
 * wd = dequant(w_packed, scales) as bf16 [N, K] (device): the 4-bit weights
 * of the pre-quantised model (Sec. 4.1; mixed-precision quantisation,
 * Sec. 3.1) brought back to the precision the matmul runs in, with the
 * format and rounding stated at the top of this file.  The same unpack and
 * rounding as inside the tcgen05 GEMM, exported so that it can be compared
 * bit for bit with that definition.
 *   w_packed_u8  [N, K/2] uint8, scales_bf16 [N, K/g] bf16, device
 *   w_bf16       [N, K] bf16, device, written in full, must not overlap the
 *                inputs
 */
int w4a16_dequant(const void* w_packed_u8, const void* scales_bf16, void* w_bf16,
                  int64_t N, int64_t K, int64_t g, void* stream);

/*
 * Quantises fp32 master weights w_f32 [N, K] (device) into w_packed_u8 and
 * scales_bf16 with the library's format: per (n, group), s = RNE_bf16(amax/7)
 * with an IEEE fp32 division, code = clamp(round_half_even(w/s), -8, 7) + 8,
 * an all-zero group gets s = 0 and code 8.  Weight preparation, not part of
 * the per-token path.
 */
int w4a16_quantize(const void* w_f32, void* w_packed_u8, void* scales_bf16,
                   int64_t N, int64_t K, int64_t g, void* stream);

/*
 * Attention prefill over a packed batch of sequences: the decoder's
 * attention between the QKV and output projections, causal within each
 * protein-ligand pair's token sequence and limited to a sliding window of
 * `window` tokens (the model's 32K window, Sec. 2.1); the paper gives no
 * further detail, so this is standard multi-head scaled dot-product
 * attention:
 *   out[i, h*d + t] = sum_j softmax_j(q_i . k_j / sqrt(d)) v_j[t]
 * over keys j of i's sequence with i - window < j <= i.
 *   qkv_bf16       [M, 3*H*d] bf16, device: the fused QKV projection output;
 *                  q of head h in columns h*d .., k at H*d + h*d, v at
 *                  2*H*d + h*d
 *   seq_start_i32  [nseq + 1] int32, device: sequence s is tokens
 *                  [seq_start[s], seq_start[s+1]); nondecreasing, within
 *                  [0, M] (else nothing is written and W4A16_ERR_INVALID_ARG
 *                  is recorded in the device status word); tokens outside
 *                  every sequence are left untouched in out
 *   d              head dimension, 128 (else W4A16_ERR_UNSUPPORTED)
 *   out_bf16       [M, H*d] bf16, device, must not overlap the inputs
 * The softmax is computed in fp32 with P rounded to bf16 for the PV product
 * (tcgen05), O accumulated in fp32, one bf16 rounding at the store.
 */
int w4a16_attention_prefill(const void* qkv_bf16, const void* seq_start_i32, int64_t nseq,
                            int64_t M, int64_t H, int64_t d, int64_t window, void* out_bf16,
                            void* stream);

/*
 * Scoring readout, the last modules of the screening pipeline (Sec. 3.3):
 * the affinity head reads one hidden state per pair of the packed batch
 * (w4a16_gather_rows, then w4a16_linear_fused with the head's weights and
 * bias), and the predicted affinities are sorted for export
 * (w4a16_topk_smallest).
 *
 * dst_bf16[p, :] = src_bf16[index_i32[p], :] for p < P.
 *   src_bf16   [src_rows, D] bf16, device
 *   index_i32  [P] int32, device (e.g. the last token of each pair)
 *   dst_bf16   [P, D] bf16, device, must not overlap src or the index
 * An index outside [0, src_rows) gives a zero row and records
 * W4A16_ERR_INVALID_ARG in the device status word (w4a16_get_device_error).
 */
int w4a16_gather_rows(const void* src_bf16, int64_t src_rows, int64_t D,
                      const void* index_i32, int64_t P, void* dst_bf16, void* stream);

/*
 * The k smallest of n scores -- predicted binding free energies in kcal/mol,
 * so the best binders -- in ascending order: out_index_i32[j] is the index
 * and out_score_f32[j] the score of the j-th.  Order: IEEE 754 totalOrder on
 * numbers (-0 before +0), every NaN after every number, equal scores by
 * ascending index; the result is unique and deterministic.
 *   scores         [n] device, fp32 (score_bits = 32) or bf16 (score_bits =
 *                  16, e.g. the head's output; widened exactly to fp32),
 *                  1 <= n < 2^31; other score_bits: W4A16_ERR_INVALID_ARG
 *   1 <= k <= n, k <= 1024 (larger k: W4A16_ERR_UNSUPPORTED)
 *   out_index_i32  [k] int32, out_score_f32 [k] fp32, device, disjoint
 * One launch of one 8-CTA thread-block cluster; no scratch memory.
 */
int w4a16_topk_smallest(const void* scores, int score_bits, int64_t n, int64_t k,
                        void* out_index_i32, void* out_score_f32, void* stream);

/*
 * Synchronises `stream`, then reads and clears the device status word.
 * Returns W4A16_OK, the first error a kernel recorded since the last read
 * (W4A16_ERR_TIMEOUT from a bounded wait that ran out, W4A16_ERR_INVALID_ARG
 * from a bad sequence table or gather index), or W4A16_ERR_CUDA if the
 * synchronisation or the copy failed.
 */
int w4a16_get_device_error(void* stream);

/*
 * Test hooks for the kernels' bounded waits; the paper has no counterpart.
 *
 * w4a16_selftest_wait_timeout launches one CTA on `stream` whose threads
 * wait, with the kernels' own wait helpers, on a shared-memory mbarrier that
 * nothing arrives on: one thread gives up after limit_ns nanoseconds of
 * global time (1e3 <= limit_ns <= 1e6, else W4A16_ERR_INVALID_ARG), raises
 * the CTA's abort flag and records W4A16_ERR_TIMEOUT; a second warp, waiting
 * with a far longer limit, must leave through that flag.  The timeout stays
 * in the status word only if both waits ended that way (else the kernel
 * records W4A16_ERR_INVALID_ARG), so w4a16_get_device_error reports it and
 * the context stays usable.
 *
 * w4a16_selftest_set_wait_limit sets the wait limit of the kernels launched
 * after it, in ns (0 < limit_ns <= 4e9; 0 restores the default of 4 s; else
 * W4A16_ERR_INVALID_ARG).  A test lowers it so that a real kernel's waits run
 * out and the kernel takes its abort path: it records W4A16_ERR_TIMEOUT,
 * waits for its own copies and MMAs in flight, frees its tensor memory and
 * returns, leaving its output incomplete.  Process-wide and not meant for
 * concurrent use with other launches.
 */
int w4a16_selftest_wait_timeout(int64_t limit_ns, void* stream);
int w4a16_selftest_set_wait_limit(int64_t limit_ns);

/* Static text for a status code; never NULL. */
const char* w4a16_status_string(int status);

/* Library version as major*10000 + minor*100 + patch. */
int w4a16_version(void);

#ifdef __cplusplus
}
#endif

#endif /* W4A16_H */
