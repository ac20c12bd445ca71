// Internal interface between the C-ABI layer (api.cu) and the kernel
// translation units.  Not part of the public ABI.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

namespace w4a16 {

// Fused epilogue of a linear layer: out = act(acc + bias) + residual, with
// act one of none, SwiGLU over interleaved (gate, up) rows (n_out = N / 2)
// or GELU.  All pointers are bf16 bits; null means absent.
struct Epilogue {
    const uint16_t* bias;      // [N]
    const uint16_t* residual;  // [M, n_out]; may be the output itself
    int act;                   // 0 none, 1 SwiGLU, 2 GELU (the ABI's w4a16_activation)
    int n_out;                 // output columns: N, or N / 2 for SwiGLU
};

// Parameters of the fused dequant + tcgen05 kernel (everything except the
// two TMA descriptors, which are passed as __grid_constant__ arguments).
struct TsParams {
    const uint16_t* scales;  // bf16 bits [N, K/g]
    uint16_t* out;           // bf16 bits [M, N]
    int* status;             // device status word (timeouts)
    int M, N, K, g;
    int num_t_tiles;         // token tiles:  ceil(M / tokens per tile)
    int num_w_tiles;         // weight tiles: ceil(N / 128)
    int num_tiles;
    int group_t;             // raster: token tiles per group
    Epilogue epi;
    uint64_t wait_ns;        // limit of every barrier wait (kWaitLimitNs unless a test lowers it)
};

// Kernel variants of the fused kernel.  Both take 128 weight rows per tile
// (the MMA's M) and 64 k per pipeline stage.
enum class TsVariant : int {
    kGemm256 = 0,   // 256 tokens per tile, persistent grid (large M)
    kGemv32 = 1,    // 32 tokens per tile, one tile per CTA (M <= 32)
    kGemmPair = 2,  // 256 tokens x 256 weight rows per CTA pair (cta_group::2), persistent
    kGemmPairWide = 3,  // 384 tokens (two 192-column accumulators) x 256 rows per CTA pair
};

int ts_tokens_per_tile(TsVariant v);
// Token rows of the x box each CTA loads (half the tile for CTA pairs).
int ts_x_box_tokens(TsVariant v);
// Fills the grid size to use for the given problem (persistent or not).
int ts_grid(TsVariant v, const TsParams& p, int sm_count);
// Whether the 384-token CTA-pair tiles take fewer unit-costs per pair than the
// 256-token ones for an M x N product (tile padding and the last wave).
bool ts_prefer_wide(int64_t M, int64_t N, int sm_count);
cudaError_t ts_launch(TsVariant v, const CUtensorMap* tmap_x, const CUtensorMap* tmap_w,
                      const TsParams& p, int grid, cudaStream_t stream);

// Parameters of the small-M streaming kernels (gemv_rows.cu, gemv_tc.cu).
struct GemvParams {
    const uint16_t* scales;  // bf16 bits [N, K/g]
    uint16_t* out;           // bf16 bits [M, N]
    int* status;
    int M, N, K, g;
    int rows_per_cta;        // RB: weight rows per CTA chunk, even, <= 352 (<= 384 tcgen05)
    int num_chunks;          // ceil(N / RB)
    int nt;                  // tcgen05 kernel: 128-row MMA tiles per chunk, ceil(RB / 128)
    Epilogue epi;
    uint64_t wait_ns;
};

// RB for N rows spread over the SMs; tokens per tile for M.
int gemv_rows_per_cta(int64_t N, int sm_count);
int gemv_tokens_per_tile(int64_t M);
cudaError_t gemv_launch(const CUtensorMap* tmap_x, const CUtensorMap* tmap_w,
                        const GemvParams& p, int sm_count, cudaStream_t stream);

// The tensor-core streaming kernel for the same regime (gemv_tc.cu): RB even,
// at most 384; x boxes of gemv_tc_tokens(M) rows x 64 k (128-byte swizzle),
// weight boxes of RB/2 rows x 64 bytes (64-byte swizzle).
int gemv_tc_rows_per_cta(int64_t N, int sm_count);
int gemv_tc_tokens(int64_t M);
cudaError_t gemv_tc_launch(const CUtensorMap* tmap_x, const CUtensorMap* tmap_w,
                           const GemvParams& p, int sm_count, cudaStream_t stream);

// Attention prefill over packed sequences (attention.cu).
struct AttnParams {
    const int32_t* seq_start;  // device [nseq + 1]
    uint16_t* out;             // bf16 bits [M, H * 128]
    int* status;
    int M, H, nseq, window;
    float scale;               // 1 / sqrt(head dim)
    uint64_t wait_ns;
};
int attention_head_dim();
// tmap_q: qkv with [128 tokens x 64 features] boxes; tmap_kv: the same
// tensor with [attention_key_block() tokens x 64 features] boxes (both with
// the 128-byte swizzle)
int attention_key_block();
cudaError_t launch_attention_prefill(const CUtensorMap* tmap_q, const CUtensorMap* tmap_kv,
                                     const AttnParams& p, cudaStream_t stream);

// Scoring readout (readout.cu).
constexpr int kTopkMaxK = 1024;  // largest k of the top-k
cudaError_t launch_topk_smallest(const void* scores, bool bf16, int64_t n, int k,
                                 int32_t* out_idx, float* out_val, cudaStream_t stream);
cudaError_t launch_gather_rows(const uint16_t* src, int64_t src_rows, int64_t D,
                               const int32_t* idx, int64_t P, uint16_t* dst, int* status,
                               int sm_count, cudaStream_t stream);

// Limit of the kernels' barrier waits for launches made now, in ns: 4 s
// unless a test lowered it (w4a16_selftest_set_wait_limit).
uint64_t wait_limit_ns();

cudaError_t launch_dequant(const uint8_t* w, const uint16_t* scales, uint16_t* wd, int64_t N,
                           int64_t K, int64_t g, cudaStream_t stream);
cudaError_t launch_quantize(const float* w, uint8_t* packed, uint16_t* scales, int64_t N,
                            int64_t K, int64_t g, cudaStream_t stream);

}  // namespace w4a16
