// C ABI of the library (declared in include/w4a16.h): argument validation,
// TMA descriptor encoding, kernel dispatch and the device status word.
#include "internal.h"
#include "ptx.cuh"
#include "w4a16.h"

#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <cmath>
#include <cstdlib>
#include <atomic>
#include <mutex>
#include <new>

namespace w4a16 {
namespace {

// Set by kernels when a bounded wait runs out; read and cleared by
// w4a16_get_device_error.
__device__ int g_status_word;

// The kernels' own wait helpers on an mbarrier that nothing arrives on:
// thread 0 of warp 0 waits alone (wait_one) with limit_ns, the whole of
// warp 1 waits (wait_warp) with a limit far beyond it, so it can only leave
// through the abort flag that warp 0 raises when it gives up.  The timeout
// that wait_one records stays in the status word only if both waits failed
// and the flag was raised; anything else overwrites it with
// W4A16_ERR_INVALID_ARG, which the test would report.
__global__ void selftest_wait_kernel(uint64_t limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    __shared__ int gave_up[2];
    if (threadIdx.x == 0) {
        mbar_init(smem_u32(&bar), 1);
        abort_flag = 0;
        gave_up[0] = gave_up[1] = 0;
        fence_mbar_init();
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5;
    if (warp == 0) {
        if (threadIdx.x == 0 &&
            !wait_one(smem_u32(&bar), 0, &abort_flag, &g_status_word, limit_ns))
            gave_up[0] = 1;
    } else if (!wait_warp(smem_u32(&bar), 0, &abort_flag, &g_status_word, 1000u * limit_ns)) {
        if ((threadIdx.x & 31) == 0) gave_up[1] = 1;
    }
    __syncthreads();
    if (threadIdx.x == 0 && !(gave_up[0] && gave_up[1] && abort_flag == 1))
        atomicExch(&g_status_word, W4A16_ERR_INVALID_ARG);
}

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

constexpr int kMaxDevices = 64;

struct DeviceState {
    bool ready = false;
    int sm_count = 0;
    int* status = nullptr;
};

std::mutex g_mutex;
DeviceState g_dev[kMaxDevices];
EncodeTiledFn g_encode = nullptr;
// Raster groups, in token tiles: 6 of 256 tokens (stack sweep 2-16: best 3
// and 6), 3 of 384 (stack at 1 / 2 / 3 / 4 / 6 / 8: 4.49 / 4.59 / 4.60-4.66 /
// 4.59 / 4.52 / 4.50 pairs/s).  W4A16_GROUP_T sets both.
int g_group_t = 6;
int g_group_t_wide = 3;
int64_t g_group_bytes = 0;  // if > 0: groups sized so that a group's x takes at most this
bool g_small_m_streaming = true;
// Small M on the tcgen05 streaming kernel from this many tokens on, on the
// warp-level mma.sync kernel below it (12288 x 49152: M = 32 94 against
// 128 us; M = 16 95 against 83 us; M = 8 95 against 68 us).
// W4A16_SMALL_M=mma / tc forces one of them.
int g_small_m_tc_from = 17;
bool g_gemm_pair = true;  // large M on CTA pairs (cta_group::2); W4A16_GEMM_PAIR=0: one CTA per tile
// CTA pairs with 384-token tiles (one dequantised weight stage serves 1.5x the
// tokens) where they take fewer unit-costs per pair than the 256-token tiles
// (ts_prefer_wide: tile padding and the last wave; 12288 x 49152: M = 4096
// 2996 against 3135 us, M = 8192 MLP projections +7%, the stack 4.51 against
// 4.32 scored pairs/s).  W4A16_GEMM_WIDE=1 / 0 forces them on or off (from this
// many tokens on; -1: chosen per call).
int64_t g_gemm_wide_from = -1;
// barrier-wait limit of the launches (test hook w4a16_selftest_set_wait_limit)
std::atomic<uint64_t> g_wait_limit_ns{kWaitLimitNs};

// Per-device set-up, done once with the device current.
int device_state(DeviceState** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return W4A16_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_mutex);
    DeviceState& st = g_dev[dev];
    if (!st.ready) {
        if (g_encode == nullptr) {
            void* fn = nullptr;
            cudaDriverEntryPointQueryResult q;
            if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000,
                                                 cudaEnableDefault, &q) != cudaSuccess ||
                q != cudaDriverEntryPointSuccess || fn == nullptr)
                return W4A16_ERR_CUDA;
            g_encode = reinterpret_cast<EncodeTiledFn>(fn);
            if (const char* e = std::getenv("W4A16_SMALL_M_TILED")) {
                if (e[0] == '1') g_small_m_streaming = false;
            }
            if (const char* e = std::getenv("W4A16_SMALL_M")) {
                if (e[0] == 'm') g_small_m_tc_from = 33;
                if (e[0] == 't') g_small_m_tc_from = 1;
            }
            if (const char* e = std::getenv("W4A16_GEMM_PAIR")) {
                if (e[0] == '1') g_gemm_pair = true;
                if (e[0] == '0') g_gemm_pair = false;
            }
            if (const char* e = std::getenv("W4A16_GEMM_WIDE")) {
                if (e[0] == '1') g_gemm_wide_from = 33;
                if (e[0] == '0') g_gemm_wide_from = int64_t{1} << 40;  // never
            }
            if (const char* e = std::getenv("W4A16_GROUP_BYTES")) {
                const long long v = std::atoll(e);
                if (v > 0) g_group_bytes = v;
            }
            if (const char* e = std::getenv("W4A16_GROUP_T")) {
                const int v = std::atoi(e);
                if (v > 0 && v <= 4096) g_group_t = g_group_t_wide = v;
            }
        }
        if (cudaDeviceGetAttribute(&st.sm_count, cudaDevAttrMultiProcessorCount, dev) !=
            cudaSuccess)
            return W4A16_ERR_CUDA;
        void* p = nullptr;
        if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return W4A16_ERR_CUDA;
        st.status = static_cast<int*>(p);
        st.ready = true;
    }
    *out = &st;
    return W4A16_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool overlaps(const void* a, int64_t na, const void* b, int64_t nb) {
    const uintptr_t a0 = reinterpret_cast<uintptr_t>(a), b0 = reinterpret_cast<uintptr_t>(b);
    return a0 < b0 + static_cast<uintptr_t>(nb) && b0 < a0 + static_cast<uintptr_t>(na);
}

constexpr int64_t kMaxDim = (int64_t{1} << 31) - 1;

int check_weights(const void* w, const void* s, int64_t N, int64_t K, int64_t g) {
    if (w == nullptr || s == nullptr) return W4A16_ERR_INVALID_ARG;
    if (N <= 0 || K <= 0 || g <= 0) return W4A16_ERR_INVALID_ARG;
    if (K % g != 0) return W4A16_ERR_INVALID_ARG;
    if (g % 64 != 0) return W4A16_ERR_UNSUPPORTED;
    if (N > kMaxDim || K > kMaxDim) return W4A16_ERR_UNSUPPORTED;
    if (!aligned16(w) || !aligned16(s)) return W4A16_ERR_ALIGNMENT;
    return W4A16_OK;
}

int check_linear(const void* x, const void* w, const void* s, const void* out, int64_t M,
                 int64_t N, int64_t K, int64_t g) {
    if (x == nullptr || out == nullptr) return W4A16_ERR_INVALID_ARG;
    if (M <= 0) return W4A16_ERR_INVALID_ARG;
    const int rc = check_weights(w, s, N, K, g);
    if (rc != W4A16_OK) return rc;
    if (M > kMaxDim) return W4A16_ERR_UNSUPPORTED;
    if (!aligned16(x) || !aligned16(out)) return W4A16_ERR_ALIGNMENT;
    const int64_t out_bytes = M * N * 2;
    if (overlaps(out, out_bytes, x, M * K * 2) || overlaps(out, out_bytes, w, N * (K / 2)) ||
        overlaps(out, out_bytes, s, N * (K / g) * 2))
        return W4A16_ERR_INVALID_ARG;
    // tile counts must fit the kernel's int arithmetic
    const int64_t tiles = ((M + 31) / 32) * ((N + 127) / 128);
    if (tiles > kMaxDim) return W4A16_ERR_UNSUPPORTED;
    return W4A16_OK;
}

Epilogue plain_epilogue(int64_t N) { return Epilogue{nullptr, nullptr, 0, static_cast<int>(N)}; }

// Arguments of w4a16_linear_fused beyond those of w4a16_linear.
int check_fused(const void* x, const void* w, const void* s, const void* bias,
                const void* residual, const void* out, int64_t M, int64_t N, int64_t K,
                int64_t g, int act) {
    if (act != W4A16_ACT_NONE && act != W4A16_ACT_SWIGLU && act != W4A16_ACT_GELU)
        return W4A16_ERR_INVALID_ARG;
    if (act == W4A16_ACT_SWIGLU && N % 2 != 0) return W4A16_ERR_INVALID_ARG;
    const int64_t n_out = act == W4A16_ACT_SWIGLU ? N / 2 : N;
    if (x == nullptr || out == nullptr) return W4A16_ERR_INVALID_ARG;
    if (M <= 0) return W4A16_ERR_INVALID_ARG;
    int rc = check_weights(w, s, N, K, g);
    if (rc != W4A16_OK) return rc;
    if (M > kMaxDim) return W4A16_ERR_UNSUPPORTED;
    if (!aligned16(x) || !aligned16(out)) return W4A16_ERR_ALIGNMENT;
    if ((bias != nullptr && !aligned16(bias)) || (residual != nullptr && !aligned16(residual)))
        return W4A16_ERR_ALIGNMENT;
    const int64_t out_bytes = M * n_out * 2;
    if (overlaps(out, out_bytes, x, M * K * 2) || overlaps(out, out_bytes, w, N * (K / 2)) ||
        overlaps(out, out_bytes, s, N * (K / g) * 2) ||
        (bias != nullptr && overlaps(out, out_bytes, bias, N * 2)))
        return W4A16_ERR_INVALID_ARG;
    // the residual is read where out is written: the same buffer, or disjoint
    if (residual != nullptr && residual != out && overlaps(out, out_bytes, residual, out_bytes))
        return W4A16_ERR_INVALID_ARG;
    const int64_t tiles = ((M + 31) / 32) * ((N + 127) / 128);
    if (tiles > kMaxDim) return W4A16_ERR_UNSUPPORTED;
    return W4A16_OK;
}

int encode_2d(CUtensorMap* map, CUtensorMapDataType dtype, const void* base, uint64_t inner,
              uint64_t outer, uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer,
              CUtensorMapSwizzle swz) {
    const cuuint64_t dims[2] = {inner, outer};
    const cuuint64_t strides[1] = {row_bytes};
    const cuuint32_t box[2] = {box_inner, box_outer};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = g_encode(map, dtype, 2, const_cast<void*>(base), dims, strides, box, estr,
                                CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS ? W4A16_OK : W4A16_ERR_CUDA;
}

// M <= 128 with g = 128: the streaming kernels (rows spread evenly over the
// SMs); the warp-level one takes at most 32 token columns.
int launch_gemv(const DeviceState& st, const void* x, const void* w, const void* s, void* out,
                int64_t M, int64_t N, int64_t K, int64_t g, const Epilogue& epi,
                cudaStream_t stream) {
    const bool tc = M > 32 || M >= g_small_m_tc_from;
    const int T = tc ? gemv_tc_tokens(M) : gemv_tokens_per_tile(M);
    const int RB = tc ? gemv_tc_rows_per_cta(N, st.sm_count) : gemv_rows_per_cta(N, st.sm_count);
    alignas(64) CUtensorMap tx;
    alignas(64) CUtensorMap tw;
    int rc = encode_2d(&tx, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, x, K, M, K * 2, 64, T,
                       CU_TENSOR_MAP_SWIZZLE_128B);
    if (rc != W4A16_OK) return rc;
    rc = encode_2d(&tw, CU_TENSOR_MAP_DATA_TYPE_UINT8, w, K / 2, N, K / 2, 64, RB / 2,
                   CU_TENSOR_MAP_SWIZZLE_64B);
    if (rc != W4A16_OK) return rc;
    GemvParams p;
    p.scales = static_cast<const uint16_t*>(s);
    p.out = static_cast<uint16_t*>(out);
    p.status = st.status;
    p.M = static_cast<int>(M);
    p.N = static_cast<int>(N);
    p.K = static_cast<int>(K);
    p.g = static_cast<int>(g);
    p.rows_per_cta = RB;
    p.num_chunks = static_cast<int>((N + RB - 1) / RB);
    p.nt = (RB + 127) / 128;
    p.epi = epi;
    p.wait_ns = wait_limit_ns();
    const cudaError_t e = tc ? gemv_tc_launch(&tx, &tw, p, st.sm_count, stream)
                             : gemv_launch(&tx, &tw, p, st.sm_count, stream);
    return e == cudaSuccess ? W4A16_OK : W4A16_ERR_CUDA;
}

// Validated arguments -> one kernel launch.
int launch_linear(const DeviceState& st, const void* x, const void* w, const void* s, void* out,
                  int64_t M, int64_t N, int64_t K, int64_t g, const Epilogue& epi,
                  cudaStream_t stream) {
    // up to 128 tokens the weights stream once per call on the streaming
    // tensor-core kernel (12288 x 49152: M = 64 103 us there against 212 on the
    // 256-token GEMM tiles, M = 128 141 against 214)
    if (M <= 128 && g == 128 && K % 128 == 0 && g_small_m_streaming)
        return launch_gemv(st, x, w, s, out, M, N, K, g, epi, stream);
    const TsVariant v = M <= 32                      ? TsVariant::kGemv32
                        : g_gemm_pair && (g_gemm_wide_from >= 0
                                              ? M >= g_gemm_wide_from
                                              : ts_prefer_wide(M, N, st.sm_count))
                            ? TsVariant::kGemmPairWide
                        : g_gemm_pair                ? TsVariant::kGemmPair
                                                     : TsVariant::kGemm256;
    const int T = ts_tokens_per_tile(v);
    alignas(64) CUtensorMap tx;
    alignas(64) CUtensorMap tw;
    int rc = encode_2d(&tx, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, x, K, M, K * 2, 64,
                       ts_x_box_tokens(v), CU_TENSOR_MAP_SWIZZLE_128B);
    if (rc != W4A16_OK) return rc;
    rc = encode_2d(&tw, CU_TENSOR_MAP_DATA_TYPE_UINT8, w, K / 2, N, K / 2, 32, 128,
                   CU_TENSOR_MAP_SWIZZLE_32B);
    if (rc != W4A16_OK) return rc;
    TsParams p;
    p.scales = static_cast<const uint16_t*>(s);
    p.out = static_cast<uint16_t*>(out);
    p.status = st.status;
    p.M = static_cast<int>(M);
    p.N = static_cast<int>(N);
    p.K = static_cast<int>(K);
    p.g = static_cast<int>(g);
    p.num_t_tiles = static_cast<int>((M + T - 1) / T);
    p.num_w_tiles = static_cast<int>((N + 127) / 128);
    p.num_tiles = p.num_t_tiles * p.num_w_tiles;
    p.group_t = v == TsVariant::kGemv32 ? 1 : v == TsVariant::kGemmPairWide ? g_group_t_wide : g_group_t;
    if (v != TsVariant::kGemv32 && g_group_bytes > 0) {
        const int64_t per_tile = static_cast<int64_t>(T) * K * 2;
        const int64_t gt = g_group_bytes / per_tile;
        p.group_t = static_cast<int>(gt < 1 ? 1 : gt > 64 ? 64 : gt);
    }
    p.epi = epi;
    p.wait_ns = wait_limit_ns();
    const int grid = ts_grid(v, p, st.sm_count);
    return ts_launch(v, &tx, &tw, p, grid, stream) == cudaSuccess ? W4A16_OK : W4A16_ERR_CUDA;
}

}  // namespace

uint64_t wait_limit_ns() { return g_wait_limit_ns.load(std::memory_order_relaxed); }

}  // namespace w4a16

using namespace w4a16;

extern "C" int w4a16_linear(const void* x_bf16, const void* w_packed_u8, const void* scales_bf16,
                            void* out_bf16, int64_t M, int64_t N, int64_t K, int64_t g,
                            void* stream) {
    int rc = check_linear(x_bf16, w_packed_u8, scales_bf16, out_bf16, M, N, K, g);
    if (rc != W4A16_OK) return rc;
    DeviceState* st = nullptr;
    rc = device_state(&st);
    if (rc != W4A16_OK) return rc;
    return launch_linear(*st, x_bf16, w_packed_u8, scales_bf16, out_bf16, M, N, K, g,
                         plain_epilogue(N), static_cast<cudaStream_t>(stream));
}

extern "C" int w4a16_linear_fused(const void* x_bf16, const void* w_packed_u8,
                                  const void* scales_bf16, const void* bias_bf16,
                                  const void* residual_bf16, void* out_bf16, int64_t M, int64_t N,
                                  int64_t K, int64_t g, int activation, void* stream) {
    int rc = check_fused(x_bf16, w_packed_u8, scales_bf16, bias_bf16, residual_bf16, out_bf16, M,
                         N, K, g, activation);
    if (rc != W4A16_OK) return rc;
    DeviceState* st = nullptr;
    rc = device_state(&st);
    if (rc != W4A16_OK) return rc;
    const Epilogue epi{static_cast<const uint16_t*>(bias_bf16),
                       static_cast<const uint16_t*>(residual_bf16), activation,
                       static_cast<int>(activation == W4A16_ACT_SWIGLU ? N / 2 : N)};
    return launch_linear(*st, x_bf16, w_packed_u8, scales_bf16, out_bf16, M, N, K, g, epi,
                         static_cast<cudaStream_t>(stream));
}

extern "C" int w4a16_linear_stack(const w4a16_layer* layers, int64_t n_layers, int64_t M,
                                  int64_t g, void* stream) {
    if (layers == nullptr || n_layers <= 0) return W4A16_ERR_INVALID_ARG;
    for (int64_t i = 0; i < n_layers; ++i) {
        const w4a16_layer& l = layers[i];
        const int rc = check_linear(l.x, l.w_packed, l.scales, l.out, M, l.N, l.K, g);
        if (rc != W4A16_OK) return rc;
    }
    DeviceState* st = nullptr;
    int rc = device_state(&st);
    if (rc != W4A16_OK) return rc;
    for (int64_t i = 0; i < n_layers; ++i) {
        const w4a16_layer& l = layers[i];
        rc = launch_linear(*st, l.x, l.w_packed, l.scales, l.out, M, l.N, l.K, g,
                           plain_epilogue(l.N), static_cast<cudaStream_t>(stream));
        if (rc != W4A16_OK) return rc;
    }
    return W4A16_OK;
}

// A captured layer stack: one CUDA graph of the stack's kernel launches.
struct w4a16_stack_graph {
    cudaGraphExec_t exec = nullptr;
    int device = 0;
};

extern "C" int w4a16_stack_graph_create(const w4a16_layer* layers, int64_t n_layers, int64_t M,
                                        int64_t g, w4a16_stack_graph** out) {
    if (out == nullptr) return W4A16_ERR_INVALID_ARG;
    *out = nullptr;
    if (layers == nullptr || n_layers <= 0) return W4A16_ERR_INVALID_ARG;
    for (int64_t i = 0; i < n_layers; ++i) {
        const w4a16_layer& l = layers[i];
        const int rc = check_linear(l.x, l.w_packed, l.scales, l.out, M, l.N, l.K, g);
        if (rc != W4A16_OK) return rc;
    }
    DeviceState* st = nullptr;
    int rc = device_state(&st);
    if (rc != W4A16_OK) return rc;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return W4A16_ERR_CUDA;
    cudaStream_t cs = nullptr;
    if (cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) != cudaSuccess) return W4A16_ERR_CUDA;
    cudaGraph_t graph = nullptr;
    cudaGraphExec_t exec = nullptr;
    rc = W4A16_OK;
    if (cudaStreamBeginCapture(cs, cudaStreamCaptureModeThreadLocal) != cudaSuccess) {
        rc = W4A16_ERR_CUDA;
    } else {
        for (int64_t i = 0; i < n_layers && rc == W4A16_OK; ++i) {
            const w4a16_layer& l = layers[i];
            rc = launch_linear(*st, l.x, l.w_packed, l.scales, l.out, M, l.N, l.K, g,
                               plain_epilogue(l.N), cs);
        }
        const cudaError_t e = cudaStreamEndCapture(cs, &graph);
        if (rc == W4A16_OK && e != cudaSuccess) rc = W4A16_ERR_CUDA;
    }
    if (rc == W4A16_OK && cudaGraphInstantiate(&exec, graph, 0) != cudaSuccess) rc = W4A16_ERR_CUDA;
    if (graph != nullptr) cudaGraphDestroy(graph);
    cudaStreamDestroy(cs);
    if (rc != W4A16_OK) {
        if (exec != nullptr) cudaGraphExecDestroy(exec);
        return rc;
    }
    w4a16_stack_graph* h = new (std::nothrow) w4a16_stack_graph;
    if (h == nullptr) {
        cudaGraphExecDestroy(exec);
        return W4A16_ERR_CUDA;
    }
    h->exec = exec;
    h->device = dev;
    *out = h;
    return W4A16_OK;
}

extern "C" int w4a16_stack_graph_launch(w4a16_stack_graph* graph, void* stream) {
    if (graph == nullptr || graph->exec == nullptr) return W4A16_ERR_INVALID_ARG;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev != graph->device) return W4A16_ERR_INVALID_ARG;
    return cudaGraphLaunch(graph->exec, static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? W4A16_OK
               : W4A16_ERR_CUDA;
}

extern "C" int w4a16_stack_graph_destroy(w4a16_stack_graph* graph) {
    if (graph == nullptr) return W4A16_ERR_INVALID_ARG;
    const cudaError_t e = graph->exec != nullptr ? cudaGraphExecDestroy(graph->exec) : cudaSuccess;
    delete graph;
    return e == cudaSuccess ? W4A16_OK : W4A16_ERR_CUDA;
}

extern "C" int w4a16_dequant(const void* w_packed_u8, const void* scales_bf16, void* w_bf16,
                             int64_t N, int64_t K, int64_t g, void* stream) {
    int rc = check_weights(w_packed_u8, scales_bf16, N, K, g);
    if (rc != W4A16_OK) return rc;
    if (w_bf16 == nullptr) return W4A16_ERR_INVALID_ARG;
    if (!aligned16(w_bf16)) return W4A16_ERR_ALIGNMENT;
    if (overlaps(w_bf16, N * K * 2, w_packed_u8, N * (K / 2)) ||
        overlaps(w_bf16, N * K * 2, scales_bf16, N * (K / g) * 2))
        return W4A16_ERR_INVALID_ARG;
    DeviceState* st = nullptr;
    rc = device_state(&st);
    if (rc != W4A16_OK) return rc;
    return launch_dequant(static_cast<const uint8_t*>(w_packed_u8),
                          static_cast<const uint16_t*>(scales_bf16),
                          static_cast<uint16_t*>(w_bf16), N, K, g,
                          static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? W4A16_OK
               : W4A16_ERR_CUDA;
}

extern "C" int w4a16_quantize(const void* w_f32, void* w_packed_u8, void* scales_bf16, int64_t N,
                              int64_t K, int64_t g, void* stream) {
    int rc = check_weights(w_packed_u8, scales_bf16, N, K, g);
    if (rc != W4A16_OK) return rc;
    if (w_f32 == nullptr) return W4A16_ERR_INVALID_ARG;
    if (!aligned16(w_f32)) return W4A16_ERR_ALIGNMENT;
    if (overlaps(w_f32, N * K * 4, w_packed_u8, N * (K / 2)) ||
        overlaps(w_f32, N * K * 4, scales_bf16, N * (K / g) * 2) ||
        overlaps(w_packed_u8, N * (K / 2), scales_bf16, N * (K / g) * 2))
        return W4A16_ERR_INVALID_ARG;
    DeviceState* st = nullptr;
    rc = device_state(&st);
    if (rc != W4A16_OK) return rc;
    return launch_quantize(static_cast<const float*>(w_f32), static_cast<uint8_t*>(w_packed_u8),
                           static_cast<uint16_t*>(scales_bf16), N, K, g,
                           static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? W4A16_OK
               : W4A16_ERR_CUDA;
}

extern "C" int w4a16_attention_prefill(const void* qkv_bf16, const void* seq_start_i32,
                                       int64_t nseq, int64_t M, int64_t H, int64_t d,
                                       int64_t window, void* out_bf16, void* stream) {
    if (qkv_bf16 == nullptr || seq_start_i32 == nullptr || out_bf16 == nullptr)
        return W4A16_ERR_INVALID_ARG;
    if (nseq <= 0 || M <= 0 || H <= 0 || d <= 0 || window <= 0) return W4A16_ERR_INVALID_ARG;
    if (d != attention_head_dim()) return W4A16_ERR_UNSUPPORTED;
    if (M > kMaxDim || nseq > kMaxDim / 2 || H > 65535 || 3 * H * d > kMaxDim)
        return W4A16_ERR_UNSUPPORTED;
    if (!aligned16(qkv_bf16) || !aligned16(seq_start_i32) || !aligned16(out_bf16))
        return W4A16_ERR_ALIGNMENT;
    const int64_t out_bytes = M * H * d * 2;
    if (overlaps(out_bf16, out_bytes, qkv_bf16, M * 3 * H * d * 2) ||
        overlaps(out_bf16, out_bytes, seq_start_i32, (nseq + 1) * 4))
        return W4A16_ERR_INVALID_ARG;
    DeviceState* st = nullptr;
    int rc = device_state(&st);
    if (rc != W4A16_OK) return rc;
    alignas(64) CUtensorMap tq;
    alignas(64) CUtensorMap tkv;
    rc = encode_2d(&tq, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, qkv_bf16, 3 * H * d, M, 3 * H * d * 2,
                   64, 128, CU_TENSOR_MAP_SWIZZLE_128B);
    if (rc != W4A16_OK) return rc;
    rc = encode_2d(&tkv, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, qkv_bf16, 3 * H * d, M, 3 * H * d * 2,
                   64, attention_key_block(), CU_TENSOR_MAP_SWIZZLE_128B);
    if (rc != W4A16_OK) return rc;
    AttnParams p;
    p.seq_start = static_cast<const int32_t*>(seq_start_i32);
    p.out = static_cast<uint16_t*>(out_bf16);
    p.status = st->status;
    p.M = static_cast<int>(M);
    p.H = static_cast<int>(H);
    p.nseq = static_cast<int>(nseq);
    p.window = window > kMaxDim ? static_cast<int>(kMaxDim) : static_cast<int>(window);
    p.scale = 1.0f / sqrtf(static_cast<float>(d));
    p.wait_ns = wait_limit_ns();
    return launch_attention_prefill(&tq, &tkv, p, static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? W4A16_OK
               : W4A16_ERR_CUDA;
}

extern "C" int w4a16_gather_rows(const void* src_bf16, int64_t src_rows, int64_t D,
                                 const void* index_i32, int64_t P, void* dst_bf16,
                                 void* stream) {
    if (src_bf16 == nullptr || index_i32 == nullptr || dst_bf16 == nullptr)
        return W4A16_ERR_INVALID_ARG;
    if (src_rows <= 0 || D <= 0 || P <= 0) return W4A16_ERR_INVALID_ARG;
    if (src_rows > kMaxDim || D > kMaxDim || P > kMaxDim) return W4A16_ERR_UNSUPPORTED;
    if (!aligned16(src_bf16) || !aligned16(index_i32) || !aligned16(dst_bf16))
        return W4A16_ERR_ALIGNMENT;
    if (overlaps(dst_bf16, P * D * 2, src_bf16, src_rows * D * 2) ||
        overlaps(dst_bf16, P * D * 2, index_i32, P * 4))
        return W4A16_ERR_INVALID_ARG;
    DeviceState* st = nullptr;
    const int rc = device_state(&st);
    if (rc != W4A16_OK) return rc;
    return launch_gather_rows(static_cast<const uint16_t*>(src_bf16), src_rows, D,
                              static_cast<const int32_t*>(index_i32), P,
                              static_cast<uint16_t*>(dst_bf16), st->status, st->sm_count,
                              static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? W4A16_OK
               : W4A16_ERR_CUDA;
}

extern "C" int w4a16_topk_smallest(const void* scores, int score_bits, int64_t n, int64_t k,
                                   void* out_index_i32, void* out_score_f32, void* stream) {
    if (scores == nullptr || out_index_i32 == nullptr || out_score_f32 == nullptr)
        return W4A16_ERR_INVALID_ARG;
    if (score_bits != 32 && score_bits != 16) return W4A16_ERR_INVALID_ARG;
    if (n <= 0 || k <= 0 || k > n) return W4A16_ERR_INVALID_ARG;
    if (k > kTopkMaxK || n > kMaxDim) return W4A16_ERR_UNSUPPORTED;
    if (!aligned16(scores) || !aligned16(out_index_i32) || !aligned16(out_score_f32))
        return W4A16_ERR_ALIGNMENT;
    const int64_t in_bytes = n * (score_bits / 8);
    if (overlaps(out_index_i32, k * 4, scores, in_bytes) ||
        overlaps(out_score_f32, k * 4, scores, in_bytes) ||
        overlaps(out_index_i32, k * 4, out_score_f32, k * 4))
        return W4A16_ERR_INVALID_ARG;
    DeviceState* st = nullptr;
    const int rc = device_state(&st);
    if (rc != W4A16_OK) return rc;
    return launch_topk_smallest(scores, score_bits == 16, n, static_cast<int>(k),
                                static_cast<int32_t*>(out_index_i32),
                                static_cast<float*>(out_score_f32),
                                static_cast<cudaStream_t>(stream)) == cudaSuccess
               ? W4A16_OK
               : W4A16_ERR_CUDA;
}

extern "C" int w4a16_get_device_error(void* stream) {
    DeviceState* st = nullptr;
    int rc = device_state(&st);
    if (rc != W4A16_OK) return rc;
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess)
        return W4A16_ERR_CUDA;
    int v = 0;
    const int zero = 0;
    if (cudaMemcpy(&v, st->status, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess ||
        cudaMemcpy(st->status, &zero, sizeof zero, cudaMemcpyHostToDevice) != cudaSuccess)
        return W4A16_ERR_CUDA;
    return v == 0 ? W4A16_OK : v;
}

extern "C" int w4a16_selftest_wait_timeout(int64_t limit_ns, void* stream) {
    if (limit_ns < 1000 || limit_ns > 1000000) return W4A16_ERR_INVALID_ARG;
    DeviceState* st = nullptr;
    const int rc = device_state(&st);
    if (rc != W4A16_OK) return rc;
    selftest_wait_kernel<<<1, 64, 0, static_cast<cudaStream_t>(stream)>>>(
        static_cast<uint64_t>(limit_ns));
    return cudaGetLastError() == cudaSuccess ? W4A16_OK : W4A16_ERR_CUDA;
}

extern "C" int w4a16_selftest_set_wait_limit(int64_t limit_ns) {
    if (limit_ns == 0) {
        g_wait_limit_ns.store(kWaitLimitNs);
        return W4A16_OK;
    }
    if (limit_ns < 0 || limit_ns > static_cast<int64_t>(kWaitLimitNs)) return W4A16_ERR_INVALID_ARG;
    g_wait_limit_ns.store(static_cast<uint64_t>(limit_ns));
    return W4A16_OK;
}

extern "C" const char* w4a16_status_string(int status) {
    switch (status) {
        case W4A16_OK: return "ok";
        case W4A16_ERR_INVALID_ARG: return "invalid argument";
        case W4A16_ERR_UNSUPPORTED: return "unsupported shape or group size";
        case W4A16_ERR_ALIGNMENT: return "pointer not 16-byte aligned";
        case W4A16_ERR_CUDA: return "CUDA error";
        case W4A16_ERR_TIMEOUT: return "kernel wait timed out";
        case W4A16_ERR_INDEX: return "index check failed (debug build)";
        default: return "unknown status";
    }
}

extern "C" int w4a16_version(void) { return 200; }
