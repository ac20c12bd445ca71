// Scoring readout for sm_103a: the last two modules of the screening pipeline
// (Sec. 3.3) -- the affinity head reads one hidden state per pair, and the
// predicted affinities are sorted for export.
//
//   gather_rows   dst[p, :] = src[idx[p], :] (bf16 rows, 16-byte copies);
//   topk_smallest the k smallest scores (best binders: lowest free energy),
//                 ascending by IEEE totalOrder with NaN last, ties by index.
//
// Top-k, GB300-first: one thread-block cluster of 8 CTAs (1024 threads each)
// does a most-significant-digit-first radix select over order-preserving
// 32-bit keys.  Each CTA histograms one contiguous eighth of the scores; CTA 0
// sums the eight histograms through distributed shared memory and picks the
// digit, four passes of 8 bits.  The selected (key, index) pairs are then
// written straight into CTA 0's shared memory -- equal keys taken in index
// order by an ordered block scan -- and CTA 0 sorts them (bitonic) and stores
// the result.  Nothing goes through global scratch memory, and the cluster
// barriers are hardware barriers among co-scheduled CTAs.
#include "internal.h"

#include <cooperative_groups.h>
#include <cuda_runtime.h>
#include <cstdint>

namespace cg = cooperative_groups;

namespace w4a16 {

namespace {

constexpr int kTopkCtas = 8;
constexpr int kTopkThreads = 1024;
constexpr int kTopkWarps = kTopkThreads / 32;

// Keys whose unsigned order is totalOrder on the scores; every NaN maps to
// the largest key.
__device__ __forceinline__ uint32_t order_key_f32(float f) {
    const uint32_t u = __float_as_uint(f);
    if ((u & 0x7F800000u) == 0x7F800000u && (u & 0x007FFFFFu) != 0u) return 0xFFFFFFFFu;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

struct TopkShared {
    uint32_t hist[256];
    uint32_t total[256];
    uint32_t warp_sum[kTopkWarps];
    uint32_t round_total;                 // block total of the last block_rank
    uint32_t digit, need;                 // written by CTA 0 each pass
    uint32_t count_lt, count_eq;          // this CTA's
    uint32_t lt_off, eq_off, eq_take;     // written by CTA 0 for this CTA
    uint32_t lt_cursor;
    unsigned long long sel[kTopkMaxK];    // CTA 0: selected (key << 32 | index)
};

// Block-wide exclusive scan of one flag per thread, in thread order;
// returns this thread's position; the block total is left in *total (shared
// memory), valid for every thread on return.
__device__ __forceinline__ uint32_t block_rank(bool flag, uint32_t* warp_sum, uint32_t* total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t ballot = __ballot_sync(0xffffffffu, flag);
    const uint32_t in_warp = __popc(ballot & ((1u << lane) - 1u));
    if (lane == 0) warp_sum[warp] = __popc(ballot);
    __syncthreads();
    if (warp == 0) {
        const uint32_t v = lane < kTopkWarps ? warp_sum[lane] : 0u;
        uint32_t incl = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t t = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += t;
        }
        if (lane < kTopkWarps) warp_sum[lane] = incl - v;  // exclusive
        if (lane == 31) *total = incl;
    }
    __syncthreads();
    const uint32_t r = warp_sum[warp] + in_warp;
    __syncthreads();
    return r;
}

// Scores are fp32, or bf16 (widened exactly: its bits are the top half of
// the fp32's).
template <bool BF16>
__device__ __forceinline__ float score_at(const void* scores, int64_t i) {
    if constexpr (BF16)
        return __uint_as_float(static_cast<uint32_t>(static_cast<const uint16_t*>(scores)[i]) << 16);
    else
        return static_cast<const float*>(scores)[i];
}

template <bool BF16>
__device__ __forceinline__ uint32_t order_key(const void* scores, int64_t i) {
    return order_key_f32(score_at<BF16>(scores, i));
}

template <bool BF16>
__global__ void __cluster_dims__(kTopkCtas, 1, 1) __launch_bounds__(kTopkThreads, 1)
    topk_smallest_kernel(const void* __restrict__ scores, int64_t n, int k,
                         int32_t* __restrict__ out_idx, float* __restrict__ out_val) {
    __shared__ TopkShared sh;
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = static_cast<int>(cluster.block_rank());
    const int tid = threadIdx.x;
    TopkShared* root = cluster.map_shared_rank(&sh, 0);

    const int64_t lo = n * rank / kTopkCtas, hi = n * (rank + 1) / kTopkCtas;
    uint32_t prefix = 0, mask = 0, need = static_cast<uint32_t>(k);

    // ---- radix select: the k-th smallest key, four digits of 8 bits
    for (int pass = 0; pass < 4; ++pass) {
        const int shift = 24 - 8 * pass;
        if (tid < 256) sh.hist[tid] = 0;
        __syncthreads();
        for (int64_t i = lo + tid; i < hi; i += kTopkThreads) {
            const uint32_t key = order_key<BF16>(scores, i);
            if ((key & mask) == prefix) atomicAdd(&sh.hist[(key >> shift) & 255u], 1u);
        }
        cluster.sync();
        if (rank == 0) {
            if (tid < 256) {
                uint32_t s = 0;
                for (int r = 0; r < kTopkCtas; ++r) s += cluster.map_shared_rank(&sh, r)->hist[tid];
                sh.total[tid] = s;
            }
            __syncthreads();
            if (tid == 0) {
                uint32_t before = 0, d = 0;
                for (; d < 255; ++d) {
                    if (before + sh.total[d] >= need) break;
                    before += sh.total[d];
                }
                sh.digit = d;
                sh.need = need - before;
            }
        }
        cluster.sync();
        const uint32_t d = root->digit;
        need = root->need;
        prefix |= d << shift;
        mask |= 255u << shift;
    }
    const uint32_t thr = prefix;        // the k-th smallest key
    const uint32_t need_eq = need;      // how many keys equal to it are taken

    // ---- per-CTA counts of keys below and equal to the threshold
    uint32_t lt = 0, eq = 0;
    for (int64_t i = lo + tid; i < hi; i += kTopkThreads) {
        const uint32_t key = order_key<BF16>(scores, i);
        lt += key < thr;
        eq += key == thr;
    }
    lt = __reduce_add_sync(0xffffffffu, lt);
    eq = __reduce_add_sync(0xffffffffu, eq);
    if ((tid & 31) == 0) sh.warp_sum[tid >> 5] = lt;
    __syncthreads();
    if (tid == 0) {
        uint32_t s = 0;
        for (int w = 0; w < kTopkWarps; ++w) s += sh.warp_sum[w];
        sh.count_lt = s;
    }
    __syncthreads();
    if ((tid & 31) == 0) sh.warp_sum[tid >> 5] = eq;
    __syncthreads();
    if (tid == 0) {
        uint32_t s = 0;
        for (int w = 0; w < kTopkWarps; ++w) s += sh.warp_sum[w];
        sh.count_eq = s;
        sh.lt_cursor = 0;
    }
    cluster.sync();
    if (rank == 0 && tid == 0) {
        // keys below the threshold first (all of them), then the first
        // need_eq equal keys in index order (CTA slices are in index order)
        uint32_t lt_off = 0, eq_seen = 0, eq_off = static_cast<uint32_t>(k) - need_eq;
        for (int r = 0; r < kTopkCtas; ++r) {
            TopkShared* o = cluster.map_shared_rank(&sh, r);
            const uint32_t take = eq_seen >= need_eq ? 0u
                                  : (o->count_eq < need_eq - eq_seen ? o->count_eq
                                                                     : need_eq - eq_seen);
            o->lt_off = lt_off;
            o->eq_off = eq_off;
            o->eq_take = take;
            lt_off += o->count_lt;
            eq_seen += o->count_eq;
            eq_off += take;
        }
    }
    cluster.sync();

    // ---- write the selected (key, index) pairs into CTA 0's shared memory
    const uint32_t eq_take = sh.eq_take;
    uint32_t eq_base = 0;
    for (int64_t base = lo; base < hi; base += kTopkThreads) {
        const int64_t i = base + tid;
        const uint32_t key = i < hi ? order_key<BF16>(scores, i) : 0xFFFFFFFFu;
        const bool is_lt = i < hi && key < thr;
        const bool is_eq = i < hi && key == thr;
        if (is_lt) {
            const uint32_t pos = sh.lt_off + atomicAdd(&sh.lt_cursor, 1u);
            root->sel[pos] = (static_cast<unsigned long long>(key) << 32) | static_cast<uint32_t>(i);
        }
        const uint32_t r = block_rank(is_eq, sh.warp_sum, &sh.round_total);
        if (is_eq && eq_base + r < eq_take)
            root->sel[sh.eq_off + eq_base + r] =
                (static_cast<unsigned long long>(key) << 32) | static_cast<uint32_t>(i);
        eq_base += sh.round_total;
    }
    cluster.sync();

    // ---- CTA 0: sort the k pairs (bitonic over the next power of two) and store
    if (rank == 0) {
        int p2 = 1;
        while (p2 < k) p2 <<= 1;
        for (int j = k + tid; j < p2; j += kTopkThreads) sh.sel[j] = ~0ull;
        __syncthreads();
        for (int size = 2; size <= p2; size <<= 1) {
            for (int stride = size >> 1; stride > 0; stride >>= 1) {
                for (int j = tid; j < p2; j += kTopkThreads) {
                    const int partner = j ^ stride;
                    if (partner > j) {
                        const bool up = (j & size) == 0;
                        const unsigned long long a = sh.sel[j], b = sh.sel[partner];
                        if ((a > b) == up) {
                            sh.sel[j] = b;
                            sh.sel[partner] = a;
                        }
                    }
                }
                __syncthreads();
            }
        }
        for (int j = tid; j < k; j += kTopkThreads) {
            const uint32_t idx = static_cast<uint32_t>(sh.sel[j] & 0xFFFFFFFFull);
            out_idx[j] = static_cast<int32_t>(idx);
            out_val[j] = score_at<BF16>(scores, idx);
        }
    }
}

__global__ void gather_rows_kernel(const uint16_t* __restrict__ src, int64_t src_rows,
                                   int64_t D, const int32_t* __restrict__ idx, int64_t P,
                                   uint16_t* __restrict__ dst, int* status) {
    for (int64_t p = blockIdx.x; p < P; p += gridDim.x) {
        const int32_t r = idx[p];
        uint16_t* d = dst + p * D;
        if (r < 0 || r >= src_rows) {
            for (int64_t j = threadIdx.x; j < D; j += blockDim.x) d[j] = 0;
            if (threadIdx.x == 0) atomicCAS(status, 0, 1 /* W4A16_ERR_INVALID_ARG; the first error is kept */);
            continue;
        }
        const uint16_t* s = src + static_cast<int64_t>(r) * D;
        if ((D & 7) == 0) {  // rows of whole 16-byte chunks (bases are 16-byte aligned)
            const uint4* s4 = reinterpret_cast<const uint4*>(s);
            uint4* d4 = reinterpret_cast<uint4*>(d);
            for (int64_t j = threadIdx.x; j < D / 8; j += blockDim.x) d4[j] = s4[j];
        } else {
            for (int64_t j = threadIdx.x; j < D; j += blockDim.x) d[j] = s[j];
        }
    }
}

}  // namespace

cudaError_t launch_topk_smallest(const void* scores, bool bf16, int64_t n, int k,
                                 int32_t* out_idx, float* out_val, cudaStream_t stream) {
    if (bf16)
        topk_smallest_kernel<true><<<kTopkCtas, kTopkThreads, 0, stream>>>(scores, n, k, out_idx,
                                                                           out_val);
    else
        topk_smallest_kernel<false><<<kTopkCtas, kTopkThreads, 0, stream>>>(scores, n, k, out_idx,
                                                                            out_val);
    return cudaGetLastError();
}

cudaError_t launch_gather_rows(const uint16_t* src, int64_t src_rows, int64_t D,
                               const int32_t* idx, int64_t P, uint16_t* dst, int* status,
                               int sm_count, cudaStream_t stream) {
    const int64_t blocks = P < 4 * sm_count ? P : 4 * sm_count;
    gather_rows_kernel<<<static_cast<int>(blocks), 256, 0, stream>>>(src, src_rows, D, idx, P,
                                                                     dst, status);
    return cudaGetLastError();
}

}  // namespace w4a16
