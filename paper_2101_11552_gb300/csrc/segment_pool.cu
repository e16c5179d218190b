// Graph pooling keyed by node_graph_index: tf_geometric's common graph
// pooling (Fig. 2a) over a BatchGraph, whose reindexing (Section 2.1.1)
// leaves the nodes of each graph contiguous and the batch vector sorted.
// This is the sorted-key reduction the paper builds from tf.math.segment_*.
//
// A CTA owns one (graph, feature tile).  It finds the graph's node range by
// binary search on the sorted batch vector, its 256 threads form
// 256 / LPR node groups that stride over the range, and the group partials
// are combined in group order through shared memory (deterministic).
#include <math_constants.h>

#include "common.cuh"

namespace tfg {
namespace {

constexpr int kPoolThreads = 256;

__global__ void check_batch(const int64_t *__restrict__ batch, int64_t n, int64_t g,
                            int32_t *status) {
    const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= n) return;
    const int64_t b = batch[i];
    if (b < 0 || b >= g) set_status(status, TFG_ERR_INDEX_RANGE);
    else if (i + 1 < n && batch[i + 1] < b) set_status(status, TFG_ERR_UNSORTED);
}

__device__ __forceinline__ int64_t lower_bound(const int64_t *batch, int64_t n, int64_t key) {
    int64_t lo = 0, hi = n;
    while (lo < hi) {
        const int64_t mid = (lo + hi) >> 1;
        if (__ldg(batch + mid) < key) lo = mid + 1;
        else hi = mid;
    }
    return lo;
}

template <typename XT, int VEC, int LPR, int RED>
__global__ void __launch_bounds__(kPoolThreads)
pool_kernel(const XT *__restrict__ x, const int64_t *__restrict__ batch, int64_t n, int64_t f,
            float *__restrict__ out) {
    constexpr int kGroups = kPoolThreads / LPR;
    constexpr int kSlots = LPR * VEC;
    __shared__ int64_t s_range[2];
    __shared__ float s_part[kGroups * kSlots];
    const int64_t gid = blockIdx.x;
    if (threadIdx.x == 0) s_range[0] = lower_bound(batch, n, gid);
    if (threadIdx.x == 32) s_range[1] = lower_bound(batch, n, gid + 1);
    __syncthreads();
    const int64_t beg = s_range[0], end = max(s_range[0], s_range[1]);
    const int grp = threadIdx.x / LPR, sub = threadIdx.x % LPR;
    const int64_t ft = static_cast<int64_t>(blockIdx.y) * kSlots;
    const int64_t f0 = ft + sub * VEC;
    const bool fok = f0 < f;
    float acc[VEC];
#pragma unroll
    for (int q = 0; q < VEC; ++q) acc[q] = RED == TFG_MAX ? -CUDART_INF_F : 0.f;
    if (fok) {
        for (int64_t v = beg + grp; v < end; v += kGroups) {
            float val[VEC];
            VecLoad<XT, VEC>::load(x + v * f + f0, val);
#pragma unroll
            for (int q = 0; q < VEC; ++q) acc[q] = RED == TFG_MAX ? fmaxf(acc[q], val[q]) : acc[q] + val[q];
        }
    }
#pragma unroll
    for (int q = 0; q < VEC; ++q) s_part[grp * kSlots + sub * VEC + q] = acc[q];
    __syncthreads();
    for (int i = threadIdx.x; i < kSlots; i += kPoolThreads) {
        const int64_t fi = ft + i;
        if (fi >= f) continue;
        float r = s_part[i];
        for (int k = 1; k < kGroups; ++k)
            r = RED == TFG_MAX ? fmaxf(r, s_part[k * kSlots + i]) : r + s_part[k * kSlots + i];
        const int64_t cnt = end - beg;
        if (cnt == 0) r = 0.f;
        else if (RED == TFG_MEAN) r = r / static_cast<float>(cnt);
        out[gid * f + fi] = r;
    }
}

template <typename XT, int VEC, int RED>
void launch_lpr(const void *x, const int64_t *batch, int64_t n, int64_t g, int64_t f, float *out,
                int lpr, cudaStream_t s) {
    const dim3 grid(static_cast<unsigned>(g), ceil_div(f, int64_t(lpr) * VEC));
    const XT *xp = static_cast<const XT *>(x);
    switch (lpr) {
        case 32: pool_kernel<XT, VEC, 32, RED><<<grid, kPoolThreads, 0, s>>>(xp, batch, n, f, out); break;
        case 16: pool_kernel<XT, VEC, 16, RED><<<grid, kPoolThreads, 0, s>>>(xp, batch, n, f, out); break;
        default: pool_kernel<XT, VEC, 8, RED><<<grid, kPoolThreads, 0, s>>>(xp, batch, n, f, out); break;
    }
}

template <typename XT, int VEC>
void launch_red(const void *x, const int64_t *batch, int64_t n, int64_t g, int64_t f, int reduce,
                float *out, int lpr, cudaStream_t s) {
    switch (reduce) {
        case TFG_MEAN: launch_lpr<XT, VEC, TFG_MEAN>(x, batch, n, g, f, out, lpr, s); break;
        case TFG_MAX: launch_lpr<XT, VEC, TFG_MAX>(x, batch, n, g, f, out, lpr, s); break;
        default: launch_lpr<XT, VEC, TFG_SUM>(x, batch, n, g, f, out, lpr, s); break;
    }
}

int lanes_for(int64_t chunks) { return chunks >= 32 ? 32 : (chunks > 8 ? 16 : 8); }

}  // namespace

cudaError_t launch_segment_pool(const void *x, int x_dtype, const int64_t *batch, int64_t n,
                                int64_t g, int64_t f, int reduce, float *out, int32_t *status,
                                cudaStream_t s) {
    cudaError_t err = cudaMemsetAsync(status, 0, sizeof(int32_t), s);
    if (err != cudaSuccess) return err;
    if (n > 0) check_batch<<<ceil_div(n, 256), 256, 0, s>>>(batch, n, g, status);
    if (g <= 0) return cudaGetLastError();
    const bool aligned = reinterpret_cast<uintptr_t>(x) % 16 == 0;
    if (x_dtype == TFG_BF16) {
        if (aligned && f % 8 == 0) launch_red<uint16_t, 8>(x, batch, n, g, f, reduce, out, lanes_for(f / 8), s);
        else launch_red<uint16_t, 1>(x, batch, n, g, f, reduce, out, lanes_for(f), s);
    } else {
        if (aligned && f % 4 == 0) launch_red<float, 4>(x, batch, n, g, f, reduce, out, lanes_for(f / 4), s);
        else launch_red<float, 1>(x, batch, n, g, f, reduce, out, lanes_for(f), s);
    }
    return cudaGetLastError();
}

}  // namespace tfg
