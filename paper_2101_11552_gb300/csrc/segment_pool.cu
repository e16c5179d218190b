// Graph pooling keyed by node_graph_index: tf_geometric's common graph
// pooling (Fig. 2a) over a BatchGraph, whose reindexing (Section 2.1.1)
// leaves the nodes of each graph contiguous and the batch vector sorted.
// This is the sorted-key reduction the paper builds from tf.math.segment_*.
//
// One (graph, feature tile) is reduced by S CTAs forming a thread-block
// cluster (S = 1 for small graphs, up to 8 for large ones).  Each CTA finds
// the graph's node range by binary search on the sorted batch vector and
// takes one contiguous S-th of it; its 256 threads form 256 / LPR node groups
// striding over that part, and the group partials are combined in group
// order in shared memory.  CTA rank 0 of the cluster then reads the other
// CTAs' partials through distributed shared memory, in rank order, and
// writes the result.  The combination order is fixed, so results are
// deterministic, and no global scratch is needed.
#include <cooperative_groups.h>
#include <math_constants.h>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace tfg {
namespace {

constexpr int kPoolThreads = 256;
constexpr int kMaxCluster = 8;

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

// Reducer ids of the kernel: TFG_SUM, TFG_MEAN, TFG_MAX, and kMeanMax, which
// keeps a sum and a max per feature in one pass and writes [mean | max]
// (the Mean-Max Pool readout of Table 2).
constexpr int kMeanMax = 3;

// op of accumulator a (0 = the sum/mean/max itself; for kMeanMax 0 = sum, 1 = max)
template <int RED>
__device__ __forceinline__ float pool_op(int a, float x, float y) {
    const bool is_max = RED == TFG_MAX || (RED == kMeanMax && a == 1);
    return is_max ? fmaxf(x, y) : x + y;
}
template <int RED>
__device__ __forceinline__ float pool_init(int a) {
    const bool is_max = RED == TFG_MAX || (RED == kMeanMax && a == 1);
    return is_max ? -CUDART_INF_F : 0.f;
}
template <int RED>
__device__ __forceinline__ float pool_final(int a, float r, int64_t cnt) {
    if (cnt == 0) return 0.f;
    const bool is_mean = RED == TFG_MEAN || (RED == kMeanMax && a == 0);
    return is_mean ? r / static_cast<float>(cnt) : r;
}

// grid = (graphs, feature tiles, S); cluster = (1, 1, S) when S > 1.
// out is [G, NA * F]: accumulator a of feature f goes to column a * F + f.
template <typename XT, int VEC, int LPR, int RED, bool CLUSTER>
__global__ void __launch_bounds__(kPoolThreads)
pool_kernel(const XT *__restrict__ x, const int64_t *__restrict__ batch, int64_t n, int64_t f,
            float *__restrict__ out) {
    constexpr int NA = RED == kMeanMax ? 2 : 1;
    constexpr int kGroups = kPoolThreads / LPR;
    constexpr int kSlots = LPR * VEC;
    __shared__ int64_t s_range[2];
    __shared__ float s_part[NA][kGroups * kSlots];
    __shared__ float s_red[NA][kSlots];
    const int64_t gid = blockIdx.x;
    const int split = blockIdx.z, nsplit = gridDim.z;
    if (threadIdx.x == 0) s_range[0] = lower_bound(batch, n, gid);
    if (threadIdx.x == 32) s_range[1] = lower_bound(batch, n, gid + 1);
    __syncthreads();
    const int64_t beg = s_range[0], end = max(s_range[0], s_range[1]);
    const int64_t len = (end - beg + nsplit - 1) / nsplit;
    const int64_t pb = min(end, beg + split * len), pe = min(end, pb + len);
    const int grp = threadIdx.x / LPR, sub = threadIdx.x % LPR;
    const int64_t ft = static_cast<int64_t>(blockIdx.y) * kSlots;
    const int64_t f0 = ft + sub * VEC;
    const bool fok = f0 < f;
    float acc[NA][VEC];
#pragma unroll
    for (int a = 0; a < NA; ++a)
#pragma unroll
        for (int q = 0; q < VEC; ++q) acc[a][q] = pool_init<RED>(a);
    if (fok) {
        for (int64_t v = pb + grp; v < pe; v += kGroups) {
            float val[VEC];
            VecLoad<XT, VEC>::load(x + v * f + f0, val);
#pragma unroll
            for (int a = 0; a < NA; ++a)
#pragma unroll
                for (int q = 0; q < VEC; ++q) acc[a][q] = pool_op<RED>(a, acc[a][q], val[q]);
        }
    }
#pragma unroll
    for (int a = 0; a < NA; ++a)
#pragma unroll
        for (int q = 0; q < VEC; ++q) s_part[a][grp * kSlots + sub * VEC + q] = acc[a][q];
    __syncthreads();
    for (int i = threadIdx.x; i < kSlots; i += kPoolThreads) {
#pragma unroll
        for (int a = 0; a < NA; ++a) {
            float r = s_part[a][i];
            for (int k = 1; k < kGroups; ++k) r = pool_op<RED>(a, r, s_part[a][k * kSlots + i]);
            s_red[a][i] = r;
        }
    }
    const int64_t cnt = end - beg;
    const int64_t ostride = NA * f;
    if constexpr (CLUSTER) {
        cg::cluster_group cluster = cg::this_cluster();
        cluster.sync();   // every CTA's partial is in its shared memory
        if (cluster.block_rank() == 0) {
            for (int i = threadIdx.x; i < kSlots; i += kPoolThreads) {
                const int64_t fi = ft + i;
#pragma unroll
                for (int a = 0; a < NA; ++a) {
                    float r = s_red[a][i];
                    for (int q = 1; q < nsplit; ++q)
                        r = pool_op<RED>(a, r, cluster.map_shared_rank(&s_red[a][0], q)[i]);
                    if (fi < f) out[gid * ostride + a * f + fi] = pool_final<RED>(a, r, cnt);
                }
            }
        }
        cluster.sync();   // keep partials alive until rank 0 has read them
    } else {
        __syncthreads();
        for (int i = threadIdx.x; i < kSlots; i += kPoolThreads) {
            const int64_t fi = ft + i;
            if (fi >= f) continue;
#pragma unroll
            for (int a = 0; a < NA; ++a)
                out[gid * ostride + a * f + fi] = pool_final<RED>(a, s_red[a][i], cnt);
        }
    }
}

template <typename XT, int VEC, int LPR, int RED>
cudaError_t launch_split(const void *x, const int64_t *batch, int64_t n, int64_t g, int64_t f,
                         float *out, int nsplit, cudaStream_t s) {
    const XT *xp = static_cast<const XT *>(x);
    const dim3 grid(static_cast<unsigned>(g), ceil_div(f, int64_t(LPR) * VEC), nsplit);
    if (nsplit == 1) {
        pool_kernel<XT, VEC, LPR, RED, false><<<grid, kPoolThreads, 0, s>>>(xp, batch, n, f, out);
        return cudaGetLastError();
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = dim3(kPoolThreads);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 1;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = nsplit;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, pool_kernel<XT, VEC, LPR, RED, true>, xp, batch, n, f, out);
}

template <typename XT, int VEC, int RED>
cudaError_t launch_lpr(const void *x, const int64_t *batch, int64_t n, int64_t g, int64_t f,
                       float *out, int lpr, int nsplit, cudaStream_t s) {
    switch (lpr) {
        case 32: return launch_split<XT, VEC, 32, RED>(x, batch, n, g, f, out, nsplit, s);
        case 16: return launch_split<XT, VEC, 16, RED>(x, batch, n, g, f, out, nsplit, s);
        default: return launch_split<XT, VEC, 8, RED>(x, batch, n, g, f, out, nsplit, s);
    }
}

template <typename XT, int VEC>
cudaError_t launch_red(const void *x, const int64_t *batch, int64_t n, int64_t g, int64_t f,
                       int reduce, float *out, int lpr, int nsplit, cudaStream_t s) {
    switch (reduce) {
        case TFG_MEAN: return launch_lpr<XT, VEC, TFG_MEAN>(x, batch, n, g, f, out, lpr, nsplit, s);
        case TFG_MAX: return launch_lpr<XT, VEC, TFG_MAX>(x, batch, n, g, f, out, lpr, nsplit, s);
        case kMeanMax: return launch_lpr<XT, VEC, kMeanMax>(x, batch, n, g, f, out, lpr, nsplit, s);
        default: return launch_lpr<XT, VEC, TFG_SUM>(x, batch, n, g, f, out, lpr, nsplit, s);
    }
}

int lanes_for(int64_t chunks) { return chunks >= 32 ? 32 : (chunks > 8 ? 16 : 8); }

// CTAs per graph: one per ~1024 nodes of an average graph, at most a portable cluster.
int splits_for(int64_t n, int64_t g) {
    const int64_t avg = g > 0 ? n / g : 0;
    int64_t s = avg / 1024;
    return static_cast<int>(s < 1 ? 1 : (s > kMaxCluster ? kMaxCluster : s));
}

}  // namespace

cudaError_t launch_segment_pool(const void *x, int x_dtype, const int64_t *batch, int64_t n,
                                int64_t g, int64_t f, int reduce, float *out, int32_t *status,
                                cudaStream_t s) {
    cudaError_t err = cudaMemsetAsync(status, 0, sizeof(int32_t), s);
    if (err != cudaSuccess) return err;
    if (n > 0) check_batch<<<ceil_div(n, 256), 256, 0, s>>>(batch, n, g, status);
    err = cudaGetLastError();
    if (err != cudaSuccess || g <= 0) return err;
    const int nsplit = splits_for(n, g);
    const bool aligned = reinterpret_cast<uintptr_t>(x) % 16 == 0;
    if (x_dtype == TFG_BF16) {
        if (aligned && f % 8 == 0)
            return launch_red<uint16_t, 8>(x, batch, n, g, f, reduce, out, lanes_for(f / 8), nsplit, s);
        return launch_red<uint16_t, 1>(x, batch, n, g, f, reduce, out, lanes_for(f), nsplit, s);
    }
    if (aligned && f % 4 == 0)
        return launch_red<float, 4>(x, batch, n, g, f, reduce, out, lanes_for(f / 4), nsplit, s);
    return launch_red<float, 1>(x, batch, n, g, f, reduce, out, lanes_for(f), nsplit, s);
}

}  // namespace tfg
