// BatchGraph construction on the device: tf_geometric's reindexing trick
// (Section 2.1.1, Fig. 4).  The j-th node of graph g becomes node
// offset[g] + j, offset[g] being the number of nodes in all earlier graphs;
// the graphs' edge lists, stacked in graph order, are shifted by their
// graph's offset; node_graph_index (the batch vector) is g for every node of
// graph g.  Graph g's edges are found from the prefix sums of the per-graph
// edge counts.
//
//   scan_counts    node_offsets = exclusive scan of node_counts (G + 1 entries,
//                  the last one the total), edge_offsets likewise
//   reindex_edges  one thread per edge: g by binary search in edge_offsets,
//                  local ids checked against node_counts[g], shifted
//   fill_batch     one thread per node: g by binary search in node_offsets
#include "common.cuh"

namespace tfg {
namespace {

constexpr int kScanT = 1024;

// One CTA scans both count arrays (G values each, in chunks of 1024 with a
// carry).  The totals are checked against the sizes the caller declared.
__global__ void __launch_bounds__(kScanT)
scan_counts(const int64_t *__restrict__ node_counts, const int64_t *__restrict__ edge_counts,
            int64_t g, int64_t total_nodes, int64_t total_edges, int64_t *__restrict__ node_off,
            int64_t *__restrict__ edge_off, int32_t *status) {
    __shared__ int64_t s_w[2][kScanT / 32];
    __shared__ int64_t s_carry[2];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) s_carry[0] = s_carry[1] = 0;
    __syncthreads();
    for (int64_t base = 0; base < g; base += kScanT) {
        const int64_t k = base + threadIdx.x;
        int64_t v[2] = {0, 0};
        if (k < g) {
            v[0] = node_counts[k];
            v[1] = edge_counts[k];
            if (v[0] < 0 || v[1] < 0) set_status(status, TFG_ERR_INDEX_RANGE);
            v[0] = max(v[0], int64_t(0));
            v[1] = max(v[1], int64_t(0));
        }
        int64_t incl[2] = {v[0], v[1]};
#pragma unroll
        for (int a = 0; a < 2; ++a) {
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int64_t y = __shfl_up_sync(kFull, incl[a], o);
                if (lane >= o) incl[a] += y;
            }
            if (lane == 31) s_w[a][warp] = incl[a];
        }
        __syncthreads();
        if (warp == 0) {
#pragma unroll
            for (int a = 0; a < 2; ++a) {
                const int64_t s = s_w[a][lane];
                int64_t si = s;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const int64_t y = __shfl_up_sync(kFull, si, o);
                    if (lane >= o) si += y;
                }
                s_w[a][lane] = si - s;
            }
        }
        __syncthreads();
        if (k < g) {
            node_off[k] = s_carry[0] + s_w[0][warp] + incl[0] - v[0];
            edge_off[k] = s_carry[1] + s_w[1][warp] + incl[1] - v[1];
        }
        __syncthreads();
        if (threadIdx.x == kScanT - 1) {
            s_carry[0] += s_w[0][warp] + incl[0];
            s_carry[1] += s_w[1][warp] + incl[1];
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        node_off[g] = s_carry[0];
        edge_off[g] = s_carry[1];
        if (s_carry[0] != total_nodes || s_carry[1] != total_edges)
            set_status(status, TFG_ERR_INDEX_RANGE);
    }
}

// Last g in [0, G) with off[g] <= v (off non-decreasing, off[0] = 0).
__device__ __forceinline__ int64_t owner(const int64_t *off, int64_t g, int64_t v) {
    int64_t lo = 0, hi = g;   // answer in [0, g - 1]
    while (hi - lo > 1) {
        const int64_t mid = (lo + hi) >> 1;
        if (__ldg(off + mid) <= v) lo = mid;
        else hi = mid;
    }
    return lo;
}

__global__ void reindex_edges(const int64_t *__restrict__ edge_index, int64_t e, int64_t g,
                              const int64_t *__restrict__ node_off,
                              const int64_t *__restrict__ edge_off,
                              int64_t *__restrict__ out, int32_t *status) {
    const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= e) return;
    const int64_t gi = owner(edge_off, g, i);
    const int64_t base = __ldg(node_off + gi), count = __ldg(node_off + gi + 1) - base;
    int64_t s = edge_index[i], d = edge_index[e + i];
    if (s < 0 || s >= count || d < 0 || d >= count) {
        set_status(status, TFG_ERR_INDEX_RANGE);
        s = 0;
        d = 0;
    }
    out[i] = base + s;
    out[e + i] = base + d;
}

__global__ void fill_batch(int64_t n, int64_t g, const int64_t *__restrict__ node_off,
                           int64_t *__restrict__ batch) {
    const int64_t v = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (v < n) batch[v] = owner(node_off, g, v);
}

}  // namespace

size_t batch_graphs_workspace_bytes(int64_t g) {
    return ((sizeof(int64_t) * size_t(g + 1)) + 255) & ~size_t(255);
}

cudaError_t launch_batch_graphs(int64_t g, const int64_t *node_counts, const int64_t *edge_counts,
                                const int64_t *edge_index, int64_t e, int64_t n,
                                int64_t *out_edge_index, int64_t *batch, int64_t *node_offsets,
                                void *ws, int32_t *status, cudaStream_t s) {
    cudaError_t err = cudaMemsetAsync(status, 0, sizeof(int32_t), s);
    if (err != cudaSuccess) return err;
    int64_t *edge_off = static_cast<int64_t *>(ws);
    scan_counts<<<1, kScanT, 0, s>>>(node_counts, edge_counts, g, n, e, node_offsets, edge_off,
                                     status);
    if (e > 0)
        reindex_edges<<<ceil_div(e, 256), 256, 0, s>>>(edge_index, e, g, node_offsets, edge_off,
                                                       out_edge_index, status);
    if (n > 0) fill_batch<<<ceil_div(n, 256), 256, 0, s>>>(n, g, node_offsets, batch);
    return cudaGetLastError();
}

}  // namespace tfg
