// Backward of the message aggregation: the gradient with respect to the node
// features x of out = aggregate(x) (the paper stresses that every
// aggregation stays differentiable, Sections 2.1.2 and 3).  For a sum with
// edge weights w, out[t] = sum over edges e = (s -> t) of w_e x[s], so
//
//   grad_x[s] = sum over edges e = (s -> t) of w_e grad_out[t]
//
// -- the same aggregation over the transposed graph.  The caller builds the
// CSR grouped by SOURCE (the radix build keyed on row 0 of edge_index: rows
// are sources, col holds targets, perm the original edge ids); the sum then
// runs on the ordinary aggregation kernels:
//
//   sum    weights w_e                      (edge_weight[perm], or 1)
//   mean   weights w_e / in_degree(t)       (the forward divides by the count)
//   GCN    dinv[s] * dinv[t] on the fly, plus fill * dinv[s]^2 grad_out[s]:
//          the symmetric normalisation is its own transpose, so the GCN
//          kernel runs unchanged on the source-grouped CSR with the forward's
//          dinv
//
// Max: the forward with argmax records, per (t, f), the original id of the
// first edge (in original order) attaining the maximum; the backward gives
// w_e grad_out[t, f] to that edge's source only.  It walks the source-grouped
// CSR, so each grad_x[s, f] is a sum in a fixed order (no atomics, bitwise
// reproducible).
#include <math_constants.h>

#include "common.cuh"

namespace tfg {
namespace {

constexpr int kBwThreads = 256;
constexpr int kBwEdges = 4;   // edges whose rows the max-with-argmax kernel requests together

// w_src[k] = (edge_weight ? edge_weight[perm_src[k]] : 1) / (mean ? max(deg[col_src[k]], 1) : 1)
__global__ void transposed_weights(const int32_t *__restrict__ perm_src,
                                   const int32_t *__restrict__ col_src,
                                   const float *__restrict__ edge_weight,
                                   const int32_t *__restrict__ in_degree, int64_t e,
                                   float *__restrict__ w_src) {
    const int64_t k = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (k >= e) return;
    float w = edge_weight ? __ldg(edge_weight + __ldg(perm_src + k)) : 1.f;
    if (in_degree) w = w / static_cast<float>(max(__ldg(in_degree + __ldg(col_src + k)), 1));
    w_src[k] = w;
}

// Forward max with argmax: one warp per target row, each lane VEC adjacent
// features (VEC = 4 when the layout allows 8- or 16-byte loads, else 1),
// lanes striding over the row, edges in CSR (= original) order; a strictly
// larger value replaces the running maximum, so ties keep the first edge.
template <typename XT, int VEC>
__global__ void __launch_bounds__(kBwThreads)
max_argmax(const int32_t *__restrict__ rowptr, const int32_t *__restrict__ col,
           const int32_t *__restrict__ perm, const float *__restrict__ w, const XT *__restrict__ x,
           int64_t n, int64_t f, float *__restrict__ out, int32_t *__restrict__ argmax) {
    const int64_t warp = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
    const int lane = threadIdx.x & 31;
    for (int64_t t = warp; t < n; t += nwarps) {
        const int64_t beg = rowptr[t], end = col ? rowptr[t + 1] : rowptr[t];
        for (int64_t f0 = static_cast<int64_t>(lane) * VEC; f0 < f; f0 += 32 * VEC) {
            float best[VEC];
            int32_t arg[VEC];
#pragma unroll
            for (int q = 0; q < VEC; ++q) {
                best[q] = -CUDART_INF_F;
                arg[q] = -1;
            }
            // kBwEdges rows requested at once, then compared in edge order
            for (int64_t k0 = beg; k0 < end; k0 += kBwEdges) {
                float v[kBwEdges][VEC];
                int32_t e[kBwEdges];
                float wk[kBwEdges];
#pragma unroll
                for (int u = 0; u < kBwEdges; ++u) {
                    const int64_t k = k0 + u < end ? k0 + u : end - 1;   // tail repeats the last edge
                    const int64_t s = __ldg(col + k);
                    e[u] = __ldg(perm + k);
                    wk[u] = w ? __ldg(w + k) : 1.f;
                    VecLoad<XT, VEC>::load(x + s * f + f0, v[u]);
                }
#pragma unroll
                for (int u = 0; u < kBwEdges; ++u) {
                    if (k0 + u >= end) break;
#pragma unroll
                    for (int q = 0; q < VEC; ++q) {
                        const float m = w ? wk[u] * v[u][q] : v[u][q];
                        if (m > best[q] || arg[q] < 0) {
                            best[q] = m;
                            arg[q] = e[u];
                        }
                    }
                }
            }
#pragma unroll
            for (int q = 0; q < VEC; ++q) {
                out[t * f + f0 + q] = arg[q] < 0 ? 0.f : best[q];
                argmax[t * f + f0 + q] = arg[q];
            }
        }
    }
}

// grad_x[s, f] = sum over the out-edges e = (s -> t) of s, in original order,
// of w_e grad_out[t, f] where argmax[t, f] == e (w_e = 1 without weights).
// VEC adjacent features per lane.
template <int VEC>
__global__ void __launch_bounds__(kBwThreads)
max_backward(const int32_t *__restrict__ rowptr_src, const int32_t *__restrict__ col_src,
             const int32_t *__restrict__ perm_src, const int32_t *__restrict__ argmax,
             const float *__restrict__ edge_weight, const float *__restrict__ grad_out, int64_t n,
             int64_t f, float *__restrict__ grad_x) {
    const int64_t warp = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 5;
    const int lane = threadIdx.x & 31;
    for (int64_t s = warp; s < n; s += nwarps) {
        const int64_t beg = rowptr_src[s], end = col_src ? rowptr_src[s + 1] : rowptr_src[s];
        for (int64_t f0 = static_cast<int64_t>(lane) * VEC; f0 < f; f0 += 32 * VEC) {
            float acc[VEC];
#pragma unroll
            for (int q = 0; q < VEC; ++q) acc[q] = 0.f;
            for (int64_t k = beg; k < end; ++k) {
                const int64_t t = __ldg(col_src + k);
                const int32_t e = __ldg(perm_src + k);
                const float we = edge_weight ? __ldg(edge_weight + e) : 1.f;
                int32_t a[VEC];
                float g[VEC];
                if constexpr (VEC == 4) {
                    const int4 a4 = __ldg(reinterpret_cast<const int4 *>(argmax + t * f + f0));
                    const float4 g4 = __ldg(reinterpret_cast<const float4 *>(grad_out + t * f + f0));
                    a[0] = a4.x; a[1] = a4.y; a[2] = a4.z; a[3] = a4.w;
                    g[0] = g4.x; g[1] = g4.y; g[2] = g4.z; g[3] = g4.w;
                } else {
                    a[0] = __ldg(argmax + t * f + f0);
                    g[0] = __ldg(grad_out + t * f + f0);
                }
#pragma unroll
                for (int q = 0; q < VEC; ++q)
                    if (a[q] == e) acc[q] = fmaf(we, g[q], acc[q]);
            }
#pragma unroll
            for (int q = 0; q < VEC; ++q) grad_x[s * f + f0 + q] = acc[q];
        }
    }
}

bool aligned(const void *p, uintptr_t b) { return reinterpret_cast<uintptr_t>(p) % b == 0; }

int rows_grid(int64_t n) {
    const int64_t warps_per_block = kBwThreads / 32;
    const int64_t want = (n + warps_per_block - 1) / warps_per_block;
    const int64_t cap = int64_t(152) * 64;
    return static_cast<int>(want < 1 ? 1 : (want < cap ? want : cap));
}

}  // namespace

size_t backward_workspace_bytes(int mode, int64_t e) {
    if (mode != TFG_SUM && mode != TFG_MEAN) return 0;
    return (sizeof(float) * static_cast<size_t>(e) + 255) & ~size_t(255);
}

cudaError_t launch_aggregate_backward(int mode, const int32_t *rowptr_src, const int32_t *col_src,
                                      const int32_t *perm_src, const float *edge_weight,
                                      const int32_t *in_degree, const float *grad_out, int64_t n,
                                      int64_t e, int64_t f, float *grad_x, void *ws,
                                      cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    float *w_src = nullptr;
    if (e > 0 && (edge_weight || mode == TFG_MEAN)) {
        w_src = static_cast<float *>(ws);
        transposed_weights<<<ceil_div(e, 256), 256, 0, s>>>(
            perm_src, col_src, edge_weight, mode == TFG_MEAN ? in_degree : nullptr, e, w_src);
        const cudaError_t err = cudaGetLastError();
        if (err != cudaSuccess) return err;
    }
    return launch_aggregate(0, rowptr_src, e > 0 ? col_src : nullptr, w_src, nullptr, grad_out,
                            TFG_F32, n, f, 0, 0.f, grad_x, s);
}

cudaError_t launch_max_argmax(const int32_t *rowptr, const int32_t *col, const int32_t *perm,
                              const float *w, const void *x, int x_dtype, int64_t n, int64_t f,
                              float *out, int32_t *argmax, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const int grid = rows_grid(n);
    const bool v4 = f % 4 == 0 && aligned(out, 16) && aligned(argmax, 16) &&
                    aligned(x, x_dtype == TFG_BF16 ? 8 : 16);
    if (x_dtype == TFG_BF16) {
        const uint16_t *xp = static_cast<const uint16_t *>(x);
        if (v4) max_argmax<uint16_t, 4><<<grid, kBwThreads, 0, s>>>(rowptr, col, perm, w, xp, n, f, out, argmax);
        else max_argmax<uint16_t, 1><<<grid, kBwThreads, 0, s>>>(rowptr, col, perm, w, xp, n, f, out, argmax);
    } else {
        const float *xp = static_cast<const float *>(x);
        if (v4) max_argmax<float, 4><<<grid, kBwThreads, 0, s>>>(rowptr, col, perm, w, xp, n, f, out, argmax);
        else max_argmax<float, 1><<<grid, kBwThreads, 0, s>>>(rowptr, col, perm, w, xp, n, f, out, argmax);
    }
    return cudaGetLastError();
}

cudaError_t launch_max_backward(const int32_t *rowptr_src, const int32_t *col_src,
                                const int32_t *perm_src, const int32_t *argmax,
                                const float *edge_weight, const float *grad_out, int64_t n,
                                int64_t f, float *grad_x, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const bool v4 = f % 4 == 0 && aligned(argmax, 16) && aligned(grad_out, 16) && aligned(grad_x, 16);
    if (v4)
        max_backward<4><<<rows_grid(n), kBwThreads, 0, s>>>(rowptr_src, col_src, perm_src, argmax,
                                                            edge_weight, grad_out, n, f, grad_x);
    else
        max_backward<1><<<rows_grid(n), kBwThreads, 0, s>>>(rowptr_src, col_src, perm_src, argmax,
                                                            edge_weight, grad_out, n, f, grad_x);
    return cudaGetLastError();
}

}  // namespace tfg
