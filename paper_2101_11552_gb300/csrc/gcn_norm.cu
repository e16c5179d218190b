// GCN symmetric normalisation of A + I (the GCN propagation rule that
// tf_geometric implements, Section 2.2; cached per graph, Section 3):
//   deg[t] = sum of the weights of the edges into t (+ fill for the implicit
//   self-loop), dinv[t] = deg[t]^-1/2 (0 when deg[t] == 0),
//   w_csr[k] = w_e * dinv[src] * dinv[t] for CSR position k of row t.
#include "common.cuh"

namespace tfg {
namespace {

constexpr int kNormThreads = 256;

__device__ __forceinline__ float inv_sqrt_or_zero(float d) {
    return d > 0.f ? 1.0f / sqrtf(d) : 0.f;  // IEEE sqrt and divide
}

// Unweighted: the degree is the row length (an integer, exact in fp32).
__global__ void dinv_unweighted(const int32_t *__restrict__ rowptr, int64_t n, int add_self,
                                float fill, float *__restrict__ dinv) {
    const int64_t t = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (t >= n) return;
    const float deg = static_cast<float>(rowptr[t + 1] - rowptr[t]) + (add_self ? fill : 0.f);
    dinv[t] = inv_sqrt_or_zero(deg);
}

// Weighted: one warp per row sums the weights in a fixed order (lane-strided
// partial sums, then a butterfly), so the result is deterministic.
__global__ void dinv_weighted(const int32_t *__restrict__ rowptr, const int32_t *__restrict__ perm,
                              const float *__restrict__ ew, int64_t n, int add_self, float fill,
                              float *__restrict__ dinv) {
    const int64_t t = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (t >= n) return;
    float s = 0.f;
    for (int64_t k = rowptr[t] + lane; k < rowptr[t + 1]; k += 32) s += __ldg(ew + perm[k]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(kFull, s, o);
    if (lane == 0) dinv[t] = inv_sqrt_or_zero(s + (add_self ? fill : 0.f));
}

__global__ void edge_weights(const int32_t *__restrict__ rowptr, const int32_t *__restrict__ col,
                             const int32_t *__restrict__ perm, const float *__restrict__ ew,
                             const float *__restrict__ dinv, int64_t n, float *__restrict__ w_csr) {
    const int64_t t = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (t >= n) return;
    const float dt = dinv[t];
    for (int64_t k = rowptr[t] + lane; k < rowptr[t + 1]; k += 32) {
        const float w = ew ? __ldg(ew + perm[k]) : 1.f;
        w_csr[k] = (w * __ldg(dinv + col[k])) * dt;
    }
}

}  // namespace

cudaError_t launch_gcn_norm(const int32_t *rowptr, const int32_t *col, const int32_t *perm,
                            const float *ew, int64_t n, int add_self, float fill, float *dinv,
                            float *w_csr, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    if (ew)
        dinv_weighted<<<ceil_div(n * 32, kNormThreads), kNormThreads, 0, s>>>(rowptr, perm, ew, n,
                                                                              add_self, fill, dinv);
    else
        dinv_unweighted<<<ceil_div(n, kNormThreads), kNormThreads, 0, s>>>(rowptr, n, add_self,
                                                                          fill, dinv);
    if (w_csr)
        edge_weights<<<ceil_div(n * 32, kNormThreads), kNormThreads, 0, s>>>(rowptr, col, perm, ew,
                                                                             dinv, n, w_csr);
    return cudaGetLastError();
}

}  // namespace tfg
