// Multi-hop propagation with the GCN-normalised adjacency: the APPNP model
// (Klicpera et al.) and its alpha = 0 special case SGC (Wu et al.), two of the
// node-level models tf_geometric provides (Section 2.2, Table 1):
//
//   h_0 = x0,   h_{k+1} = (1 - alpha) * Ahat h_k + alpha * x0,   out = h_K
//
// with Ahat = D^-1/2 (A + fill I) D^-1/2, its weights formed on the fly from
// dinv (or read from w_csr), exactly as in the one-hop GCN aggregation.
//
// Hop k is one launch of the GCN-mode aggregation kernel (agg.cuh) with the
// teleport term fused into its epilogue, so a hop reads the edge list, the
// gathered rows of h_k and the row of x0, and writes h_{k+1} once.  The hops
// need every row of h_k before any row of h_{k+1} can start, so each is its
// own launch (stream order is the barrier).  They alternate between out and
// one fp32 workspace buffer [N, F], arranged so that the last hop lands in
// out; hop 0 reads x0 in its storage type, later hops read fp32 iterates.
// K = 0 widens x0 into out.
#include "agg.cuh"

namespace tfg {
namespace {

template <typename XT>
__global__ void widen_kernel(const XT *__restrict__ x, int64_t count, float *__restrict__ out) {
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < count;
         i += stride) {
        float v[1];
        VecLoad<XT, 1>::load(x + i, v);
        out[i] = v[0];
    }
}

bool aligned_to(const void *p, uintptr_t b) { return reinterpret_cast<uintptr_t>(p) % b == 0; }

// One hop.  x = h_k (x0 itself for k = 0), a.out = h_{k+1}.
template <typename X0T>
cudaError_t launch_hop(AggArgs a, bool first, cudaStream_t s) {
    const int64_t f = a.f;
    const bool out16 = aligned_to(a.out, 16);
    if (first) {   // h_0 = x0: the gathered rows and the teleport rows share one type
        if constexpr (sizeof(X0T) == 2) {
            if (out16 && aligned_to(a.x, 16) && f % 8 == 0)
                return launch_lpr<X0T, 8, kAppnp, X0T>(a, lanes_per_row(f / 8), s);
            return launch_lpr<X0T, 1, kAppnp, X0T>(a, lanes_per_row(f), s);
        } else {
            if (out16 && aligned_to(a.x, 16) && f % 4 == 0)
                return launch_lpr<float, 4, kAppnp, float>(a, lanes_per_row(f / 4), s);
            return launch_lpr<float, 1, kAppnp, float>(a, lanes_per_row(f), s);
        }
    }
    // fp32 iterate; x0 rows are read 4 at a time (16 bytes fp32, 8 bytes bf16)
    if (out16 && aligned_to(a.x, 16) && f % 4 == 0 && aligned_to(a.x0, 4 * sizeof(X0T)))
        return launch_lpr<float, 4, kAppnp, X0T>(a, lanes_per_row(f / 4), s);
    return launch_lpr<float, 1, kAppnp, X0T>(a, lanes_per_row(f), s);
}

}  // namespace

size_t propagate_workspace_bytes(int64_t n, int64_t f, int64_t hops) {
    if (hops < 2 || n <= 0) return 0;
    return (sizeof(float) * static_cast<size_t>(n) * static_cast<size_t>(f) + 255) & ~size_t(255);
}

cudaError_t launch_propagate(const int32_t *rowptr, const int32_t *col, const float *w,
                             const float *dinv, const void *x0, int x_dtype, int64_t n, int64_t f,
                             int64_t hops, float alpha, int add_self, float fill, float *out,
                             void *ws, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    if (hops == 0) {
        const int64_t count = n * f;
        const int grid = static_cast<int>(min64((count + 255) / 256, int64_t(152) * 32));
        if (x_dtype == TFG_BF16)
            widen_kernel<uint16_t><<<grid, 256, 0, s>>>(static_cast<const uint16_t *>(x0), count, out);
        else
            widen_kernel<float><<<grid, 256, 0, s>>>(static_cast<const float *>(x0), count, out);
        return cudaGetLastError();
    }
    const float beta = static_cast<float>(1.0 - static_cast<double>(alpha));
    float *spare = static_cast<float *>(ws);
    const void *h = x0;
    for (int64_t k = 0; k < hops; ++k) {
        float *dst = ((hops - 1 - k) % 2 == 0) ? out : spare;
        AggArgs a{rowptr, col, w, dinv, h, dst, n, f, 0, add_self, fill, x0, alpha, beta, kRegimeAny};
        const cudaError_t err = x_dtype == TFG_BF16 ? launch_hop<uint16_t>(a, k == 0, s)
                                                    : launch_hop<float>(a, k == 0, s);
        if (err != cudaSuccess) return err;
        h = dst;
    }
    return cudaSuccess;
}

}  // namespace tfg
