// Edge-softmax (GAT) aggregation: the map-reduce workflow of tf_geometric
// Fig. 5a (Section 2.1.2) fused with the attention-weighted sum it feeds.
//
//   node scores  s_src[n,h] = <x[n,h,:], a_src[h,:]>, s_dst likewise  (prologue)
//   map          l = LeakyReLU(s_src[src,h] + s_dst[t,h])
//   reduce       m = max over row t of l; den = sum over row t of exp(l - m)
//   map          alpha = exp(l - m) / den
//   aggregate    out[t,h,:] = sum over row t of alpha * x[src,h,:]
//
// One warp owns a target row; lane L covers features f0 = 32*VEC*tile +
// L*VEC (all of them inside head f0 / C).  Pass 1 finds the row maximum of
// each head, pass 2 accumulates exp(l - m) and exp(l - m) * x in fp32, and
// the result is divided by the denominator once.  With alpha requested a
// third pass writes the normalised weights.  Every lane of a head computes
// the same logits from the same inputs in the same order, so the values are
// consistent across lanes and deterministic.
#include <math_constants.h>

#include "common.cuh"

namespace tfg {
namespace {

constexpr int kSmThreads = 256;
constexpr int kSmUnroll = 4;

__global__ void node_scores(const float *__restrict__ x, int64_t n, int heads, int channels,
                            const float *__restrict__ a_src, const float *__restrict__ a_dst,
                            float *__restrict__ s_src, float *__restrict__ s_dst) {
    const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= n * heads) return;
    const int64_t v = i / heads;
    const int h = static_cast<int>(i % heads);
    const float *xr = x + v * heads * channels + static_cast<int64_t>(h) * channels;
    const float *as = a_src + h * channels, *ad = a_dst + h * channels;
    float a = 0.f, b = 0.f;
    for (int c = 0; c < channels; ++c) {
        const float xv = __ldg(xr + c);
        a = fmaf(xv, __ldg(as + c), a);
        b = fmaf(xv, __ldg(ad + c), b);
    }
    s_src[i] = a;
    s_dst[i] = b;
}

__device__ __forceinline__ float leaky(float v, float slope) { return v > 0.f ? v : slope * v; }

template <int VEC>
__global__ void __launch_bounds__(kSmThreads)
softmax_aggregate(const int32_t *__restrict__ rowptr, const int32_t *__restrict__ col,
                  const float *__restrict__ x, int64_t n, int heads, int channels, float slope,
                  const float *__restrict__ s_src, const float *__restrict__ s_dst,
                  float *__restrict__ out, float *__restrict__ alpha) {
    const int64_t t = (static_cast<int64_t>(blockIdx.x) * kSmThreads + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (t >= n) return;
    const int64_t f = static_cast<int64_t>(heads) * channels;
    const int64_t beg = rowptr[t], end = rowptr[t + 1];
    for (int64_t ft = 0; ft < f; ft += 32 * VEC) {
        const int64_t f0 = ft + lane * VEC;
        const bool fok = f0 < f;
        const int h = fok ? static_cast<int>(f0 / channels) : 0;
        const float sd = __ldg(s_dst + t * heads + h);

        // pass 1: per-head maximum of the logits of this row
        float m = -CUDART_INF_F;
        for (int64_t base = beg; base < end; base += 32) {
            const int cnt = static_cast<int>(min64(32, end - base));
            const int c = lane < cnt ? __ldg(col + base + lane) : 0;
            for (int j = 0; j < cnt; ++j) {
                const int src = __shfl_sync(kFull, c, j);
                m = fmaxf(m, leaky(__ldg(s_src + static_cast<int64_t>(src) * heads + h) + sd, slope));
            }
        }

        // pass 2: denominator and exp-weighted feature sum, blocked in two
        // levels (32-edge chunk, 32 chunks, total) to keep fp32 chains short
        float den = 0.f, den_sup = 0.f;
        float acc[VEC], sup[VEC], part[VEC];
#pragma unroll
        for (int q = 0; q < VEC; ++q) acc[q] = sup[q] = 0.f;
        int chunks = 0;
        for (int64_t base = beg; base < end; base += 32) {
            const int cnt = static_cast<int>(min64(32, end - base));
            const int c = lane < cnt ? __ldg(col + base + lane) : 0;
            float den_part = 0.f;
#pragma unroll
            for (int q = 0; q < VEC; ++q) part[q] = 0.f;
            for (int j = 0; j < cnt; j += kSmUnroll) {
                int src[kSmUnroll];
                float p[kSmUnroll];
                float v[kSmUnroll][VEC];
#pragma unroll
                for (int u = 0; u < kSmUnroll; ++u) {
                    src[u] = __shfl_sync(kFull, c, (j + u) & 31);
                    p[u] = 0.f;
                    if (j + u < cnt) {
                        const float l = leaky(__ldg(s_src + static_cast<int64_t>(src[u]) * heads + h) + sd, slope);
                        p[u] = __expf(l - m);
                        if (fok) VecLoad<float, VEC>::load(x + static_cast<int64_t>(src[u]) * f + f0, v[u]);
                    }
                }
#pragma unroll
                for (int u = 0; u < kSmUnroll; ++u) {
                    if (j + u >= cnt) continue;
                    den_part += p[u];
                    if (fok) {
#pragma unroll
                        for (int q = 0; q < VEC; ++q) part[q] = fmaf(p[u], v[u][q], part[q]);
                    }
                }
            }
            den_sup += den_part;
#pragma unroll
            for (int q = 0; q < VEC; ++q) sup[q] += part[q];
            if (++chunks == 32) {
                den += den_sup;
                den_sup = 0.f;
#pragma unroll
                for (int q = 0; q < VEC; ++q) {
                    acc[q] += sup[q];
                    sup[q] = 0.f;
                }
                chunks = 0;
            }
        }
        den += den_sup;
#pragma unroll
        for (int q = 0; q < VEC; ++q) acc[q] += sup[q];
        if (fok) {
            float *o = out + t * f + f0;
#pragma unroll
            for (int q = 0; q < VEC; ++q) o[q] = end > beg ? acc[q] / den : 0.f;
        }

        // pass 3 (optional): normalised attention weights, one writer per head
        if (alpha && fok && (f0 % channels) == 0) {
            for (int64_t k = beg; k < end; ++k) {
                const int src = __ldg(col + k);
                const float l = leaky(__ldg(s_src + static_cast<int64_t>(src) * heads + h) + sd, slope);
                alpha[k * heads + h] = __expf(l - m) / den;
            }
        }
    }
}

size_t align256(size_t b) { return (b + 255) & ~size_t(255); }

}  // namespace

size_t softmax_workspace_bytes(int64_t n, int heads) {
    return 2 * align256(sizeof(float) * size_t(n > 0 ? n : 1) * size_t(heads));
}

cudaError_t launch_edge_softmax(const int32_t *rowptr, const int32_t *col, const float *x,
                                int64_t n, int heads, int channels, const float *a_src,
                                const float *a_dst, float slope, float *out, float *alpha,
                                void *ws, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    float *s_src = static_cast<float *>(ws);
    float *s_dst = reinterpret_cast<float *>(static_cast<char *>(ws) +
                                             align256(sizeof(float) * size_t(n) * size_t(heads)));
    node_scores<<<ceil_div(n * heads, 256), 256, 0, s>>>(x, n, heads, channels, a_src, a_dst,
                                                        s_src, s_dst);
    const bool vec = (channels % 4 == 0) && (reinterpret_cast<uintptr_t>(x) % 16 == 0) &&
                     (reinterpret_cast<uintptr_t>(out) % 16 == 0);
    const int grid = ceil_div(n * 32, kSmThreads);
    if (vec)
        softmax_aggregate<4><<<grid, kSmThreads, 0, s>>>(rowptr, col, x, n, heads, channels, slope,
                                                         s_src, s_dst, out, alpha);
    else
        softmax_aggregate<1><<<grid, kSmThreads, 0, s>>>(rowptr, col, x, n, heads, channels, slope,
                                                         s_src, s_dst, out, alpha);
    return cudaGetLastError();
}

}  // namespace tfg
