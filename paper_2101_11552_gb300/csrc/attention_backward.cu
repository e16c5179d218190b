// Backward of the GAT edge-softmax aggregation (Fig. 5a workflow): the
// gradients with respect to the node features x and the attention vectors
// a_src, a_dst, given grad_out = dL/dout and the forward's output out.  The
// paper keeps graph construction and mini-batching differentiable (Sections
// 2.1.1 and 2.1.3); with alpha the softmax weights of the forward:
//
//   dalpha[e,h] = <grad_out[t,h,:], x[s,h,:]>                 (e = s -> t)
//   beta[t,h]   = sum over e into t of alpha dalpha = <grad_out[t,h,:], out[t,h,:]>
//   dz[e,h]     = alpha (dalpha - beta[t,h]) * (z > 0 ? 1 : slope)
//   grad_x[s,h,:] = sum over e out of s of alpha grad_out[t,h,:]
//                   + ds_src[s,h] a_src[h,:] + ds_dst[s,h] a_dst[h,:]
//   ds_src[s,h] = sum over e out of s of dz,   ds_dst[t,h] = sum over e into t of dz
//   grad_a_src[h,c] = sum_v ds_src[v,h] x[v,h,c],  grad_a_dst likewise.
//
// Kernels (each warp owns one row, lanes cover the features in tiles of 32,
// a head's dot products are finished by a butterfly over its lanes):
//   node_scores         s_src, s_dst in base-2 units, as in the forward
//   bwd_targets         per target t (CSR by target): the softmax statistics
//                       m, den of the forward, beta from out, and ds_dst
//   bwd_sources         per source s (CSR by source): alpha recomputed from the
//                       statistics, grad_x and ds_src
//   bwd_vectors_*       grad_a_src / grad_a_dst: per-block column sums, then
//                       the blocks' sums added in block order (deterministic)
#include <math_constants.h>

#include "common.cuh"

namespace tfg {
namespace {

constexpr int kBwThreads = 256;
constexpr int kBwWarps = kBwThreads / 32;
constexpr int kBwMaxTiles = 8;                 // F <= 256
constexpr int kBwRowsPerBlock = 512;           // node rows per block of the vector sums

__device__ __forceinline__ float bw_leaky(float v, float slope) { return v > 0.f ? v : slope * v; }

// Sum of v over the lanes holding the same head.  Heads of C <= 32 channels
// are aligned groups of C lanes inside a 32-feature tile; heads of C >= 32
// channels span whole tiles, whose full-warp sums are added over the tiles
// of the head.  Every lane of a head receives the head's sum.
template <int NT>
__device__ __forceinline__ void head_sums(float (&v)[NT], int channels) {
    if (channels <= 32) {
#pragma unroll
        for (int i = 0; i < NT; ++i)
            for (int o = 1; o < channels; o <<= 1) v[i] += __shfl_xor_sync(kFull, v[i], o);
    } else {
#pragma unroll
        for (int i = 0; i < NT; ++i)
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) v[i] += __shfl_xor_sync(kFull, v[i], o);
        const int per = channels / 32;             // tiles per head
        float tot[NT];
#pragma unroll
        for (int i = 0; i < NT; ++i) {
            tot[i] = 0.f;
#pragma unroll
            for (int j = 0; j < NT; ++j)
                if (j / per == i / per) tot[i] += v[j];
        }
#pragma unroll
        for (int i = 0; i < NT; ++i) v[i] = tot[i];
    }
}

struct BwArgs {
    const int32_t *rowptr, *col;          // CSR by target
    const int32_t *rowptr_src, *col_src;  // CSR by source (col_src holds targets)
    const void *x;
    int64_t n;
    int heads, channels;
    float slope;
    const float *a_src, *a_dst;
    const float *out, *grad_out;
    const float *s_src, *s_dst;           // base-2 node scores
    float *m, *den, *beta, *ds_dst, *ds_src;   // [N, H] each
    float *grad_x;
};

// Per target t: the forward's softmax statistics (running maximum in base-2
// units and denominator), beta = <grad_out[t], out[t]> per head, and
// ds_dst[t] = sum of dz over the in-edges.
template <typename XT, int NT>
__global__ void __launch_bounds__(kBwThreads) bwd_targets(BwArgs a) {
    const int lane = threadIdx.x & 31;
    const int64_t t = static_cast<int64_t>(blockIdx.x) * kBwWarps + (threadIdx.x >> 5);
    if (t >= a.n) return;
    const int f = a.heads * a.channels;
    const XT *x = static_cast<const XT *>(a.x);
    float g[NT], sd[NT], beta[NT];
    int hd[NT];
    bool ok[NT];
#pragma unroll
    for (int i = 0; i < NT; ++i) {
        const int fi = 32 * i + lane;
        ok[i] = fi < f;
        hd[i] = ok[i] ? fi / a.channels : 0;
        g[i] = ok[i] ? a.grad_out[t * f + fi] : 0.f;
        beta[i] = ok[i] ? g[i] * a.out[t * f + fi] : 0.f;
        sd[i] = __ldg(a.s_dst + t * a.heads + hd[i]);
    }
    head_sums<NT>(beta, a.channels);
    const int32_t beg = a.rowptr[t], end = a.rowptr[t + 1];
    // pass 1: maximum and denominator of each head's logits (base 2)
    float m[NT], den[NT];
#pragma unroll
    for (int i = 0; i < NT; ++i) {
        m[i] = -CUDART_INF_F;
        den[i] = 0.f;
    }
    for (int32_t k = beg; k < end; ++k) {
        const int64_t s = __ldg(a.col + k);
#pragma unroll
        for (int i = 0; i < NT; ++i) {
            const float l = bw_leaky(__ldg(a.s_src + s * a.heads + hd[i]) + sd[i], a.slope);
            if (l > m[i]) {
                den[i] = (m[i] == -CUDART_INF_F ? 0.f : den[i] * exp2f(m[i] - l));
                m[i] = l;
            }
            den[i] += exp2f(l - m[i]);
        }
    }
    // pass 2: dz of every in-edge, summed into ds_dst
    // (sums blocked per 32 edges to keep fp32 chains short)
    float dsd[NT];
#pragma unroll
    for (int i = 0; i < NT; ++i) dsd[i] = 0.f;
    for (int32_t k0 = beg; k0 < end; k0 += 32) {
        const int32_t k1 = min(end, k0 + 32);
        float part[NT];
#pragma unroll
        for (int i = 0; i < NT; ++i) part[i] = 0.f;
        for (int32_t k = k0; k < k1; ++k) {
            const int64_t s = __ldg(a.col + k);
            float d[NT], z[NT];
#pragma unroll
            for (int i = 0; i < NT; ++i) {
                float xv[1] = {0.f};
                if (ok[i]) VecLoad<XT, 1>::load(x + s * f + 32 * i + lane, xv);
                d[i] = g[i] * xv[0];
                z[i] = __ldg(a.s_src + s * a.heads + hd[i]) + sd[i];
            }
            head_sums<NT>(d, a.channels);
#pragma unroll
            for (int i = 0; i < NT; ++i) {
                const float alpha = exp2f(bw_leaky(z[i], a.slope) - m[i]) / den[i];
                part[i] += alpha * (d[i] - beta[i]) * (z[i] > 0.f ? 1.f : a.slope);
            }
        }
#pragma unroll
        for (int i = 0; i < NT; ++i) dsd[i] += part[i];
    }
    // one lane per head writes the head's values
#pragma unroll
    for (int i = 0; i < NT; ++i) {
        const int fi = 32 * i + lane;
        if (ok[i] && fi % a.channels == 0) {
            const int64_t o = t * a.heads + hd[i];
            a.m[o] = m[i];
            a.den[o] = den[i];
            a.beta[o] = beta[i];
            a.ds_dst[o] = dsd[i];
        }
    }
}

// Per source s: alpha of every out-edge from the statistics of its target,
// the weighted sum of the targets' gradients, ds_src, and grad_x[s].
template <typename XT, int NT>
__global__ void __launch_bounds__(kBwThreads) bwd_sources(BwArgs a) {
    const int lane = threadIdx.x & 31;
    const int64_t s = static_cast<int64_t>(blockIdx.x) * kBwWarps + (threadIdx.x >> 5);
    if (s >= a.n) return;
    const int f = a.heads * a.channels;
    const XT *x = static_cast<const XT *>(a.x);
    float xs[NT], ss[NT], acc[NT], dss[NT];
    int hd[NT];
    bool ok[NT];
#pragma unroll
    for (int i = 0; i < NT; ++i) {
        const int fi = 32 * i + lane;
        ok[i] = fi < f;
        hd[i] = ok[i] ? fi / a.channels : 0;
        float xv[1] = {0.f};
        if (ok[i]) VecLoad<XT, 1>::load(x + s * f + fi, xv);
        xs[i] = xv[0];
        ss[i] = __ldg(a.s_src + s * a.heads + hd[i]);
        acc[i] = 0.f;
        dss[i] = 0.f;
    }
    const int32_t beg = a.rowptr_src[s], end = a.rowptr_src[s + 1];
    for (int32_t k0 = beg; k0 < end; k0 += 32) {          // sums blocked per 32 edges
        const int32_t k1 = min(end, k0 + 32);
        float pa[NT], pd[NT];
#pragma unroll
        for (int i = 0; i < NT; ++i) pa[i] = pd[i] = 0.f;
        for (int32_t k = k0; k < k1; ++k) {
            const int64_t t = __ldg(a.col_src + k);
            float gt[NT], d[NT];
#pragma unroll
            for (int i = 0; i < NT; ++i) {
                gt[i] = ok[i] ? __ldg(a.grad_out + t * f + 32 * i + lane) : 0.f;
                d[i] = gt[i] * xs[i];
            }
            head_sums<NT>(d, a.channels);
#pragma unroll
            for (int i = 0; i < NT; ++i) {
                const int64_t th = t * a.heads + hd[i];
                const float z = ss[i] + __ldg(a.s_dst + th);
                const float alpha = exp2f(bw_leaky(z, a.slope) - __ldg(a.m + th)) / __ldg(a.den + th);
                pa[i] = fmaf(alpha, gt[i], pa[i]);
                pd[i] += alpha * (d[i] - __ldg(a.beta + th)) * (z > 0.f ? 1.f : a.slope);
            }
        }
#pragma unroll
        for (int i = 0; i < NT; ++i) {
            acc[i] += pa[i];
            dss[i] += pd[i];
        }
    }
#pragma unroll
    for (int i = 0; i < NT; ++i) {
        const int fi = 32 * i + lane;
        if (!ok[i]) continue;
        const float dsd = __ldg(a.ds_dst + s * a.heads + hd[i]);
        a.grad_x[s * f + fi] = acc[i] + dss[i] * __ldg(a.a_src + fi) + dsd * __ldg(a.a_dst + fi);
        if (fi % a.channels == 0) a.ds_src[s * a.heads + hd[i]] = dss[i];
    }
}

// Column sums of ds[v, head(f)] * x[v, f] over a block of rows, for both
// vectors: part[b][0:F] (a_src) and part[b][F:2F] (a_dst).
template <typename XT>
__global__ void __launch_bounds__(kBwThreads) bwd_vectors_partial(const XT *__restrict__ x,
                                                                  int64_t n, int heads,
                                                                  int channels,
                                                                  const float *__restrict__ ds_src,
                                                                  const float *__restrict__ ds_dst,
                                                                  float *__restrict__ part) {
    const int f = heads * channels;
    const int64_t v0 = static_cast<int64_t>(blockIdx.x) * kBwRowsPerBlock;
    const int64_t v1 = min64(n, v0 + kBwRowsPerBlock);
    for (int fi = threadIdx.x; fi < f; fi += kBwThreads) {
        const int h = fi / channels;
        float s1 = 0.f, s2 = 0.f;
        for (int64_t v = v0; v < v1; ++v) {
            float xv[1];
            VecLoad<XT, 1>::load(x + v * f + fi, xv);
            s1 = fmaf(__ldg(ds_src + v * heads + h), xv[0], s1);
            s2 = fmaf(__ldg(ds_dst + v * heads + h), xv[0], s2);
        }
        part[static_cast<int64_t>(blockIdx.x) * 2 * f + fi] = s1;
        part[static_cast<int64_t>(blockIdx.x) * 2 * f + f + fi] = s2;
    }
}

__global__ void __launch_bounds__(kBwThreads) bwd_vectors_final(const float *__restrict__ part,
                                                                int blocks, int f,
                                                                float *__restrict__ ga_src,
                                                                float *__restrict__ ga_dst) {
    const int fi = blockIdx.x * kBwThreads + threadIdx.x;
    if (fi >= 2 * f) return;
    float s = 0.f;
    for (int b = 0; b < blocks; ++b) s += part[static_cast<int64_t>(b) * 2 * f + fi];
    if (fi < f) ga_src[fi] = s;
    else ga_dst[fi - f] = s;
}

size_t bw_align(size_t b) { return (b + 255) & ~size_t(255); }

int bw_blocks(int64_t n) { return static_cast<int>((n + kBwRowsPerBlock - 1) / kBwRowsPerBlock); }

template <typename XT, int NT>
cudaError_t launch_bw(const BwArgs &a, float *part, float *ga_src, float *ga_dst,
                      cudaStream_t s) {
    const int rows = ceil_div(a.n, kBwWarps);
    bwd_targets<XT, NT><<<rows, kBwThreads, 0, s>>>(a);
    bwd_sources<XT, NT><<<rows, kBwThreads, 0, s>>>(a);
    const int f = a.heads * a.channels;
    const int nb = bw_blocks(a.n);
    bwd_vectors_partial<XT><<<nb, kBwThreads, 0, s>>>(static_cast<const XT *>(a.x), a.n, a.heads,
                                                      a.channels, a.ds_src, a.ds_dst, part);
    bwd_vectors_final<<<ceil_div(2 * f, kBwThreads), kBwThreads, 0, s>>>(part, nb, f, ga_src, ga_dst);
    return cudaGetLastError();
}

template <typename XT>
cudaError_t launch_bw_tiles(const BwArgs &a, float *part, float *ga_src, float *ga_dst,
                            cudaStream_t s) {
    const int nt = ceil_div(static_cast<int64_t>(a.heads) * a.channels, 32);
    switch (nt) {
        case 1: return launch_bw<XT, 1>(a, part, ga_src, ga_dst, s);
        case 2: return launch_bw<XT, 2>(a, part, ga_src, ga_dst, s);
        case 3: return launch_bw<XT, 3>(a, part, ga_src, ga_dst, s);
        case 4: return launch_bw<XT, 4>(a, part, ga_src, ga_dst, s);
        case 5: return launch_bw<XT, 5>(a, part, ga_src, ga_dst, s);
        case 6: return launch_bw<XT, 6>(a, part, ga_src, ga_dst, s);
        case 7: return launch_bw<XT, 7>(a, part, ga_src, ga_dst, s);
        default: return launch_bw<XT, 8>(a, part, ga_src, ga_dst, s);
    }
}

}  // namespace

bool attention_backward_layout_ok(int heads, int channels) {
    const int64_t f = static_cast<int64_t>(heads) * channels;
    const bool heads_fit = channels <= 32 ? (32 % channels == 0) : (channels % 32 == 0);
    return heads >= 1 && channels >= 1 && f <= 32 * kBwMaxTiles && heads_fit;
}

size_t attention_backward_workspace_bytes(int64_t n, int heads, int channels) {
    const size_t nh = bw_align(sizeof(float) * size_t(n > 0 ? n : 1) * size_t(heads));
    const size_t f = static_cast<size_t>(heads) * channels;
    return 7 * nh + bw_align(sizeof(float) * 2 * f * size_t(bw_blocks(n > 0 ? n : 1)));
}

// edge_softmax.cu's node-score launcher (the same scores as the forward)
cudaError_t launch_node_scores(const void *x, int x_dtype, int64_t n, int heads, int channels,
                               const float *a_src, const float *a_dst, float *s_src, float *s_dst,
                               cudaStream_t s);

cudaError_t launch_edge_softmax_backward(const int32_t *rowptr, const int32_t *col,
                                         const int32_t *rowptr_src, const int32_t *col_src,
                                         const void *x, int x_dtype, int64_t n, int heads,
                                         int channels, const float *a_src, const float *a_dst,
                                         float slope, const float *out, const float *grad_out,
                                         float *grad_x, float *grad_a_src, float *grad_a_dst,
                                         void *ws, cudaStream_t s) {
    const size_t f = static_cast<size_t>(heads) * channels;
    if (n <= 0) {   // no nodes: the vector gradients are zero
        cudaError_t err = cudaMemsetAsync(grad_a_src, 0, sizeof(float) * f, s);
        if (err == cudaSuccess) err = cudaMemsetAsync(grad_a_dst, 0, sizeof(float) * f, s);
        return err;
    }
    const size_t nh = bw_align(sizeof(float) * size_t(n) * size_t(heads));
    char *w = static_cast<char *>(ws);
    float *buf[7];
    for (int i = 0; i < 7; ++i) buf[i] = reinterpret_cast<float *>(w + i * nh);
    float *part = reinterpret_cast<float *>(w + 7 * nh);
    BwArgs a{rowptr, col, rowptr_src, col_src, x, n, heads, channels, slope, a_src, a_dst,
             out, grad_out, buf[0], buf[1], buf[2], buf[3], buf[4], buf[5], buf[6], grad_x};
    cudaError_t err = launch_node_scores(x, x_dtype, n, heads, channels, a_src, a_dst, buf[0],
                                         buf[1], s);
    if (err != cudaSuccess) return err;
    return x_dtype == TFG_BF16 ? launch_bw_tiles<uint16_t>(a, part, grad_a_src, grad_a_dst, s)
                               : launch_bw_tiles<float>(a, part, grad_a_src, grad_a_dst, s);
}

}  // namespace tfg
