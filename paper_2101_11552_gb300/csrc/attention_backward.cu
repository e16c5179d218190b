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
// Kernels, one warp per row:
//   node_scores         s_src, s_dst in base-2 units, as in the forward
//   fast_bwd_targets    (the forward's fast layout) per target t, CSR by
//                       target: one online pass gives the softmax statistics
//                       and ds_dst; statistics stored per (node, head)
//   fast_bwd_sources    per source s, CSR by source: alpha from the
//                       statistics, grad_x and ds_src
//   bwd_targets,        the same two passes for any other layout: lanes cover
//   bwd_sources         the features in tiles of 32, a head's dot products
//                       finished by a butterfly over its lanes
//   bwd_vectors_*       grad_a_src / grad_a_dst: per-block column sums, then
//                       the blocks' sums added in block order (deterministic)
// The same file holds the backward of the dot-product form (below).
#include <math_constants.h>

#include "common.cuh"

namespace tfg {
namespace {

constexpr int kBwThreads = 256;
constexpr int kBwWarps = kBwThreads / 32;
constexpr int kBwMaxTiles = 8;                 // F <= 256
constexpr int kBwRowsPerBlock = 512;           // node rows per block of the vector sums
constexpr int kBwUnroll = 4;                   // in-edges whose rows are in flight together
constexpr int kBwUnrollSrc = 2;                // out-edges whose target rows are in flight

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
    // (ids of 32 edges loaded together, kBwUnroll edges' scores in flight)
    for (int32_t k0 = beg; k0 < end; k0 += 32) {
        const int cnt = min(32, end - k0);
        const int c = lane < cnt ? __ldg(a.col + k0 + lane) : 0;
        for (int j = 0; j < cnt; j += kBwUnroll) {
            float l[kBwUnroll][NT];
#pragma unroll
            for (int u = 0; u < kBwUnroll; ++u) {
                const int64_t s = __shfl_sync(kFull, c, (j + u) & 31);
#pragma unroll
                for (int i = 0; i < NT; ++i)
                    l[u][i] = bw_leaky(__ldg(a.s_src + s * a.heads + hd[i]) + sd[i], a.slope);
            }
#pragma unroll
            for (int u = 0; u < kBwUnroll; ++u) {
                if (j + u >= cnt) break;                 // warp-uniform
#pragma unroll
                for (int i = 0; i < NT; ++i) {
                    if (l[u][i] > m[i]) {
                        den[i] = (m[i] == -CUDART_INF_F ? 0.f : den[i] * exp2f(m[i] - l[u][i]));
                        m[i] = l[u][i];
                    }
                    den[i] += exp2f(l[u][i] - m[i]);
                }
            }
        }
    }
    // pass 2: dz of every in-edge, summed into ds_dst
    // (sums blocked per 32 edges to keep fp32 chains short)
    float dsd[NT];
#pragma unroll
    for (int i = 0; i < NT; ++i) dsd[i] = 0.f;
    for (int32_t k0 = beg; k0 < end; k0 += 32) {
        const int cnt = min(32, end - k0);
        const int c = lane < cnt ? __ldg(a.col + k0 + lane) : 0;
        float part[NT];
#pragma unroll
        for (int i = 0; i < NT; ++i) part[i] = 0.f;
        for (int j = 0; j < cnt; j += kBwUnroll) {
            float d[kBwUnroll][NT], z[kBwUnroll][NT];
#pragma unroll
            for (int u = 0; u < kBwUnroll; ++u) {
                const int64_t s = __shfl_sync(kFull, c, (j + u) & 31);
#pragma unroll
                for (int i = 0; i < NT; ++i) {
                    float xv[1] = {0.f};
                    if (ok[i]) VecLoad<XT, 1>::load(x + s * f + 32 * i + lane, xv);
                    d[u][i] = g[i] * xv[0];
                    z[u][i] = __ldg(a.s_src + s * a.heads + hd[i]) + sd[i];
                }
            }
#pragma unroll
            for (int u = 0; u < kBwUnroll; ++u) {
                if (j + u >= cnt) break;                 // warp-uniform
                head_sums<NT>(d[u], a.channels);
#pragma unroll
                for (int i = 0; i < NT; ++i) {
                    const float alpha = exp2f(bw_leaky(z[u][i], a.slope) - m[i]) / den[i];
                    part[i] += alpha * (d[u][i] - beta[i]) * (z[u][i] > 0.f ? 1.f : a.slope);
                }
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
        const int cnt = min(32, end - k0);
        const int c = lane < cnt ? __ldg(a.col_src + k0 + lane) : 0;
        float pa[NT], pd[NT];
#pragma unroll
        for (int i = 0; i < NT; ++i) pa[i] = pd[i] = 0.f;
        for (int j = 0; j < cnt; j += kBwUnrollSrc) {
            float gt[kBwUnrollSrc][NT], zt[kBwUnrollSrc][NT], mt[kBwUnrollSrc][NT],
                dt[kBwUnrollSrc][NT], bt[kBwUnrollSrc][NT];
#pragma unroll
            for (int u = 0; u < kBwUnrollSrc; ++u) {
                const int64_t t = __shfl_sync(kFull, c, (j + u) & 31);
#pragma unroll
                for (int i = 0; i < NT; ++i) {
                    const int64_t th = t * a.heads + hd[i];
                    gt[u][i] = ok[i] ? __ldg(a.grad_out + t * f + 32 * i + lane) : 0.f;
                    zt[u][i] = ss[i] + __ldg(a.s_dst + th);
                    mt[u][i] = __ldg(a.m + th);
                    dt[u][i] = __ldg(a.den + th);
                    bt[u][i] = __ldg(a.beta + th);
                }
            }
#pragma unroll
            for (int u = 0; u < kBwUnrollSrc; ++u) {
                if (j + u >= cnt) break;                 // warp-uniform
                float d[NT];
#pragma unroll
                for (int i = 0; i < NT; ++i) d[i] = gt[u][i] * xs[i];
                head_sums<NT>(d, a.channels);
#pragma unroll
                for (int i = 0; i < NT; ++i) {
                    const float z = zt[u][i];
                    const float alpha = exp2f(bw_leaky(z, a.slope) - mt[u][i]) / dt[u][i];
                    pa[i] = fmaf(alpha, gt[u][i], pa[i]);
                    pd[i] += alpha * (d[i] - bt[u][i]) * (z > 0.f ? 1.f : a.slope);
                }
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

// ---------------------------------------------------------------------------
// Fast form, on the forward's fast layout: H divides 32, channels / VEC a
// power of two (a lane's VEC features lie in one head), one feature tile per
// row.  Score lanes (se, sh) = (lane / H, lane % H) evaluate each (edge, head)
// once; feature lanes gather 16-byte slices of the rows and finish a head's
// dot product with a butterfly over its channels / VEC lanes.
//
// Target pass (CSR by target), one warp per row t and ONE online pass over the
// in-edges, as in the forward: the running maximum m and denominator den of
// each head, and the rescaled sum of w (dalpha - beta), w = exp(l - m) times
// the LeakyReLU slope at z; ds_dst[t] = that sum / den.  The row's statistics
// go to stats[t, h] = (s_dst, m, 1 / den, beta) for the source pass.
//
// Source pass (CSR by source), one warp per row s: alpha of each out-edge
// from stats[t] (score lanes), the fp32 rows grad_out[t] gathered 16 bytes
// per lane (feature lanes), then grad_x[s] and ds_src[s].
// ---------------------------------------------------------------------------
struct FastBwArgs {
    const int32_t *rowptr, *col;          // CSR by target
    const int32_t *rowptr_src, *col_src;  // CSR by source
    const void *x;
    int64_t n;
    int heads, channels;
    float slope;
    const float *a_src, *a_dst, *out, *grad_out;
    const float *s_src, *s_dst;           // base-2 node scores
    float4 *stats;                        // [N, H]: (s_dst, m, 1 / den, beta)
    float *ds_dst, *ds_src, *grad_x;
};

constexpr int64_t kFbMinWork = 2048;   // edges + rows per CTA, at least
#ifndef TFG_FB_STAGE
#define TFG_FB_STAGE 1             // source pass: per-chunk weights staged in shared memory
#endif
#ifndef TFG_FB_UNROLL_TGT
#define TFG_FB_UNROLL_TGT 4        // row gathers in flight per lane, target pass
#endif
#ifndef TFG_FB_UNROLL_SRC
#define TFG_FB_UNROLL_SRC 4        // row gathers in flight per lane, source pass
#endif
constexpr int kFbUnroll = TFG_FB_UNROLL_TGT;
constexpr int kFbUnrollSrc = TFG_FB_UNROLL_SRC;
// Measured on the 114.6M-edge graph (bf16, 8 heads x 16): 3 / 3 CTAs per SM
// 13.43 ms, 4 target / 3 source 13.20, 3 / 4 12.60, 4 / 4 12.37.
#ifndef TFG_FB_TGT_BLOCKS
#define TFG_FB_TGT_BLOCKS 4        // resident CTAs per SM of the fast target pass
#endif
#ifndef TFG_FB_SRC_BLOCKS
#define TFG_FB_SRC_BLOCKS 4        // resident CTAs per SM of the fast source pass
#endif

// Sum over the aligned groups of hl lanes (hl a power of two).
__device__ __forceinline__ float group_sum(float v, int hl) {
    for (int o = 1; o < hl; o <<= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}

template <typename XT, int VEC, int LPR, int H>
__device__ __forceinline__ void fast_bwd_target(const FastBwArgs &a, int64_t t, int lane) {
    using V = VecLoad<XT, VEC>;
    constexpr int G = 32 / LPR;     // edges per feature step
    constexpr int ES = 32 / H;      // edges per score step
    constexpr int R = H;            // score steps per 32-edge chunk
    static_assert(ES % G == 0, "score step must hold whole feature steps");
    static_assert(G * kFbUnroll <= 32 && 32 % (G * kFbUnroll) == 0,
                  "feature steps of G * kFbUnroll slots must tile the 32-edge chunk");
    const int se = lane / H, sh = lane % H;
    const int g = lane / LPR, sub = lane % LPR;
    const int f = H * a.channels;
    const int hl = a.channels / VEC;
    const int f0 = sub * VEC;
    const bool fok = f0 < f;
    const int fh = fok ? f0 / a.channels : 0;
    const int fo = fok ? f0 : 0;
    const char *xb = reinterpret_cast<const char *>(static_cast<const XT *>(a.x) + fo);
    const uint32_t row_bytes = static_cast<uint32_t>(f) * static_cast<uint32_t>(sizeof(XT));
    auto gather = [&](uint32_t src) {
        return V::raw(reinterpret_cast<const XT *>(xb + static_cast<uint64_t>(src) * row_bytes));
    };
    const int64_t beg = a.rowptr[t], end = a.rowptr[t + 1];
    const float sd = __ldg(a.s_dst + t * H + sh);
    // the lane's slice of grad_out[t] and beta = <grad_out[t, h], out[t, h]>
    float gt[VEC], beta = 0.f;
#pragma unroll
    for (int q = 0; q < VEC; q += 4) {
        const float4 g4 = __ldg(reinterpret_cast<const float4 *>(a.grad_out + t * f + fo + q));
        const float4 o4 = __ldg(reinterpret_cast<const float4 *>(a.out + t * f + fo + q));
        gt[q] = fok ? g4.x : 0.f;
        gt[q + 1] = fok ? g4.y : 0.f;
        gt[q + 2] = fok ? g4.z : 0.f;
        gt[q + 3] = fok ? g4.w : 0.f;
        beta = fmaf(gt[q], o4.x, beta);
        beta = fmaf(gt[q + 1], o4.y, beta);
        beta = fmaf(gt[q + 2], o4.z, beta);
        beta = fmaf(gt[q + 3], o4.w, beta);
    }
    beta = group_sum(beta, hl);

    float m = -CUDART_INF_F, den = 0.f, acc = 0.f;
    int cnext = beg + lane < end ? ld_stream(a.col + beg + lane) : 0;
    for (int64_t base = beg; base < end; base += 32) {
        const int cnt = static_cast<int>(min64(32, end - base));
        const int c = cnext;
        cnext = base + 32 + lane < end ? ld_stream(a.col + base + 32 + lane) : 0;
        typename V::Raw raw0[kFbUnroll];
#pragma unroll
        for (int u = 0; u < kFbUnroll; ++u)
            raw0[u] = gather(static_cast<uint32_t>(__shfl_sync(kFull, c, (u * G + g) & 31)));
        float l[R], w[R];
        float cm = -CUDART_INF_F;
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int k = r * ES + se;
            const int src = __shfl_sync(kFull, c, k);
            const float z = __ldg(a.s_src + static_cast<int64_t>(src) * H + sh) + sd;
            l[r] = k < cnt ? bw_leaky(z, a.slope) : -CUDART_INF_F;
            w[r] = z > 0.f ? 1.f : a.slope;
            cm = fmaxf(cm, l[r]);
        }
#pragma unroll
        for (int o = H; o < 32; o <<= 1) cm = fmaxf(cm, __shfl_xor_sync(kFull, cm, o));
        const bool rises = cm > m;
        if (__any_sync(kFull, rises)) {   // warp-uniform; rare after the first chunks
            const float sc = rises ? (m == -CUDART_INF_F ? 0.f : exp2f(m - cm)) : 1.f;
            den *= sc;
            acc *= __shfl_sync(kFull, sc, fh);   // lane fh scores head fh
            m = fmaxf(m, cm);
        }
        float den_part = 0.f;
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const float p = r * ES + se < cnt ? exp2f(l[r] - m) : 0.f;
            den_part += p;
            w[r] *= p;
        }
        den += den_part;
        float part = 0.f;
#pragma unroll
        for (int e = 0; e < 32; e += G * kFbUnroll) {
            if (e >= cnt) break;   // warp-uniform
            typename V::Raw raw[kFbUnroll];
            float ww[kFbUnroll];
#pragma unroll
            for (int u = 0; u < kFbUnroll; ++u) {
                const int k0 = e + u * G;
                const int k = k0 + g;
                ww[u] = __shfl_sync(kFull, w[k0 / ES], ((k0 % ES) + g) * H + fh);
                if (e == 0) raw[u] = raw0[u];
                else raw[u] = gather(static_cast<uint32_t>(__shfl_sync(kFull, c, k & 31)));
            }
#pragma unroll
            for (int u = 0; u < kFbUnroll; ++u) {
                float v[VEC];
                V::widen(raw[u], v);
                float d = 0.f;
#pragma unroll
                for (int q = 0; q < VEC; ++q) d = fmaf(gt[q], v[q], d);
                d = group_sum(d, hl);
                part = fmaf(ww[u], d - beta, part);
            }
        }
        acc += part;
    }
#pragma unroll
    for (int o = H; o < 32; o <<= 1) den += __shfl_xor_sync(kFull, den, o);
#pragma unroll
    for (int o = LPR; o < 32; o <<= 1) acc += __shfl_xor_sync(kFull, acc, o);
    const float dh = __shfl_sync(kFull, den, fh);
    const float bh = __shfl_sync(kFull, beta, (sh * hl) & 31);   // group-0 lane of head sh
    if (lane < LPR && fok && f0 % a.channels == 0)
        a.ds_dst[t * H + fh] = end > beg ? acc / dh : 0.f;
    if (lane < H) a.stats[t * H + sh] = make_float4(sd, m, den > 0.f ? 1.f / den : 0.f, bh);
}

// (Splitting the heads over several launches, so that the slice of grad_out
// each one gathers stays in L2, measured no faster on the 114.6M-edge graph:
// 14.65 ms in one launch, 14.59 in two, 15.06 in four -- the pass is bound by
// latency, not by DRAM bytes.)
template <typename XT, int LPR, int H>
__device__ __forceinline__ void fast_bwd_source(const FastBwArgs &a, int64_t s, int lane,
                                                float4 *__restrict__ stage) {
    constexpr int G = 32 / LPR;     // edges per feature step
    constexpr int ES = 32 / H;      // edges per score step
    constexpr int R = H;
    static_assert(ES % G == 0, "score step must hold whole feature steps");
    static_assert(G * kFbUnrollSrc <= 32 && 32 % (G * kFbUnrollSrc) == 0,
                  "feature steps of G * kFbUnrollSrc slots must tile the 32-edge chunk");
    const int se = lane / H, sh = lane % H;
    const int g = lane / LPR, sub = lane % LPR;
    const int f = H * a.channels;
    const int hl = a.channels / 4;
    const int f0 = sub * 4;
    const bool fok = f0 < f;
    const int fh = fok ? f0 / a.channels : 0;
    const int fo = fok ? f0 : 0;
    float xs[4];
    VecLoad<XT, 4>::load(static_cast<const XT *>(a.x) + s * f + fo, xs);
    const float ss = __ldg(a.s_src + s * H + sh);
    const char *gb = reinterpret_cast<const char *>(a.grad_out + fo);
    const uint32_t row_bytes = static_cast<uint32_t>(f) * 4u;
    auto gather = [&](uint32_t t) {
        return VecLoad<float, 4>::raw(reinterpret_cast<const float *>(gb + static_cast<uint64_t>(t) * row_bytes));
    };
    const int64_t beg = a.rowptr_src[s], end = a.rowptr_src[s + 1];
    float px[4] = {0.f, 0.f, 0.f, 0.f}, pdz = 0.f;
    int cnext = beg + lane < end ? ld_stream(a.col_src + beg + lane) : 0;
    for (int64_t base = beg; base < end; base += 32) {
        const int cnt = static_cast<int>(min64(32, end - base));
        const int c = cnext;
        cnext = base + 32 + lane < end ? ld_stream(a.col_src + base + 32 + lane) : 0;
        float4 raw0[kFbUnrollSrc];
#pragma unroll
        for (int u = 0; u < kFbUnrollSrc; ++u)
            raw0[u] = gather(static_cast<uint32_t>(__shfl_sync(kFull, c, (u * G + g) & 31)));
        // alpha, af = alpha * slope(z) and ab = af * beta of (edge, head)
#if TFG_FB_STAGE
        // score lanes stage them per (edge, head) in the warp's shared-memory
        // slots (lane-consecutive: conflict-free); feature lanes read their
        // (edge, head) with one 16-byte load instead of three shuffles
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int k = r * ES + se;
            const int t = __shfl_sync(kFull, c, k);
            float4 v = make_float4(0.f, 0.f, 0.f, 0.f);
            if (k < cnt) {
                const float4 st = __ldg(a.stats + static_cast<int64_t>(t) * H + sh);
                const float z = ss + st.x;
                v.x = exp2f(bw_leaky(z, a.slope) - st.y) * st.z;
                v.y = v.x * (z > 0.f ? 1.f : a.slope);
                v.z = v.y * st.w;
            }
            stage[k * H + sh] = v;
        }
        __syncwarp();
#else
        float al[R], af[R], ab[R];
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int k = r * ES + se;
            const int t = __shfl_sync(kFull, c, k);
            al[r] = af[r] = ab[r] = 0.f;
            if (k < cnt) {
                const float4 st = __ldg(a.stats + static_cast<int64_t>(t) * H + sh);
                const float z = ss + st.x;
                al[r] = exp2f(bw_leaky(z, a.slope) - st.y) * st.z;
                af[r] = al[r] * (z > 0.f ? 1.f : a.slope);
                ab[r] = af[r] * st.w;
            }
        }
#endif
        float part[4] = {0.f, 0.f, 0.f, 0.f}, partd = 0.f;
#pragma unroll
        for (int e = 0; e < 32; e += G * kFbUnrollSrc) {
            if (e >= cnt) break;   // warp-uniform
            float4 raw[kFbUnrollSrc];
#if !TFG_FB_STAGE
            float wa[kFbUnrollSrc], wf[kFbUnrollSrc], wb[kFbUnrollSrc];
#endif
#pragma unroll
            for (int u = 0; u < kFbUnrollSrc; ++u) {
                const int k0 = e + u * G;
                const int k = k0 + g;
#if !TFG_FB_STAGE
                const int from = ((k0 % ES) + g) * H + fh;
                wa[u] = __shfl_sync(kFull, al[k0 / ES], from);
                wf[u] = __shfl_sync(kFull, af[k0 / ES], from);
                wb[u] = __shfl_sync(kFull, ab[k0 / ES], from);
#endif
                if (e == 0) raw[u] = raw0[u];
                else raw[u] = gather(static_cast<uint32_t>(__shfl_sync(kFull, c, k & 31)));
            }
#pragma unroll
            for (int u = 0; u < kFbUnrollSrc; ++u) {
#if TFG_FB_STAGE
                // the staged weights are read when the row is used, so only
                // the row slices are live while the gathers are in flight
                const float4 w4 = stage[(e + u * G + g) * H + fh];
                const float wa_u = w4.x, wf_u = w4.y, wb_u = w4.z;
#else
                const float wa_u = wa[u], wf_u = wf[u], wb_u = wb[u];
#endif
                const float gv[4] = {raw[u].x, raw[u].y, raw[u].z, raw[u].w};
                float d = 0.f;
#pragma unroll
                for (int q = 0; q < 4; ++q) d = fmaf(gv[q], xs[q], d);
                d = group_sum(d, hl);
#pragma unroll
                for (int q = 0; q < 4; ++q) part[q] = fmaf(wa_u, gv[q], part[q]);
                partd += fmaf(wf_u, d, -wb_u);
            }
        }
#pragma unroll
        for (int q = 0; q < 4; ++q) px[q] += part[q];
        pdz += partd;
#if TFG_FB_STAGE
        __syncwarp();   // every lane has read the stage before the next chunk writes it
#endif
    }
#pragma unroll
    for (int o = LPR; o < 32; o <<= 1) {
#pragma unroll
        for (int q = 0; q < 4; ++q) px[q] += __shfl_xor_sync(kFull, px[q], o);
        pdz += __shfl_xor_sync(kFull, pdz, o);
    }
    if (lane < LPR && fok) {
        const int64_t sh_g = s * H + fh;
        const float dsd = __ldg(a.ds_dst + sh_g);
        const float4 as = __ldg(reinterpret_cast<const float4 *>(a.a_src + fo));
        const float4 ad = __ldg(reinterpret_cast<const float4 *>(a.a_dst + fo));
        float4 o;
        o.x = px[0] + pdz * as.x + dsd * ad.x;
        o.y = px[1] + pdz * as.y + dsd * ad.y;
        o.z = px[2] + pdz * as.z + dsd * ad.z;
        o.w = px[3] + pdz * as.w + dsd * ad.w;
        *reinterpret_cast<float4 *>(a.grad_x + s * f + fo) = o;
        if (f0 % a.channels == 0) a.ds_src[sh_g] = pdz;
    }
}

template <typename XT, int VEC, int LPR, int H>
__global__ void __launch_bounds__(kBwThreads, TFG_FB_TGT_BLOCKS) fast_bwd_targets(FastBwArgs a) {
    for_each_row(a.rowptr, a.n, [&](int64_t t, int lane) { fast_bwd_target<XT, VEC, LPR, H>(a, t, lane); });
}

template <typename XT, int LPR, int H>
__global__ void __launch_bounds__(kBwThreads, TFG_FB_SRC_BLOCKS) fast_bwd_sources(FastBwArgs a) {
    __shared__ float4 s_stage[TFG_FB_STAGE ? kBwWarps : 1][TFG_FB_STAGE ? 32 * H : 1];
    float4 *stage = s_stage[TFG_FB_STAGE ? (threadIdx.x >> 5) : 0];
    for_each_row(a.rowptr_src, a.n, [&](int64_t s, int lane) { fast_bwd_source<XT, LPR, H>(a, s, lane, stage); });
}

// ---------------------------------------------------------------------------
// Backward of the dot-product attention (l = scale <q[t], k[s]> per head):
//   dalpha = <grad_out[t,h,:], v[s,h,:]>,  beta[t,h] = <grad_out[t,h,:], out[t,h,:]>
//   dl = alpha (dalpha - beta)
//   grad_q[t] = scale sum over e into t of dl k[s];  grad_k[s] = scale sum over
//   e out of s of dl q[t];  grad_v[s] = sum over e out of s of alpha grad_out[t].
// Logits are recomputed in base-2 units (scale2 = scale log2 e) with the same
// lane layout in both kernels, so both see the same weights.
// ---------------------------------------------------------------------------
struct DotBwArgs {
    const int32_t *rowptr, *col, *rowptr_src, *col_src;
    const void *q, *k, *v;
    int64_t n;
    int heads, channels;
    float scale, scale2;
    const float *out, *grad_out;
    float *m, *den, *beta;                // [N, H] each
    float *grad_q, *grad_k, *grad_v;
};

template <typename XT, int NT>
__device__ __forceinline__ void load_row(const XT *base, int64_t row, int f, int lane,
                                         const bool (&ok)[NT], float (&r)[NT]) {
#pragma unroll
    for (int i = 0; i < NT; ++i) {
        float xv[1] = {0.f};
        if (ok[i]) VecLoad<XT, 1>::load(base + row * f + 32 * i + lane, xv);
        r[i] = xv[0];
    }
}

// Per target t: the softmax statistics, beta and grad_q[t].
template <typename XT, int NT>
__global__ void __launch_bounds__(kBwThreads) dot_bwd_targets(DotBwArgs a) {
    const int lane = threadIdx.x & 31;
    const int64_t t = static_cast<int64_t>(blockIdx.x) * kBwWarps + (threadIdx.x >> 5);
    if (t >= a.n) return;
    const int f = a.heads * a.channels;
    const XT *qp = static_cast<const XT *>(a.q), *kp = static_cast<const XT *>(a.k),
             *vp = static_cast<const XT *>(a.v);
    bool ok[NT];
    int hd[NT];
    float qt[NT], g[NT], beta[NT], m[NT], den[NT], dq[NT];
#pragma unroll
    for (int i = 0; i < NT; ++i) {
        const int fi = 32 * i + lane;
        ok[i] = fi < f;
        hd[i] = ok[i] ? fi / a.channels : 0;
        g[i] = ok[i] ? a.grad_out[t * f + fi] : 0.f;
        beta[i] = ok[i] ? g[i] * a.out[t * f + fi] : 0.f;
        m[i] = -CUDART_INF_F;
        den[i] = 0.f;
        dq[i] = 0.f;
    }
    load_row<XT, NT>(qp, t, f, lane, ok, qt);
    head_sums<NT>(beta, a.channels);
    const int32_t beg = a.rowptr[t], end = a.rowptr[t + 1];
    for (int32_t k = beg; k < end; ++k) {                 // pass 1: maximum and denominator
        float kr[NT];
        load_row<XT, NT>(kp, __ldg(a.col + k), f, lane, ok, kr);
        float l[NT];
#pragma unroll
        for (int i = 0; i < NT; ++i) l[i] = qt[i] * kr[i];
        head_sums<NT>(l, a.channels);
#pragma unroll
        for (int i = 0; i < NT; ++i) {
            const float l2 = l[i] * a.scale2;
            if (l2 > m[i]) {
                den[i] = (m[i] == -CUDART_INF_F ? 0.f : den[i] * exp2f(m[i] - l2));
                m[i] = l2;
            }
            den[i] += exp2f(l2 - m[i]);
        }
    }
    for (int32_t k0 = beg; k0 < end; k0 += 32) {          // pass 2: grad_q (blocked sums)
        const int32_t k1 = min(end, k0 + 32);
        float part[NT];
#pragma unroll
        for (int i = 0; i < NT; ++i) part[i] = 0.f;
        for (int32_t k = k0; k < k1; ++k) {
            const int64_t s = __ldg(a.col + k);
            float kr[NT], vr[NT], l[NT], d[NT];
            load_row<XT, NT>(kp, s, f, lane, ok, kr);
            load_row<XT, NT>(vp, s, f, lane, ok, vr);
#pragma unroll
            for (int i = 0; i < NT; ++i) {
                l[i] = qt[i] * kr[i];
                d[i] = g[i] * vr[i];
            }
            head_sums<NT>(l, a.channels);
            head_sums<NT>(d, a.channels);
#pragma unroll
            for (int i = 0; i < NT; ++i) {
                const float alpha = exp2f(l[i] * a.scale2 - m[i]) / den[i];
                part[i] = fmaf(a.scale * alpha * (d[i] - beta[i]), kr[i], part[i]);
            }
        }
#pragma unroll
        for (int i = 0; i < NT; ++i) dq[i] += part[i];
    }
#pragma unroll
    for (int i = 0; i < NT; ++i) {
        const int fi = 32 * i + lane;
        if (!ok[i]) continue;
        a.grad_q[t * f + fi] = dq[i];
        if (fi % a.channels == 0) {
            const int64_t o = t * a.heads + hd[i];
            a.m[o] = m[i];
            a.den[o] = den[i];
            a.beta[o] = beta[i];
        }
    }
}

// Per source s: grad_k[s] and grad_v[s] from the out-edges' weights.
template <typename XT, int NT>
__global__ void __launch_bounds__(kBwThreads) dot_bwd_sources(DotBwArgs a) {
    const int lane = threadIdx.x & 31;
    const int64_t s = static_cast<int64_t>(blockIdx.x) * kBwWarps + (threadIdx.x >> 5);
    if (s >= a.n) return;
    const int f = a.heads * a.channels;
    const XT *qp = static_cast<const XT *>(a.q), *kp = static_cast<const XT *>(a.k),
             *vp = static_cast<const XT *>(a.v);
    bool ok[NT];
    int hd[NT];
    float ks[NT], vs[NT], dk[NT], dv[NT];
#pragma unroll
    for (int i = 0; i < NT; ++i) {
        const int fi = 32 * i + lane;
        ok[i] = fi < f;
        hd[i] = ok[i] ? fi / a.channels : 0;
        dk[i] = dv[i] = 0.f;
    }
    load_row<XT, NT>(kp, s, f, lane, ok, ks);
    load_row<XT, NT>(vp, s, f, lane, ok, vs);
    const int32_t beg = a.rowptr_src[s], end = a.rowptr_src[s + 1];
    for (int32_t k0 = beg; k0 < end; k0 += 32) {          // sums blocked per 32 edges
        const int32_t k1 = min(end, k0 + 32);
        float pk[NT], pv[NT];
#pragma unroll
        for (int i = 0; i < NT; ++i) pk[i] = pv[i] = 0.f;
        for (int32_t k = k0; k < k1; ++k) {
            const int64_t t = __ldg(a.col_src + k);
            float qr[NT], gr[NT], l[NT], d[NT];
            load_row<XT, NT>(qp, t, f, lane, ok, qr);
#pragma unroll
            for (int i = 0; i < NT; ++i) {
                gr[i] = ok[i] ? __ldg(a.grad_out + t * f + 32 * i + lane) : 0.f;
                l[i] = qr[i] * ks[i];
                d[i] = gr[i] * vs[i];
            }
            head_sums<NT>(l, a.channels);
            head_sums<NT>(d, a.channels);
#pragma unroll
            for (int i = 0; i < NT; ++i) {
                const int64_t th = t * a.heads + hd[i];
                const float alpha = exp2f(l[i] * a.scale2 - __ldg(a.m + th)) / __ldg(a.den + th);
                pk[i] = fmaf(a.scale * alpha * (d[i] - __ldg(a.beta + th)), qr[i], pk[i]);
                pv[i] = fmaf(alpha, gr[i], pv[i]);
            }
        }
#pragma unroll
        for (int i = 0; i < NT; ++i) {
            dk[i] += pk[i];
            dv[i] += pv[i];
        }
    }
#pragma unroll
    for (int i = 0; i < NT; ++i) {
        if (!ok[i]) continue;
        a.grad_k[s * f + 32 * i + lane] = dk[i];
        a.grad_v[s * f + 32 * i + lane] = dv[i];
    }
}

// Fast form of the dot-product backward, on the forward's fast layout
// (channels = lh * VEC, lh a power of two, 16-byte aligned rows): a lane
// holds VEC features of one head, the lh lanes of a head finish each dot
// product with a butterfly, G = 32 / LPR lane groups take every G-th edge
// and merge their states at the end; tiles of LPR * VEC features loop.
//  * target pass (CSR by target): per row t the running maximum m and
//    denominator den of each head and the rescaled sum
//    acc = sum of exp(l - m) (dalpha - beta) k[s], in one pass;
//    grad_q[t] = scale * acc / den; stats[t, h] = (m, 1 / den, beta, 0).
//  * source pass (CSR by source): per row s, alpha of each out-edge from
//    stats[t]; grad_k[s] = scale * sum dl q[t], grad_v[s] = sum alpha grad_out[t].
// Measured on the 114.6M-edge graph (bf16, 8 x 16): 4 / 2 edges in flight
// (target / source) at 2 CTAs per SM 21.60 ms, 4 / 4 20.95 ms (kept), 2 / 2
// 23.32 ms, 2 / 1 at 3 CTAs 23.23 ms, 8 / 2 at 1 CTA 35.65 ms.
#ifndef TFG_DB_UNROLL_TGT
#define TFG_DB_UNROLL_TGT 4       // edges in flight per lane, target pass
#endif
#ifndef TFG_DB_UNROLL_SRC
#define TFG_DB_UNROLL_SRC 4       // edges in flight per lane, source pass
#endif
constexpr int kDbUnroll = TFG_DB_UNROLL_TGT;
constexpr int kDbUnrollSrc = TFG_DB_UNROLL_SRC;
#ifndef TFG_DB_BLOCKS
#define TFG_DB_BLOCKS 3           // resident CTAs per SM of the fast passes, fp32
#endif
#ifndef TFG_DB_BLOCKS16
#define TFG_DB_BLOCKS16 2         // the same for bf16 (8 features a lane: 3 spill)
#endif

struct DotFastBwArgs {
    const int32_t *rowptr, *col, *rowptr_src, *col_src;
    const void *q, *k, *v;
    int64_t n;
    int heads, channels, lh;
    float scale, scale2;              // natural and base-2 (scale * log2 e)
    const float *out, *grad_out;
    float4 *stats;                    // [N, H]: (m, 1 / den, beta, 0)
    float *grad_q, *grad_k, *grad_v;
};

template <int VEC>
__device__ __forceinline__ float vec_dot(const float (&a)[VEC], const float (&b)[VEC]) {
    float2 d = make_float2(0.f, 0.f);
#pragma unroll
    for (int i = 0; i < VEC; i += 2) d = fma2(make_float2(a[i], a[i + 1]), make_float2(b[i], b[i + 1]), d);
    return d.x + d.y;
}

template <int VEC>
__device__ __forceinline__ void vec_axpy(float (&acc)[VEC], float w, const float (&v)[VEC]) {
    const float2 w2 = make_float2(w, w);
#pragma unroll
    for (int i = 0; i < VEC; i += 2) {
        const float2 r = fma2(make_float2(v[i], v[i + 1]), w2, make_float2(acc[i], acc[i + 1]));
        acc[i] = r.x;
        acc[i + 1] = r.y;
    }
}

template <int VEC>
__device__ __forceinline__ void load_f32(const float *p, float (&r)[VEC]) {
#pragma unroll
    for (int i = 0; i < VEC; i += 4) {
        const float4 v = __ldg(reinterpret_cast<const float4 *>(p + i));
        r[i] = v.x; r[i + 1] = v.y; r[i + 2] = v.z; r[i + 3] = v.w;
    }
}

template <typename XT, int VEC, int LPR>
__device__ __forceinline__ void dot_fast_bwd_target(const DotFastBwArgs &a, int64_t t, int lane) {
    using V = VecLoad<XT, VEC>;
    constexpr int G = 32 / LPR;
    static_assert(G * kDbUnroll <= 32, "a step must stay inside the 32-edge chunk");
    const int g = lane / LPR, sub = lane % LPR;
    const int64_t f = static_cast<int64_t>(a.heads) * a.channels;
    const XT *qp = static_cast<const XT *>(a.q), *kp = static_cast<const XT *>(a.k),
             *vp = static_cast<const XT *>(a.v);
    const int64_t beg = a.rowptr[t], end = a.rowptr[t + 1];
    const uint32_t row_bytes = static_cast<uint32_t>(f) * static_cast<uint32_t>(sizeof(XT));
    for (int64_t ft = 0; ft < f; ft += LPR * VEC) {
        const int64_t f0 = ft + sub * VEC;
        const bool fok = f0 < f;
        const int64_t fl = fok ? f0 : 0;
        float qv[VEC], gt[VEC], ov[VEC];
        V::load(qp + t * f + fl, qv);
        load_f32<VEC>(a.grad_out + t * f + fl, gt);
        load_f32<VEC>(a.out + t * f + fl, ov);
        if (!fok) {
#pragma unroll
            for (int i = 0; i < VEC; ++i) qv[i] = gt[i] = 0.f;
        }
        const float beta = group_sum(vec_dot(gt, ov), a.lh);
        const char *kb = reinterpret_cast<const char *>(kp + fl);
        const char *vb = reinterpret_cast<const char *>(vp + fl);
        float m = -CUDART_INF_F, den = 0.f, acc[VEC];
#pragma unroll
        for (int i = 0; i < VEC; ++i) acc[i] = 0.f;
        int cnext = beg + lane < end ? ld_stream(a.col + beg + lane) : 0;
        for (int64_t base = beg; base < end; base += 32) {
            const int cnt = static_cast<int>(min64(32, end - base));
            const int c = cnext;
            cnext = base + 32 + lane < end ? ld_stream(a.col + base + 32 + lane) : 0;
            float den_part = 0.f, part[VEC];
#pragma unroll
            for (int i = 0; i < VEC; ++i) part[i] = 0.f;
            for (int j = 0; j < cnt; j += G * kDbUnroll) {
                typename V::Raw rk[kDbUnroll], rv[kDbUnroll];
                bool ok[kDbUnroll];
#pragma unroll
                for (int u = 0; u < kDbUnroll; ++u) {
                    const int k = j + u * G + g;
                    const uint64_t off = static_cast<uint64_t>(
                        static_cast<uint32_t>(__shfl_sync(kFull, c, k & 31))) * row_bytes;
                    ok[u] = k < cnt;
                    rk[u] = ok[u] ? V::raw(reinterpret_cast<const XT *>(kb + off)) : V::zero();
                    rv[u] = ok[u] ? V::raw(reinterpret_cast<const XT *>(vb + off)) : V::zero();
                }
                float l[kDbUnroll], da[kDbUnroll];
                float mc = -CUDART_INF_F;
#pragma unroll
                for (int u = 0; u < kDbUnroll; ++u) {
                    float kv[VEC], vv[VEC];
                    V::widen(rk[u], kv);
                    V::widen(rv[u], vv);
                    l[u] = group_sum(vec_dot(qv, kv), a.lh);
                    da[u] = group_sum(vec_dot(gt, vv), a.lh);
                    l[u] = ok[u] ? l[u] * a.scale2 : -CUDART_INF_F;
                    mc = fmaxf(mc, l[u]);
                }
                if (mc > m) {   // new running maximum for this lane's head
                    const float sc = m == -CUDART_INF_F ? 0.f : exp2f(m - mc);
                    den *= sc;
                    den_part *= sc;
#pragma unroll
                    for (int i = 0; i < VEC; ++i) {
                        acc[i] *= sc;
                        part[i] *= sc;
                    }
                    m = mc;
                }
#pragma unroll
                for (int u = 0; u < kDbUnroll; ++u) {
                    const float p = ok[u] ? exp2f(l[u] - m) : 0.f;
                    den_part += p;
                    float kv[VEC];
                    V::widen(rk[u], kv);
                    vec_axpy(part, p * (da[u] - beta), kv);
                }
            }
            den += den_part;
#pragma unroll
            for (int i = 0; i < VEC; ++i) acc[i] += part[i];
        }
        // merge the G groups' states in a fixed butterfly order
#pragma unroll
        for (int o = LPR; o < 32; o <<= 1) {
            const float mo = __shfl_xor_sync(kFull, m, o);
            const float dn = __shfl_xor_sync(kFull, den, o);
            const float mm = fmaxf(m, mo);
            const float x = m == -CUDART_INF_F ? 0.f : exp2f(m - mm);
            const float y = mo == -CUDART_INF_F ? 0.f : exp2f(mo - mm);
            den = den * x + dn * y;
#pragma unroll
            for (int i = 0; i < VEC; ++i) {
                const float ao = __shfl_xor_sync(kFull, acc[i], o);
                acc[i] = acc[i] * x + ao * y;
            }
            m = mm;
        }
        if (lane < LPR && fok) {
            const float w = end > beg ? a.scale / den : 0.f;
#pragma unroll
            for (int i = 0; i < VEC; i += 4)
                *reinterpret_cast<float4 *>(a.grad_q + t * f + f0 + i) =
                    make_float4(acc[i] * w, acc[i + 1] * w, acc[i + 2] * w, acc[i + 3] * w);
            if (sub % a.lh == 0)
                a.stats[t * a.heads + f0 / a.channels] =
                    make_float4(m, den > 0.f ? 1.f / den : 0.f, beta, 0.f);
        }
    }
}

template <typename XT, int VEC, int LPR>
__device__ __forceinline__ void dot_fast_bwd_source(const DotFastBwArgs &a, int64_t s, int lane) {
    using V = VecLoad<XT, VEC>;
    constexpr int G = 32 / LPR;
    static_assert(G * kDbUnrollSrc <= 32, "a step must stay inside the 32-edge chunk");
    const int g = lane / LPR, sub = lane % LPR;
    const int64_t f = static_cast<int64_t>(a.heads) * a.channels;
    const XT *qp = static_cast<const XT *>(a.q), *kp = static_cast<const XT *>(a.k),
             *vp = static_cast<const XT *>(a.v);
    const int64_t beg = a.rowptr_src[s], end = a.rowptr_src[s + 1];
    const uint32_t row_bytes = static_cast<uint32_t>(f) * static_cast<uint32_t>(sizeof(XT));
    const uint32_t grow_bytes = static_cast<uint32_t>(f) * 4u;
    for (int64_t ft = 0; ft < f; ft += LPR * VEC) {
        const int64_t f0 = ft + sub * VEC;
        const bool fok = f0 < f;
        const int64_t fl = fok ? f0 : 0;
        const int h = static_cast<int>(fl / a.channels);
        float ks[VEC], vs[VEC];
        V::load(kp + s * f + fl, ks);
        V::load(vp + s * f + fl, vs);
        const char *qb = reinterpret_cast<const char *>(qp + fl);
        const char *gb = reinterpret_cast<const char *>(a.grad_out + fl);
        float dk[VEC], dv[VEC];
#pragma unroll
        for (int i = 0; i < VEC; ++i) dk[i] = dv[i] = 0.f;
        int cnext = beg + lane < end ? ld_stream(a.col_src + beg + lane) : 0;
        for (int64_t base = beg; base < end; base += 32) {
            const int cnt = static_cast<int>(min64(32, end - base));
            const int c = cnext;
            cnext = base + 32 + lane < end ? ld_stream(a.col_src + base + 32 + lane) : 0;
            float pk[VEC], pv[VEC];
#pragma unroll
            for (int i = 0; i < VEC; ++i) pk[i] = pv[i] = 0.f;
            for (int j = 0; j < cnt; j += G * kDbUnrollSrc) {
                typename V::Raw rq[kDbUnrollSrc];
                float gr[kDbUnrollSrc][VEC];
                float4 st[kDbUnrollSrc];
                bool ok[kDbUnrollSrc];
#pragma unroll
                for (int u = 0; u < kDbUnrollSrc; ++u) {
                    const int k = j + u * G + g;
                    const uint32_t t = static_cast<uint32_t>(__shfl_sync(kFull, c, k & 31));
                    ok[u] = k < cnt;
                    rq[u] = ok[u] ? V::raw(reinterpret_cast<const XT *>(qb + uint64_t(t) * row_bytes)) : V::zero();
                    if (ok[u]) {
                        load_f32<VEC>(reinterpret_cast<const float *>(gb + uint64_t(t) * grow_bytes), gr[u]);
                        st[u] = __ldg(a.stats + static_cast<int64_t>(t) * a.heads + h);
                    } else {
#pragma unroll
                        for (int i = 0; i < VEC; ++i) gr[u][i] = 0.f;
                        st[u] = make_float4(0.f, 0.f, 0.f, 0.f);
                    }
                }
#pragma unroll
                for (int u = 0; u < kDbUnrollSrc; ++u) {
                    float qv[VEC];
                    V::widen(rq[u], qv);
                    const float l = group_sum(vec_dot(qv, ks), a.lh) * a.scale2;
                    const float da = group_sum(vec_dot(gr[u], vs), a.lh);
                    const float alpha = ok[u] ? exp2f(l - st[u].x) * st[u].y : 0.f;
                    vec_axpy(pk, alpha * (da - st[u].z), qv);
                    vec_axpy(pv, alpha, gr[u]);
                }
            }
#pragma unroll
            for (int i = 0; i < VEC; ++i) {
                dk[i] += pk[i];
                dv[i] += pv[i];
            }
        }
#pragma unroll
        for (int o = LPR; o < 32; o <<= 1)
#pragma unroll
            for (int i = 0; i < VEC; ++i) {
                dk[i] += __shfl_xor_sync(kFull, dk[i], o);
                dv[i] += __shfl_xor_sync(kFull, dv[i], o);
            }
        if (lane < LPR && fok) {
#pragma unroll
            for (int i = 0; i < VEC; i += 4) {
                *reinterpret_cast<float4 *>(a.grad_k + s * f + f0 + i) =
                    make_float4(dk[i] * a.scale, dk[i + 1] * a.scale, dk[i + 2] * a.scale,
                                dk[i + 3] * a.scale);
                *reinterpret_cast<float4 *>(a.grad_v + s * f + f0 + i) =
                    make_float4(dv[i], dv[i + 1], dv[i + 2], dv[i + 3]);
            }
        }
    }
}

template <typename XT, int VEC, int LPR>
__global__ void __launch_bounds__(kBwThreads, VEC >= 8 ? TFG_DB_BLOCKS16 : TFG_DB_BLOCKS) dot_fast_bwd_targets(DotFastBwArgs a) {
    for_each_row(a.rowptr, a.n, [&](int64_t t, int lane) { dot_fast_bwd_target<XT, VEC, LPR>(a, t, lane); });
}

template <typename XT, int VEC, int LPR>
__global__ void __launch_bounds__(kBwThreads, VEC >= 8 ? TFG_DB_BLOCKS16 : TFG_DB_BLOCKS) dot_fast_bwd_sources(DotFastBwArgs a) {
    for_each_row(a.rowptr_src, a.n, [&](int64_t s, int lane) { dot_fast_bwd_source<XT, VEC, LPR>(a, s, lane); });
}

template <typename XT, int VEC>
void launch_dot_fast_bw(const DotFastBwArgs &a, int64_t e, cudaStream_t s) {
    const int64_t chunks = static_cast<int64_t>(a.heads) * a.channels / VEC;
    const int grid = balanced_grid(a.n, e, kFbMinWork);
    if (chunks >= 32 || a.lh > 16) {
        dot_fast_bwd_targets<XT, VEC, 32><<<grid, kBwThreads, 0, s>>>(a);
        dot_fast_bwd_sources<XT, VEC, 32><<<grid, kBwThreads, 0, s>>>(a);
    } else if (chunks > 8 || a.lh > 8) {
        dot_fast_bwd_targets<XT, VEC, 16><<<grid, kBwThreads, 0, s>>>(a);
        dot_fast_bwd_sources<XT, VEC, 16><<<grid, kBwThreads, 0, s>>>(a);
    } else {
        dot_fast_bwd_targets<XT, VEC, 8><<<grid, kBwThreads, 0, s>>>(a);
        dot_fast_bwd_sources<XT, VEC, 8><<<grid, kBwThreads, 0, s>>>(a);
    }
}

template <typename XT, int NT>
cudaError_t launch_dot_bw(const DotBwArgs &a, cudaStream_t s) {
    const int rows = ceil_div(a.n, kBwWarps);
    dot_bwd_targets<XT, NT><<<rows, kBwThreads, 0, s>>>(a);
    dot_bwd_sources<XT, NT><<<rows, kBwThreads, 0, s>>>(a);
    return cudaGetLastError();
}

template <typename XT>
cudaError_t launch_dot_bw_tiles(const DotBwArgs &a, cudaStream_t s) {
    switch (ceil_div(static_cast<int64_t>(a.heads) * a.channels, 32)) {
        case 1: return launch_dot_bw<XT, 1>(a, s);
        case 2: return launch_dot_bw<XT, 2>(a, s);
        case 3: return launch_dot_bw<XT, 3>(a, s);
        case 4: return launch_dot_bw<XT, 4>(a, s);
        case 5: return launch_dot_bw<XT, 5>(a, s);
        case 6: return launch_dot_bw<XT, 6>(a, s);
        case 7: return launch_dot_bw<XT, 7>(a, s);
        default: return launch_dot_bw<XT, 8>(a, s);
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

// Fast passes when the layout allows them (both or neither); false means
// "use the general kernels".
template <typename XT, int VEC, int H>
bool launch_fast_bw_heads(const FastBwArgs &a, int64_t e, cudaStream_t s) {
    const int f = H * a.channels;
    const int lt = f / VEC <= 8 ? 8 : (f / VEC <= 16 ? 16 : 32);   // target pass lanes per row
    const int ls = f / 4 <= 8 ? 8 : (f / 4 <= 16 ? 16 : 32);       // source pass lanes per row
    if ((32 / H) % (32 / lt) != 0 || (32 / H) % (32 / ls) != 0) return false;
    const int grid = balanced_grid(a.n, e, kFbMinWork);
    switch (lt) {
        case 8:
            if constexpr ((32 / H) % 4 == 0)
                fast_bwd_targets<XT, VEC, 8, H><<<grid, kBwThreads, 0, s>>>(a);
            break;
        case 16:
            if constexpr ((32 / H) % 2 == 0)
                fast_bwd_targets<XT, VEC, 16, H><<<grid, kBwThreads, 0, s>>>(a);
            break;
        default:
            if constexpr (VEC == 4) fast_bwd_targets<XT, VEC, 32, H><<<grid, kBwThreads, 0, s>>>(a);
            break;
    }
    switch (ls) {
        case 8:
            if constexpr ((32 / H) % 4 == 0)
                fast_bwd_sources<XT, 8, H><<<grid, kBwThreads, 0, s>>>(a);
            break;
        case 16:
            if constexpr ((32 / H) % 2 == 0)
                fast_bwd_sources<XT, 16, H><<<grid, kBwThreads, 0, s>>>(a);
            break;
        default: fast_bwd_sources<XT, 32, H><<<grid, kBwThreads, 0, s>>>(a); break;
    }
    return true;
}

template <typename XT, int VEC>
bool launch_fast_bw(const FastBwArgs &a, int heads, int64_t e, cudaStream_t s) {
    const int c = a.channels;
    const int hl = c / VEC;
    if (c % VEC != 0 || (hl & (hl - 1)) != 0 || static_cast<int64_t>(heads) * c > 128) return false;
    switch (heads) {
        case 1: return launch_fast_bw_heads<XT, VEC, 1>(a, e, s);
        case 2: return launch_fast_bw_heads<XT, VEC, 2>(a, e, s);
        case 4: return launch_fast_bw_heads<XT, VEC, 4>(a, e, s);
        case 8: return launch_fast_bw_heads<XT, VEC, 8>(a, e, s);
        default: return false;
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
    return 8 * nh + bw_align(sizeof(float) * 2 * f * size_t(bw_blocks(n > 0 ? n : 1)));
}

size_t dot_attention_backward_workspace_bytes(int64_t n, int heads) {
    return 4 * bw_align(sizeof(float) * size_t(n > 0 ? n : 1) * size_t(heads));
}

cudaError_t launch_dot_softmax_backward(const int32_t *rowptr, const int32_t *col,
                                        const int32_t *rowptr_src, const int32_t *col_src,
                                        const void *q, const void *k, const void *v, int x_dtype,
                                        int64_t n, int64_t e, int heads, int channels, float scale,
                                        const float *out, const float *grad_out, float *grad_q,
                                        float *grad_k, float *grad_v, void *ws, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const size_t nh = bw_align(sizeof(float) * size_t(n) * size_t(heads));
    char *w = static_cast<char *>(ws);
    auto a16 = [](const void *p) { return reinterpret_cast<uintptr_t>(p) % 16 == 0; };
    const int vec = x_dtype == TFG_BF16 ? 8 : 4;
    const int lh = channels / vec;
    if (a16(q) && a16(k) && a16(v) && a16(out) && a16(grad_out) && a16(grad_q) && a16(grad_k) &&
        a16(grad_v) && channels % vec == 0 && lh >= 1 && lh <= 32 && (lh & (lh - 1)) == 0) {
        // workspace: the [N, H] float4 statistics (4 * nh bytes)
        const DotFastBwArgs fa{rowptr, col, rowptr_src, col_src, q, k, v, n, heads, channels, lh,
                               scale, scale * 1.4426950408889634f, out, grad_out,
                               reinterpret_cast<float4 *>(w), grad_q, grad_k, grad_v};
        if (x_dtype == TFG_BF16) launch_dot_fast_bw<uint16_t, 8>(fa, e, s);
        else launch_dot_fast_bw<float, 4>(fa, e, s);
        return cudaGetLastError();
    }
    DotBwArgs a{rowptr, col, rowptr_src, col_src, q, k, v, n, heads, channels, scale,
                scale * 1.4426950408889634f, out, grad_out,
                reinterpret_cast<float *>(w), reinterpret_cast<float *>(w + nh),
                reinterpret_cast<float *>(w + 2 * nh), grad_q, grad_k, grad_v};
    return x_dtype == TFG_BF16 ? launch_dot_bw_tiles<uint16_t>(a, s) : launch_dot_bw_tiles<float>(a, s);
}

// edge_softmax.cu's node-score launcher (the same scores as the forward)
cudaError_t launch_node_scores(const void *x, int x_dtype, int64_t n, int heads, int channels,
                               const float *a_src, const float *a_dst, float *s_src, float *s_dst,
                               cudaStream_t s);

cudaError_t launch_edge_softmax_backward(const int32_t *rowptr, const int32_t *col,
                                         const int32_t *rowptr_src, const int32_t *col_src,
                                         const void *x, int x_dtype, int64_t n, int64_t e,
                                         int heads, int channels, const float *a_src,
                                         const float *a_dst,
                                         float slope, const float *out, const float *grad_out,
                                         float *grad_x, float *grad_a_src, float *grad_a_dst,
                                         void *ws, cudaStream_t s) {
    const size_t f = static_cast<size_t>(heads) * channels;
    if (n <= 0) {   // no nodes: the vector gradients are zero
        cudaError_t err = cudaMemsetAsync(grad_a_src, 0, sizeof(float) * f, s);
        if (err == cudaSuccess) err = cudaMemsetAsync(grad_a_dst, 0, sizeof(float) * f, s);
        return err;
    }
    // workspace: s_src, s_dst, four [N, H] buffers (the fast form's float4
    // statistics, or m, den, beta and ds_dst), two more, the vector partials
    const size_t nh = bw_align(sizeof(float) * size_t(n) * size_t(heads));
    char *w = static_cast<char *>(ws);
    float *buf[8];
    for (int i = 0; i < 8; ++i) buf[i] = reinterpret_cast<float *>(w + i * nh);
    float *part = reinterpret_cast<float *>(w + 8 * nh);
    cudaError_t err = launch_node_scores(x, x_dtype, n, heads, channels, a_src, a_dst, buf[0],
                                         buf[1], s);
    if (err != cudaSuccess) return err;
    auto a16 = [](const void *p) { return reinterpret_cast<uintptr_t>(p) % 16 == 0; };
    const bool aligned = a16(x) && a16(out) && a16(grad_out) && a16(grad_x) && a16(a_src) &&
                         a16(a_dst);
    if (aligned) {
        FastBwArgs fa{rowptr, col, rowptr_src, col_src, x, n, heads, channels, slope, a_src, a_dst,
                      out, grad_out, buf[0], buf[1], reinterpret_cast<float4 *>(buf[2]), buf[6],
                      buf[7], grad_x};
        const bool fast = x_dtype == TFG_BF16 ? launch_fast_bw<uint16_t, 8>(fa, heads, e, s)
                                              : launch_fast_bw<float, 4>(fa, heads, e, s);
        if (fast) {
            const int fdim = heads * channels;
            const int nb = bw_blocks(n);
            if (x_dtype == TFG_BF16)
                bwd_vectors_partial<uint16_t><<<nb, kBwThreads, 0, s>>>(
                    static_cast<const uint16_t *>(x), n, heads, channels, buf[7], buf[6], part);
            else
                bwd_vectors_partial<float><<<nb, kBwThreads, 0, s>>>(
                    static_cast<const float *>(x), n, heads, channels, buf[7], buf[6], part);
            bwd_vectors_final<<<ceil_div(2 * fdim, kBwThreads), kBwThreads, 0, s>>>(
                part, nb, fdim, grad_a_src, grad_a_dst);
            return cudaGetLastError();
        }
    }
    BwArgs a{rowptr, col, rowptr_src, col_src, x, n, heads, channels, slope, a_src, a_dst,
             out, grad_out, buf[0], buf[1], buf[2], buf[3], buf[4], buf[5], buf[6], grad_x};
    return x_dtype == TFG_BF16 ? launch_bw_tiles<uint16_t>(a, part, grad_a_src, grad_a_dst, s)
                               : launch_bw_tiles<float>(a, part, grad_a_src, grad_a_dst, s);
}

}  // namespace tfg
