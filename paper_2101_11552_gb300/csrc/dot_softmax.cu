// Dot-product (Transformer-style) edge-softmax aggregation: the attention
// form of the GAT that tf_geometric ships (Section 4.2 names it a
// Transformer-based GAT), on the same map-reduce workflow as Fig. 5a:
//
//   map      l[k, h] = scale * <q[t, h, :], k[src, h, :]>   for position k of row t
//   reduce   m = max over row t of l[., h];  den = sum of exp(l - m)
//   map      alpha[k, h] = exp(l[k, h] - m) / den
//   aggregate out[t, h, :] = sum over row t of alpha[k, h] * v[src, h, :]
//
// Unlike the additive form there is no per-node score to precompute: every
// logit is a dot product of a gathered key row with the target's query row,
// so each edge gathers a key row and a value row.  One warp owns a target row
// and makes one pass with the running-maximum softmax (the running sums are
// rescaled by exp(m_old - m_new) when the maximum rises; the result is
// unchanged), blocked per 32-edge chunk to keep fp32 chains short.
//
//  * fast form (channels = LH * VEC with LH a power of two <= 32, 16-byte
//    aligned rows): a row tile of LPR * VEC features holds whole heads; a
//    lane holds VEC features of one head, the LH lanes of a head finish the
//    dot product with a butterfly, so every lane of a head sees the same
//    logit.  G = 32 / LPR lane groups take every G-th edge and merge their
//    (m, den, acc) states at the end.  Tiles loop when F > LPR * VEC.
//  * general form (any channels <= 256, any alignment): the warp walks the
//    heads of the row one at a time, lanes striding over the channels of the
//    head (NCH chunks of 32), the logit finished by a full-warp butterfly.
#include <math_constants.h>

#include <type_traits>

#include "common.cuh"

namespace tfg {
namespace {

constexpr int kDotThreads = 256;
// Tuning knobs (compile-time; the defaults are the measured best on GB300).
#ifndef TFG_DOT_UNROLL
#define TFG_DOT_UNROLL 8   // edges gathered per lane per step (key + value rows)
#endif
#ifndef TFG_DOT_MINB
#define TFG_DOT_MINB 2     // resident CTAs per SM asked of the compiler, 16-byte bf16 path
#endif
// (the fp32 path, with half the features per load, keeps 4 in flight: 8 spill there)
template <int VEC>
__host__ __device__ constexpr int dot_unroll() { return VEC >= 8 ? TFG_DOT_UNROLL : 4; }
constexpr int64_t kDotMinWork = 2048;      // edges + rows per CTA, at least
constexpr int kDotMaxChannels = 256;

// Logits are kept in base-2 units: the launcher folds log2(e) into the
// scale once, so every logit, maximum and difference is log2(e) times its
// natural-log value and exp(l - m) = exp2f(l2 - m2) -- the CUDA math
// library's base-2 exponential (documented maximum error 2 ulp over its
// whole range), so the weights' error is set by the fp32 logits alone.
constexpr float kDotLog2e = 1.4426950408889634f;

// 2^(m_old - m_new), with 2^(-inf - anything) = 0 (an empty state has m = -inf).
__device__ __forceinline__ float dot_rescale(float m_old, float m_new) {
    return m_old == -CUDART_INF_F ? 0.f : exp2f(m_old - m_new);
}

struct DotArgs {
    const int32_t *rowptr;
    const int32_t *col;
    const void *q, *k, *v;
    int64_t n;
    int heads, channels;
    float scale;
    float *out;
    float *alpha;
};

// Rows of a work-balanced range (edges + rows split evenly across CTAs),
// taken one at a time by the CTA's warps from a shared counter.
template <typename RowFn>
__device__ __forceinline__ void dot_rows(const int32_t *rowptr, int64_t n, RowFn fn) {
    __shared__ int s_next;
    int64_t r0, r1;
    balanced_rows(rowptr, n, gridDim.x, blockIdx.x, r0, r1);
    if (threadIdx.x == 0) s_next = 0;
    __syncthreads();
    const int lane = threadIdx.x & 31;
    for (;;) {
        int i = 0;
        if (lane == 0) i = atomicAdd(&s_next, 1);
        i = __shfl_sync(kFull, i, 0);
        if (i >= r1 - r0) break;
        fn(r0 + i, lane);
    }
}

// This lane's share of a head's dot product: two interleaved fp32 chains
// through the packed fma (even and odd channels), added at the end.
template <int VEC>
__device__ __forceinline__ float lane_dot(const float (&q)[VEC], const float (&k)[VEC]) {
    if constexpr (VEC % 2 == 0) {
        float2 d = make_float2(0.f, 0.f);
#pragma unroll
        for (int i = 0; i < VEC; i += 2)
            d = fma2(make_float2(q[i], q[i + 1]), make_float2(k[i], k[i + 1]), d);
        return d.x + d.y;
    } else {
        float d = 0.f;
#pragma unroll
        for (int i = 0; i < VEC; ++i) d = fmaf(q[i], k[i], d);
        return d;
    }
}

// part += p * v through the packed fma.
template <int VEC>
__device__ __forceinline__ void axpy_vec(float (&part)[VEC], float p, const float (&v)[VEC]) {
    if constexpr (VEC % 2 == 0) {
        const float2 p2 = make_float2(p, p);
#pragma unroll
        for (int i = 0; i < VEC; i += 2) {
            const float2 r = fma2(make_float2(v[i], v[i + 1]), p2, make_float2(part[i], part[i + 1]));
            part[i] = r.x;
            part[i + 1] = r.y;
        }
    } else {
#pragma unroll
        for (int i = 0; i < VEC; ++i) part[i] = fmaf(p, v[i], part[i]);
    }
}

// LH > 0: lanes per head fixed at compile time (the butterfly unrolls);
// LH = 0 takes lh_arg.
template <typename XT, int VEC, int LPR, int LH>
__device__ __forceinline__ void dot_fast_row(const DotArgs &a, int lh_arg, int64_t t, int lane) {
    const int lh = LH > 0 ? LH : lh_arg;
    using V = VecLoad<XT, VEC>;
    constexpr int G = 32 / LPR;
    constexpr int kDotUnroll = dot_unroll<VEC>();
    // a step's slots j + u * G + g must stay inside one 32-edge chunk: full
    // chunks take no slot test, so a wider step would add edges twice
    static_assert(G * kDotUnroll <= 32 && 32 % (G * kDotUnroll) == 0,
                  "steps of G * kDotUnroll slots must tile the 32-edge chunk");
    const int g = lane / LPR, sub = lane % LPR;
    const int64_t f = static_cast<int64_t>(a.heads) * a.channels;
    const XT *qp = static_cast<const XT *>(a.q);
    const XT *kp = static_cast<const XT *>(a.k);
    const XT *vp = static_cast<const XT *>(a.v);
    const int64_t beg = a.rowptr[t], end = a.col ? a.rowptr[t + 1] : a.rowptr[t];
    for (int64_t ft = 0; ft < f; ft += LPR * VEC) {
        const int64_t f0 = ft + sub * VEC;
        const bool fok = f0 < f;
        const int64_t fl = fok ? f0 : 0;       // lanes past F read (and never store) feature 0
        float qv[VEC];
        V::load(qp + t * f + fl, qv);
        if (!fok) {
#pragma unroll
            for (int q = 0; q < VEC; ++q) qv[q] = 0.f;
        }
        float m = -CUDART_INF_F, den = 0.f, acc[VEC];
#pragma unroll
        for (int q = 0; q < VEC; ++q) acc[q] = 0.f;
        // key and value row slices of node src, addressed in bytes (one wide
        // multiply-add per gather)
        const char *kb = reinterpret_cast<const char *>(kp + fl);
        const char *vb = reinterpret_cast<const char *>(vp + fl);
        const uint32_t row_bytes = static_cast<uint32_t>(f) * static_cast<uint32_t>(sizeof(XT));
        // one 32-edge chunk; FULL chunks (all 32 slots used) skip every slot test
        // c: the chunk's column ids (lane j: edge j; any valid id past cnt)
        auto chunk = [&](auto full_tag, int c, int cnt) {
            constexpr bool FULL = decltype(full_tag)::value;
            float den_part = 0.f, part[VEC];
#pragma unroll
            for (int q = 0; q < VEC; ++q) part[q] = 0.f;
#pragma unroll
            for (int j = 0; j < (FULL ? 32 : cnt); j += G * kDotUnroll) {
                typename V::Raw rk[kDotUnroll], rv[kDotUnroll];
                bool ok[kDotUnroll];
#pragma unroll
                for (int u = 0; u < kDotUnroll; ++u) {
                    const int k = j + u * G + g;
                    const uint64_t off = static_cast<uint64_t>(
                        static_cast<uint32_t>(__shfl_sync(kFull, c, k & 31))) * row_bytes;
                    ok[u] = FULL || k < cnt;
                    rk[u] = ok[u] ? V::raw(reinterpret_cast<const XT *>(kb + off)) : V::zero();
                    rv[u] = ok[u] ? V::raw(reinterpret_cast<const XT *>(vb + off)) : V::zero();
                }
                float l[kDotUnroll];
                float mc = -CUDART_INF_F;
#pragma unroll
                for (int u = 0; u < kDotUnroll; ++u) {
                    float kv[VEC];
                    V::widen(rk[u], kv);
                    float d = lane_dot(qv, kv);
#pragma unroll
                    for (int o = 1; o < lh; o <<= 1) d += __shfl_xor_sync(kFull, d, o);
                    l[u] = ok[u] ? d * a.scale : -CUDART_INF_F;
                    mc = fmaxf(mc, l[u]);
                }
                if (mc > m) {   // new running maximum for this lane's head
                    const float sc = dot_rescale(m, mc);
                    den *= sc;
                    den_part *= sc;
#pragma unroll
                    for (int q = 0; q < VEC; ++q) {
                        acc[q] *= sc;
                        part[q] *= sc;
                    }
                    m = mc;
                }
#pragma unroll
                for (int u = 0; u < kDotUnroll; ++u) {
                    const float p = ok[u] ? exp2f(l[u] - m) : 0.f;
                    den_part += p;
                    float vv[VEC];
                    V::widen(rv[u], vv);
                    axpy_vec(part, p, vv);
                }
            }
            den += den_part;
#pragma unroll
            for (int q = 0; q < VEC; ++q) acc[q] += part[q];
        };
        // the next chunk's column ids are requested before this chunk's rows
        int cnext = (a.col && beg + lane < end) ? ld_stream(a.col + beg + lane) : 0;
        for (int64_t base = beg; base < end; base += 32) {
            const int cnt = static_cast<int>(min64(32, end - base));
            const int c = cnext;
            cnext = (base + 32 + lane < end) ? ld_stream(a.col + base + 32 + lane) : 0;
            if (cnt == 32) chunk(std::true_type{}, c, 32);
            else chunk(std::false_type{}, c, cnt);
        }
        // merge the G groups' states in a fixed butterfly order
#pragma unroll
        for (int s = LPR; s < 32; s <<= 1) {
            const float mo = __shfl_xor_sync(kFull, m, s);
            const float dn = __shfl_xor_sync(kFull, den, s);
            const float mm = fmaxf(m, mo);
            const float x = dot_rescale(m, mm), y = dot_rescale(mo, mm);
            den = den * x + dn * y;
#pragma unroll
            for (int q = 0; q < VEC; ++q) {
                const float ao = __shfl_xor_sync(kFull, acc[q], s);
                acc[q] = acc[q] * x + ao * y;
            }
            m = mm;
        }
        if (lane < LPR && fok) {
            float *o = a.out + t * f + f0;
#pragma unroll
            for (int q = 0; q < VEC; ++q) o[q] = end > beg ? acc[q] / den : 0.f;
        }
        if (a.alpha) {   // recompute each logit; one writer per (edge, head)
            const int h = static_cast<int>(fl / a.channels);
            const int64_t steps = (end - beg + G - 1) / G;   // the same for every lane
            for (int64_t it = 0; it < steps; ++it) {
                const int64_t k = beg + it * G + g;
                const bool ok = k < end;
                const int64_t src = ok ? __ldg(a.col + k) : 0;
                float kv[VEC];
                V::load(kp + src * f + fl, kv);
                float d = lane_dot(qv, kv);
                for (int o = 1; o < lh; o <<= 1) d += __shfl_xor_sync(kFull, d, o);
                if (ok && fok && sub % lh == 0)
                    a.alpha[k * a.heads + h] = exp2f(d * a.scale - m) / den;
            }
        }
    }
}

// General form: one head at a time, lanes over its channels (NCH chunks of 32).
template <typename XT, int NCH>
__device__ __forceinline__ void dot_general_row(const DotArgs &a, int64_t t, int lane) {
    using V1 = VecLoad<XT, 1>;
    const int C = a.channels;
    const int64_t f = static_cast<int64_t>(a.heads) * C;
    const XT *qp = static_cast<const XT *>(a.q);
    const XT *kp = static_cast<const XT *>(a.k);
    const XT *vp = static_cast<const XT *>(a.v);
    const int64_t beg = a.rowptr[t], end = a.col ? a.rowptr[t + 1] : a.rowptr[t];
    for (int h = 0; h < a.heads; ++h) {
        const int64_t hb = static_cast<int64_t>(h) * C;
        float qv[NCH];
#pragma unroll
        for (int j = 0; j < NCH; ++j) {
            const int ch = j * 32 + lane;
            float x[1] = {0.f};
            if (ch < C) V1::load(qp + t * f + hb + ch, x);
            qv[j] = x[0];
        }
        float m = -CUDART_INF_F, den = 0.f, acc[NCH];
#pragma unroll
        for (int j = 0; j < NCH; ++j) acc[j] = 0.f;
        for (int64_t base = beg; base < end; base += 32) {
            const int cnt = static_cast<int>(min64(32, end - base));
            const int c = lane < cnt ? ld_stream(a.col + base + lane) : 0;
            float den_part = 0.f, part[NCH];
#pragma unroll
            for (int j = 0; j < NCH; ++j) part[j] = 0.f;
            for (int e = 0; e < cnt; ++e) {
                const int64_t src = __shfl_sync(kFull, c, e);
                float kv[NCH], vv[NCH];
#pragma unroll
                for (int j = 0; j < NCH; ++j) {
                    const int ch = j * 32 + lane;
                    float x[1] = {0.f}, y[1] = {0.f};
                    if (ch < C) {
                        V1::load(kp + src * f + hb + ch, x);
                        V1::load(vp + src * f + hb + ch, y);
                    }
                    kv[j] = x[0];
                    vv[j] = y[0];
                }
                float d = 0.f;
#pragma unroll
                for (int j = 0; j < NCH; ++j) d = fmaf(qv[j], kv[j], d);
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) d += __shfl_xor_sync(kFull, d, o);
                const float l = d * a.scale;
                if (l > m) {
                    const float sc = dot_rescale(m, l);
                    den *= sc;
                    den_part *= sc;
#pragma unroll
                    for (int j = 0; j < NCH; ++j) {
                        acc[j] *= sc;
                        part[j] *= sc;
                    }
                    m = l;
                }
                const float p = exp2f(l - m);
                den_part += p;
#pragma unroll
                for (int j = 0; j < NCH; ++j) part[j] = fmaf(p, vv[j], part[j]);
            }
            den += den_part;
#pragma unroll
            for (int j = 0; j < NCH; ++j) acc[j] += part[j];
        }
#pragma unroll
        for (int j = 0; j < NCH; ++j) {
            const int ch = j * 32 + lane;
            if (ch < C) a.out[t * f + hb + ch] = end > beg ? acc[j] / den : 0.f;
        }
        if (a.alpha) {
            for (int64_t k = beg; k < end; ++k) {
                const int64_t src = __ldg(a.col + k);
                float d = 0.f;
#pragma unroll
                for (int j = 0; j < NCH; ++j) {
                    const int ch = j * 32 + lane;
                    float x[1] = {0.f};
                    if (ch < C) V1::load(kp + src * f + hb + ch, x);
                    d = fmaf(qv[j], x[0], d);
                }
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) d += __shfl_xor_sync(kFull, d, o);
                if (lane == 0) a.alpha[k * a.heads + h] = exp2f(d * a.scale - m) / den;
            }
        }
    }
}

// 16-byte bf16 rows hold twice the features per gather: two resident CTAs
// per SM leave the registers for kDotUnroll key + value gathers in flight.
template <typename XT, int VEC, int LPR, int LH>
__global__ void __launch_bounds__(kDotThreads, VEC >= 8 ? TFG_DOT_MINB : 3) dot_fast(DotArgs a, int lh) {
    dot_rows(a.rowptr, a.n, [&](int64_t t, int lane) { dot_fast_row<XT, VEC, LPR, LH>(a, lh, t, lane); });
}

template <typename XT, int NCH>
__global__ void __launch_bounds__(kDotThreads, 3) dot_general(DotArgs a) {
    dot_rows(a.rowptr, a.n, [&](int64_t t, int lane) { dot_general_row<XT, NCH>(a, t, lane); });
}

#ifndef TFG_DOT_STATIC_LH
#define TFG_DOT_STATIC_LH 1   // one kernel per lanes-per-head count
#endif

// lh (a power of two <= LPR) picks the kernel with that many lanes per head.
template <typename XT, int VEC, int LPR>
void launch_fast_lpr(const DotArgs &a, int lh, int grid, cudaStream_t s) {
    if constexpr (!TFG_DOT_STATIC_LH) {
        dot_fast<XT, VEC, LPR, 0><<<grid, kDotThreads, 0, s>>>(a, lh);
        return;
    }
    switch (lh) {
        case 1: dot_fast<XT, VEC, LPR, 1><<<grid, kDotThreads, 0, s>>>(a, lh); break;
        case 2: dot_fast<XT, VEC, LPR, 2><<<grid, kDotThreads, 0, s>>>(a, lh); break;
        case 4: dot_fast<XT, VEC, LPR, 4><<<grid, kDotThreads, 0, s>>>(a, lh); break;
        case 8: dot_fast<XT, VEC, LPR, 8><<<grid, kDotThreads, 0, s>>>(a, lh); break;
        default:
            if constexpr (LPR >= 16) {
                if (lh == 16) {
                    dot_fast<XT, VEC, LPR, 16><<<grid, kDotThreads, 0, s>>>(a, lh);
                    break;
                }
            }
            if constexpr (LPR >= 32) dot_fast<XT, VEC, LPR, 32><<<grid, kDotThreads, 0, s>>>(a, lh);
            break;
    }
}

template <typename XT, int VEC>
void launch_fast_vec(const DotArgs &a, int lh, int grid, cudaStream_t s) {
    const int64_t chunks = static_cast<int64_t>(a.heads) * a.channels / VEC;
    if (chunks >= 32 || lh > 16) launch_fast_lpr<XT, VEC, 32>(a, lh, grid, s);
    else if (chunks > 8 || lh > 8) launch_fast_lpr<XT, VEC, 16>(a, lh, grid, s);
    else launch_fast_lpr<XT, VEC, 8>(a, lh, grid, s);
}

template <typename XT>
void launch_general(const DotArgs &a, int grid, cudaStream_t s) {
    const int nch = (a.channels + 31) / 32;
    if (nch <= 1) dot_general<XT, 1><<<grid, kDotThreads, 0, s>>>(a);
    else if (nch <= 2) dot_general<XT, 2><<<grid, kDotThreads, 0, s>>>(a);
    else if (nch <= 4) dot_general<XT, 4><<<grid, kDotThreads, 0, s>>>(a);
    else dot_general<XT, 8><<<grid, kDotThreads, 0, s>>>(a);
}

bool is_pow2_upto32(int x) { return x >= 1 && x <= 32 && (x & (x - 1)) == 0; }

}  // namespace

int dot_softmax_max_channels() { return kDotMaxChannels; }

cudaError_t launch_dot_softmax(const int32_t *rowptr, const int32_t *col, const void *q,
                               const void *k, const void *v, int x_dtype, int64_t n, int64_t e,
                               int heads, int channels, float scale, float *out, float *alpha,
                               cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const DotArgs a{rowptr, col, q, k, v, n, heads, channels, scale * kDotLog2e, out, alpha};
    const int grid = balanced_grid(n, e, kDotMinWork);
    auto a16 = [](const void *p) { return reinterpret_cast<uintptr_t>(p) % 16 == 0; };
    const bool aligned = a16(q) && a16(k) && a16(v) && a16(out);
    const int vec = x_dtype == TFG_BF16 ? 8 : 4;
    if (aligned && channels % vec == 0 && is_pow2_upto32(channels / vec)) {
        if (x_dtype == TFG_BF16) launch_fast_vec<uint16_t, 8>(a, channels / 8, grid, s);
        else launch_fast_vec<float, 4>(a, channels / 4, grid, s);
    } else {
        if (x_dtype == TFG_BF16) launch_general<uint16_t>(a, grid, s);
        else launch_general<float>(a, grid, s);
    }
    return cudaGetLastError();
}

}  // namespace tfg
