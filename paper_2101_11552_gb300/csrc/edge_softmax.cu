// Edge-softmax (GAT) aggregation: the map-reduce workflow of tf_geometric
// Fig. 5a (Section 2.1.2) fused with the attention-weighted sum it feeds.
//
//   node scores  s_src[n,h] = <x[n,h,:], a_src[h,:]>, s_dst likewise  (prologue)
//   map          l = LeakyReLU(s_src[src,h] + s_dst[t,h])
//   reduce       m = max over row t of l; den = sum over row t of exp(l - m)
//   map          alpha = exp(l - m) / den
//   aggregate    out[t,h,:] = sum over row t of alpha * x[src,h,:]
//
// The paper's workflow runs map, reduce and map as separate passes over the
// edges.  Here one warp owns a target row and makes a single pass with the
// running-maximum form of the softmax: when an edge raises the row maximum m
// of a head, the running denominator and weighted sum are rescaled by
// exp(m_old - m_new), which leaves alpha and out mathematically unchanged.
// A row is split among G = 32 / LPR lane groups (each group covers LPR * VEC
// features and takes every G-th edge); the groups' (m, den, acc) triples are
// merged by a butterfly at the end.  Sums are blocked per 32-edge chunk to
// keep fp32 chains short.  Every lane of a head evaluates the same logits in
// the same order, so the lanes agree and results are deterministic.  With
// alpha requested, a second pass over the row writes the normalised weights.
//
// Logits are kept in base-2 units: the node scores are multiplied by log2(e)
// once, and since LeakyReLU(c v) = c LeakyReLU(v) for c > 0 every logit,
// maximum and difference is log2(e) times its natural-log value, so
// exp(l - m) = exp2f(l2 - m2).  exp2f is the CUDA math library's base-2
// exponential (documented maximum error 2 ulp over its whole range), so the
// relative error of each weight is set by the fp32 rounding of the logits,
// not by an approximate exponential.
#include <math_constants.h>

#include <mutex>
#include <type_traits>

#include "common.cuh"

namespace tfg {
namespace {

constexpr int kSmThreads = 256;
#ifndef TFG_SM_UNROLL
#define TFG_SM_UNROLL 4   // gathers in flight per lane (tuning knob)
#endif
constexpr int kSmUnroll = TFG_SM_UNROLL;   // fast kernel
// 1: the next chunk's column ids are requested one chunk ahead; 2: also its
// node scores s_src, gathered while this chunk's rows are summed (measured on
// the 114.6M-edge graph: 2.29 ms with 2, 2.40-2.50 ms with 1, 2.44-2.57 ms with 0)
#ifndef TFG_SM_PREFETCH
#define TFG_SM_PREFETCH 2
#endif
#ifndef TFG_SM_FULL_CHUNKS
#define TFG_SM_FULL_CHUNKS 1   // separate code for full 32-edge chunks (no slot tests)
#endif
constexpr bool kSmFullChunks = TFG_SM_FULL_CHUNKS != 0;
constexpr int kGenUnroll = 4;               // generic kernel
constexpr float kLog2e = 1.4426950408889634f;   // log2(e): natural-log units -> base-2 units

// Compensated dot product (the "Dot2" scheme of Ogita, Rump and Oishi,
// "Accurate sum and dot product", SIAM J. Sci. Comput. 2005): each product
// is split exactly into p + e with one fma, each running sum into s + e with
// the error-free two-sum, and the collected errors are added at the end.  The
// result is as accurate as a dot product in twice the working precision,
// rounded once -- node scores feed every logit, so their error would become a
// relative error in every attention weight.
struct Dot2 {
    float s = 0.f, c = 0.f;
    __device__ __forceinline__ void add(float a, float b) {
        const float p = a * b;
        const float pe = fmaf(a, b, -p);       // a * b = p + pe exactly
        const float t = s + p;
        const float z = t - s;
        const float se = (s - (t - z)) + (p - z);  // s + p = t + se exactly
        s = t;
        c += pe + se;
    }
    __device__ __forceinline__ float value() const { return s + c; }
};

template <typename XT>
__global__ void node_scores(const XT *__restrict__ x, int64_t n, int heads, int channels,
                            const float *__restrict__ a_src, const float *__restrict__ a_dst,
                            float *__restrict__ s_src, float *__restrict__ s_dst) {
    const int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (i >= n * heads) return;
    const int64_t v = i / heads;
    const int h = static_cast<int>(i % heads);
    const XT *xr = x + v * heads * channels + static_cast<int64_t>(h) * channels;
    const float *as = a_src + h * channels, *ad = a_dst + h * channels;
    Dot2 a, b;
    for (int c = 0; c < channels; ++c) {
        float xv[1];
        VecLoad<XT, 1>::load(xr + c, xv);
        a.add(xv[0], __ldg(as + c));
        b.add(xv[0], __ldg(ad + c));
    }
    s_src[i] = a.value() * kLog2e;
    s_dst[i] = b.value() * kLog2e;
}

__device__ __forceinline__ float leaky(float v, float slope) { return v > 0.f ? v : slope * v; }

// 2^(m_old - m_new) for base-2 maxima, with 2^(-inf - anything) = 0 (an
// empty group has m = -inf).
__device__ __forceinline__ float rescale(float m_old, float m_new) {
    return m_old == -CUDART_INF_F ? 0.f : exp2f(m_old - m_new);
}

template <typename XT, int VEC, int LPR>
__device__ __forceinline__ void generic_row(const int32_t *__restrict__ rowptr,
                                            const int32_t *__restrict__ col,
                                            const XT *__restrict__ x, int heads, int channels,
                                            float slope, const float *__restrict__ s_src,
                                            const float *__restrict__ s_dst,
                                            float *__restrict__ out, float *__restrict__ alpha,
                                            int64_t t, int lane) {
    using V = VecLoad<XT, VEC>;
    constexpr int G = 32 / LPR;
    const int g = lane / LPR, sub = lane % LPR;
    const int64_t f = static_cast<int64_t>(heads) * channels;
    const int64_t beg = rowptr[t], end = col ? rowptr[t + 1] : rowptr[t];
    for (int64_t ft = 0; ft < f; ft += LPR * VEC) {
        const int64_t f0 = ft + sub * VEC;
        const bool fok = f0 < f;
        const int h = fok ? static_cast<int>(f0 / channels) : 0;
        const float sd = __ldg(s_dst + t * heads + h);

        float m = -CUDART_INF_F, den = 0.f;
        float acc[VEC];
#pragma unroll
        for (int q = 0; q < VEC; ++q) acc[q] = 0.f;
        for (int64_t base = beg; base < end; base += 32) {
            const int cnt = static_cast<int>(min64(32, end - base));
            const int c = lane < cnt ? ld_stream(col + base + lane) : 0;
            float den_part = 0.f, part[VEC];
#pragma unroll
            for (int q = 0; q < VEC; ++q) part[q] = 0.f;
            for (int j = 0; j < cnt; j += G * kGenUnroll) {
                float l[kGenUnroll];
                typename V::Raw raw[kGenUnroll];
#pragma unroll
                for (int u = 0; u < kGenUnroll; ++u) {
                    const int k = j + u * G + g;
                    const int src = __shfl_sync(kFull, c, k & 31);
                    const bool ok = k < cnt;
                    l[u] = ok ? leaky(__ldg(s_src + static_cast<int64_t>(src) * heads + h) + sd, slope)
                              : -CUDART_INF_F;
                    raw[u] = (ok && fok) ? V::raw(x + static_cast<int64_t>(src) * f + f0) : V::zero();
                }
#pragma unroll
                for (int u = 0; u < kGenUnroll; ++u) {
                    if (l[u] == -CUDART_INF_F) continue;   // empty slot
                    if (l[u] > m) {                        // new running maximum
                        const float sc = rescale(m, l[u]);
                        den *= sc;
                        den_part *= sc;
#pragma unroll
                        for (int q = 0; q < VEC; ++q) {
                            acc[q] *= sc;
                            part[q] *= sc;
                        }
                        m = l[u];
                    }
                    const float p = exp2f(l[u] - m);
                    den_part += p;
                    float v[VEC];
                    V::widen(raw[u], v);
#pragma unroll
                    for (int q = 0; q < VEC; ++q) part[q] = fmaf(p, v[q], part[q]);
                }
            }
            den += den_part;
#pragma unroll
            for (int q = 0; q < VEC; ++q) acc[q] += part[q];
        }
        // merge the G groups: (m, den, acc) in a fixed butterfly order
#pragma unroll
        for (int s = LPR; s < 32; s <<= 1) {
            const float mo = __shfl_xor_sync(kFull, m, s);
            const float dn = __shfl_xor_sync(kFull, den, s);
            const float mm = fmaxf(m, mo);
            const float a = rescale(m, mm), b = rescale(mo, mm);
            den = den * a + dn * b;
#pragma unroll
            for (int q = 0; q < VEC; ++q) {
                const float ao = __shfl_xor_sync(kFull, acc[q], s);
                acc[q] = acc[q] * a + ao * b;
            }
            m = mm;
        }
        if (lane < LPR && fok) {
            float *o = out + t * f + f0;
#pragma unroll
            for (int q = 0; q < VEC; ++q) o[q] = end > beg ? acc[q] / den : 0.f;
        }
        // normalised attention weights, one writer per (edge, head)
        if (alpha && lane < LPR && fok && (f0 % channels) == 0) {
            for (int64_t k = beg; k < end; ++k) {
                const int src = __ldg(col + k);
                const float l = leaky(__ldg(s_src + static_cast<int64_t>(src) * heads + h) + sd, slope);
                alpha[k * heads + h] = exp2f(l - m) / den;
            }
        }
    }
}

// Fast form for the common layout: H divides 32, every lane's VEC features
// lie in one head, and one feature tile covers the row (F <= LPR * VEC).
// One pass over the row in 32-edge chunks:
//  * score lanes: lane (se, sh) = (lane / H, lane % H) evaluates the logit of
//    edge slot se and head sh -- each (edge, head) logit and exponential is
//    computed once.  The chunk's maximum per head (butterfly over the lanes
//    of a head) updates the running maximum m; when m rises, the sums so far
//    are rescaled by exp(m_old - m_new) (a warp-uniform branch, taken a few
//    times per row).  p = exp(l - m) then feeds the denominator.
//  * feature lanes: group g = lane / LPR gathers every G-th edge, fetches the
//    p of its (edge, head) from the score lane holding it with one shuffle,
//    and accumulates p * x into fp32 per-chunk partials.
template <typename XT, int VEC, int LPR, int H>
__device__ __forceinline__ void fast_row(const int32_t *__restrict__ rowptr,
                                         const int32_t *__restrict__ col,
                                         const XT *__restrict__ x, int channels, float slope,
                                         const float *__restrict__ s_src,
                                         const float *__restrict__ s_dst, float *__restrict__ out,
                                         float *__restrict__ alpha, int64_t t, int lane) {
    using V = VecLoad<XT, VEC>;
    constexpr int G = 32 / LPR;     // edges per feature step
    constexpr int ES = 32 / H;      // edges per score step
    constexpr int R = 32 / ES;      // score steps per 32-edge chunk (= H)
    static_assert(ES % G == 0, "score step must hold whole feature steps");
    // a step's slots e + u * G + g must stay inside one 32-edge chunk (full
    // chunks take no slot test, and p[k0 / ES] must stay inside p[R])
    static_assert(G * kSmUnroll <= 32 && 32 % (G * kSmUnroll) == 0,
                  "steps of G * kSmUnroll slots must tile the 32-edge chunk");
    const int se = lane / H, sh = lane % H;
    const int g = lane / LPR, sub = lane % LPR;
    const int f = H * channels;
    const int f0 = sub * VEC;
    const bool fok = f0 < f;
    const int fh = fok ? f0 / channels : 0;
    const char *xb = reinterpret_cast<const char *>(x + (fok ? f0 : 0));
    const uint32_t row_bytes = static_cast<uint32_t>(f) * static_cast<uint32_t>(sizeof(XT));
    // row slice of node src, addressed in bytes (one wide multiply-add per gather)
    auto gather = [&](uint32_t src) {
        return V::raw(reinterpret_cast<const XT *>(xb + static_cast<uint64_t>(src) * row_bytes));
    };
    const int64_t beg = rowptr[t], end = col ? rowptr[t + 1] : rowptr[t];
    const float sd = __ldg(s_dst + t * H + sh);

    // one pass over the row, 32 edges at a time: the score lanes form the
    // chunk's logits, the running maximum m of each head absorbs the chunk's
    // maximum (earlier sums are rescaled by exp(m_old - m_new) when it rises),
    // then p = exp(l - m) weights the chunk's gathered rows
    float m = -CUDART_INF_F, den = 0.f, acc[VEC];
#pragma unroll
    for (int q = 0; q < VEC; ++q) acc[q] = 0.f;
#if TFG_SM_PREFETCH
    int cnext = 0;   // the next chunk's column ids (lane j: edge j of that chunk)
#endif
#if TFG_SM_PREFETCH >= 2
    float sv[R];     // s_src of the chunk about to run, for (edge r * ES + se, head sh)
#endif
    // one 32-edge chunk with its column ids in c (lane j: edge base + j; any
    // valid id past cnt); FULL chunks (all 32 slots used) skip every slot test
    auto chunk = [&](auto full_tag, int c, int cnt) {
        constexpr bool FULL = decltype(full_tag)::value;
        // the first step's row gathers need only the column ids: issue them
        // before the scores so that their latency overlaps the score work
        typename V::Raw raw0[kSmUnroll];
#pragma unroll
        for (int u = 0; u < kSmUnroll; ++u)
            raw0[u] = gather(static_cast<uint32_t>(__shfl_sync(kFull, c, (u * G + g) & 31)));
        float p[R];
        float cm = -CUDART_INF_F;
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int k = r * ES + se;
#if TFG_SM_PREFETCH >= 2
            const float ss = sv[r];                  // gathered during the previous chunk
#else
            const float ss = __ldg(s_src + static_cast<int64_t>(__shfl_sync(kFull, c, k)) * H + sh);
#endif
            p[r] = (FULL || k < cnt) ? leaky(ss + sd, slope) : -CUDART_INF_F;
            cm = fmaxf(cm, p[r]);
        }
#pragma unroll
        for (int o = H; o < 32; o <<= 1) cm = fmaxf(cm, __shfl_xor_sync(kFull, cm, o));
        const bool rises = cm > m;
        if (__any_sync(kFull, rises)) {   // warp-uniform; rare after the first chunks
            const float sc = rises ? (m == -CUDART_INF_F ? 0.f : exp2f(m - cm)) : 1.f;
            den *= sc;
            const float fsc = __shfl_sync(kFull, sc, fh);   // lane fh scores head fh
#pragma unroll
            for (int q = 0; q < VEC; ++q) acc[q] *= fsc;
            m = fmaxf(m, cm);
        }
        float den_part = 0.f;
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int k = r * ES + se;
            p[r] = (FULL || k < cnt) ? exp2f(p[r] - m) : 0.f;
            den_part += p[r];
        }
        den += den_part;
#if TFG_SM_PREFETCH >= 2
        // the next chunk's node scores, requested before this chunk's rows
#pragma unroll
        for (int r = 0; r < R; ++r)
            sv[r] = __ldg(s_src + static_cast<int64_t>(__shfl_sync(kFull, cnext, r * ES + se)) * H + sh);
#endif
        float part[VEC];
#pragma unroll
        for (int q = 0; q < VEC; ++q) part[q] = 0.f;
#pragma unroll
        for (int e = 0; e < 32; e += G * kSmUnroll) {
            if (!FULL && e >= cnt) break;   // warp-uniform
            typename V::Raw raw[kSmUnroll];
            float pw[kSmUnroll];
#pragma unroll
            for (int u = 0; u < kSmUnroll; ++u) {
                const int k0 = e + u * G;              // edge of group 0 in this step
                const int k = k0 + g;
                // p of (edge k, head fh) sits in lane (k % ES) * H + fh, register k / ES
                pw[u] = __shfl_sync(kFull, p[k0 / ES], ((k0 % ES) + g) * H + fh);
                if (e == 0) raw[u] = raw0[u];
                else raw[u] = gather(static_cast<uint32_t>(__shfl_sync(kFull, c, k & 31)));
            }
#pragma unroll
            for (int u = 0; u < kSmUnroll; ++u) {
                float v[VEC];
                V::widen(raw[u], v);
                if constexpr (VEC % 2 == 0) {
                    const float2 w2 = make_float2(pw[u], pw[u]);
#pragma unroll
                    for (int q = 0; q < VEC; q += 2) {
                        const float2 r2 = fma2(make_float2(v[q], v[q + 1]), w2,
                                               make_float2(part[q], part[q + 1]));
                        part[q] = r2.x;
                        part[q + 1] = r2.y;
                    }
                } else {
#pragma unroll
                    for (int q = 0; q < VEC; ++q) part[q] = fmaf(pw[u], v[q], part[q]);
                }
            }
        }
#pragma unroll
        for (int q = 0; q < VEC; ++q) acc[q] += part[q];
    };
#if TFG_SM_PREFETCH
    // the next chunk's column ids are requested before this chunk's rows
    cnext = (col && beg + lane < end) ? ld_stream(col + beg + lane) : 0;
#endif
#if TFG_SM_PREFETCH >= 2
#pragma unroll
    for (int r = 0; r < R; ++r)
        sv[r] = __ldg(s_src + static_cast<int64_t>(__shfl_sync(kFull, cnext, r * ES + se)) * H + sh);
#endif
    for (int64_t base = beg; base < end; base += 32) {
        const int cnt = static_cast<int>(min64(32, end - base));
#if TFG_SM_PREFETCH
        const int c = cnext;
        cnext = (base + 32 + lane < end) ? ld_stream(col + base + 32 + lane) : 0;
#else
        const int c = lane < cnt ? ld_stream(col + base + lane) : 0;
#endif
        if (kSmFullChunks && cnt == 32) chunk(std::true_type{}, c, 32);
        else chunk(std::false_type{}, c, cnt);
    }
#pragma unroll
    for (int o = H; o < 32; o <<= 1) den += __shfl_xor_sync(kFull, den, o);
#pragma unroll
    for (int o = LPR; o < 32; o <<= 1)
#pragma unroll
        for (int q = 0; q < VEC; ++q) acc[q] += __shfl_xor_sync(kFull, acc[q], o);
    const float dh = __shfl_sync(kFull, den, fh);   // lane fh holds head fh's denominator
    if (lane < LPR && fok) {
        float *o = out + t * f + f0;
#pragma unroll
        for (int q = 0; q < VEC; ++q) o[q] = end > beg ? acc[q] / dh : 0.f;
    }
    if (alpha) {
        for (int64_t base = beg; base < end; base += 32) {
            const int cnt = static_cast<int>(min64(32, end - base));
            const int c = lane < cnt ? __ldg(col + base + lane) : 0;
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const int k = r * ES + se;
                const int src = __shfl_sync(kFull, c, k);
                if (k < cnt) {
                    const float l = leaky(__ldg(s_src + static_cast<int64_t>(src) * H + sh) + sd, slope);
                    alpha[(base + k) * H + sh] = exp2f(l - m) / den;
                }
            }
        }
    }
}

// ---------------------------------------------------------------------------
// Merge-path form of the fast kernel (same layout conditions).  The work is
// split as in aggregate_mp_kernel: whole rows per CTA, an equal number of
// edges + row ends per warp inside it, so a hub row is shared by the warps it
// spans; the next chunk's column ids are loaded before this chunk is
// gathered.  A warp's part of a row is the running state (m, den, acc) of
// fast_row; the owner of a row begun by earlier warps merges their parts and
// its own in warp order after the CTA's one barrier:
//   m = max(m1, m2),  den = den1 2^(m1 - m) + den2 2^(m2 - m),  acc likewise.
// ---------------------------------------------------------------------------
#ifndef TFG_SM_MP
#define TFG_SM_MP 1          // 0: the fast layout takes softmax_fast (side-by-side timing)
#endif
#ifndef TFG_SMP_BLOCKS
#define TFG_SMP_BLOCKS 3     // resident CTAs per SM
#endif
constexpr int kSmpBlocks = TFG_SMP_BLOCKS;
// Measured: on the 169,343-node graph (mean in-degree 6.9) the merge-path form
// takes 0.24 ms against 0.26 ms; on the 114.6M-edge graph (mean 492) 3.15 ms
// against 2.62 ms for softmax_fast, whose per-row work is already balanced
// by its long rows.  Graphs with a mean in-degree below this take it.
constexpr int64_t kSmpMaxDegree = 32;
constexpr int kSmWarps = kSmThreads / 32;

// (M, D, A) absorbs another part (m2, d2, a2) of the same row and head.
template <int VEC>
__device__ __forceinline__ void merge_state(float &M, float &D, float (&A)[VEC], float m2,
                                            float d2, const float *a2) {
    const float mn = fmaxf(M, m2);
    const float sa = M == -CUDART_INF_F ? 0.f : exp2f(M - mn);
    const float sb = m2 == -CUDART_INF_F ? 0.f : exp2f(m2 - mn);
    D = D * sa + d2 * sb;
#pragma unroll
    for (int q = 0; q < VEC; ++q) A[q] = A[q] * sa + (a2 ? a2[q] * sb : 0.f);
    M = mn;
}

template <typename XT, int VEC, int LPR, int H>
struct SmMp {
    using V = VecLoad<XT, VEC>;
    static constexpr int G = 32 / LPR;     // edges per feature step
    static constexpr int ES = 32 / H;      // edges per score step
    static constexpr int R = 32 / ES;      // score steps per 32-edge chunk (= H)
    static constexpr int kF = LPR * VEC;
    static_assert(ES % G == 0, "score step must hold whole feature steps");
    static_assert(G * kSmUnroll <= 32 && 32 % (G * kSmUnroll) == 0,
                  "steps of G * kSmUnroll slots must tile the 32-edge chunk");

    // One chunk of up to 32 edges of one row (ids in c, lane j holds edge j):
    // the logits of the chunk (score lanes), the running maximum, then the
    // weighted rows (feature lanes), exactly as in fast_row.
    static __device__ __forceinline__ void chunk(const XT *xf, uint32_t fs,
                                                 const float *__restrict__ s_src, float sd,
                                                 float slope, int c, int cnt, int lane, int fh,
                                                 float &m, float &den, float (&acc)[VEC]) {
        const int se = lane / H, sh = lane % H, g = lane / LPR;
        typename V::Raw raw0[kSmUnroll];
#pragma unroll
        for (int u = 0; u < kSmUnroll; ++u) {
            const uint32_t src = static_cast<uint32_t>(__shfl_sync(kFull, c, u * G + g));
            raw0[u] = V::raw(xf + static_cast<uint64_t>(src) * fs);
        }
        float p[R];
        float cm = -CUDART_INF_F;
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int k = r * ES + se;
            const uint32_t src = static_cast<uint32_t>(__shfl_sync(kFull, c, k));
            p[r] = k < cnt ? leaky(__ldg(s_src + static_cast<uint64_t>(src) * H + sh) + sd, slope)
                           : -CUDART_INF_F;
            cm = fmaxf(cm, p[r]);
        }
#pragma unroll
        for (int o = H; o < 32; o <<= 1) cm = fmaxf(cm, __shfl_xor_sync(kFull, cm, o));
        const bool rises = cm > m;
        if (__any_sync(kFull, rises)) {   // warp-uniform; rare after the first chunks
            const float sc = rises ? (m == -CUDART_INF_F ? 0.f : exp2f(m - cm)) : 1.f;
            den *= sc;
            const float fsc = __shfl_sync(kFull, sc, fh);   // lane fh scores head fh
#pragma unroll
            for (int q = 0; q < VEC; ++q) acc[q] *= fsc;
            m = fmaxf(m, cm);
        }
        float den_part = 0.f;
#pragma unroll
        for (int r = 0; r < R; ++r) {
            const int k = r * ES + se;
            p[r] = k < cnt ? exp2f(p[r] - m) : 0.f;
            den_part += p[r];
        }
        den += den_part;
        float part[VEC];
#pragma unroll
        for (int q = 0; q < VEC; ++q) part[q] = 0.f;
#pragma unroll
        for (int e = 0; e < 32; e += G * kSmUnroll) {
            if (e >= cnt) break;   // warp-uniform
            typename V::Raw raw[kSmUnroll];
            float pw[kSmUnroll];
#pragma unroll
            for (int u = 0; u < kSmUnroll; ++u) {
                const int k0 = e + u * G;              // edge of group 0 in this step
                // p of (edge k0 + g, head fh) sits in lane ((k0 + g) % ES) * H + fh, register k0 / ES
                pw[u] = __shfl_sync(kFull, p[k0 / ES], ((k0 % ES) + g) * H + fh);
                if (e == 0) {
                    raw[u] = raw0[u];
                } else {
                    const uint32_t src = static_cast<uint32_t>(__shfl_sync(kFull, c, k0 + g));
                    raw[u] = V::raw(xf + static_cast<uint64_t>(src) * fs);
                }
            }
#pragma unroll
            for (int u = 0; u < kSmUnroll; ++u) {
                float v[VEC];
                V::widen(raw[u], v);
                if constexpr (VEC % 2 == 0) {
                    const float2 w2 = make_float2(pw[u], pw[u]);
#pragma unroll
                    for (int q = 0; q < VEC; q += 2) {
                        const float2 r2 = fma2(make_float2(v[q], v[q + 1]), w2,
                                               make_float2(part[q], part[q + 1]));
                        part[q] = r2.x;
                        part[q + 1] = r2.y;
                    }
                } else {
#pragma unroll
                    for (int q = 0; q < VEC; ++q) part[q] = fmaf(pw[u], v[q], part[q]);
                }
            }
        }
#pragma unroll
        for (int q = 0; q < VEC; ++q) acc[q] += part[q];
    }

    // Normalised weights of every edge of row t, given the row's final
    // maximum M and denominator D of this lane's score head.
    static __device__ void write_alpha(const int32_t *__restrict__ rowptr,
                                       const int32_t *__restrict__ col,
                                       const float *__restrict__ s_src, float sd, float slope,
                                       float M, float D, float *__restrict__ alpha, int32_t t,
                                       int lane) {
        const int se = lane / H, sh = lane % H;
        const int32_t beg = __ldg(rowptr + t), end = __ldg(rowptr + t + 1);
        for (int32_t base = beg; base < end; base += 32) {
            const int cnt = min(32, end - base);
            const int c = lane < cnt ? __ldg(col + base + lane) : 0;
#pragma unroll
            for (int r = 0; r < R; ++r) {
                const int k = r * ES + se;
                const uint32_t src = static_cast<uint32_t>(__shfl_sync(kFull, c, k));
                if (k < cnt) {
                    const float l = leaky(__ldg(s_src + static_cast<uint64_t>(src) * H + sh) + sd, slope);
                    alpha[(static_cast<int64_t>(base) + k) * H + sh] = exp2f(l - M) / D;
                }
            }
        }
    }
};

template <typename XT, int VEC, int LPR, int H>
__global__ void __launch_bounds__(kSmThreads, kSmpBlocks)
softmax_mp(const int32_t *__restrict__ rowptr, const int32_t *__restrict__ col,
           const XT *__restrict__ x, int64_t n, int channels, float slope,
           const float *__restrict__ s_src, const float *__restrict__ s_dst,
           float *__restrict__ out, float *__restrict__ alpha) {
    using S = SmMp<XT, VEC, LPR, H>;
    constexpr int kF = S::kF;
    __shared__ float s_tacc[kSmWarps][kF], s_hacc[kSmWarps][kF];
    __shared__ float s_tm[kSmWarps][H], s_tden[kSmWarps][H], s_hm[kSmWarps][H], s_hden[kSmWarps][H];
    __shared__ int32_t s_tail_row[kSmWarps], s_head_row[kSmWarps];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sh = lane % H, sub = lane % LPR;
    const int f = H * channels;
    const int f0 = sub * VEC;
    const bool fok = f0 < f;
    const int fh = fok ? f0 / channels : 0;
    const XT *xf = x + (fok ? f0 : 0);
    const uint32_t fs = static_cast<uint32_t>(f);

    // node ids and edge positions fit int32 (the ABI caps N and E below 2^31)
    int64_t r0l, r1l;
    balanced_rows(rowptr, n, gridDim.x, blockIdx.x, r0l, r1l);
    const int32_t r0 = static_cast<int32_t>(r0l), r1 = static_cast<int32_t>(r1l);
    const int64_t q0 = static_cast<int64_t>(__ldg(rowptr + r0)) + r0;
    const int64_t q1 = static_cast<int64_t>(__ldg(rowptr + r1)) + r1;
    const int64_t per = (q1 - q0 + kSmWarps - 1) / kSmWarps;
    const int64_t qa = min64(q1, q0 + warp * per), qb = min64(q1, qa + per);
    const int32_t ta = last_row_at(rowptr, r0, r1, qa);
    const int32_t tb = last_row_at(rowptr, ta, r1, qb);
    const int32_t ka = static_cast<int32_t>(qa - ta), kb = static_cast<int32_t>(qb - tb);
    const bool head_split = ka > __ldg(rowptr + ta);   // row ta begun by an earlier warp
    if (lane == 0) s_head_row[warp] = -1;

    float m = -CUDART_INF_F, den = 0.f, acc[VEC];
#pragma unroll
    for (int q = 0; q < VEC; ++q) acc[q] = 0.f;
    int32_t t = ta, k = ka;                            // this warp's edges are [ka, kb)
    int32_t rend = t < tb ? __ldg(rowptr + t + 1) : kb;
    float sd = t < n ? __ldg(s_dst + static_cast<int64_t>(t) * H + sh) : 0.f;
    int cnext = (col && k + lane < kb) ? __ldg(col + k + lane) : 0;
    for (;;) {
        while (k >= rend) {                            // row t has no edges left here
            if (t >= tb) break;
#pragma unroll
            for (int o = H; o < 32; o <<= 1) den += __shfl_xor_sync(kFull, den, o);
#pragma unroll
            for (int o = LPR; o < 32; o <<= 1)
#pragma unroll
                for (int q = 0; q < VEC; ++q) acc[q] += __shfl_xor_sync(kFull, acc[q], o);
            if (t == ta && head_split) {               // parts of it sit with earlier warps
                if (lane < H) {
                    s_hm[warp][lane] = m;
                    s_hden[warp][lane] = den;
                }
                if (lane < LPR) {
#pragma unroll
                    for (int q = 0; q < VEC; ++q) s_hacc[warp][f0 + q] = acc[q];
                }
                if (lane == 0) s_head_row[warp] = t;
            } else {
                const float dh = __shfl_sync(kFull, den, fh);   // lane fh: head fh's denominator
                const bool any = __ldg(rowptr + t + 1) > __ldg(rowptr + t);
                if (lane < LPR && fok) {
                    float *o = out + static_cast<int64_t>(t) * f + f0;
#pragma unroll
                    for (int q = 0; q < VEC; ++q) o[q] = any ? acc[q] / dh : 0.f;
                }
                if (alpha && any) S::write_alpha(rowptr, col, s_src, sd, slope, m, den, alpha, t, lane);
            }
            m = -CUDART_INF_F;
            den = 0.f;
#pragma unroll
            for (int q = 0; q < VEC; ++q) acc[q] = 0.f;
            ++t;
            rend = t < tb ? __ldg(rowptr + t + 1) : kb;
            sd = t < n ? __ldg(s_dst + static_cast<int64_t>(t) * H + sh) : 0.f;
        }
        if (k >= rend) break;                          // t == tb and its edges are done
        const int cnt = min(32, rend - k);
        const int c = cnext;
        const int32_t kn = k + cnt;                    // the next chunk starts here
        cnext = (kn + lane < kb) ? __ldg(col + kn + lane) : 0;
        S::chunk(xf, fs, s_src, sd, slope, c, cnt, lane, fh, m, den, acc);
        k = kn;
    }
    // this warp's part of row tb (empty when the range ends on a row end)
#pragma unroll
    for (int o = H; o < 32; o <<= 1) den += __shfl_xor_sync(kFull, den, o);
#pragma unroll
    for (int o = LPR; o < 32; o <<= 1)
#pragma unroll
        for (int q = 0; q < VEC; ++q) acc[q] += __shfl_xor_sync(kFull, acc[q], o);
    if (lane < H) {
        s_tm[warp][lane] = m;
        s_tden[warp][lane] = den;
    }
    if (lane < LPR) {
#pragma unroll
        for (int q = 0; q < VEC; ++q) s_tacc[warp][f0 + q] = acc[q];
    }
    if (lane == 0) s_tail_row[warp] = tb;
    __syncthreads();
    const int32_t hr = s_head_row[warp];
    if (hr < 0) return;
    // earlier warps' parts in warp order, then ours: (Ms, Ds) for the score
    // head sh, (Mf, Df, A) for the feature head fh
    float Ms = -CUDART_INF_F, Ds = 0.f, Mf = -CUDART_INF_F, Df = 0.f, A[VEC];
    float none[1] = {0.f};
#pragma unroll
    for (int q = 0; q < VEC; ++q) A[q] = 0.f;
    for (int w = 0; w < warp; ++w) {
        if (s_tail_row[w] != hr) continue;
        merge_state<1>(Ms, Ds, none, s_tm[w][sh], s_tden[w][sh], nullptr);
        merge_state<VEC>(Mf, Df, A, s_tm[w][fh], s_tden[w][fh], &s_tacc[w][fok ? f0 : 0]);
    }
    merge_state<1>(Ms, Ds, none, s_hm[warp][sh], s_hden[warp][sh], nullptr);
    merge_state<VEC>(Mf, Df, A, s_hm[warp][fh], s_hden[warp][fh], &s_hacc[warp][fok ? f0 : 0]);
    if (lane < LPR && fok) {
        float *o = out + static_cast<int64_t>(hr) * f + f0;
#pragma unroll
        for (int q = 0; q < VEC; ++q) o[q] = A[q] / Df;   // a split row has edges
    }
    if (alpha) {
        const float sdr = __ldg(s_dst + static_cast<int64_t>(hr) * H + sh);
        S::write_alpha(rowptr, col, s_src, sdr, slope, Ms, Ds, alpha, hr, lane);
    }
}

template <typename XT, int VEC, int LPR>
__global__ void __launch_bounds__(kSmThreads, 3)
softmax_aggregate(const int32_t *__restrict__ rowptr, const int32_t *__restrict__ col,
                  const XT *__restrict__ x, int64_t n, int heads, int channels, float slope,
                  const float *__restrict__ s_src, const float *__restrict__ s_dst,
                  float *__restrict__ out, float *__restrict__ alpha) {
    for_each_row(rowptr, n, [&](int64_t t, int lane) {
        generic_row<XT, VEC, LPR>(rowptr, col, x, heads, channels, slope, s_src, s_dst, out,
                                  alpha, t, lane);
    });
}

// Measured on the 114.6M-edge graph (bf16, 8 heads x 16), ids and scores
// requested one chunk ahead: 3 CTAs per SM with 4 gathers in flight per lane
// 2.29 ms; 4 CTAs 2.31 ms; 3 CTAs with 8 in flight 2.52 ms.  Without the
// early requests: 4 CTAs / 4 in flight 2.44-2.50 ms, 3 / 8 2.62 ms, 2 / 8 3.48 ms.
#ifndef TFG_SMF_BLOCKS
#define TFG_SMF_BLOCKS 3     // resident CTAs per SM of softmax_fast
#endif

template <typename XT, int VEC, int LPR, int H>
__global__ void __launch_bounds__(kSmThreads, TFG_SMF_BLOCKS)
softmax_fast(const int32_t *__restrict__ rowptr, const int32_t *__restrict__ col,
             const XT *__restrict__ x, int64_t n, int channels, float slope,
             const float *__restrict__ s_src, const float *__restrict__ s_dst,
             float *__restrict__ out, float *__restrict__ alpha) {
    for_each_row(rowptr, n, [&](int64_t t, int lane) {
        fast_row<XT, VEC, LPR, H>(rowptr, col, x, channels, slope, s_src, s_dst, out, alpha, t,
                                  lane);
    });
}

constexpr int64_t kSmMinWork = 2048;   // edges + rows per CTA, at least

size_t align256(size_t b) { return (b + 255) & ~size_t(255); }

// Launch the fast form when the layout allows it; false means "use the generic one".
template <typename XT, int VEC, int LPR>
bool launch_fast_lpr(const int32_t *rowptr, const int32_t *col, const void *x, int64_t n, int64_t e,
                     int heads, int channels, float slope, const float *s_src, const float *s_dst,
                     float *out, float *alpha, cudaStream_t s) {
    constexpr int G = 32 / LPR;
    const int grid = balanced_grid(n, e, kSmMinWork);
    const XT *xp = static_cast<const XT *>(x);
    const int mp_grid = static_cast<int>(min64(n, static_cast<int64_t>(sm_count()) * kSmpBlocks));
#define TFG_FAST(HH)                                                                              \
    if (heads == HH) {                                                                            \
        if constexpr ((32 / HH) % G == 0) {                                                       \
            if (TFG_SM_MP && e < kSmpMaxDegree * n)                                              \
                softmax_mp<XT, VEC, LPR, HH><<<mp_grid, kSmThreads, 0, s>>>(                      \
                    rowptr, col, xp, n, channels, slope, s_src, s_dst, out, alpha);               \
            else                                                                                  \
                softmax_fast<XT, VEC, LPR, HH><<<grid, kSmThreads, 0, s>>>(                       \
                    rowptr, col, xp, n, channels, slope, s_src, s_dst, out, alpha);               \
            return true;                                                                          \
        }                                                                                         \
        return false;                                                                             \
    }
    TFG_FAST(1)
    TFG_FAST(2)
    TFG_FAST(4)
    TFG_FAST(8)
    TFG_FAST(16)
#undef TFG_FAST
    return false;
}

template <typename XT, int VEC>
bool launch_fast(const int32_t *rowptr, const int32_t *col, const void *x, int64_t n, int64_t e,
                 int heads, int channels, float slope, const float *s_src, const float *s_dst,
                 float *out, float *alpha, cudaStream_t s) {
    const int64_t f = static_cast<int64_t>(heads) * channels;
    if (channels % VEC != 0 || f > 32 * VEC) return false;
    const int64_t chunks = f / VEC;
    if (chunks > 16) return launch_fast_lpr<XT, VEC, 32>(rowptr, col, x, n, e, heads, channels, slope, s_src, s_dst, out, alpha, s);
    if (chunks > 8) return launch_fast_lpr<XT, VEC, 16>(rowptr, col, x, n, e, heads, channels, slope, s_src, s_dst, out, alpha, s);
    return launch_fast_lpr<XT, VEC, 8>(rowptr, col, x, n, e, heads, channels, slope, s_src, s_dst, out, alpha, s);
}

template <typename XT, int VEC>
void launch_main(const int32_t *rowptr, const int32_t *col, const void *x, int64_t n, int64_t e,
                 int heads, int channels, float slope, const float *s_src, const float *s_dst,
                 float *out, float *alpha, cudaStream_t s) {
    const int64_t chunks = static_cast<int64_t>(heads) * channels / VEC;
    const int grid = balanced_grid(n, e, kSmMinWork);
    const XT *xp = static_cast<const XT *>(x);
    if (chunks >= 32)
        softmax_aggregate<XT, VEC, 32><<<grid, kSmThreads, 0, s>>>(rowptr, col, xp, n, heads, channels,
                                                                   slope, s_src, s_dst, out, alpha);
    else if (chunks > 8)
        softmax_aggregate<XT, VEC, 16><<<grid, kSmThreads, 0, s>>>(rowptr, col, xp, n, heads, channels,
                                                                   slope, s_src, s_dst, out, alpha);
    else
        softmax_aggregate<XT, VEC, 8><<<grid, kSmThreads, 0, s>>>(rowptr, col, xp, n, heads, channels,
                                                                  slope, s_src, s_dst, out, alpha);
}

// Scratch of tfg_edge_softmax_aggregate_noalloc: the node scores s_src and
// s_dst of up to kNoAllocNodeHeads (node, head) pairs each, 16 MiB in all,
// resident on every GPU that loads the library for as long as it stays
// loaded.  Every call overwrites the part it uses, so nothing needs clearing.
constexpr int64_t kNoAllocNodeHeads = int64_t(1) << 21;
static __device__ __align__(256) float g_noalloc_scores[2 * kNoAllocNodeHeads];

}  // namespace

int64_t noalloc_softmax_max_node_heads() { return kNoAllocNodeHeads; }

// Device address of the scratch array on the current device.  Host code
// cannot use the array's name as a device pointer, so the address is looked
// up once per device with that device current (the lookup may load the
// module, which is why the first call on a device must not be captured into
// a CUDA graph) and cached.
cudaError_t noalloc_softmax_scratch(void **ptr, size_t *bytes) {
    constexpr int kMaxDevices = 64;
    static std::mutex mu;
    static void *addr[kMaxDevices] = {};
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    if (addr[dev] == nullptr) {
        void *p = nullptr;
        err = cudaGetSymbolAddress(&p, g_noalloc_scores);
        if (err != cudaSuccess) return err;
        addr[dev] = p;
    }
    *ptr = addr[dev];
    *bytes = sizeof(g_noalloc_scores);
    return cudaSuccess;
}

cudaError_t launch_node_scores(const void *x, int x_dtype, int64_t n, int heads, int channels,
                               const float *a_src, const float *a_dst, float *s_src, float *s_dst,
                               cudaStream_t s) {
    const int sgrid = ceil_div(n * heads, 256);
    if (x_dtype == TFG_BF16)
        node_scores<uint16_t><<<sgrid, 256, 0, s>>>(static_cast<const uint16_t *>(x), n, heads,
                                                    channels, a_src, a_dst, s_src, s_dst);
    else
        node_scores<float><<<sgrid, 256, 0, s>>>(static_cast<const float *>(x), n, heads, channels,
                                                 a_src, a_dst, s_src, s_dst);
    return cudaGetLastError();
}

size_t softmax_workspace_bytes(int64_t n, int heads) {
    return 2 * align256(sizeof(float) * size_t(n > 0 ? n : 1) * size_t(heads));
}

cudaError_t launch_edge_softmax(const int32_t *rowptr, const int32_t *col, const void *x,
                                int x_dtype, int64_t n, int64_t e, int heads, int channels,
                                const float *a_src, const float *a_dst, float slope, float *out,
                                float *alpha, void *ws, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    float *s_src = static_cast<float *>(ws);
    float *s_dst = reinterpret_cast<float *>(static_cast<char *>(ws) +
                                             align256(sizeof(float) * size_t(n) * size_t(heads)));
    const int sgrid = ceil_div(n * heads, 256);
    const bool aligned = (reinterpret_cast<uintptr_t>(x) % 16 == 0) &&
                         (reinterpret_cast<uintptr_t>(out) % 16 == 0);
    if (x_dtype == TFG_BF16) {
        node_scores<uint16_t><<<sgrid, 256, 0, s>>>(static_cast<const uint16_t *>(x), n, heads,
                                                    channels, a_src, a_dst, s_src, s_dst);
        if (aligned && channels % 8 == 0) {
            if (!launch_fast<uint16_t, 8>(rowptr, col, x, n, e, heads, channels, slope, s_src, s_dst, out, alpha, s))
                launch_main<uint16_t, 8>(rowptr, col, x, n, e, heads, channels, slope, s_src, s_dst, out, alpha, s);
        } else {
            launch_main<uint16_t, 1>(rowptr, col, x, n, e, heads, channels, slope, s_src, s_dst, out, alpha, s);
        }
    } else {
        node_scores<float><<<sgrid, 256, 0, s>>>(static_cast<const float *>(x), n, heads, channels,
                                                 a_src, a_dst, s_src, s_dst);
        if (aligned && channels % 4 == 0) {
            if (!launch_fast<float, 4>(rowptr, col, x, n, e, heads, channels, slope, s_src, s_dst, out, alpha, s))
                launch_main<float, 4>(rowptr, col, x, n, e, heads, channels, slope, s_src, s_dst, out, alpha, s);
        } else {
            launch_main<float, 1>(rowptr, col, x, n, e, heads, channels, slope, s_src, s_dst, out, alpha, s);
        }
    }
    return cudaGetLastError();
}

}  // namespace tfg
