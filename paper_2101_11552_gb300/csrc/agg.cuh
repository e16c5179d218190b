// Fused gather * weight * reduce over a CSR grouped by target: the message
// aggregation of tf_geometric (Fig. 1) with the reducer of Fig. 5b, which the
// paper implements as tf.math.unsorted_segment_* over the edge list
// (Section 2.1.2).  Grouping by target first turns the scatter-reduce into
// owner-computes row reductions: no atomics, a fixed summation order, and
// bit-identical results from run to run.
//
// Work layout
//  * A CTA (8 warps) owns a contiguous range of target rows holding an equal
//    share of edges + rows (a merge-path split of rowptr), so a hub row does
//    not leave one CTA running long after the others.  Its warps take rows
//    one at a time from a shared counter.  A row is split among
//    G = 32 / LPR lane groups: each group of LPR lanes covers LPR * VEC
//    features (16-byte loads when the layout allows) and takes every G-th
//    edge of the row; the groups' partials are then combined by a butterfly.
//  * Rows longer than kHeavyDeg (power-law hubs) are set aside and done after
//    the light rows by the whole CTA: each warp takes one contiguous slice of
//    the row, and the eight warp partials are combined in warp order through
//    shared memory.  No global scratch and no inter-CTA waiting.
//  * Column ids (and weights) of 32 edges are loaded by the 32 lanes at once
//    and broadcast with shuffles; kUnroll gathers are kept in flight per lane.
//  * GCN mode without w_csr forms the weight on the fly:  out[t] = dinv[t] *
//    (sum_k dinv[col[k]] * x[col[k]] + fill * dinv[t] * x[t]), so no per-edge
//    weight array is read.  With w_csr it adds fill * dinv[t]^2 * x[t] to the
//    weighted sum.
//  * APPNP mode (one propagation step, Klicpera et al., the APPNP model the
//    paper lists in Section 2.2 and Table 1) is GCN mode with an epilogue:
//    out[t] = (1 - alpha) * gcn(h)[t] + alpha * x0[t], x0 read in its own
//    storage type X0T.  alpha = 0 is one SGC step.
//
// Shared by aggregate.cu (one-hop entry points) and propagate.cu (multi-hop);
// each translation unit instantiates the variants it launches.
#pragma once
#include <math_constants.h>

#include "common.cuh"

namespace tfg {
namespace {

constexpr int kAggWarps = 8;
constexpr int kAggThreads = kAggWarps * 32;
// Tuning knobs (compile-time; the defaults are the measured best on GB300).
#ifndef TFG_HEAVY_DEG
#define TFG_HEAVY_DEG 2048
#endif
#ifndef TFG_AGG_UNROLL
#define TFG_AGG_UNROLL 4
#endif
#ifndef TFG_AGG_MINB
#define TFG_AGG_MINB 4   // resident CTAs per SM asked of the compiler, 16-byte bf16 path
#endif
constexpr int kHeavyDeg = TFG_HEAVY_DEG;
constexpr int kMaxHeavy = 64;   // hub rows a CTA sets aside; more are done warp by warp
// gathers in flight per lane: deeper for the 16-byte bf16 sum path (measured
// faster there), 4 elsewhere (keeps the other variants free of spills)
template <int VEC, bool IS_MAX>
constexpr int unroll_for() { return (VEC >= 8 && !IS_MAX) ? TFG_AGG_UNROLL : 4; }

struct AggArgs {
    const int32_t *rowptr;
    const int32_t *col;
    const float *w;     // CSR-order weights or null (sum / mean / max)
    const float *dinv;  // GCN mode
    const void *x;
    float *out;
    int64_t n;
    int64_t f;
    int mean;
    int add_self;
    float fill;
    const void *x0;     // APPNP mode: the teleport features x0 [N, F]
    float alpha;        // APPNP mode: teleport weight
    float beta;         // APPNP mode: 1 - alpha, rounded once on the host
    int regime;         // kRegimeAny, or the degree regime the launched kernel serves
};

#ifndef TFG_MP_F32_DEGREE
#define TFG_MP_F32_DEGREE 32   // mean in-degree splitting the fp32 sum regimes
#endif
constexpr int kRegimeAny = 0;      // the kernel runs whatever the degree
constexpr int kRegimeShort = 1;    // runs only when E < TFG_MP_F32_DEGREE * N
constexpr int kRegimeLong = 2;     // runs only when E >= TFG_MP_F32_DEGREE * N

// True when a kernel launched for one degree regime finds the graph in the
// other (the same answer in every thread: the caller returns before any
// barrier).
__device__ __forceinline__ bool other_regime(const int32_t *rowptr, int64_t n, int regime,
                                             int64_t degree) {
    if (regime == kRegimeAny) return false;
    const bool short_rows = static_cast<int64_t>(__ldg(rowptr + n)) < degree * n;
    return short_rows != (regime == kRegimeShort);
}

enum Kind { kSumLike = 0, kMax = 1, kGcn = 2, kAppnp = 3 };

// The layouts whose launch splits by degree regime: fp32 sums in 16-byte slices.
template <typename XT, int VEC, int KIND>
constexpr bool kSplitsRegimes = sizeof(XT) == 4 && VEC == 4 && KIND != kMax;

template <typename XT, int VEC, int LPR, int KIND, typename X0T = XT>
struct Agg {
    static constexpr int G = 32 / LPR;
    static constexpr bool kIsMax = KIND == kMax;
    static constexpr bool kGcnLike = KIND == kGcn || KIND == kAppnp;
    static constexpr int kUnroll = unroll_for<VEC, kIsMax>();
    // a step's slots j + u * G + g must stay inside one 32-edge chunk: full
    // chunks take no slot test, so a wider step would add edges twice
    static_assert(G * kUnroll <= 32 && 32 % (G * kUnroll) == 0,
                  "steps of G * kUnroll slots must tile the 32-edge chunk");

    static __device__ __forceinline__ float identity() { return kIsMax ? -CUDART_INF_F : 0.f; }

    static __device__ __forceinline__ float combine(float a, float b) {
        return kIsMax ? fmaxf(a, b) : a + b;
    }

    // part[q] += w * v[q] for one gathered vector (pairs through fma2).
    static __device__ __forceinline__ void axpy(float (&part)[VEC], float w,
                                                const typename VecLoad<XT, VEC>::Raw &raw) {
        float v[VEC];
        VecLoad<XT, VEC>::widen(raw, v);
        if constexpr (VEC % 2 == 0) {
            const float2 w2 = make_float2(w, w);
#pragma unroll
            for (int q = 0; q < VEC; q += 2) {
                const float2 r = fma2(make_float2(v[q], v[q + 1]), w2, make_float2(part[q], part[q + 1]));
                part[q] = r.x;
                part[q + 1] = r.y;
            }
        } else {
#pragma unroll
            for (int q = 0; q < VEC; ++q) part[q] = fmaf(w, v[q], part[q]);
        }
    }

    // One 32-edge chunk of a sum: group g takes edges g, g + G, ...  FULL
    // chunks need no bounds checks; in a partial chunk the slots past cnt get
    // weight 0 and read row 0 (always valid), contributing an exact zero.
    // Lanes whose features lie past F read the row's first features instead
    // (in bounds); their partials are never stored.
    template <bool FULL>
    static __device__ __forceinline__ void sum_chunk(const XT *xf, uint32_t fs, int c, float ww,
                                                     int cnt, int g, bool weighted,
                                                     float (&part)[VEC]) {
        using V = VecLoad<XT, VEC>;
        for (int j = 0; j < (FULL ? 32 : cnt); j += G * kUnroll) {
            typename V::Raw raw[kUnroll];
            float wt[kUnroll];
            // all row gathers first (they need only the column ids), then the
            // weights, whose loads may still be in flight
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int k = j + u * G + g;
                const uint32_t src = static_cast<uint32_t>(__shfl_sync(kFull, c, k & 31));
                raw[u] = V::raw(xf + static_cast<uint64_t>(src) * fs);
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int k = j + u * G + g;
                wt[u] = weighted ? __shfl_sync(kFull, ww, k & 31) : 1.f;
                if (!FULL && k >= cnt) wt[u] = 0.f;
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) axpy(part, wt[u], raw[u]);
        }
    }

    // Accumulate edges [beg, end) into acc (this lane's VEC features at f0).
    // Each 32-edge chunk is summed into its own partial before it is added to
    // acc, so an fp32 chain is at most 32 / G + deg / 32 additions long.  The
    // order is fixed, so results are deterministic.
    static __device__ __forceinline__ void edges(const AggArgs &a, int64_t beg, int64_t end,
                                                 int64_t f0, bool fok, float (&acc)[VEC],
                                                 int lane) {
        using V = VecLoad<XT, VEC>;
        const XT *x = static_cast<const XT *>(a.x);
        const XT *xf = x + (fok ? f0 : 0);
        const uint32_t fs = static_cast<uint32_t>(a.f);
        const int g = lane / LPR;
        const bool weighted = kGcnLike || a.w != nullptr;
        if (a.col == nullptr) return;   // a graph without edges
        for (int64_t base = beg; base < end; base += 32) {
            const int cnt = static_cast<int>(min64(32, end - base));
            int c = 0;
            float ww = 1.f;
            if (lane < cnt) {
                c = ld_stream(a.col + base + lane);
                if (a.w) ww = ld_stream(a.w + base + lane);
                else if (kGcnLike) ww = __ldg(a.dinv + c);
            }
            if constexpr (kIsMax) {
                for (int j = 0; j < cnt; j += G * kUnroll) {
                    typename V::Raw raw[kUnroll];
                    float wt[kUnroll];
                    bool ok[kUnroll];
#pragma unroll
                    for (int u = 0; u < kUnroll; ++u) {
                        const int k = j + u * G + g;
                        const uint32_t src = static_cast<uint32_t>(__shfl_sync(kFull, c, k & 31));
                        wt[u] = weighted ? __shfl_sync(kFull, ww, k & 31) : 1.f;
                        ok[u] = fok && (k < cnt);
                        raw[u] = ok[u] ? V::raw(xf + static_cast<uint64_t>(src) * fs) : V::zero();
                    }
#pragma unroll
                    for (int u = 0; u < kUnroll; ++u) {
                        if (!ok[u]) continue;
                        float v[VEC];
                        V::widen(raw[u], v);
#pragma unroll
                        for (int q = 0; q < VEC; ++q) acc[q] = fmaxf(acc[q], wt[u] * v[q]);
                    }
                }
            } else {
                float part[VEC];
#pragma unroll
                for (int q = 0; q < VEC; ++q) part[q] = 0.f;
                if (cnt == 32) sum_chunk<true>(xf, fs, c, ww, cnt, g, weighted, part);
                else sum_chunk<false>(xf, fs, c, ww, cnt, g, weighted, part);
#pragma unroll
                for (int q = 0; q < VEC; ++q) acc[q] += part[q];
            }
        }
    }

    static __device__ __forceinline__ void reduce_groups(float (&acc)[VEC]) {
#pragma unroll
        for (int s = LPR; s < 32; s <<= 1)
#pragma unroll
            for (int q = 0; q < VEC; ++q) acc[q] = combine(acc[q], __shfl_xor_sync(kFull, acc[q], s));
    }

    // Final value of one feature of row t from its reduced accumulator.
    static __device__ __forceinline__ float finish(const AggArgs &a, int64_t t, int64_t deg,
                                                   float acc, float xt, float dt, float x0t) {
        if (kGcnLike) {
            float r;
            if (a.w) r = a.add_self ? acc + (a.fill * dt) * dt * xt : acc;
            else r = a.add_self ? dt * (acc + a.fill * dt * xt) : dt * acc;
            if (KIND == kAppnp) r = fmaf(a.alpha, x0t, a.beta * r);
            return r;
        }
        if (deg == 0) return 0.f;
        if (a.mean) return acc / static_cast<float>(deg);
        return acc;
    }

    static __device__ void warp_row(const AggArgs &a, int64_t t, int lane) {
        const int64_t beg = a.rowptr[t], end = a.rowptr[t + 1];
        const int sub = lane % LPR;
        const float dt = kGcnLike ? __ldg(a.dinv + t) : 1.f;
        for (int64_t ft = 0; ft < a.f; ft += LPR * VEC) {
            const int64_t f0 = ft + sub * VEC;
            const bool fok = f0 < a.f;
            float acc[VEC];
#pragma unroll
            for (int q = 0; q < VEC; ++q) acc[q] = identity();
            edges(a, beg, end, f0, fok, acc, lane);
            reduce_groups(acc);
            if (lane < LPR && fok) {
                float xt[VEC], x0t[VEC];
#pragma unroll
                for (int q = 0; q < VEC; ++q) xt[q] = x0t[q] = 0.f;
                if (kGcnLike && a.add_self)
                    VecLoad<XT, VEC>::load(static_cast<const XT *>(a.x) + t * a.f + f0, xt);
                if (KIND == kAppnp)
                    VecLoad<X0T, VEC>::load(static_cast<const X0T *>(a.x0) + t * a.f + f0, x0t);
                float *o = a.out + t * a.f + f0;
                float r[VEC];
#pragma unroll
                for (int q = 0; q < VEC; ++q)
                    r[q] = finish(a, t, end - beg, acc[q], xt[q], dt, x0t[q]);
                if constexpr (VEC % 4 == 0) {
#pragma unroll
                    for (int q = 0; q < VEC; q += 4)
                        *reinterpret_cast<float4 *>(o + q) = make_float4(r[q], r[q + 1], r[q + 2], r[q + 3]);
                } else {
#pragma unroll
                    for (int q = 0; q < VEC; ++q) o[q] = r[q];
                }
            }
        }
    }

    // A hub row done by all warps of the CTA; partials combined in warp order.
    static __device__ void cta_row(const AggArgs &a, int64_t t, float *s_part) {
        const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, sub = lane % LPR;
        const int64_t beg = a.rowptr[t], end = a.rowptr[t + 1], deg = end - beg;
        const int64_t per = ((deg + kAggWarps - 1) / kAggWarps + 31) / 32 * 32;
        const int64_t wb = min(end, beg + warp * per), we = min(end, wb + per);
        const float dt = kGcnLike ? __ldg(a.dinv + t) : 1.f;
        constexpr int kSlots = LPR * VEC;
        for (int64_t ft = 0; ft < a.f; ft += kSlots) {
            const int64_t f0 = ft + sub * VEC;
            const bool fok = f0 < a.f;
            float acc[VEC];
#pragma unroll
            for (int q = 0; q < VEC; ++q) acc[q] = identity();
            edges(a, wb, we, f0, fok, acc, lane);
            reduce_groups(acc);
            if (lane < LPR) {
#pragma unroll
                for (int q = 0; q < VEC; ++q) s_part[warp * kSlots + sub * VEC + q] = acc[q];
            }
            __syncthreads();
            for (int i = threadIdx.x; i < kSlots; i += kAggThreads) {
                const int64_t fi = ft + i;
                if (fi < a.f) {
                    float r = s_part[i];
                    for (int w = 1; w < kAggWarps; ++w) r = combine(r, s_part[w * kSlots + i]);
                    float one[1] = {0.f}, x0t[1] = {0.f};
                    if (kGcnLike && a.add_self)
                        VecLoad<XT, 1>::load(static_cast<const XT *>(a.x) + t * a.f + fi, one);
                    if (KIND == kAppnp)
                        VecLoad<X0T, 1>::load(static_cast<const X0T *>(a.x0) + t * a.f + fi, x0t);
                    a.out[t * a.f + fi] = finish(a, t, deg, r, one[0], dt, x0t[0]);
                }
            }
            __syncthreads();
        }
    }
};

template <typename XT, int VEC, int LPR, int KIND, typename X0T>
__global__ void __launch_bounds__(kAggThreads, VEC >= 8 ? TFG_AGG_MINB : 4) aggregate_kernel(AggArgs a) {
    using A = Agg<XT, VEC, LPR, KIND, X0T>;
    __shared__ int s_next, s_nheavy;
    __shared__ int64_t s_heavy[kMaxHeavy];
    __shared__ float s_part[kAggWarps * LPR * VEC];
    if constexpr (kSplitsRegimes<XT, VEC, KIND>) {
        if (other_regime(a.rowptr, a.n, a.regime, TFG_MP_F32_DEGREE)) return;
    }
    int64_t r0, r1;
    balanced_rows(a.rowptr, a.n, gridDim.x, blockIdx.x, r0, r1);
    const int64_t nrows = r1 - r0;
    if (threadIdx.x == 0) {
        s_next = 0;
        s_nheavy = 0;
    }
    __syncthreads();
    const int lane = threadIdx.x & 31;
    for (;;) {
        int i = 0;
        if (lane == 0) i = atomicAdd(&s_next, 1);
        i = __shfl_sync(kFull, i, 0);
        if (i >= nrows) break;
        const int64_t t = r0 + i;
        if (a.col != nullptr && a.rowptr[t + 1] - a.rowptr[t] > kHeavyDeg) {
            int slot = 0;
            if (lane == 0) slot = atomicAdd(&s_nheavy, 1);
            slot = __shfl_sync(kFull, slot, 0);
            if (slot < kMaxHeavy) {
                if (lane == 0) s_heavy[slot] = t;
                continue;
            }
        }
        A::warp_row(a, t, lane);
    }
    __syncthreads();
    const int nh = min(s_nheavy, kMaxHeavy);
    for (int h = 0; h < nh; ++h) A::cta_row(a, s_heavy[h], s_part);
}

// ---------------------------------------------------------------------------
// Merge-path kernel for rows that fit one feature tile (F <= LPR * VEC).
//
//  * A persistent grid of mp_blocks CTAs per SM.  CTA b owns whole rows, an
//    equal share of rows + edges (balanced_rows).  Inside the CTA the same
//    split is made again at the granularity of edges: warp w takes the
//    items [qa, qb) of the CTA's merge coordinates Q(t) = rowptr[t] + t, so
//    each warp gets an equal number of edges + row ends whatever the degree
//    distribution, and a hub row is shared by as many warps as it needs.
//  * A warp walks its range row by row in chunks of up to 32 edges; the next
//    chunk's column ids are loaded before this chunk's rows are gathered,
//    kMpDepth 16-byte gathers are in flight per lane.
//  * A row that a warp finishes is written at once, unless earlier warps hold
//    parts of it: then its owner (the warp holding its last edge) parks its
//    own part in shared memory, and after the CTA's one barrier adds the
//    earlier warps' parts and its own in warp order and writes the row.  No
//    global scratch, one barrier per CTA, a fixed summation order.
// ---------------------------------------------------------------------------
#ifndef TFG_AGG_MP
#define TFG_AGG_MP 1       // 0: every layout takes aggregate_kernel (for side-by-side timing)
#endif
// Measured on the 114.6M-edge graph (bf16, F = 128, ids and weights staged in
// shared memory): GCN 1.82 ms at 4 CTAs per SM and 4 gathers in flight per
// lane (3 CTAs and 8 in flight: 1.84 ms; 2 CTAs and 16: 2.06 ms; the
// row-per-warp aggregate_kernel: 1.95 ms); max 2.84 ms (aggregate_kernel
// 3.34 ms).  bf16 rows as 8-byte slices (4 features per lane, up to 16 in
// flight) measured 1.90-3.04 ms.
// fp32 rows (16-byte slices of 4 features) depend on the degree.  On the
// same graph in fp32 (mean in-degree 493) the GCN sum takes 2.99-3.04 ms in
// aggregate_kernel against 3.15-3.31 ms here, at 2-4 CTAs per SM and 4-8 in
// flight; max takes 3.35 ms here against 4.32 ms.  On graphs of mean
// in-degree 4-8 (2,708 nodes F = 64; 169,343 nodes F = 128; 1,024 molecule
// graphs F = 128) this kernel is 21-38% faster for sums and 26-42% for max.
// So fp32 max always comes here, and an fp32 sum launches both kernels with
// a degree regime: each reads E = rowptr[N] and returns at once unless the
// mean in-degree E / N is on its side of TFG_MP_F32_DEGREE (the entry points
// are not given E on the host, and reading it back would stall the stream).
#ifndef TFG_MP_BLOCKS
#define TFG_MP_BLOCKS 4    // resident CTAs per SM for sums (64 registers per thread)
#endif
#ifndef TFG_MP_DEPTH
#define TFG_MP_DEPTH 4     // 16-byte gathers in flight per lane for sums
#endif
template <bool IS_MAX>
constexpr int mp_blocks() { return IS_MAX ? 4 : TFG_MP_BLOCKS; }
template <int VEC, bool IS_MAX>
constexpr int mp_depth() { return IS_MAX ? 4 : TFG_MP_DEPTH; }


template <typename XT, int VEC, int LPR, int KIND, typename X0T>
struct MpAgg {
    using A = Agg<XT, VEC, LPR, KIND, X0T>;
    using V = VecLoad<XT, VEC>;
    static constexpr int G = 32 / LPR;
    static constexpr int kSlots = 32 / G;                       // edges of a group per chunk
    static constexpr int kDepth = kSlots < mp_depth<VEC, A::kIsMax>() ? kSlots
                                                                      : mp_depth<VEC, A::kIsMax>();
    static constexpr int kF = LPR * VEC;
    static_assert(G * kDepth <= 32 && kSlots % kDepth == 0 && kDepth % 2 == 0,
                  "batches of kDepth slots (pairs) must tile a group's slots of the chunk");

    // Write the finished row t from the lane groups' reduced accumulator.
    static __device__ __forceinline__ void store_row(const AggArgs &a, int64_t t,
                                                     const float (&acc)[VEC], int64_t f0,
                                                     bool fok, int lane) {
        if (lane >= LPR || !fok) return;
        const int64_t deg = static_cast<int64_t>(a.rowptr[t + 1]) - a.rowptr[t];
        const float dt = A::kGcnLike ? __ldg(a.dinv + t) : 1.f;
        float xt[VEC], x0t[VEC];
#pragma unroll
        for (int q = 0; q < VEC; ++q) xt[q] = x0t[q] = 0.f;
        if (A::kGcnLike && a.add_self)
            V::load(static_cast<const XT *>(a.x) + t * a.f + f0, xt);
        if (KIND == kAppnp)
            VecLoad<X0T, VEC>::load(static_cast<const X0T *>(a.x0) + t * a.f + f0, x0t);
        float *o = a.out + t * a.f + f0;
        float r[VEC];
#pragma unroll
        for (int q = 0; q < VEC; ++q) r[q] = A::finish(a, t, deg, acc[q], xt[q], dt, x0t[q]);
        if constexpr (VEC % 4 == 0) {
#pragma unroll
            for (int q = 0; q < VEC; q += 4)
                *reinterpret_cast<float4 *>(o + q) = make_float4(r[q], r[q + 1], r[q + 2], r[q + 3]);
        } else {
#pragma unroll
            for (int q = 0; q < VEC; ++q) o[q] = r[q];
        }
    }

    // Row slice of node src: byte offsets (one wide multiply-add per gather).
    static __device__ __forceinline__ typename V::Raw gather(const char *xb, uint32_t row_bytes,
                                                            uint32_t src) {
        return V::raw(reinterpret_cast<const XT *>(xb + static_cast<uint64_t>(src) * row_bytes));
    }

    // Slot of edge k of a chunk in the warp's staging buffer: each lane group's
    // edges k = i * G + g sit at g * kSlots + i, so a group reads the
    // (id, weight) pairs of two consecutive edges with one 16-byte load.
    static __device__ __forceinline__ int stage_slot(int k) { return (k % G) * kSlots + k / G; }

    // One chunk of a sum: edges [k, k + cnt) of one row.  Lane j stages the id
    // and weight of edge k + j (weight 0 past cnt, so those slots add an exact
    // zero from a valid row); each group then reads its edges' pairs two at a
    // time from shared memory instead of two shuffles per edge.
    static __device__ __forceinline__ void chunk_sum(const char *xb, uint32_t row_bytes,
                                                     float2 *stage, int c, float ww, int cnt,
                                                     int lane, int g, float (&part)[VEC]) {
        __syncwarp();                                      // the previous chunk's reads are done
        stage[stage_slot(lane)] = make_float2(__int_as_float(c), lane < cnt ? ww : 0.f);
        __syncwarp();
        const float4 *mine = reinterpret_cast<const float4 *>(stage + g * kSlots);
#pragma unroll
        for (int j = 0; j < kSlots; j += kDepth) {
            if (j * G >= cnt) break;                       // warp-uniform
            typename V::Raw raw[kDepth];
            float wt[kDepth];
#pragma unroll
            for (int u = 0; u < kDepth; u += 2) {
                const float4 cw = mine[(j + u) / 2];       // (id, w) of slots j + u, j + u + 1
                raw[u] = gather(xb, row_bytes, static_cast<uint32_t>(__float_as_int(cw.x)));
                raw[u + 1] = gather(xb, row_bytes, static_cast<uint32_t>(__float_as_int(cw.z)));
                wt[u] = cw.y;
                wt[u + 1] = cw.w;
            }
#pragma unroll
            for (int u = 0; u < kDepth; ++u) A::axpy(part, wt[u], raw[u]);
        }
    }

    // One chunk of a max: edges [k, k + cnt) of one row, column ids in c
    // (lane j holds the id of edge k + j), per-edge weights in ww.
    static __device__ __forceinline__ void chunk(const XT *xf, uint32_t fs, int c, float ww,
                                                 int cnt, int g, bool fok, float (&part)[VEC]) {
#pragma unroll
        for (int j = 0; j < kSlots; j += kDepth) {
            if (j * G >= cnt) break;                       // warp-uniform
            typename V::Raw raw[kDepth];
#pragma unroll
            for (int u = 0; u < kDepth; ++u) {
                const int k = (j + u) * G + g;
                const uint32_t src = static_cast<uint32_t>(__shfl_sync(kFull, c, k));
                raw[u] = V::raw(xf + static_cast<uint64_t>(src) * fs);
            }
#pragma unroll
            for (int u = 0; u < kDepth; ++u) {
                const int k = (j + u) * G + g;
                float wt = __shfl_sync(kFull, ww, k);   // ww = 1 without weights
                if constexpr (A::kIsMax) {
                    if (k < cnt && fok) {
                        float v[VEC];
                        V::widen(raw[u], v);
#pragma unroll
                        for (int q = 0; q < VEC; ++q) part[q] = fmaxf(part[q], wt * v[q]);
                    }
                } else {
                    if (k >= cnt) wt = 0.f;
                    A::axpy(part, wt, raw[u]);
                }
            }
        }
    }
};

template <typename XT, int VEC, int LPR, int KIND, typename X0T>
__global__ void __launch_bounds__(kAggThreads, mp_blocks<KIND == kMax>()) aggregate_mp_kernel(AggArgs a) {
    using M = MpAgg<XT, VEC, LPR, KIND, X0T>;
    using A = typename M::A;
    constexpr int kF = M::kF;
    __shared__ float s_tail[kAggWarps][kF];    // each warp's part of its last, unfinished row
    __shared__ float s_head[kAggWarps][kF];    // an owner's own part of a row begun by others
    __shared__ int32_t s_tail_row[kAggWarps], s_head_row[kAggWarps];
    __shared__ __align__(16) float2 s_stage[kAggWarps][32];   // a chunk's (id, weight) pairs
    if constexpr (kSplitsRegimes<XT, VEC, KIND>) {
        if (other_regime(a.rowptr, a.n, a.regime, TFG_MP_F32_DEGREE)) return;
    }
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int g = lane / LPR, sub = lane % LPR;
    const int64_t f0 = static_cast<int64_t>(sub) * VEC;
    const bool fok = f0 < a.f;
    const XT *xf = static_cast<const XT *>(a.x) + (fok ? f0 : 0);
    const uint32_t fs = static_cast<uint32_t>(a.f);
    const char *xb = reinterpret_cast<const char *>(xf);
    const uint32_t row_bytes = fs * static_cast<uint32_t>(sizeof(XT));

    // node ids and edge positions fit int32 (the ABI caps N and E below 2^31)
    int64_t r0l, r1l;
    balanced_rows(a.rowptr, a.n, gridDim.x, blockIdx.x, r0l, r1l);
    const int32_t r0 = static_cast<int32_t>(r0l), r1 = static_cast<int32_t>(r1l);
    const int64_t q0 = static_cast<int64_t>(__ldg(a.rowptr + r0)) + r0;
    const int64_t q1 = static_cast<int64_t>(__ldg(a.rowptr + r1)) + r1;
    const int64_t per = (q1 - q0 + kAggWarps - 1) / kAggWarps;
    const int64_t qa = min64(q1, q0 + warp * per), qb = min64(q1, qa + per);
    const int32_t ta = last_row_at(a.rowptr, r0, r1, qa);
    const int32_t tb = last_row_at(a.rowptr, ta, r1, qb);
    const int32_t ka = static_cast<int32_t>(qa - ta), kb = static_cast<int32_t>(qb - tb);
    const bool head_split = ka > __ldg(a.rowptr + ta);   // row ta begun by an earlier warp
    if (lane == 0) s_head_row[warp] = -1;

    float acc[VEC];
#pragma unroll
    for (int q = 0; q < VEC; ++q) acc[q] = A::identity();
    int32_t t = ta, k = ka;                            // this warp's edges are [ka, kb)
    int32_t rend = t < tb ? __ldg(a.rowptr + t + 1) : kb;
    int cnext = (k + lane < kb) ? __ldg(a.col + k + lane) : 0;
    for (;;) {
        while (k >= rend) {                            // row t has no edges left here
            if (t >= tb) break;
            A::reduce_groups(acc);
            if (t == ta && head_split) {               // parts of it sit with earlier warps
                if (lane < LPR) {
#pragma unroll
                    for (int q = 0; q < VEC; ++q) s_head[warp][sub * VEC + q] = acc[q];
                }
                if (lane == 0) s_head_row[warp] = t;
            } else {
                M::store_row(a, t, acc, f0, fok, lane);
            }
#pragma unroll
            for (int q = 0; q < VEC; ++q) acc[q] = A::identity();
            ++t;
            rend = t < tb ? __ldg(a.rowptr + t + 1) : kb;
        }
        if (k >= rend) break;                          // t == tb and its edges are done
        const int cnt = min(32, rend - k);
        const int c = cnext;
        float ww = 1.f;
        if (lane < cnt) {
            if (a.w) ww = __ldg(a.w + k + lane);
            else if (A::kGcnLike) ww = __ldg(a.dinv + c);
        }
        const int32_t kn = k + cnt;                    // the next chunk starts here
        cnext = (kn + lane < kb) ? __ldg(a.col + kn + lane) : 0;
        float part[VEC];
#pragma unroll
        for (int q = 0; q < VEC; ++q) part[q] = A::identity();
        if constexpr (A::kIsMax) M::chunk(xf, fs, c, ww, cnt, g, fok, part);
        else M::chunk_sum(xb, row_bytes, s_stage[warp], c, ww, cnt, lane, g, part);
#pragma unroll
        for (int q = 0; q < VEC; ++q) acc[q] = A::combine(acc[q], part[q]);
        k = kn;
    }
    // the part of row tb held here (empty when the range ends on a row end)
    A::reduce_groups(acc);
    if (lane < LPR) {
#pragma unroll
        for (int q = 0; q < VEC; ++q) s_tail[warp][sub * VEC + q] = acc[q];
    }
    if (lane == 0) s_tail_row[warp] = tb;
    __syncthreads();
    const int32_t hr = s_head_row[warp];
    if (hr >= 0) {                                     // earlier parts in warp order, then ours
        float r[VEC];
#pragma unroll
        for (int q = 0; q < VEC; ++q) r[q] = A::identity();
        if (lane < LPR) {
            for (int w = 0; w < warp; ++w) {
                if (s_tail_row[w] != hr) continue;
#pragma unroll
                for (int q = 0; q < VEC; ++q) r[q] = A::combine(r[q], s_tail[w][sub * VEC + q]);
            }
#pragma unroll
            for (int q = 0; q < VEC; ++q) r[q] = A::combine(r[q], s_head[warp][sub * VEC + q]);
        }
        M::store_row(a, hr, r, f0, fok, lane);
    }
}

template <typename XT, int VEC, int LPR, int KIND, typename X0T>
cudaError_t launch_mp(const AggArgs &a, cudaStream_t s) {
    const int grid = static_cast<int>(
        min64(a.n, static_cast<int64_t>(sm_count()) * mp_blocks<KIND == kMax>()));
    aggregate_mp_kernel<XT, VEC, LPR, KIND, X0T><<<grid, kAggThreads, 0, s>>>(a);
    return cudaGetLastError();
}

template <typename XT, int VEC, int LPR, int KIND, typename X0T>
cudaError_t launch_rows(const AggArgs &a, cudaStream_t s) {
    aggregate_kernel<XT, VEC, LPR, KIND, X0T><<<balanced_grid(a.n, 0, 1), kAggThreads, 0, s>>>(a);
    return cudaGetLastError();
}

template <typename XT, int VEC, int LPR, int KIND, typename X0T>
cudaError_t launch_agg(const AggArgs &a, cudaStream_t s) {
    // E is not known on the host; the kernels read rowptr[N] for the split.
    // Rows of one feature tile in 16-byte slices take the merge-path kernel:
    // bf16 always, fp32 for max, and fp32 sums on graphs of short rows (the
    // row-per-warp kernel is launched beside it for the long-row regime).
    constexpr bool bf16 = sizeof(XT) == 2 && VEC == 8;
    constexpr bool f32 = sizeof(XT) == 4 && VEC == 4;
    if constexpr (bf16 || f32) {
        if (TFG_AGG_MP && static_cast<int64_t>(LPR) * VEC >= a.f) {
            if constexpr (!kSplitsRegimes<XT, VEC, KIND>) return launch_mp<XT, VEC, LPR, KIND, X0T>(a, s);
            AggArgs shortr = a, longr = a;
            shortr.regime = kRegimeShort;
            longr.regime = kRegimeLong;
            const cudaError_t err = launch_mp<XT, VEC, LPR, KIND, X0T>(shortr, s);
            if (err != cudaSuccess) return err;
            return launch_rows<XT, VEC, LPR, KIND, X0T>(longr, s);
        }
    }
    return launch_rows<XT, VEC, LPR, KIND, X0T>(a, s);
}

template <typename XT, int VEC, int KIND, typename X0T = XT>
cudaError_t launch_lpr(const AggArgs &a, int lpr, cudaStream_t s) {
    switch (lpr) {
        case 32: return launch_agg<XT, VEC, 32, KIND, X0T>(a, s);
        case 16: return launch_agg<XT, VEC, 16, KIND, X0T>(a, s);
        default: return launch_agg<XT, VEC, 8, KIND, X0T>(a, s);
    }
}

inline int lanes_per_row(int64_t chunks) { return chunks >= 32 ? 32 : (chunks > 8 ? 16 : 8); }

}  // namespace
}  // namespace tfg
