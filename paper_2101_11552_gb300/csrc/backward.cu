// Backward of the message aggregation: the gradient with respect to the node
// features x of out = aggregate(x) (the paper keeps graph construction and
// mini-batching differentiable, Sections 2.1.1 and 2.1.3, so gradients flow
// through the aggregation to the features).  For a sum with edge weights w,
// out[t] = sum over edges e = (s -> t) of w_e x[s], so
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

// ---- max with argmax, and its backward ------------------------------------
// Both kernels walk CSR rows in 32-edge chunks: one coalesced load brings the
// chunk's indices (and weights) and lanes pass them on by shuffle; the
// forward has kMxUnroll row gathers per lane group in flight before any is
// used.  Each CTA owns a work-balanced range of rows (balanced_rows); its
// warps take rows from a shared counter.  A row longer than kMxHeavyDeg is
// set aside and then split over all the CTA's warps in contiguous edge
// segments, whose states are merged, so the result is what one warp walking
// the row in order would give.
constexpr int kMxWarps = 8;
constexpr int kMxThreads = kMxWarps * 32;
#ifndef TFG_MXF_UNROLL
#define TFG_MXF_UNROLL 4   // forward: feature-row gathers in flight per lane group
#endif
#ifndef TFG_MXF_VEC8
#define TFG_MXF_VEC8 1     // forward, bf16: 8 features per lane and lane groups
#endif
constexpr int kMxUnroll = TFG_MXF_UNROLL;
constexpr int64_t kMxHeavyDeg = 1024;
constexpr int kMxMaxHeavy = 64;

struct MaxArgs {
    const int32_t *rowptr, *col, *perm;
    const float *w;   // forward: w_csr (CSR order); backward: edge_weight (original order)
    const void *x;    // forward: features; backward: grad_out
    const int32_t *argmax_in;   // backward only
    int64_t n, f;
    float *out;
    int32_t *argmax_out;        // forward only
    const uint8_t *mark;        // backward: bit j of mark[e] when edge e wins some (t, f) of feature group j
    int64_t e;                  // backward: edges (the extent of mark)
    int group;                  // backward: features per group (a multiple of 4, at most 8 groups)
};

// Forward state of VEC features over an edge range, in CSR order (= original
// order for a CSR from tfg_build_csr).  The running maximum keeps the CSR
// POSITION of its edge; the original id is looked up once per row (perm) when
// the result is stored.  The row's first edge is taken whatever its value
// (NaN included); after that only a strictly larger value replaces the
// maximum, so ties keep the earliest edge and a NaN is only ever held from
// the first edge.  The G = 32 / LPR lane groups of a warp take every G-th
// edge of a chunk; their states, like those of the segments of a split hub
// row, combine by max_combine, which depends only on values and positions:
// the larger value wins, equal values go to the smaller position, and a NaN
// held from the row's first edge wins over everything.  That is exactly what
// one pass over the row in order gives.
__device__ __forceinline__ void max_combine(float &b, int32_t &p, float ob, int32_t op,
                                            int32_t row_beg) {
    if (op < 0) return;
    const bool mine_first_nan = p == row_beg && isnan(b);
    const bool other_first_nan = op == row_beg && isnan(ob);
    bool take;
    if (p < 0 || other_first_nan) take = true;
    else if (mine_first_nan) take = false;
    else take = ob > b || (ob == b && op < p);
    if (take) {
        b = ob;
        p = op;
    }
}

template <typename XT, int VEC, int LPR>
struct MaxFwd {
    static constexpr int kVec = VEC, kLpr = LPR, kGroups = 32 / LPR;
    float best[VEC];
    int32_t pos[VEC];

    __device__ void init() {
#pragma unroll
        for (int q = 0; q < VEC; ++q) {
            best[q] = -CUDART_INF_F;
            pos[q] = -1;
        }
    }

    // edges [k0, k1) of the row; first = k0 is the row's first edge
    __device__ void scan(const MaxArgs &a, int64_t k0, int64_t k1, int64_t fl, bool first,
                         int lane) {
        using V = VecLoad<XT, VEC>;
        constexpr int G = kGroups;
        const int g = lane / LPR;
        const XT *x = static_cast<const XT *>(a.x);
        for (int64_t base = k0; base < k1; base += 32) {
            const int cnt = static_cast<int>(min64(32, k1 - base));
            const bool mine = lane < cnt;
            const int c = mine ? ld_stream(a.col + base + lane) : 0;
            const float wc = a.w ? (mine ? ld_stream(a.w + base + lane) : 0.f) : 1.f;
            for (int j = 0; j < cnt; j += G * kMxUnroll) {
                typename V::Raw raw[kMxUnroll];
#pragma unroll
                for (int u = 0; u < kMxUnroll; ++u) {
                    const int k = j + u * G + g;
                    const int64_t src = __shfl_sync(kFull, c, k & 31);
                    raw[u] = k < cnt ? V::raw(x + src * a.f + fl) : V::zero();
                }
#pragma unroll
                for (int u = 0; u < kMxUnroll; ++u) {
                    const int k = j + u * G + g;
                    const float wk = __shfl_sync(kFull, wc, k & 31);
                    if (k < cnt) {
                        float v[VEC];
                        V::widen(raw[u], v);
                        const bool take_any = first && base == k0 && k == 0;
                        const int32_t kp = static_cast<int32_t>(base + k);
#pragma unroll
                        for (int q = 0; q < VEC; ++q) {
                            const float m = a.w ? wk * v[q] : v[q];
                            if (m > best[q] || take_any) {
                                best[q] = m;
                                pos[q] = kp;
                            }
                        }
                    }
                }
            }
        }
    }

    // fold the lane groups together (every lane ends with the row's state)
    __device__ void finish(int32_t row_beg) {
#pragma unroll
        for (int sh = LPR; sh < 32; sh <<= 1) {
#pragma unroll
            for (int q = 0; q < VEC; ++q) {
                const float ob = __shfl_xor_sync(kFull, best[q], sh);
                const int32_t op = __shfl_xor_sync(kFull, pos[q], sh);
                max_combine(best[q], pos[q], ob, op, row_beg);
            }
        }
    }

    // the state of another segment of the same row
    __device__ void merge(const float (&b)[VEC], const int32_t (&p)[VEC], int32_t row_beg) {
#pragma unroll
        for (int q = 0; q < VEC; ++q) max_combine(best[q], pos[q], b[q], p[q], row_beg);
    }

    __device__ float *values() { return best; }
    __device__ int32_t *positions() { return pos; }

    __device__ void store(const MaxArgs &a, int64_t t, int64_t f0) const {
#pragma unroll
        for (int q = 0; q < VEC; ++q) {
            a.out[t * a.f + f0 + q] = pos[q] < 0 ? 0.f : best[q];
            a.argmax_out[t * a.f + f0 + q] = pos[q] < 0 ? -1 : __ldg(a.perm + pos[q]);
        }
    }
};

// Backward state: grad_x[s, f] = sum over the out-edges e = (s -> t) of s,
// in CSR (= original) order, of w_e grad_out[t, f] where argmax[t, f] == e.
#ifndef TFG_MXB_DEPTH
#define TFG_MXB_DEPTH 4        // backward with win marks: marked out-edges in flight per warp
#endif
#ifndef TFG_MXB_DEPTH_ALL
#define TFG_MXB_DEPTH_ALL 4    // backward over every out-edge: edges in flight per warp
#endif
#ifndef TFG_MXB_MINB
#define TFG_MXB_MINB 4         // backward: resident CTAs per SM (64 registers per thread)
#endif
#ifndef TFG_MXB_GROUPS
#define TFG_MXB_GROUPS 1       // 1: a marked edge's lanes read only the feature groups it wins
#endif

// Two ways to find the (edge, feature) pairs that contribute, with the same
// sums in the same order:
//  * every out-edge: a lane requests its slice of the argmax row and of the
//    gradient row of t together (one round trip, D edges in flight) and
//    adds where the argmax names the edge;
//  * win marks (MASKED): the features are cut into at most 8 groups, and bit
//    j of mark[e] is set when edge e is the argmax of some (t, f) with f in
//    group j.  A chunk's edges with no bit set are skipped, and for the
//    others only the lanes whose group bit is set read their slices.  On
//    long rows few edges win anything and a winner wins few features, so
//    most row reads disappear; the marks take a byte per edge and stay in
//    L2.  A bit can come from another row's argmax naming the edge: the
//    argmax check decides, as in the full walk.
template <int VEC, bool MASKED>
struct MaxBwd {
    static constexpr int kVec = VEC, kLpr = 32;
    float acc[VEC];

    __device__ void init() {
#pragma unroll
        for (int q = 0; q < VEC; ++q) acc[q] = 0.f;
    }

    // A chunk's loads: its target ids and edge ids, then (given the edge
    // ids) its marks and weights.  Requesting the next chunk's ids and marks
    // before this chunk's rows measured slower (more registers, spills).
    struct Chunk {
        int c;
        int32_t ec;
    };
    static __device__ __forceinline__ Chunk ids(const MaxArgs &a, int64_t base, int64_t k1, int lane) {
        Chunk r{0, 0};
        if (base + lane < k1) {
            r.c = ld_stream(a.col + base + lane);
            r.ec = __ldg(a.perm + base + lane);
        }
        return r;
    }
    static __device__ __forceinline__ uint32_t mark_of(const MaxArgs &a, int64_t base, int64_t k1,
                                                       int lane, int32_t ec) {
        const bool mine = base + lane < k1;
        if constexpr (MASKED)
            return mine && static_cast<uint64_t>(ec) < static_cast<uint64_t>(a.e) ? __ldg(a.mark + ec) : 0u;
        return mine ? 0xffu : 0u;
    }
    static __device__ __forceinline__ float weight_of(const MaxArgs &a, uint32_t mk, int32_t ec) {
        return a.w ? (mk != 0 ? __ldg(a.w + ec) : 0.f) : 1.f;
    }

    __device__ void scan(const MaxArgs &a, int64_t k0, int64_t k1, int64_t fl, bool, int lane) {
        constexpr int D = MASKED ? TFG_MXB_DEPTH : TFG_MXB_DEPTH_ALL;
        const float *g = static_cast<const float *>(a.x);
        const uint32_t my_bit =
            MASKED && TFG_MXB_GROUPS ? 1u << static_cast<uint32_t>(fl / a.group) : 0xffu;
        for (int64_t base = k0; base < k1; base += 32) {
            const Chunk ch = ids(a, base, k1, lane);
            const int c = ch.c;
            const int32_t ec = ch.ec;
            const uint32_t mk = mark_of(a, base, k1, lane, ec);
            const float wc = weight_of(a, mk, ec);
            const bool win = mk != 0;
            // the chunk's edges that may contribute, D at a time in chunk order
            for (uint32_t m = __ballot_sync(kFull, win); m != 0;) {
                int64_t t[D];
                int32_t ed[D];
                float we[D];
                bool ok[D];
#pragma unroll
                for (int d = 0; d < D; ++d) {
                    const bool any = m != 0;
                    const int k = any ? __ffs(m) - 1 : 0;
                    m &= m - 1;
                    t[d] = __shfl_sync(kFull, c, k);
                    ed[d] = __shfl_sync(kFull, ec, k);
                    we[d] = __shfl_sync(kFull, wc, k);
                    ok[d] = any && (__shfl_sync(kFull, mk, k) & my_bit) != 0;   // per lane
                }
                int32_t am[D][VEC];
                float gv[D][VEC];
#pragma unroll
                for (int d = 0; d < D; ++d) {
                    if (!ok[d]) continue;
                    if constexpr (VEC == 4) {
                        const int4 v = __ldg(reinterpret_cast<const int4 *>(a.argmax_in + t[d] * a.f + fl));
                        const float4 w4 = __ldg(reinterpret_cast<const float4 *>(g + t[d] * a.f + fl));
                        am[d][0] = v.x; am[d][1] = v.y; am[d][2] = v.z; am[d][3] = v.w;
                        gv[d][0] = w4.x; gv[d][1] = w4.y; gv[d][2] = w4.z; gv[d][3] = w4.w;
                    } else {
                        am[d][0] = __ldg(a.argmax_in + t[d] * a.f + fl);
                        gv[d][0] = __ldg(g + t[d] * a.f + fl);
                    }
                }
#pragma unroll
                for (int d = 0; d < D; ++d) {
                    if (!ok[d]) continue;
#pragma unroll
                    for (int q = 0; q < VEC; ++q)
                        if (am[d][q] == ed[d]) acc[q] = fmaf(we[d], gv[d][q], acc[q]);
                }
            }
        }
    }

    __device__ void finish(int32_t) {}

    // the sum over a later segment of the same row
    __device__ void merge(const float (&b)[VEC], const int32_t (&)[VEC], int32_t) {
#pragma unroll
        for (int q = 0; q < VEC; ++q) acc[q] += b[q];
    }

    __device__ float *values() { return acc; }
    __device__ int32_t *positions() { return nullptr; }

    __device__ void store(const MaxArgs &a, int64_t s, int64_t f0) const {
#pragma unroll
        for (int q = 0; q < VEC; ++q) a.out[s * a.f + f0 + q] = acc[q];
    }
};

// One row by one warp, feature tiles of LPR * VEC.
template <typename State>
__device__ void max_warp_row(const MaxArgs &a, int64_t t, int lane) {
    constexpr int VEC = State::kVec, LPR = State::kLpr;
    const int64_t beg = a.rowptr[t], end = a.col ? a.rowptr[t + 1] : a.rowptr[t];
    for (int64_t ft = 0; ft < a.f; ft += LPR * VEC) {
        const int64_t f0 = ft + static_cast<int64_t>(lane % LPR) * VEC;
        const bool fok = f0 < a.f;
        State st;
        st.init();
        st.scan(a, beg, end, fok ? f0 : 0, true, lane);
        st.finish(static_cast<int32_t>(beg));
        if (fok && lane < LPR) st.store(a, t, f0);
    }
}

// One long row by all warps of the CTA: warp w takes the w-th of kMxWarps
// contiguous edge segments; warp 0 folds the other segments into its own,
// in segment order.  Every thread of the CTA calls this.
template <typename State>
__device__ void max_cta_row(const MaxArgs &a, int64_t t, float *s_val, int32_t *s_pos) {
    constexpr int VEC = State::kVec, LPR = State::kLpr;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int64_t beg = a.rowptr[t], end = a.rowptr[t + 1], d = end - beg;
    const int64_t k0 = beg + d * warp / kMxWarps, k1 = beg + d * (warp + 1) / kMxWarps;
    const int32_t rb = static_cast<int32_t>(beg);
    for (int64_t ft = 0; ft < a.f; ft += LPR * VEC) {
        const int64_t f0 = ft + static_cast<int64_t>(lane % LPR) * VEC;
        const bool fok = f0 < a.f;
        State st;
        st.init();
        st.scan(a, k0, k1, fok ? f0 : 0, warp == 0, lane);
        st.finish(rb);
        if (warp > 0 && lane < LPR) {
            const int32_t *ps = st.positions();
#pragma unroll
            for (int q = 0; q < VEC; ++q) {
                s_val[(warp * LPR + lane) * VEC + q] = st.values()[q];
                if (ps) s_pos[(warp * LPR + lane) * VEC + q] = ps[q];
            }
        }
        __syncthreads();
        if (warp == 0 && lane < LPR) {
            for (int w = 1; w < kMxWarps; ++w) {
                float b[VEC];
                int32_t p[VEC];
#pragma unroll
                for (int q = 0; q < VEC; ++q) {
                    b[q] = s_val[(w * LPR + lane) * VEC + q];
                    p[q] = st.positions() ? s_pos[(w * LPR + lane) * VEC + q] : 0;
                }
                st.merge(b, p, rb);
            }
            if (fok) st.store(a, t, f0);
        }
        __syncthreads();
    }
}

template <typename State>
__device__ __forceinline__ void max_rows(const MaxArgs &a) {
    __shared__ int s_next, s_nheavy;
    __shared__ int64_t s_heavy[kMxMaxHeavy];
    __shared__ float s_val[kMxWarps * State::kLpr * State::kVec];
    __shared__ int32_t s_pos[kMxWarps * State::kLpr * State::kVec];
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
        if (a.col != nullptr && a.rowptr[t + 1] - a.rowptr[t] > kMxHeavyDeg) {
            int slot = 0;
            if (lane == 0) slot = atomicAdd(&s_nheavy, 1);
            slot = __shfl_sync(kFull, slot, 0);
            if (slot < kMxMaxHeavy) {
                if (lane == 0) s_heavy[slot] = t;
                continue;
            }
        }
        max_warp_row<State>(a, t, lane);
    }
    __syncthreads();
    const int nh = min(s_nheavy, kMxMaxHeavy);
    for (int h = 0; h < nh; ++h) max_cta_row<State>(a, s_heavy[h], s_val, s_pos);
}

// The forward keeps the compiler's register choice; the backward is held
// to TFG_MXB_MINB resident CTAs per SM (64 registers per thread).
template <typename State>
__global__ void __launch_bounds__(kMxThreads) max_rows_kernel(MaxArgs a) { max_rows<State>(a); }

template <typename State>
__global__ void __launch_bounds__(kMxThreads, TFG_MXB_MINB) max_bwd_kernel(MaxArgs a) {
    max_rows<State>(a);
}

bool aligned(const void *p, uintptr_t b) { return reinterpret_cast<uintptr_t>(p) % b == 0; }

// Win marks of the max backward.  Every (t, f) has one winning edge (none
// for a row without edges); a row of in-degree d has at most min(d, F)
// distinct winners, so on long rows most out-edges win nothing and a
// winner wins few features.  Two launches write the marks: zero them, then
// for each e = argmax[t, f] set bit f / group of mark[e] (atomicOr on the
// word holding the byte).  Ids outside [0, E) are ignored.
__global__ void max_marks_zero(uint8_t *__restrict__ mark, int64_t bytes) {
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    const int64_t i0 = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    const int64_t n16 = reinterpret_cast<uintptr_t>(mark) % 16 == 0 ? bytes / 16 : 0;
    uint4 *m16 = reinterpret_cast<uint4 *>(mark);
    for (int64_t i = i0; i < n16; i += stride) m16[i] = make_uint4(0, 0, 0, 0);
    for (int64_t i = n16 * 16 + i0; i < bytes; i += stride) mark[i] = 0;
}

__global__ void max_marks_set(const int32_t *__restrict__ argmax, int64_t n, int64_t f, int64_t e,
                              int group, uint8_t *__restrict__ mark) {
    uint32_t *words = reinterpret_cast<uint32_t *>(mark);   // 4-byte aligned (checked by the caller)
    // rows t over the grid, features over the threads of a block
    for (int64_t t = blockIdx.x; t < n; t += gridDim.x)
        for (int64_t c = threadIdx.x; c < f; c += blockDim.x) {
            const int32_t k = __ldg(argmax + t * f + c);
            if (static_cast<uint64_t>(k) >= static_cast<uint64_t>(e)) continue;
            const uint32_t bit = 1u << static_cast<uint32_t>(c / group);
            atomicOr(words + (k >> 2), bit << (8 * (k & 3)));
        }
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
    const MaxArgs a{rowptr, col, perm, w, x, nullptr, n, f, out, argmax};
    // E is not known on the host; the kernel reads rowptr[N] for the split
    const int grid = balanced_grid(n, 0, 1);
    if (x_dtype == TFG_BF16) {
        if (TFG_MXF_VEC8 && f % 8 == 0 && aligned(x, 16)) {   // 16-byte row slices: 8 features per lane
            const int64_t lanes = f / 8;
            if (lanes >= 32) max_rows_kernel<MaxFwd<uint16_t, 8, 32>><<<grid, kMxThreads, 0, s>>>(a);
            else if (lanes > 8) max_rows_kernel<MaxFwd<uint16_t, 8, 16>><<<grid, kMxThreads, 0, s>>>(a);
            else max_rows_kernel<MaxFwd<uint16_t, 8, 8>><<<grid, kMxThreads, 0, s>>>(a);
        } else if (f % 4 == 0 && aligned(x, 8)) {
            max_rows_kernel<MaxFwd<uint16_t, 4, 32>><<<grid, kMxThreads, 0, s>>>(a);
        } else {
            max_rows_kernel<MaxFwd<uint16_t, 1, 32>><<<grid, kMxThreads, 0, s>>>(a);
        }
    } else {
        if (f % 4 == 0 && aligned(x, 16)) max_rows_kernel<MaxFwd<float, 4, 32>><<<grid, kMxThreads, 0, s>>>(a);
        else max_rows_kernel<MaxFwd<float, 1, 32>><<<grid, kMxThreads, 0, s>>>(a);
    }
    return cudaGetLastError();
}

// The win marks pay when most edges win nothing in a row tile of kMxbSpan
// features: an edge into a row of in-degree d wins a given feature with
// probability about 1 / d, so it is visited in a tile with probability
// about 1 - exp(-span / d), span = min(F, kMxbSpan).  They are used when
// the mean in-degree E / N is at least span.  Measured: 114.6M edges, mean
// in-degree 492, bf16: 1.7-2x faster for F = 128-2048, 1.4x at F = 4096;
// 12.0M edges over the same nodes (mean in-degree 51.5, F = 128): 0.94 ms
// for the marked walk + 0.15 ms for the marks against 0.91 ms unmarked
// (ncu, serialised); 1.17M edges, mean in-degree 6.9: 2-60 % slower for F =
// 8-128.
#ifndef TFG_MXB_SPAN
#define TFG_MXB_SPAN 128
#endif
constexpr int64_t kMxbSpan = TFG_MXB_SPAN;

size_t max_backward_workspace_bytes(int64_t n, int64_t e, int64_t f) {
    if (n <= 0 || e <= 0 || f <= 0 || e < n * (f < kMxbSpan ? f : kMxbSpan)) return 0;
    return (static_cast<size_t>(e) + 255) & ~size_t(255);
}

// Features per mark bit: at most 8 groups, each a multiple of 4 features so
// that a lane's 16-byte slice lies in one group.
int mark_group(int64_t f) { return static_cast<int>(((f + 7) / 8 + 3) / 4 * 4); }

cudaError_t launch_max_backward_marked(const int32_t *rowptr_src, const int32_t *col_src,
                                       const int32_t *perm_src, const int32_t *argmax,
                                       const float *edge_weight, const float *grad_out, int64_t n,
                                       int64_t e, int64_t f, float *grad_x, void *ws,
                                       cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const bool marked = ws != nullptr && col_src != nullptr && max_backward_workspace_bytes(n, e, f) > 0;
    uint8_t *mark = marked ? static_cast<uint8_t *>(ws) : nullptr;
    const int group = mark_group(f);
    if (marked) {
        const int grid = sm_count() * 8;
        max_marks_zero<<<grid, 256, 0, s>>>(mark, e);
        max_marks_set<<<grid, f >= 256 ? 256 : 128, 0, s>>>(argmax, n, f, e, group, mark);
    }
    const MaxArgs a{rowptr_src, col_src, perm_src, edge_weight, grad_out, argmax, n, f, grad_x,
                    nullptr, mark, e, group};
    const int grid = balanced_grid(n, 0, 1);
    const bool v4 = f % 4 == 0 && aligned(argmax, 16) && aligned(grad_out, 16) && aligned(grad_x, 16);
    if (marked) {
        if (v4) max_bwd_kernel<MaxBwd<4, true>><<<grid, kMxThreads, 0, s>>>(a);
        else max_bwd_kernel<MaxBwd<1, true>><<<grid, kMxThreads, 0, s>>>(a);
    } else {
        if (v4) max_bwd_kernel<MaxBwd<4, false>><<<grid, kMxThreads, 0, s>>>(a);
        else max_bwd_kernel<MaxBwd<1, false>><<<grid, kMxThreads, 0, s>>>(a);
    }
    return cudaGetLastError();
}

cudaError_t launch_max_backward(const int32_t *rowptr_src, const int32_t *col_src,
                                const int32_t *perm_src, const int32_t *argmax,
                                const float *edge_weight, const float *grad_out, int64_t n,
                                int64_t f, float *grad_x, cudaStream_t s) {
    return launch_max_backward_marked(rowptr_src, col_src, perm_src, argmax, edge_weight, grad_out,
                                      n, 0, f, grad_x, nullptr, s);
}

}  // namespace tfg
