// Internal helpers shared by the kernels of libtfg (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "../../include/tfg.h"

namespace tfg {

constexpr unsigned kFull = 0xffffffffu;

// First error wins: a kernel that finds bad data records its code once.
__device__ __forceinline__ void set_status(int32_t *status, int32_t code) {
    if (status) atomicCAS(status, 0, code);
}

// bf16 -> fp32 is exact: the 16 stored bits are the high half of the fp32 word.
__device__ __forceinline__ float bf16_lo(uint32_t packed) { return __uint_as_float(packed << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t packed) { return __uint_as_float(packed & 0xffff0000u); }

// L2 residency of the two kinds of data the aggregation kernels read: the
// CSR column array is streamed once per call, the gathered feature rows are
// reused by every edge that names them.  TFG_L2_HINTS=1 marks the stream
// evict-first (and keeps it out of L1) and the rows evict-last; measured on
// GB300 the policy loads slowed the row gather (1.16 -> 1.30 ms for the
// 114.6M-edge gather) and the GCN kernel, so the default is plain loads.
#ifndef TFG_L2_HINTS
#define TFG_L2_HINTS 0
#endif
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
    uint64_t p;
    asm("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
    return p;
}
__device__ __forceinline__ uint64_t l2_policy_evict_last() {
    uint64_t p;
    asm("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
    return p;
}
// One element of a streamed index array (col, CSR-order weights).
__device__ __forceinline__ int32_t ld_stream(const int32_t *p) {
#if TFG_L2_HINTS
    int32_t v;
    asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.b32 %0, [%1], %2;"
                 : "=r"(v) : "l"(p), "l"(l2_policy_evict_first()));
    return v;
#else
    return __ldg(p);
#endif
}
__device__ __forceinline__ float ld_stream(const float *p) {
    return __int_as_float(ld_stream(reinterpret_cast<const int32_t *>(p)));
}
// A 16-byte slice of a gathered row.
__device__ __forceinline__ uint4 ld_row16(const void *p) {
#if TFG_L2_HINTS
    uint4 v;
    asm volatile("ld.global.nc.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p), "l"(l2_policy_evict_last()));
    return v;
#else
    return __ldg(reinterpret_cast<const uint4 *>(p));
#endif
}

// VEC consecutive features of one row: a raw load (kept packed in registers
// while the load is in flight) and its widening to fp32.
template <typename XT, int VEC> struct VecLoad;

template <> struct VecLoad<float, 4> {
    using Raw = float4;
    static __device__ __forceinline__ Raw raw(const float *p) {
        const uint4 v = ld_row16(p);
        return make_float4(__uint_as_float(v.x), __uint_as_float(v.y), __uint_as_float(v.z),
                           __uint_as_float(v.w));
    }
    static __device__ __forceinline__ Raw zero() { return make_float4(0.f, 0.f, 0.f, 0.f); }
    static __device__ __forceinline__ void widen(const Raw &q, float (&v)[4]) {
        v[0] = q.x; v[1] = q.y; v[2] = q.z; v[3] = q.w;
    }
    static __device__ __forceinline__ void load(const float *p, float (&v)[4]) { widen(raw(p), v); }
};
template <> struct VecLoad<float, 1> {
    using Raw = float;
    static __device__ __forceinline__ Raw raw(const float *p) { return __ldg(p); }
    static __device__ __forceinline__ Raw zero() { return 0.f; }
    static __device__ __forceinline__ void widen(const Raw &q, float (&v)[1]) { v[0] = q; }
    static __device__ __forceinline__ void load(const float *p, float (&v)[1]) { v[0] = __ldg(p); }
};
template <> struct VecLoad<uint16_t, 8> {
    using Raw = uint4;
    static __device__ __forceinline__ Raw raw(const uint16_t *p) { return ld_row16(p); }
    static __device__ __forceinline__ Raw zero() { return make_uint4(0u, 0u, 0u, 0u); }
    static __device__ __forceinline__ void widen(const Raw &q, float (&v)[8]) {
        v[0] = bf16_lo(q.x); v[1] = bf16_hi(q.x);
        v[2] = bf16_lo(q.y); v[3] = bf16_hi(q.y);
        v[4] = bf16_lo(q.z); v[5] = bf16_hi(q.z);
        v[6] = bf16_lo(q.w); v[7] = bf16_hi(q.w);
    }
    static __device__ __forceinline__ void load(const uint16_t *p, float (&v)[8]) { widen(raw(p), v); }
};
template <> struct VecLoad<uint16_t, 4> {
    using Raw = uint2;
    static __device__ __forceinline__ Raw raw(const uint16_t *p) {
        return __ldg(reinterpret_cast<const uint2 *>(p));
    }
    static __device__ __forceinline__ Raw zero() { return make_uint2(0u, 0u); }
    static __device__ __forceinline__ void widen(const Raw &q, float (&v)[4]) {
        v[0] = bf16_lo(q.x); v[1] = bf16_hi(q.x);
        v[2] = bf16_lo(q.y); v[3] = bf16_hi(q.y);
    }
    static __device__ __forceinline__ void load(const uint16_t *p, float (&v)[4]) { widen(raw(p), v); }
};
template <> struct VecLoad<uint16_t, 1> {
    using Raw = uint32_t;
    static __device__ __forceinline__ Raw raw(const uint16_t *p) {
        return static_cast<uint32_t>(__ldg(p)) << 16;
    }
    static __device__ __forceinline__ Raw zero() { return 0u; }
    static __device__ __forceinline__ void widen(const Raw &q, float (&v)[1]) { v[0] = __uint_as_float(q); }
    static __device__ __forceinline__ void load(const uint16_t *p, float (&v)[1]) { widen(raw(p), v); }
};

// acc += a * b on a pair of fp32 lanes: one packed fma.rn.f32x2 on sm_100+
// (each half is an ordinary correctly rounded fp32 fma, so the result is
// bit-identical to two fmaf calls).  TFG_NO_PACKED_FMA selects the scalar form.
__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) {
#if !defined(TFG_NO_PACKED_FMA)
    float2 d;
    asm("{\n\t.reg .b64 ra, rb, rc, rd;\n\t"
        "mov.b64 ra, {%2, %3};\n\tmov.b64 rb, {%4, %5};\n\tmov.b64 rc, {%6, %7};\n\t"
        "fma.rn.f32x2 rd, ra, rb, rc;\n\tmov.b64 {%0, %1}, rd;\n\t}"
        : "=f"(d.x), "=f"(d.y)
        : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
    return d;
#else
    return make_float2(fmaf(a.x, b.x, c.x), fmaf(a.y, b.y, c.y));
#endif
}

__host__ __device__ constexpr int ceil_div(int64_t a, int64_t b) { return (int)((a + b - 1) / b); }
__host__ __device__ constexpr int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }

// Work-balanced row ranges.  A CTA b of nb owns the rows t whose merge-path
// coordinate rowptr[t] + t (edges before t plus rows before t) falls in
// [b * W, (b + 1) * W), W = ceil((E + N) / nb): every CTA gets about the same
// number of edges plus rows, whatever the degree distribution, and every row
// belongs to exactly one CTA.  rowptr[t] + t is strictly increasing in t.
__device__ __forceinline__ int64_t first_row_at(const int32_t *rowptr, int64_t n, int64_t target) {
    int64_t lo = 0, hi = n;   // first t in [0, n] with rowptr[t] + t >= target
    while (lo < hi) {
        const int64_t mid = (lo + hi) >> 1;
        if (static_cast<int64_t>(__ldg(rowptr + mid)) + mid < target) lo = mid + 1;
        else hi = mid;
    }
    return lo;
}

// Last t in [lo, hi] with rowptr[t] + t <= q (rowptr[lo] + lo <= q holds):
// the row open at merge coordinate q; q - t is the CSR position reached.
__device__ __forceinline__ int32_t last_row_at(const int32_t *rowptr, int32_t lo, int32_t hi,
                                               int64_t q) {
    while (lo < hi) {
        const int32_t mid = lo + (hi - lo + 1) / 2;
        if (static_cast<int64_t>(__ldg(rowptr + mid)) + mid <= q) lo = mid;
        else hi = mid - 1;
    }
    return lo;
}

__device__ __forceinline__ void balanced_rows(const int32_t *rowptr, int64_t n, int64_t nb,
                                              int64_t b, int64_t &r0, int64_t &r1) {
    const int64_t total = static_cast<int64_t>(__ldg(rowptr + n)) + n;
    const int64_t w = (total + nb - 1) / nb;
    r0 = first_row_at(rowptr, n, b * w);
    r1 = b + 1 == nb ? n : first_row_at(rowptr, n, (b + 1) * w);
}

// Each CTA owns a work-balanced range of rows (edges + rows split evenly
// across CTAs); its warps take rows one at a time from a shared counter.
template <typename RowFn>
__device__ __forceinline__ void for_each_row(const int32_t *rowptr, int64_t n, RowFn fn) {
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

}  // namespace tfg

// Number of CTAs for a balanced launch over E edges and N rows: enough for
// several resident CTAs per SM, and at least min_work units of work each.
namespace tfg {
int balanced_grid(int64_t n, int64_t e, int64_t min_work);
int sm_count();   // multiprocessors of the current device
}

// Host-side launchers implemented in the kernel files; api.cu validates
// arguments before calling them.  Each returns cudaSuccess or the launch error.
namespace tfg {
size_t csr_workspace_bytes(int64_t n, int64_t e);
cudaError_t launch_build_csr(const int64_t *edge_index, int64_t e, int64_t n, int32_t *rowptr,
                             int32_t *col, int32_t *perm, int32_t *in_degree, void *ws,
                             int32_t *status, cudaStream_t s, bool by_source = false);
cudaError_t launch_gcn_norm(const int32_t *rowptr, const int32_t *col, const int32_t *perm,
                            const float *ew, int64_t n, int add_self, float fill, float *dinv,
                            float *w_csr, cudaStream_t s);
// mode: 0 = sum, 1 = mean, 2 = max, 3 = gcn sum
cudaError_t launch_aggregate(int mode, const int32_t *rowptr, const int32_t *col, const float *w,
                             const float *dinv, const void *x, int x_dtype, int64_t n, int64_t f,
                             int add_self, float fill, float *out, cudaStream_t s);
size_t backward_workspace_bytes(int mode, int64_t e);
cudaError_t launch_aggregate_backward(int mode, const int32_t *rowptr_src, const int32_t *col_src,
                                      const int32_t *perm_src, const float *edge_weight,
                                      const int32_t *in_degree, const float *grad_out, int64_t n,
                                      int64_t e, int64_t f, float *grad_x, void *ws,
                                      cudaStream_t s);
cudaError_t launch_max_argmax(const int32_t *rowptr, const int32_t *col, const int32_t *perm,
                              const float *w, const void *x, int x_dtype, int64_t n, int64_t f,
                              float *out, int32_t *argmax, cudaStream_t s);
cudaError_t launch_max_backward(const int32_t *rowptr_src, const int32_t *col_src,
                                const int32_t *perm_src, const int32_t *argmax,
                                const float *edge_weight, const float *grad_out, int64_t n,
                                int64_t f, float *grad_x, cudaStream_t s);
size_t propagate_workspace_bytes(int64_t n, int64_t f, int64_t hops);
cudaError_t launch_propagate(const int32_t *rowptr, const int32_t *col, const float *w,
                             const float *dinv, const void *x0, int x_dtype, int64_t n, int64_t f,
                             int64_t hops, float alpha, int add_self, float fill, float *out,
                             void *ws, cudaStream_t s);
int dot_softmax_max_channels();
cudaError_t launch_dot_softmax(const int32_t *rowptr, const int32_t *col, const void *q,
                               const void *k, const void *v, int x_dtype, int64_t n, int64_t e,
                               int heads, int channels, float scale, float *out, float *alpha,
                               cudaStream_t s);
size_t softmax_workspace_bytes(int64_t n, int heads);
cudaError_t launch_edge_softmax(const int32_t *rowptr, const int32_t *col, const void *x,
                                int x_dtype, int64_t n, int64_t e, int heads, int channels,
                                const float *a_src, const float *a_dst, float slope, float *out,
                                float *alpha, void *ws, cudaStream_t s);
size_t batch_graphs_workspace_bytes(int64_t g);
cudaError_t launch_batch_graphs(int64_t g, const int64_t *node_counts, const int64_t *edge_counts,
                                const int64_t *edge_index, int64_t e, int64_t n,
                                int64_t *out_edge_index, int64_t *batch, int64_t *node_offsets,
                                void *ws, int32_t *status, cudaStream_t s);
int64_t noalloc_softmax_max_node_heads();
cudaError_t noalloc_softmax_scratch(void **ptr, size_t *bytes);
bool attention_backward_layout_ok(int heads, int channels);
size_t attention_backward_workspace_bytes(int64_t n, int heads, int channels);
cudaError_t launch_edge_softmax_backward(const int32_t *rowptr, const int32_t *col,
                                         const int32_t *rowptr_src, const int32_t *col_src,
                                         const void *x, int x_dtype, int64_t n, int64_t e,
                                         int heads, int channels, const float *a_src,
                                         const float *a_dst,
                                         float slope, const float *out, const float *grad_out,
                                         float *grad_x, float *grad_a_src, float *grad_a_dst,
                                         void *ws, cudaStream_t s);
size_t dot_attention_backward_workspace_bytes(int64_t n, int heads);
cudaError_t launch_dot_softmax_backward(const int32_t *rowptr, const int32_t *col,
                                        const int32_t *rowptr_src, const int32_t *col_src,
                                        const void *q, const void *k, const void *v, int x_dtype,
                                        int64_t n, int64_t e, int heads, int channels, float scale,
                                        const float *out, const float *grad_out, float *grad_q,
                                        float *grad_k, float *grad_v, void *ws, cudaStream_t s);
cudaError_t launch_gather_xor(const int32_t *col, int64_t e, const void *x, int64_t row_bytes,
                              uint32_t *out, cudaStream_t s);
cudaError_t launch_segment_pool(const void *x, int x_dtype, const int64_t *batch, int64_t n,
                                int64_t g, int64_t f, int reduce, float *out, int32_t *status,
                                cudaStream_t s);
}  // namespace tfg
