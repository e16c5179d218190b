// Gather-only floor of the row aggregations (a measurement kernel, not a step
// of the paper's method).
//
// Every aggregation of this library reads, for each edge of a CSR, the whole
// feature row of the edge's source node: for the benchmark graph that is
// 114.6M rows of 256 bytes from an array that fits in L2, i.e. ~29 GB moved
// from L2 to the SMs per call against ~0.6 GB from HBM.  The HBM roofline
// therefore does not bound those kernels; the rate at which the SMs can pull
// gathered rows out of L2 does.  This kernel measures that rate on the same
// column array and feature rows with nothing else to do: each warp takes
// 32-edge chunks of col, gathers the source rows as 16-byte vectors and folds
// them with XOR (one instruction per vector, no floating point) -- with the
// same L2 policies as the aggregation kernels (col streamed, rows kept) -- and the
// folds of all warps are XOR-combined into one output row.  Its time is the
// floor that the aggregation kernels are compared against; its result (the
// XOR of all gathered rows) is exact and order-free, so it is testable.
#include "common.cuh"

namespace tfg {
namespace {

constexpr int kGfThreads = 256;
constexpr int kGfWarps = kGfThreads / 32;
// The shape measured fastest on GB300 for 256-byte rows: a persistent grid
// of 4 CTAs of 256 threads per SM, 8 16-byte gathers in flight per lane, and
// the next chunk's column ids loaded before this chunk's rows are gathered
// (1.16 ms for 114.6M rows; 16 in flight per lane: 1.30 ms, 4: 1.39 ms, one
// chunk per warp without the persistent loop: 2.77 ms).
#ifndef TFG_GF_DEPTH
#define TFG_GF_DEPTH 8    // 16-byte gathers in flight per lane (tuning knob)
#endif
constexpr int kGfDepth = TFG_GF_DEPTH;

// LPR lanes cover one row (LPR = 16-byte vectors per row, a power of two
// <= 32); the G = 32 / LPR lane groups take every G-th edge of a chunk.
template <int LPR>
__global__ void __launch_bounds__(kGfThreads, 4)
gather_xor_kernel(const int32_t *__restrict__ col, int64_t e, const uint4 *__restrict__ x,
                  uint32_t *__restrict__ out) {
    constexpr int G = 32 / LPR;
    constexpr int kSteps = 32 / G;                       // slots of a group per chunk
    constexpr int kDepth = kGfDepth < kSteps ? kGfDepth : kSteps;
    __shared__ uint4 s_fold[kGfWarps][LPR];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = lane / LPR, sub = lane % LPR;
    uint4 acc = make_uint4(0u, 0u, 0u, 0u);
    const int64_t chunks = (e + 31) / 32;
    const int64_t nwarps = static_cast<int64_t>(gridDim.x) * kGfWarps;
    int64_t c = static_cast<int64_t>(blockIdx.x) * kGfWarps + warp;
    int next = (c < chunks && c * 32 + lane < e) ? ld_stream(col + c * 32 + lane) : 0;
    for (; c < chunks; c += nwarps) {
        const int64_t base = c * 32;
        const int cnt = static_cast<int>(min64(32, e - base));
        const int src_l = next;
        const int64_t cn = c + nwarps;                   // prefetch the next chunk's ids
        next = (cn < chunks && cn * 32 + lane < e) ? ld_stream(col + cn * 32 + lane) : 0;
#pragma unroll
        for (int j = 0; j < kSteps; j += kDepth) {
            uint4 raw[kDepth];
#pragma unroll
            for (int u = 0; u < kDepth; ++u) {
                const int k = (j + u) * G + g;
                const uint32_t src = static_cast<uint32_t>(__shfl_sync(kFull, src_l, k));
                raw[u] = k < cnt ? ld_row16(x + static_cast<uint64_t>(src) * LPR + sub)
                                 : make_uint4(0u, 0u, 0u, 0u);
            }
#pragma unroll
            for (int u = 0; u < kDepth; ++u) {
                acc.x ^= raw[u].x;
                acc.y ^= raw[u].y;
                acc.z ^= raw[u].z;
                acc.w ^= raw[u].w;
            }
        }
    }
    // fold the lane groups, then the CTA's warps, then the CTAs (atomics)
#pragma unroll
    for (int s = LPR; s < 32; s <<= 1) {
        acc.x ^= __shfl_xor_sync(kFull, acc.x, s);
        acc.y ^= __shfl_xor_sync(kFull, acc.y, s);
        acc.z ^= __shfl_xor_sync(kFull, acc.z, s);
        acc.w ^= __shfl_xor_sync(kFull, acc.w, s);
    }
    if (lane < LPR) s_fold[warp][lane] = acc;
    __syncthreads();
    if (threadIdx.x < LPR) {
        uint4 r = s_fold[0][threadIdx.x];
        for (int w = 1; w < kGfWarps; ++w) {
            const uint4 o = s_fold[w][threadIdx.x];
            r.x ^= o.x;
            r.y ^= o.y;
            r.z ^= o.z;
            r.w ^= o.w;
        }
        uint32_t *o = out + threadIdx.x * 4;
        if (r.x) atomicXor(o + 0, r.x);
        if (r.y) atomicXor(o + 1, r.y);
        if (r.z) atomicXor(o + 2, r.z);
        if (r.w) atomicXor(o + 3, r.w);
    }
}

template <int LPR>
cudaError_t launch_gf(const int32_t *col, int64_t e, const void *x, uint32_t *out, cudaStream_t s) {
    int dev = 0, sms = 0, per_sm = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err == cudaSuccess) err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    if (err == cudaSuccess)
        err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, gather_xor_kernel<LPR>,
                                                            kGfThreads, 0);
    if (err != cudaSuccess) return err;
    const int64_t chunks = (e + 31) / 32;
    const int64_t want = (chunks + kGfWarps - 1) / kGfWarps;
    const int64_t cap = static_cast<int64_t>(sms) * (per_sm > 0 ? per_sm : 1);
    const int grid = static_cast<int>(want < cap ? want : cap);
    gather_xor_kernel<LPR><<<grid, kGfThreads, 0, s>>>(col, e, static_cast<const uint4 *>(x), out);
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gather_xor(const int32_t *col, int64_t e, const void *x, int64_t row_bytes,
                              uint32_t *out, cudaStream_t s) {
    cudaError_t err = cudaMemsetAsync(out, 0, static_cast<size_t>(row_bytes), s);
    if (err != cudaSuccess || e == 0) return err;
    switch (row_bytes / 16) {
        case 1: return launch_gf<1>(col, e, x, out, s);
        case 2: return launch_gf<2>(col, e, x, out, s);
        case 4: return launch_gf<4>(col, e, x, out, s);
        case 8: return launch_gf<8>(col, e, x, out, s);
        case 16: return launch_gf<16>(col, e, x, out, s);
        default: return launch_gf<32>(col, e, x, out, s);
    }
}

}  // namespace tfg
