// One-hop entry points of the fused gather * weight * reduce (the kernels
// themselves are in agg.cuh): sum / mean / max with optional CSR-order
// weights, and GCN sum with symmetric-normalised weights formed on the fly.
#include "agg.cuh"

namespace tfg {
namespace {

template <typename XT, int VEC>
cudaError_t launch_kind(const AggArgs &a, int kind, int lpr, cudaStream_t s) {
    switch (kind) {
        case kMax: return launch_lpr<XT, VEC, kMax>(a, lpr, s);
        case kGcn: return launch_lpr<XT, VEC, kGcn>(a, lpr, s);
        default: return launch_lpr<XT, VEC, kSumLike>(a, lpr, s);
    }
}

}  // namespace

cudaError_t launch_aggregate(int mode, const int32_t *rowptr, const int32_t *col, const float *w,
                             const float *dinv, const void *x, int x_dtype, int64_t n, int64_t f,
                             int add_self, float fill, float *out, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    AggArgs a{rowptr, col, w, dinv, x, out, n, f, mode == 1, add_self, fill, nullptr, 0.f, 1.f,
              kRegimeAny};
    const int kind = mode == 2 ? kMax : (mode == 3 ? kGcn : kSumLike);
    const bool aligned = (reinterpret_cast<uintptr_t>(x) % 16 == 0) &&
                         (reinterpret_cast<uintptr_t>(out) % 16 == 0);
    if (x_dtype == TFG_BF16) {
        if (aligned && f % 8 == 0) return launch_kind<uint16_t, 8>(a, kind, lanes_per_row(f / 8), s);
        return launch_kind<uint16_t, 1>(a, kind, lanes_per_row(f), s);
    }
    if (aligned && f % 4 == 0) return launch_kind<float, 4>(a, kind, lanes_per_row(f / 4), s);
    return launch_kind<float, 1>(a, kind, lanes_per_row(f), s);
}

}  // namespace tfg
