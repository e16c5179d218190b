// C ABI of libtfg: host-side argument checks, then the launchers.
// Every entry point validates before it touches the GPU, so a rejected call
// enqueues nothing.  See include/tfg.h for the contract of each call.
#include <cstdarg>
#include <cstdio>

#include "common.cuh"

// NVTX ranges (header-only NVTX 3; no-ops unless a profiler is attached):
// every entry point opens a range named after itself around its host work
// and launches, so ncu / nsys timelines show which call enqueued which
// kernels.  TFG_NVTX=0 compiles them out.
#ifndef TFG_NVTX
#define TFG_NVTX 1
#endif
#if TFG_NVTX
#include <nvtx3/nvToolsExt.h>
namespace {
struct NvtxRange {
    explicit NvtxRange(const char *name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
    NvtxRange(const NvtxRange &) = delete;
    NvtxRange &operator=(const NvtxRange &) = delete;
};
}  // namespace
#define TFG_RANGE(name) NvtxRange tfg_nvtx_range_(name)
#else
#define TFG_RANGE(name) \
    do {                \
    } while (0)
#endif

// Helpers of the bounds-checked debug build (check_bounds.cu), the CSR
// build over an int32 edge list (csr_build.cu) and the max backward with
// win marks (backward.cu).
namespace tfg {
size_t max_backward_workspace_bytes(int64_t n, int64_t e, int64_t f);
cudaError_t launch_max_backward_marked(const int32_t *rowptr_src, const int32_t *col_src,
                                       const int32_t *perm_src, const int32_t *argmax,
                                       const float *edge_weight, const float *grad_out, int64_t n,
                                       int64_t e, int64_t f, float *grad_x, void *ws,
                                       cudaStream_t s);
cudaError_t launch_build_csr32(const int32_t *edge_index, int64_t e, int64_t n, int32_t *rowptr,
                               int32_t *col, int32_t *perm, int32_t *in_degree, void *ws,
                               int32_t *status, cudaStream_t s, bool by_source);
bool allocation_range(const void *p, uintptr_t *base, size_t *size);
cudaError_t csr_ends(const int32_t *rowptr, int64_t n, int32_t *first, int32_t *last,
                     cudaStream_t s);
cudaError_t validate_csr(const int32_t *rowptr, const int32_t *col, const int32_t *perm,
                         int64_t n, int64_t e, int *flags, cudaStream_t s);
}  // namespace tfg

namespace {

thread_local char g_err[512];

int fail(int code, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof(g_err), fmt, ap);
    va_end(ap);
    return code;
}

int ok() {
    g_err[0] = '\0';
    return TFG_OK;
}

int cuda_result(cudaError_t e, const char *where) {
    if (e != cudaSuccess) return fail(TFG_ERR_CUDA, "%s: %s", where, cudaGetErrorString(e));
    return ok();
}

constexpr int64_t kIndexLimit = int64_t(1) << 31;  // CSR ids are int32

int check_counts(const char *fn, int64_t n, int64_t e) {
    if (n < 0 || e < 0) return fail(TFG_ERR_INVALID_ARG, "%s: negative size (N=%lld, E=%lld)", fn,
                                    (long long)n, (long long)e);
    if (n >= kIndexLimit || e >= kIndexLimit)
        return fail(TFG_ERR_TOO_LARGE, "%s: N and E must be < 2^31 (N=%lld, E=%lld)", fn,
                    (long long)n, (long long)e);
    if (e > 0 && n == 0) return fail(TFG_ERR_INVALID_ARG, "%s: edges given but N == 0", fn);
    return TFG_OK;
}

int check_features(const char *fn, int64_t n, int64_t f) {
    if (f < 1 || f > (int64_t(1) << 24))
        return fail(TFG_ERR_INVALID_ARG, "%s: feature count must be in [1, 2^24] (F=%lld)", fn,
                    (long long)f);
    if (n * f >= (int64_t(1) << 46))
        return fail(TFG_ERR_TOO_LARGE, "%s: N*F too large", fn);
    return TFG_OK;
}

int check_dtype(const char *fn, int dtype) {
    if (dtype != TFG_F32 && dtype != TFG_BF16)
        return fail(TFG_ERR_INVALID_ARG, "%s: unknown dtype %d", fn, dtype);
    return TFG_OK;
}

#define TFG_TRY(expr)                    \
    do {                                 \
        int rc_ = (expr);                \
        if (rc_ != TFG_OK) return rc_;   \
    } while (0)

#define TFG_NEED(ptr, cond, fn, name)                                                  \
    do {                                                                               \
        if ((cond) && (ptr) == nullptr)                                                \
            return fail(TFG_ERR_INVALID_ARG, "%s: %s must not be NULL", fn, name);    \
    } while (0)

// ---- bounds-checked debug build (TFG_CHECK_BOUNDS=1) ----------------------
// Before any launch, every device buffer is checked against the allocation
// that holds it (the bytes the call will touch must lie inside it), and every
// caller-built index array is read once on the device: rowptr[0] = 0,
// rowptr[N] = E, rowptr non-decreasing, col ids in [0, N), perm ids in
// [0, E).  A violation returns TFG_ERR_INDEX_RANGE with the reason and
// launches nothing, so no kernel reads out of bounds.  Each check copies a
// few values to the host and synchronises the stream: a debugging aid, not a
// production mode.  The default build compiles none of it.
#ifndef TFG_CHECK_BOUNDS
#define TFG_CHECK_BOUNDS 0
#endif

#if TFG_CHECK_BOUNDS
int debug_extent(const char *fn, const char *name, const void *p, size_t bytes) {
    if (p == nullptr || bytes == 0) return TFG_OK;
    uintptr_t base = 0;
    size_t size = 0;
    if (!tfg::allocation_range(p, &base, &size))
        return fail(TFG_ERR_INVALID_ARG, "%s: %s is not device memory of the current context", fn,
                    name);
    const uintptr_t a = reinterpret_cast<uintptr_t>(p);
    if (a + bytes > base + size)
        return fail(TFG_ERR_INDEX_RANGE,
                    "%s: %s must hold %zu bytes, its allocation ends %zu bytes after it", fn, name,
                    bytes, static_cast<size_t>(base + size - a));
    return TFG_OK;
}

// rowptr [N + 1] (or NULL: col ids only, E = e_given), col [E] and perm [E]
// each NULL when the call does not read it (a NULL col that the call reads
// is refused when E > 0); e_given < 0 takes E from rowptr[N].  E is returned
// in *e_out.
int debug_csr(const char *fn, const char *which, const int32_t *rowptr, const int32_t *col,
              const int32_t *perm, int64_t n, int64_t e_given, int64_t *e_out,
              tfg_stream_t stream, bool col_read = true) {
    cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    int64_t e = e_given;
    if (rowptr) {
        TFG_TRY(debug_extent(fn, "rowptr", rowptr, sizeof(int32_t) * size_t(n + 1)));
        int32_t first = 0, last = 0;
        cudaError_t err = tfg::csr_ends(rowptr, n, &first, &last, s);
        if (err != cudaSuccess) return cuda_result(err, fn);
        if (first != 0 || last < 0 || (e_given >= 0 && last != e_given))
            return fail(TFG_ERR_INDEX_RANGE, "%s: %s rowptr[0] = %d, rowptr[N] = %d (E = %lld)",
                        fn, which, first, last, (long long)e_given);
        e = last;
    }
    if (e_out) *e_out = e;
    if (e > 0 && col_read && col == nullptr)
        return fail(TFG_ERR_INVALID_ARG, "%s: %s is NULL but the graph has %lld edges", fn, which,
                    (long long)e);
    if (e > 0) {
        TFG_TRY(debug_extent(fn, "col", col, sizeof(int32_t) * size_t(e)));
        TFG_TRY(debug_extent(fn, "perm", perm, sizeof(int32_t) * size_t(e)));
    }
    int flags = 0;
    cudaError_t err = tfg::validate_csr(rowptr, col, perm, n, e, &flags, s);
    if (err != cudaSuccess) return cuda_result(err, fn);
    if (flags & 1) return fail(TFG_ERR_INDEX_RANGE, "%s: %s rowptr decreases", fn, which);
    if (flags & 2) return fail(TFG_ERR_INDEX_RANGE, "%s: a %s id lies outside [0, N)", fn, which);
    if (flags & 4) return fail(TFG_ERR_INDEX_RANGE, "%s: a %s perm id lies outside [0, E)", fn, which);
    return TFG_OK;
}
#define TFG_DEBUG(expr) TFG_TRY(expr)

size_t elem_bytes(int dtype) { return dtype == TFG_BF16 ? 2 : 4; }
#else
#define TFG_DEBUG(expr) \
    do {                \
    } while (0)
#endif

int aggregate_common(const char *fn, int mode, const int32_t *rowptr, const int32_t *col,
                     const float *w, const float *dinv, const void *x, int dtype, int64_t n,
                     int64_t f, int add_self, float fill, float *out, tfg_stream_t stream) {
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, n, 0));
    TFG_TRY(check_features(fn, n, f));
    TFG_TRY(check_dtype(fn, dtype));
    TFG_NEED(rowptr, true, fn, "rowptr");
    TFG_NEED(x, n > 0, fn, "x");
    TFG_NEED(out, n > 0, fn, "out");
    TFG_NEED(dinv, mode == 3 && n > 0, fn, "dinv");
#if TFG_CHECK_BOUNDS
    {
        int64_t e = 0;
        TFG_DEBUG(debug_csr(fn, "col", rowptr, col, nullptr, n, -1, &e, stream));
        TFG_DEBUG(debug_extent(fn, "w_csr", w, sizeof(float) * size_t(e)));
        TFG_DEBUG(debug_extent(fn, "dinv", dinv, sizeof(float) * size_t(n)));
        TFG_DEBUG(debug_extent(fn, "x", x, elem_bytes(dtype) * size_t(n * f)));
        TFG_DEBUG(debug_extent(fn, "out", out, sizeof(float) * size_t(n * f)));
    }
#endif
    return cuda_result(tfg::launch_aggregate(mode, rowptr, col, w, dinv, x, dtype, n, f, add_self,
                                             fill, out, reinterpret_cast<cudaStream_t>(stream)),
                       fn);
}

constexpr int kMaxHops = 1024;

int propagate_common(const char *fn, const int32_t *rowptr, const int32_t *col, const float *dinv,
                     const float *w, const void *x0, int dtype, int64_t n, int64_t f, int64_t hops,
                     float alpha, int add_self, float fill, float *out, void *ws, size_t ws_bytes,
                     tfg_stream_t stream) {
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, n, 0));
    TFG_TRY(check_features(fn, n, f));
    TFG_TRY(check_dtype(fn, dtype));
    if (hops < 0 || hops > kMaxHops)
        return fail(TFG_ERR_INVALID_ARG, "%s: num_hops must be in [0, %d]", fn, kMaxHops);
    if (!(alpha >= 0.f && alpha <= 1.f))
        return fail(TFG_ERR_INVALID_ARG, "%s: alpha must be in [0, 1]", fn);
    TFG_NEED(rowptr, hops > 0, fn, "rowptr");
    TFG_NEED(dinv, hops > 0 && n > 0, fn, "dinv");
    TFG_NEED(x0, n > 0, fn, "x0");
    TFG_NEED(out, n > 0, fn, "out");
    const size_t need = tfg::propagate_workspace_bytes(n, f, hops);
    if (need > 0) {
        if (ws == nullptr || ws_bytes < need)
            return fail(TFG_ERR_WORKSPACE, "%s: workspace of %zu bytes needed, %zu given", fn, need,
                        ws ? ws_bytes : size_t(0));
        if (reinterpret_cast<uintptr_t>(ws) % 16 != 0)
            return fail(TFG_ERR_INVALID_ARG, "%s: workspace must be 16-byte aligned", fn);
    }
#if TFG_CHECK_BOUNDS
    if (hops > 0) {
        int64_t e = 0;
        TFG_DEBUG(debug_csr(fn, "col", rowptr, col, nullptr, n, -1, &e, stream));
        TFG_DEBUG(debug_extent(fn, "w_csr", w, sizeof(float) * size_t(e)));
        TFG_DEBUG(debug_extent(fn, "dinv", dinv, sizeof(float) * size_t(n)));
    }
    TFG_DEBUG(debug_extent(fn, "x0", x0, elem_bytes(dtype) * size_t(n * f)));
    TFG_DEBUG(debug_extent(fn, "out", out, sizeof(float) * size_t(n * f)));
    TFG_DEBUG(debug_extent(fn, "workspace", ws, need));
#endif
    return cuda_result(tfg::launch_propagate(rowptr, col, w, dinv, x0, dtype, n, f, hops, alpha,
                                             add_self, fill, out, ws,
                                             reinterpret_cast<cudaStream_t>(stream)),
                       fn);
}

}  // namespace

namespace tfg {
int sm_count() {
    thread_local int sms = 0, sms_dev = -1;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) dev = 0;
    if (sms == 0 || sms_dev != dev) {
        if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0)
            sms = 148;
        sms_dev = dev;
    }
    return sms;
}

int balanced_grid(int64_t n, int64_t e, int64_t min_work) {
    const int sms = sm_count();
    const int64_t by_work = (n + e + min_work - 1) / min_work;
    const int64_t cap = int64_t(sms) * 16;
    const int64_t g = by_work < cap ? by_work : cap;
    return static_cast<int>(g < 1 ? 1 : g);
}
}  // namespace tfg

extern "C" {

int tfg_version(void) { return 300; }

int tfg_check_bounds_enabled(void) { return TFG_CHECK_BOUNDS; }

const char *tfg_last_error(void) { return g_err; }

int tfg_build_csr_workspace_size(int64_t num_nodes, int64_t num_edges, size_t *bytes) {
    const char *fn = "tfg_build_csr_workspace_size";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, num_edges));
    TFG_NEED(bytes, true, fn, "bytes");
    *bytes = tfg::csr_workspace_bytes(num_nodes, num_edges);
    return ok();
}

namespace {
// edge_index: int64 [2, E], or int32 [2, E] when id32
int build_csr_common(const char *fn, bool by_source, const void *edge_index, bool id32, int64_t num_edges,
                     int64_t num_nodes, int32_t *rowptr, int32_t *col, int32_t *perm,
                     int32_t *in_degree, void *workspace, size_t workspace_bytes, int32_t *status,
                     tfg_stream_t stream) {
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, num_edges));
    TFG_NEED(edge_index, num_edges > 0, fn, "edge_index");
    TFG_NEED(rowptr, true, fn, "rowptr");
    TFG_NEED(col, num_edges > 0, fn, "col");
    TFG_NEED(perm, num_edges > 0, fn, "perm");
    TFG_NEED(in_degree, num_nodes > 0, fn, "in_degree");
    TFG_NEED(status, true, fn, "status");
    const size_t need = tfg::csr_workspace_bytes(num_nodes, num_edges);
    if (num_edges > 0) {
        if (workspace == nullptr || workspace_bytes < need)
            return fail(TFG_ERR_WORKSPACE, "%s: workspace of %zu bytes needed, %zu given", fn, need,
                        workspace ? workspace_bytes : size_t(0));
        if (reinterpret_cast<uintptr_t>(workspace) % 256 != 0)
            return fail(TFG_ERR_INVALID_ARG, "%s: workspace must be 256-byte aligned", fn);
    }
    TFG_DEBUG(debug_extent(fn, "edge_index", edge_index,
                           (id32 ? sizeof(int32_t) : sizeof(int64_t)) * 2 * size_t(num_edges)));
    TFG_DEBUG(debug_extent(fn, "rowptr", rowptr, sizeof(int32_t) * size_t(num_nodes + 1)));
    TFG_DEBUG(debug_extent(fn, "col", col, sizeof(int32_t) * size_t(num_edges)));
    TFG_DEBUG(debug_extent(fn, "perm", perm, sizeof(int32_t) * size_t(num_edges)));
    TFG_DEBUG(debug_extent(fn, "in_degree", in_degree, sizeof(int32_t) * size_t(num_nodes)));
    TFG_DEBUG(debug_extent(fn, "workspace", num_edges > 0 ? workspace : nullptr, need));
    const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    return cuda_result(
        id32 ? tfg::launch_build_csr32(static_cast<const int32_t *>(edge_index), num_edges,
                                       num_nodes, rowptr, col, perm, in_degree, workspace, status,
                                       s, by_source)
             : tfg::launch_build_csr(static_cast<const int64_t *>(edge_index), num_edges,
                                     num_nodes, rowptr, col, perm, in_degree, workspace, status,
                                     s, by_source),
        fn);
}
}  // namespace

int tfg_build_csr(const int64_t *edge_index, int64_t num_edges, int64_t num_nodes,
                  int32_t *rowptr, int32_t *col, int32_t *perm, int32_t *in_degree,
                  void *workspace, size_t workspace_bytes, int32_t *status,
                  tfg_stream_t stream) {
    return build_csr_common("tfg_build_csr", false, edge_index, false, num_edges, num_nodes, rowptr,
                            col, perm, in_degree, workspace, workspace_bytes, status, stream);
}

int tfg_build_csr32(const int32_t *edge_index, int64_t num_edges, int64_t num_nodes,
                    int32_t *rowptr, int32_t *col, int32_t *perm, int32_t *in_degree,
                    void *workspace, size_t workspace_bytes, int32_t *status,
                    tfg_stream_t stream) {
    return build_csr_common("tfg_build_csr32", false, edge_index, true, num_edges, num_nodes,
                            rowptr, col, perm, in_degree, workspace, workspace_bytes, status,
                            stream);
}

int tfg_build_csr32_by_source(const int32_t *edge_index, int64_t num_edges, int64_t num_nodes,
                              int32_t *rowptr_src, int32_t *col_src, int32_t *perm_src,
                              int32_t *out_degree, void *workspace, size_t workspace_bytes,
                              int32_t *status, tfg_stream_t stream) {
    return build_csr_common("tfg_build_csr32_by_source", true, edge_index, true, num_edges,
                            num_nodes, rowptr_src, col_src, perm_src, out_degree, workspace,
                            workspace_bytes, status, stream);
}

int tfg_build_csr_by_source(const int64_t *edge_index, int64_t num_edges, int64_t num_nodes,
                            int32_t *rowptr_src, int32_t *col_src, int32_t *perm_src,
                            int32_t *out_degree, void *workspace, size_t workspace_bytes,
                            int32_t *status, tfg_stream_t stream) {
    return build_csr_common("tfg_build_csr_by_source", true, edge_index, false, num_edges, num_nodes,
                            rowptr_src, col_src, perm_src, out_degree, workspace, workspace_bytes,
                            status, stream);
}

int tfg_gcn_norm(const int32_t *rowptr, const int32_t *col, const int32_t *perm,
                 const float *edge_weight, int64_t num_nodes, int64_t num_edges,
                 int add_self_loops, float self_loop_fill, float *dinv, float *w_csr,
                 tfg_stream_t stream) {
    const char *fn = "tfg_gcn_norm";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, num_edges));
    TFG_NEED(rowptr, true, fn, "rowptr");
    TFG_NEED(dinv, num_nodes > 0, fn, "dinv");
    TFG_NEED(col, w_csr != nullptr && num_edges > 0, fn, "col");
    TFG_NEED(perm, (w_csr != nullptr || edge_weight != nullptr) && num_edges > 0, fn, "perm");
    TFG_DEBUG(debug_csr(fn, "col", rowptr, w_csr ? col : nullptr, w_csr || edge_weight ? perm : nullptr,
                        num_nodes, num_edges, nullptr, stream, w_csr != nullptr));
    TFG_DEBUG(debug_extent(fn, "edge_weight", edge_weight, sizeof(float) * size_t(num_edges)));
    TFG_DEBUG(debug_extent(fn, "dinv", dinv, sizeof(float) * size_t(num_nodes)));
    TFG_DEBUG(debug_extent(fn, "w_csr", w_csr, sizeof(float) * size_t(num_edges)));
    return cuda_result(tfg::launch_gcn_norm(rowptr, col, perm, edge_weight, num_nodes,
                                            add_self_loops, self_loop_fill, dinv, w_csr,
                                            reinterpret_cast<cudaStream_t>(stream)),
                       fn);
}

int tfg_aggregate_sum(const int32_t *rowptr, const int32_t *col, const float *w_csr,
                      const void *x, int x_dtype, int64_t num_nodes, int64_t num_features,
                      float *out, tfg_stream_t stream) {
    return aggregate_common("tfg_aggregate_sum", 0, rowptr, col, w_csr, nullptr, x, x_dtype,
                            num_nodes, num_features, 0, 0.f, out, stream);
}

int tfg_aggregate_mean(const int32_t *rowptr, const int32_t *col, const float *w_csr,
                       const void *x, int x_dtype, int64_t num_nodes, int64_t num_features,
                       float *out, tfg_stream_t stream) {
    return aggregate_common("tfg_aggregate_mean", 1, rowptr, col, w_csr, nullptr, x, x_dtype,
                            num_nodes, num_features, 0, 0.f, out, stream);
}

int tfg_aggregate_max(const int32_t *rowptr, const int32_t *col, const float *w_csr,
                      const void *x, int x_dtype, int64_t num_nodes, int64_t num_features,
                      float *out, tfg_stream_t stream) {
    return aggregate_common("tfg_aggregate_max", 2, rowptr, col, w_csr, nullptr, x, x_dtype,
                            num_nodes, num_features, 0, 0.f, out, stream);
}

int tfg_gcn_aggregate_sum(const int32_t *rowptr, const int32_t *col, const float *dinv,
                          const float *w_csr, const void *x, int x_dtype, int64_t num_nodes,
                          int64_t num_features, int add_self_loops, float self_loop_fill,
                          float *out, tfg_stream_t stream) {
    return aggregate_common("tfg_gcn_aggregate_sum", 3, rowptr, col, w_csr, dinv, x, x_dtype,
                            num_nodes, num_features, add_self_loops, self_loop_fill, out, stream);
}

int tfg_aggregate_backward_workspace_size(int reduce, int64_t num_edges, size_t *bytes) {
    const char *fn = "tfg_aggregate_backward_workspace_size";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, 1, num_edges));
    if (reduce != TFG_SUM && reduce != TFG_MEAN)
        return fail(TFG_ERR_INVALID_ARG, "%s: reduce must be TFG_SUM or TFG_MEAN", fn);
    TFG_NEED(bytes, true, fn, "bytes");
    *bytes = tfg::backward_workspace_bytes(reduce, num_edges);
    return ok();
}

int tfg_aggregate_backward(int reduce, const int32_t *rowptr_src, const int32_t *col_src,
                           const int32_t *perm_src, const float *edge_weight,
                           const int32_t *in_degree, const float *grad_out, int64_t num_nodes,
                           int64_t num_edges, int64_t num_features, float *grad_x,
                           void *workspace, size_t workspace_bytes, tfg_stream_t stream) {
    const char *fn = "tfg_aggregate_backward";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, num_edges));
    TFG_TRY(check_features(fn, num_nodes, num_features));
    if (reduce != TFG_SUM && reduce != TFG_MEAN)
        return fail(TFG_ERR_INVALID_ARG, "%s: reduce must be TFG_SUM or TFG_MEAN", fn);
    TFG_NEED(rowptr_src, true, fn, "rowptr_src");
    TFG_NEED(col_src, num_edges > 0, fn, "col_src");
    TFG_NEED(perm_src, num_edges > 0 && (edge_weight != nullptr || reduce == TFG_MEAN), fn,
             "perm_src");
    TFG_NEED(in_degree, reduce == TFG_MEAN && num_edges > 0, fn, "in_degree");
    TFG_NEED(grad_out, num_nodes > 0, fn, "grad_out");
    TFG_NEED(grad_x, num_nodes > 0, fn, "grad_x");
    const bool weighted = num_edges > 0 && (edge_weight != nullptr || reduce == TFG_MEAN);
    const size_t need = weighted ? tfg::backward_workspace_bytes(reduce, num_edges) : 0;
    if (need > 0 && (workspace == nullptr || workspace_bytes < need))
        return fail(TFG_ERR_WORKSPACE, "%s: workspace of %zu bytes needed, %zu given", fn, need,
                    workspace ? workspace_bytes : size_t(0));
    TFG_DEBUG(debug_csr(fn, "col_src", rowptr_src, col_src, weighted ? perm_src : nullptr, num_nodes,
                        num_edges, nullptr, stream));
    TFG_DEBUG(debug_extent(fn, "edge_weight", edge_weight, sizeof(float) * size_t(num_edges)));
    TFG_DEBUG(debug_extent(fn, "in_degree", reduce == TFG_MEAN ? in_degree : nullptr,
                           sizeof(int32_t) * size_t(num_nodes)));
    TFG_DEBUG(debug_extent(fn, "grad_out", grad_out, sizeof(float) * size_t(num_nodes * num_features)));
    TFG_DEBUG(debug_extent(fn, "grad_x", grad_x, sizeof(float) * size_t(num_nodes * num_features)));
    TFG_DEBUG(debug_extent(fn, "workspace", need ? workspace : nullptr, need));
    return cuda_result(tfg::launch_aggregate_backward(reduce, rowptr_src, col_src, perm_src,
                                                      edge_weight, in_degree, grad_out, num_nodes,
                                                      num_edges, num_features, grad_x, workspace,
                                                      reinterpret_cast<cudaStream_t>(stream)),
                       fn);
}

int tfg_gcn_aggregate_backward(const int32_t *rowptr_src, const int32_t *col_src,
                               const float *dinv, const float *grad_out, int64_t num_nodes,
                               int64_t num_features, int add_self_loops, float self_loop_fill,
                               float *grad_x, tfg_stream_t stream) {
    return aggregate_common("tfg_gcn_aggregate_backward", 3, rowptr_src, col_src, nullptr, dinv,
                            grad_out, TFG_F32, num_nodes, num_features, add_self_loops,
                            self_loop_fill, grad_x, stream);
}

int tfg_aggregate_max_argmax(const int32_t *rowptr, const int32_t *col, const int32_t *perm,
                             const float *w_csr, const void *x, int x_dtype, int64_t num_nodes,
                             int64_t num_features, float *out, int32_t *argmax,
                             tfg_stream_t stream) {
    const char *fn = "tfg_aggregate_max_argmax";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, 0));
    TFG_TRY(check_features(fn, num_nodes, num_features));
    TFG_TRY(check_dtype(fn, x_dtype));
    TFG_NEED(rowptr, true, fn, "rowptr");
    TFG_NEED(perm, col != nullptr, fn, "perm");
    TFG_NEED(x, num_nodes > 0, fn, "x");
    TFG_NEED(out, num_nodes > 0, fn, "out");
    TFG_NEED(argmax, num_nodes > 0, fn, "argmax");
#if TFG_CHECK_BOUNDS
    {
        int64_t e = 0;
        TFG_DEBUG(debug_csr(fn, "col", rowptr, col, perm, num_nodes, -1, &e, stream));
        TFG_DEBUG(debug_extent(fn, "w_csr", w_csr, sizeof(float) * size_t(e)));
        TFG_DEBUG(debug_extent(fn, "x", x, elem_bytes(x_dtype) * size_t(num_nodes * num_features)));
        TFG_DEBUG(debug_extent(fn, "out", out, sizeof(float) * size_t(num_nodes * num_features)));
        TFG_DEBUG(debug_extent(fn, "argmax", argmax, sizeof(int32_t) * size_t(num_nodes * num_features)));
    }
#endif
    return cuda_result(tfg::launch_max_argmax(rowptr, col, perm, w_csr, x, x_dtype, num_nodes,
                                              num_features, out, argmax,
                                              reinterpret_cast<cudaStream_t>(stream)),
                       fn);
}

int tfg_aggregate_max_backward_workspace_size(int64_t num_nodes, int64_t num_edges,
                                              int64_t num_features, size_t *bytes) {
    const char *fn = "tfg_aggregate_max_backward_workspace_size";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, num_edges));
    TFG_TRY(check_features(fn, num_nodes, num_features));
    TFG_NEED(bytes, true, fn, "bytes");
    *bytes = tfg::max_backward_workspace_bytes(num_nodes, num_edges, num_features);
    return ok();
}

int tfg_aggregate_max_backward(const int32_t *rowptr_src, const int32_t *col_src,
                               const int32_t *perm_src, const int32_t *argmax,
                               const float *edge_weight, const float *grad_out,
                               int64_t num_nodes, int64_t num_edges, int64_t num_features,
                               float *grad_x, void *workspace, size_t workspace_bytes,
                               tfg_stream_t stream) {
    const char *fn = "tfg_aggregate_max_backward";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, num_edges));
    TFG_TRY(check_features(fn, num_nodes, num_features));
    TFG_NEED(rowptr_src, true, fn, "rowptr_src");
    TFG_NEED(col_src, num_edges > 0, fn, "col_src");
    TFG_NEED(perm_src, num_edges > 0, fn, "perm_src");
    TFG_NEED(argmax, num_nodes > 0, fn, "argmax");
    TFG_NEED(grad_out, num_nodes > 0, fn, "grad_out");
    TFG_NEED(grad_x, num_nodes > 0, fn, "grad_x");
    const size_t need =
        workspace ? tfg::max_backward_workspace_bytes(num_nodes, num_edges, num_features) : 0;
    if (need > 0 && workspace_bytes < need)
        return fail(TFG_ERR_WORKSPACE, "%s: workspace of %zu bytes needed, %zu given", fn, need,
                    workspace_bytes);
    if (need > 0 && reinterpret_cast<uintptr_t>(workspace) % 16 != 0)
        return fail(TFG_ERR_INVALID_ARG, "%s: workspace must be 16-byte aligned", fn);
    TFG_DEBUG(debug_csr(fn, "col_src", rowptr_src, col_src, perm_src, num_nodes, num_edges,
                        nullptr, stream));
    TFG_DEBUG(debug_extent(fn, "edge_weight", edge_weight, sizeof(float) * size_t(num_edges)));
    TFG_DEBUG(debug_extent(fn, "argmax", argmax, sizeof(int32_t) * size_t(num_nodes * num_features)));
    TFG_DEBUG(debug_extent(fn, "grad_out", grad_out, sizeof(float) * size_t(num_nodes * num_features)));
    TFG_DEBUG(debug_extent(fn, "grad_x", grad_x, sizeof(float) * size_t(num_nodes * num_features)));
    TFG_DEBUG(debug_extent(fn, "workspace", need ? workspace : nullptr, need));
    const int32_t *col = num_edges > 0 ? col_src : nullptr;
    const cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
    return cuda_result(
        need ? tfg::launch_max_backward_marked(rowptr_src, col, perm_src, argmax, edge_weight,
                                               grad_out, num_nodes, num_edges, num_features, grad_x,
                                               workspace, s)
             : tfg::launch_max_backward(rowptr_src, col, perm_src, argmax, edge_weight, grad_out,
                                        num_nodes, num_features, grad_x, s),
        fn);
}

int tfg_propagate_workspace_size(int64_t num_nodes, int64_t num_features, int64_t num_hops,
                                 size_t *bytes) {
    const char *fn = "tfg_propagate_workspace_size";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, 0));
    TFG_TRY(check_features(fn, num_nodes, num_features));
    if (num_hops < 0 || num_hops > kMaxHops)
        return fail(TFG_ERR_INVALID_ARG, "%s: num_hops must be in [0, %d]", fn, kMaxHops);
    TFG_NEED(bytes, true, fn, "bytes");
    *bytes = tfg::propagate_workspace_bytes(num_nodes, num_features, num_hops);
    return ok();
}

int tfg_appnp_propagate(const int32_t *rowptr, const int32_t *col, const float *dinv,
                        const float *w_csr, const void *x0, int x_dtype, int64_t num_nodes,
                        int64_t num_features, int64_t num_hops, float alpha, int add_self_loops,
                        float self_loop_fill, float *out, void *workspace,
                        size_t workspace_bytes, tfg_stream_t stream) {
    return propagate_common("tfg_appnp_propagate", rowptr, col, dinv, w_csr, x0, x_dtype,
                            num_nodes, num_features, num_hops, alpha, add_self_loops,
                            self_loop_fill, out, workspace, workspace_bytes, stream);
}

int tfg_sgc_propagate(const int32_t *rowptr, const int32_t *col, const float *dinv,
                      const float *w_csr, const void *x0, int x_dtype, int64_t num_nodes,
                      int64_t num_features, int64_t num_hops, int add_self_loops,
                      float self_loop_fill, float *out, void *workspace, size_t workspace_bytes,
                      tfg_stream_t stream) {
    return propagate_common("tfg_sgc_propagate", rowptr, col, dinv, w_csr, x0, x_dtype,
                            num_nodes, num_features, num_hops, 0.f, add_self_loops,
                            self_loop_fill, out, workspace, workspace_bytes, stream);
}

int tfg_edge_softmax_workspace_size(int64_t num_nodes, int heads, size_t *bytes) {
    const char *fn = "tfg_edge_softmax_workspace_size";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, 0));
    if (heads < 1) return fail(TFG_ERR_INVALID_ARG, "%s: heads must be >= 1", fn);
    TFG_NEED(bytes, true, fn, "bytes");
    *bytes = tfg::softmax_workspace_bytes(num_nodes, heads);
    return ok();
}

int tfg_edge_softmax_aggregate(const int32_t *rowptr, const int32_t *col, const void *x,
                               int x_dtype, int64_t num_nodes, int64_t num_edges, int heads,
                               int channels,
                               const float *a_src, const float *a_dst, float negative_slope,
                               float *out, float *alpha, void *workspace,
                               size_t workspace_bytes, tfg_stream_t stream) {
    const char *fn = "tfg_edge_softmax_aggregate";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, num_edges));
    if (heads < 1 || channels < 1)
        return fail(TFG_ERR_INVALID_ARG, "%s: heads and channels must be >= 1", fn);
    TFG_TRY(check_features(fn, num_nodes, int64_t(heads) * channels));
    TFG_TRY(check_dtype(fn, x_dtype));
    TFG_NEED(rowptr, true, fn, "rowptr");
    TFG_NEED(col, num_edges > 0, fn, "col");
    TFG_NEED(x, num_nodes > 0, fn, "x");
    TFG_NEED(out, num_nodes > 0, fn, "out");
    TFG_NEED(a_src, true, fn, "a_src");
    TFG_NEED(a_dst, true, fn, "a_dst");
    const size_t need = tfg::softmax_workspace_bytes(num_nodes, heads);
    if (num_nodes > 0 && (workspace == nullptr || workspace_bytes < need))
        return fail(TFG_ERR_WORKSPACE, "%s: workspace of %zu bytes needed, %zu given", fn, need,
                    workspace ? workspace_bytes : size_t(0));
    TFG_DEBUG(debug_csr(fn, "col", rowptr, col, nullptr, num_nodes, num_edges, nullptr, stream));
    TFG_DEBUG(debug_extent(fn, "x", x, elem_bytes(x_dtype) * size_t(num_nodes * heads * channels)));
    TFG_DEBUG(debug_extent(fn, "out", out, sizeof(float) * size_t(num_nodes * heads * channels)));
    TFG_DEBUG(debug_extent(fn, "alpha", alpha, sizeof(float) * size_t(num_edges * heads)));
    TFG_DEBUG(debug_extent(fn, "a_src", a_src, sizeof(float) * size_t(heads * channels)));
    TFG_DEBUG(debug_extent(fn, "a_dst", a_dst, sizeof(float) * size_t(heads * channels)));
    TFG_DEBUG(debug_extent(fn, "workspace", num_nodes > 0 ? workspace : nullptr, need));
    return cuda_result(tfg::launch_edge_softmax(rowptr, num_edges > 0 ? col : nullptr, x, x_dtype,
                                                num_nodes, num_edges, heads, channels, a_src, a_dst,
                                                negative_slope, out, alpha, workspace,
                                                reinterpret_cast<cudaStream_t>(stream)),
                       fn);
}

int tfg_edge_softmax_backward_workspace_size(int64_t num_nodes, int heads, int channels,
                                             size_t *bytes) {
    const char *fn = "tfg_edge_softmax_backward_workspace_size";
    TFG_RANGE(fn);
    TFG_NEED(bytes, true, fn, "bytes");
    TFG_TRY(check_counts(fn, num_nodes, 0));
    if (!tfg::attention_backward_layout_ok(heads, channels))
        return fail(TFG_ERR_INVALID_ARG,
                    "%s: channels must be a power of two up to 32 or a multiple of 32, H*C <= 256",
                    fn);
    *bytes = tfg::attention_backward_workspace_bytes(num_nodes, heads, channels);
    return ok();
}

int tfg_edge_softmax_aggregate_backward(const int32_t *rowptr, const int32_t *col,
                                        const int32_t *rowptr_src, const int32_t *col_src,
                                        const void *x, int x_dtype, int64_t num_nodes,
                                        int64_t num_edges, int heads, int channels,
                                        const float *a_src, const float *a_dst,
                                        float negative_slope, const float *out,
                                        const float *grad_out, float *grad_x, float *grad_a_src,
                                        float *grad_a_dst, void *workspace,
                                        size_t workspace_bytes, tfg_stream_t stream) {
    const char *fn = "tfg_edge_softmax_aggregate_backward";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, num_edges));
    if (!tfg::attention_backward_layout_ok(heads, channels))
        return fail(TFG_ERR_INVALID_ARG,
                    "%s: channels must be a power of two up to 32 or a multiple of 32, H*C <= 256",
                    fn);
    TFG_TRY(check_features(fn, num_nodes, int64_t(heads) * channels));
    TFG_TRY(check_dtype(fn, x_dtype));
    TFG_NEED(rowptr, true, fn, "rowptr");
    TFG_NEED(rowptr_src, true, fn, "rowptr_src");
    TFG_NEED(col, num_edges > 0, fn, "col");
    TFG_NEED(col_src, num_edges > 0, fn, "col_src");
    TFG_NEED(x, num_nodes > 0, fn, "x");
    TFG_NEED(out, num_nodes > 0, fn, "out");
    TFG_NEED(grad_out, num_nodes > 0, fn, "grad_out");
    TFG_NEED(grad_x, num_nodes > 0, fn, "grad_x");
    TFG_NEED(a_src, true, fn, "a_src");
    TFG_NEED(a_dst, true, fn, "a_dst");
    TFG_NEED(grad_a_src, true, fn, "grad_a_src");
    TFG_NEED(grad_a_dst, true, fn, "grad_a_dst");
    const size_t need = tfg::attention_backward_workspace_bytes(num_nodes, heads, channels);
    if (workspace == nullptr || workspace_bytes < need)
        return fail(TFG_ERR_WORKSPACE, "%s: workspace of %zu bytes needed, %zu given", fn, need,
                    workspace ? workspace_bytes : size_t(0));
#if TFG_CHECK_BOUNDS
    {
        const size_t nf = size_t(num_nodes) * size_t(heads) * size_t(channels);
        TFG_DEBUG(debug_csr(fn, "col", rowptr, col, nullptr, num_nodes, num_edges, nullptr, stream));
        TFG_DEBUG(debug_csr(fn, "col_src", rowptr_src, col_src, nullptr, num_nodes, num_edges,
                            nullptr, stream));
        TFG_DEBUG(debug_extent(fn, "x", x, elem_bytes(x_dtype) * nf));
        TFG_DEBUG(debug_extent(fn, "out", out, sizeof(float) * nf));
        TFG_DEBUG(debug_extent(fn, "grad_out", grad_out, sizeof(float) * nf));
        TFG_DEBUG(debug_extent(fn, "grad_x", grad_x, sizeof(float) * nf));
        TFG_DEBUG(debug_extent(fn, "workspace", workspace, need));
    }
#endif
    return cuda_result(tfg::launch_edge_softmax_backward(
                           rowptr, col, rowptr_src, col_src, x, x_dtype, num_nodes,
                           num_edges, heads, channels, a_src, a_dst, negative_slope, out, grad_out, grad_x,
                           grad_a_src, grad_a_dst, workspace, reinterpret_cast<cudaStream_t>(stream)),
                       fn);
}

int tfg_dot_edge_softmax_backward_workspace_size(int64_t num_nodes, int heads, int channels,
                                                 size_t *bytes) {
    const char *fn = "tfg_dot_edge_softmax_backward_workspace_size";
    TFG_RANGE(fn);
    TFG_NEED(bytes, true, fn, "bytes");
    TFG_TRY(check_counts(fn, num_nodes, 0));
    if (!tfg::attention_backward_layout_ok(heads, channels))
        return fail(TFG_ERR_INVALID_ARG,
                    "%s: channels must be a power of two up to 32 or a multiple of 32, H*C <= 256",
                    fn);
    *bytes = tfg::dot_attention_backward_workspace_bytes(num_nodes, heads);
    return TFG_OK;
}

int tfg_dot_edge_softmax_aggregate_backward(const int32_t *rowptr, const int32_t *col,
                                            const int32_t *rowptr_src, const int32_t *col_src,
                                            const void *q, const void *k, const void *v,
                                            int x_dtype, int64_t num_nodes, int64_t num_edges,
                                            int heads, int channels, float scale,
                                            const float *out, const float *grad_out,
                                            float *grad_q, float *grad_k, float *grad_v,
                                            void *workspace, size_t workspace_bytes,
                                            tfg_stream_t stream) {
    const char *fn = "tfg_dot_edge_softmax_aggregate_backward";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, num_edges));
    if (!tfg::attention_backward_layout_ok(heads, channels))
        return fail(TFG_ERR_INVALID_ARG,
                    "%s: channels must be a power of two up to 32 or a multiple of 32, H*C <= 256",
                    fn);
    TFG_TRY(check_features(fn, num_nodes, int64_t(heads) * channels));
    TFG_TRY(check_dtype(fn, x_dtype));
    if (!(scale == scale) || scale == INFINITY || scale == -INFINITY)
        return fail(TFG_ERR_INVALID_ARG, "%s: scale must be finite", fn);
    TFG_NEED(rowptr, true, fn, "rowptr");
    TFG_NEED(rowptr_src, true, fn, "rowptr_src");
    TFG_NEED(col, num_edges > 0, fn, "col");
    TFG_NEED(col_src, num_edges > 0, fn, "col_src");
    TFG_NEED(q, num_nodes > 0, fn, "q");
    TFG_NEED(k, num_nodes > 0, fn, "k");
    TFG_NEED(v, num_nodes > 0, fn, "v");
    TFG_NEED(out, num_nodes > 0, fn, "out");
    TFG_NEED(grad_out, num_nodes > 0, fn, "grad_out");
    TFG_NEED(grad_q, num_nodes > 0, fn, "grad_q");
    TFG_NEED(grad_k, num_nodes > 0, fn, "grad_k");
    TFG_NEED(grad_v, num_nodes > 0, fn, "grad_v");
    const size_t need = tfg::dot_attention_backward_workspace_bytes(num_nodes, heads);
    if (workspace == nullptr || workspace_bytes < need)
        return fail(TFG_ERR_WORKSPACE, "%s: workspace of %zu bytes needed, %zu given", fn, need,
                    workspace ? workspace_bytes : size_t(0));
#if TFG_CHECK_BOUNDS
    {
        const size_t nf = size_t(num_nodes) * size_t(heads) * size_t(channels);
        TFG_DEBUG(debug_csr(fn, "col", rowptr, col, nullptr, num_nodes, num_edges, nullptr, stream));
        TFG_DEBUG(debug_csr(fn, "col_src", rowptr_src, col_src, nullptr, num_nodes, num_edges,
                            nullptr, stream));
        TFG_DEBUG(debug_extent(fn, "q", q, elem_bytes(x_dtype) * nf));
        TFG_DEBUG(debug_extent(fn, "k", k, elem_bytes(x_dtype) * nf));
        TFG_DEBUG(debug_extent(fn, "v", v, elem_bytes(x_dtype) * nf));
        TFG_DEBUG(debug_extent(fn, "out", out, sizeof(float) * nf));
        TFG_DEBUG(debug_extent(fn, "grad_out", grad_out, sizeof(float) * nf));
        TFG_DEBUG(debug_extent(fn, "grad_q", grad_q, sizeof(float) * nf));
        TFG_DEBUG(debug_extent(fn, "grad_k", grad_k, sizeof(float) * nf));
        TFG_DEBUG(debug_extent(fn, "grad_v", grad_v, sizeof(float) * nf));
        TFG_DEBUG(debug_extent(fn, "workspace", workspace, need));
    }
#endif
    return cuda_result(tfg::launch_dot_softmax_backward(
                           rowptr, col, rowptr_src, col_src, q, k, v, x_dtype, num_nodes,
                           num_edges, heads, channels, scale, out, grad_out, grad_q, grad_k,
                           grad_v, workspace, reinterpret_cast<cudaStream_t>(stream)),
                       fn);
}

int tfg_dot_edge_softmax_aggregate(const int32_t *rowptr, const int32_t *col, const void *q,
                                   const void *k, const void *v, int x_dtype, int64_t num_nodes,
                                   int64_t num_edges, int heads, int channels, float scale,
                                   float *out, float *alpha, tfg_stream_t stream) {
    const char *fn = "tfg_dot_edge_softmax_aggregate";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, num_edges));
    if (heads < 1 || channels < 1)
        return fail(TFG_ERR_INVALID_ARG, "%s: heads and channels must be >= 1", fn);
    if (channels > tfg::dot_softmax_max_channels())
        return fail(TFG_ERR_TOO_LARGE, "%s: at most %d channels per head", fn,
                    tfg::dot_softmax_max_channels());
    TFG_TRY(check_features(fn, num_nodes, int64_t(heads) * channels));
    TFG_TRY(check_dtype(fn, x_dtype));
    if (!(scale == scale) || scale == INFINITY || scale == -INFINITY)
        return fail(TFG_ERR_INVALID_ARG, "%s: scale must be finite", fn);
    TFG_NEED(rowptr, true, fn, "rowptr");
    TFG_NEED(col, num_edges > 0, fn, "col");
    TFG_NEED(q, num_nodes > 0, fn, "q");
    TFG_NEED(k, num_nodes > 0, fn, "k");
    TFG_NEED(v, num_nodes > 0, fn, "v");
    TFG_NEED(out, num_nodes > 0, fn, "out");
#if TFG_CHECK_BOUNDS
    {
        const size_t nf = size_t(num_nodes) * size_t(heads) * size_t(channels);
        TFG_DEBUG(debug_csr(fn, "col", rowptr, col, nullptr, num_nodes, num_edges, nullptr, stream));
        TFG_DEBUG(debug_extent(fn, "q", q, elem_bytes(x_dtype) * nf));
        TFG_DEBUG(debug_extent(fn, "k", k, elem_bytes(x_dtype) * nf));
        TFG_DEBUG(debug_extent(fn, "v", v, elem_bytes(x_dtype) * nf));
        TFG_DEBUG(debug_extent(fn, "out", out, sizeof(float) * nf));
        TFG_DEBUG(debug_extent(fn, "alpha", alpha, sizeof(float) * size_t(num_edges * heads)));
    }
#endif
    return cuda_result(tfg::launch_dot_softmax(rowptr, num_edges > 0 ? col : nullptr, q, k, v,
                                               x_dtype, num_nodes, num_edges, heads, channels,
                                               scale, out, alpha,
                                               reinterpret_cast<cudaStream_t>(stream)),
                       fn);
}

int tfg_edge_softmax_aggregate_noalloc(const int32_t *rowptr, const int32_t *col, const void *x,
                                       int x_dtype, int64_t num_nodes, int64_t num_edges,
                                       int heads, int channels, const float *a_src,
                                       const float *a_dst, float negative_slope, float *out,
                                       float *alpha, tfg_stream_t stream) {
    const char *fn = "tfg_edge_softmax_aggregate_noalloc";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, num_edges));
    if (heads < 1 || channels < 1)
        return fail(TFG_ERR_INVALID_ARG, "%s: heads and channels must be >= 1", fn);
    const int64_t limit = tfg::noalloc_softmax_max_node_heads();
    if (num_nodes * heads > limit)
        return fail(TFG_ERR_TOO_LARGE,
                    "%s: num_nodes * heads = %lld exceeds the built-in scratch of %lld node-head "
                    "pairs; use tfg_edge_softmax_aggregate with a caller workspace",
                    fn, (long long)(num_nodes * heads), (long long)limit);
    TFG_TRY(check_features(fn, num_nodes, int64_t(heads) * channels));
    TFG_TRY(check_dtype(fn, x_dtype));
    TFG_NEED(rowptr, true, fn, "rowptr");
    TFG_NEED(col, num_edges > 0, fn, "col");
    TFG_NEED(x, num_nodes > 0, fn, "x");
    TFG_NEED(out, num_nodes > 0, fn, "out");
    TFG_NEED(a_src, true, fn, "a_src");
    TFG_NEED(a_dst, true, fn, "a_dst");
    if (num_nodes == 0) return ok();
    TFG_DEBUG(debug_csr(fn, "col", rowptr, col, nullptr, num_nodes, num_edges, nullptr, stream));
    TFG_DEBUG(debug_extent(fn, "x", x, elem_bytes(x_dtype) * size_t(num_nodes * heads * channels)));
    TFG_DEBUG(debug_extent(fn, "out", out, sizeof(float) * size_t(num_nodes * heads * channels)));
    TFG_DEBUG(debug_extent(fn, "alpha", alpha, sizeof(float) * size_t(num_edges * heads)));
    void *scratch = nullptr;
    size_t scratch_bytes = 0;
    cudaError_t err = tfg::noalloc_softmax_scratch(&scratch, &scratch_bytes);
    if (err != cudaSuccess) return cuda_result(err, fn);
    if (tfg::softmax_workspace_bytes(num_nodes, heads) > scratch_bytes)
        return fail(TFG_ERR_TOO_LARGE, "%s: scratch too small", fn);
    return cuda_result(tfg::launch_edge_softmax(rowptr, num_edges > 0 ? col : nullptr, x, x_dtype,
                                                num_nodes, num_edges, heads, channels, a_src, a_dst,
                                                negative_slope, out, alpha, scratch,
                                                reinterpret_cast<cudaStream_t>(stream)),
                       fn);
}

int tfg_segment_pool_meanmax(const void *x, int x_dtype, const int64_t *batch,
                             int64_t num_nodes, int64_t num_graphs, int64_t num_features,
                             float *out, int32_t *status, tfg_stream_t stream) {
    const char *fn = "tfg_segment_pool_meanmax";
    TFG_RANGE(fn);
    if (num_nodes < 0 || num_graphs < 0)
        return fail(TFG_ERR_INVALID_ARG, "%s: negative size", fn);
    if (num_graphs >= kIndexLimit) return fail(TFG_ERR_TOO_LARGE, "%s: too many graphs", fn);
    TFG_TRY(check_features(fn, num_nodes > num_graphs ? num_nodes : num_graphs, num_features));
    TFG_TRY(check_dtype(fn, x_dtype));
    if (num_features > int64_t(65535) * 8)
        return fail(TFG_ERR_TOO_LARGE, "%s: at most %d features", fn, 65535 * 8);
    TFG_NEED(x, num_nodes > 0, fn, "x");
    TFG_NEED(batch, num_nodes > 0, fn, "batch");
    TFG_NEED(out, num_graphs > 0, fn, "out");
    TFG_NEED(status, true, fn, "status");
    TFG_DEBUG(debug_extent(fn, "x", x, elem_bytes(x_dtype) * size_t(num_nodes * num_features)));
    TFG_DEBUG(debug_extent(fn, "batch", batch, sizeof(int64_t) * size_t(num_nodes)));
    TFG_DEBUG(debug_extent(fn, "out", out, sizeof(float) * 2 * size_t(num_graphs * num_features)));
    return cuda_result(tfg::launch_segment_pool(x, x_dtype, batch, num_nodes, num_graphs,
                                                num_features, 3 /* mean | max */, out, status,
                                                reinterpret_cast<cudaStream_t>(stream)),
                       fn);
}

int tfg_batch_graphs_workspace_size(int64_t num_graphs, size_t *bytes) {
    const char *fn = "tfg_batch_graphs_workspace_size";
    TFG_RANGE(fn);
    if (num_graphs < 0) return fail(TFG_ERR_INVALID_ARG, "%s: negative size", fn);
    TFG_NEED(bytes, true, fn, "bytes");
    *bytes = tfg::batch_graphs_workspace_bytes(num_graphs);
    return ok();
}

int tfg_batch_graphs(int64_t num_graphs, const int64_t *node_counts, const int64_t *edge_counts,
                     const int64_t *edge_index, int64_t total_edges, int64_t total_nodes,
                     int64_t *out_edge_index, int64_t *batch, int64_t *node_offsets,
                     void *workspace, size_t workspace_bytes, int32_t *status,
                     tfg_stream_t stream) {
    const char *fn = "tfg_batch_graphs";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, total_nodes, total_edges));
    if (num_graphs < 0) return fail(TFG_ERR_INVALID_ARG, "%s: negative graph count", fn);
    if (num_graphs >= kIndexLimit) return fail(TFG_ERR_TOO_LARGE, "%s: too many graphs", fn);
    if (num_graphs == 0 && (total_nodes > 0 || total_edges > 0))
        return fail(TFG_ERR_INVALID_ARG, "%s: nodes or edges given for zero graphs", fn);
    TFG_NEED(node_counts, num_graphs > 0, fn, "node_counts");
    TFG_NEED(edge_counts, num_graphs > 0, fn, "edge_counts");
    TFG_NEED(edge_index, total_edges > 0, fn, "edge_index");
    TFG_NEED(out_edge_index, total_edges > 0, fn, "out_edge_index");
    TFG_NEED(batch, total_nodes > 0, fn, "batch");
    TFG_NEED(node_offsets, true, fn, "node_offsets");
    TFG_NEED(status, true, fn, "status");
    const size_t need = tfg::batch_graphs_workspace_bytes(num_graphs);
    if (workspace == nullptr || workspace_bytes < need)
        return fail(TFG_ERR_WORKSPACE, "%s: workspace of %zu bytes needed, %zu given", fn, need,
                    workspace ? workspace_bytes : size_t(0));
    TFG_DEBUG(debug_extent(fn, "node_counts", node_counts, sizeof(int64_t) * size_t(num_graphs)));
    TFG_DEBUG(debug_extent(fn, "edge_counts", edge_counts, sizeof(int64_t) * size_t(num_graphs)));
    TFG_DEBUG(debug_extent(fn, "edge_index", edge_index, sizeof(int64_t) * 2 * size_t(total_edges)));
    TFG_DEBUG(debug_extent(fn, "out_edge_index", out_edge_index,
                           sizeof(int64_t) * 2 * size_t(total_edges)));
    TFG_DEBUG(debug_extent(fn, "batch", batch, sizeof(int64_t) * size_t(total_nodes)));
    TFG_DEBUG(debug_extent(fn, "node_offsets", node_offsets, sizeof(int64_t) * size_t(num_graphs + 1)));
    return cuda_result(tfg::launch_batch_graphs(num_graphs, node_counts, edge_counts, edge_index,
                                                total_edges, total_nodes, out_edge_index, batch,
                                                node_offsets, workspace, status,
                                                reinterpret_cast<cudaStream_t>(stream)),
                       fn);
}

int tfg_segment_pool(const void *x, int x_dtype, const int64_t *batch, int64_t num_nodes,
                     int64_t num_graphs, int64_t num_features, int reduce, float *out,
                     int32_t *status, tfg_stream_t stream) {
    const char *fn = "tfg_segment_pool";
    TFG_RANGE(fn);
    if (num_nodes < 0 || num_graphs < 0)
        return fail(TFG_ERR_INVALID_ARG, "%s: negative size", fn);
    if (num_graphs >= kIndexLimit) return fail(TFG_ERR_TOO_LARGE, "%s: too many graphs", fn);
    TFG_TRY(check_features(fn, num_nodes > num_graphs ? num_nodes : num_graphs, num_features));
    TFG_TRY(check_dtype(fn, x_dtype));
    if (num_features > int64_t(65535) * 8)
        return fail(TFG_ERR_TOO_LARGE, "%s: at most %d features", fn, 65535 * 8);
    if (reduce != TFG_SUM && reduce != TFG_MEAN && reduce != TFG_MAX)
        return fail(TFG_ERR_INVALID_ARG, "%s: unknown reducer %d", fn, reduce);
    TFG_NEED(x, num_nodes > 0, fn, "x");
    TFG_NEED(batch, num_nodes > 0, fn, "batch");
    TFG_NEED(out, num_graphs > 0, fn, "out");
    TFG_NEED(status, true, fn, "status");
    TFG_DEBUG(debug_extent(fn, "x", x, elem_bytes(x_dtype) * size_t(num_nodes * num_features)));
    TFG_DEBUG(debug_extent(fn, "batch", batch, sizeof(int64_t) * size_t(num_nodes)));
    TFG_DEBUG(debug_extent(fn, "out", out, sizeof(float) * size_t(num_graphs * num_features)));
    return cuda_result(tfg::launch_segment_pool(x, x_dtype, batch, num_nodes, num_graphs,
                                                num_features, reduce, out, status,
                                                reinterpret_cast<cudaStream_t>(stream)),
                       fn);
}

int tfg_gather_xor(const int32_t *col, int64_t num_edges, const void *x, int64_t num_nodes,
                   int64_t row_bytes, uint32_t *out, tfg_stream_t stream) {
    const char *fn = "tfg_gather_xor";
    TFG_RANGE(fn);
    TFG_TRY(check_counts(fn, num_nodes, num_edges));
    if (row_bytes < 16 || row_bytes > 512 || (row_bytes & (row_bytes - 1)) != 0)
        return fail(TFG_ERR_INVALID_ARG, "%s: row_bytes must be a power of two in [16, 512] (%lld)",
                    fn, (long long)row_bytes);
    TFG_NEED(col, num_edges > 0, fn, "col");
    TFG_NEED(x, num_edges > 0, fn, "x");
    TFG_NEED(out, true, fn, "out");
    if (reinterpret_cast<uintptr_t>(x) % 16 != 0)
        return fail(TFG_ERR_INVALID_ARG, "%s: x must be 16-byte aligned", fn);
    TFG_DEBUG(debug_csr(fn, "col", nullptr, col, nullptr, num_nodes, num_edges, nullptr, stream));
    TFG_DEBUG(debug_extent(fn, "x", num_edges > 0 ? x : nullptr, size_t(num_nodes) * size_t(row_bytes)));
    TFG_DEBUG(debug_extent(fn, "out", out, size_t(row_bytes)));
    return cuda_result(tfg::launch_gather_xor(col, num_edges, x, row_bytes, out,
                                              reinterpret_cast<cudaStream_t>(stream)),
                       fn);
}

}  // extern "C"
