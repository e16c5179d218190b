/*
 * tfg.h -- C ABI of the GB300 (sm_103a) graph message-aggregation library.
 *
 * The library implements the data-parallel core of the graph map-reduce
 * framework of tf_geometric (arXiv:2101.11552): gathering source-node
 * features along the edges of a COO edge list, weighting them, and reducing
 * them per target node (sum / mean / max, GCN normalisation, additive and
 * dot-product attention, multi-hop APPNP / SGC propagation, and the
 * gradients of the aggregations); plus BatchGraph construction and the
 * per-graph segment reductions used for graph pooling.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - edge_index is the COO adjacency of Section 2.1.1 ("Graph Data
 *    Structure"): int64 [2, E] row-major, row 0 = source node of each edge,
 *    row 1 = target node.  An entry A_ij > 0 is an edge i -> j; messages flow
 *    from source to target and are reduced at the target (Fig. 1).
 *  - The "reduce key" of the map-reduce framework (Section 2.1.2, Fig. 5b) is
 *    the target node.  tfg_build_csr groups the edges by that key once; every
 *    aggregation then reads the grouped form (rowptr, col).
 *  - Node features are dense row-major [N, F]; fp32, or bf16 storage where a
 *    dtype argument allows it.  Every reduction accumulates in fp32.
 *  - Pointers marked (device) are device memory owned by the caller; the
 *    library never allocates, frees or keeps them.  Workspace buffers are
 *    caller-provided device memory of at least the queried size.
 *  - Every call is stateless (the functional style of Section 2.1.5): all
 *    parameters, including attention vectors, are passed per call.  The
 *    graph-level cache of Section 3 is the caller keeping the outputs of
 *    tfg_build_csr / tfg_gcn_norm and passing them back.
 *  - Calls enqueue work on `stream` (NULL = the legacy default stream) and
 *    return immediately; results are ready once the stream reaches them.
 *  - Return value: TFG_OK (0) or a negative tfg_status.  Host-side checks
 *    (null pointers, sizes, workspace) fail before anything is enqueued;
 *    tfg_last_error() then describes the failure (thread-local).
 *  - Checks that need the data (edge ids outside [0, N), an unsorted batch
 *    vector) run on the device: the call first sets *status to 0 and a kernel
 *    that finds a bad value writes the error code there.  Out-of-range
 *    values are clamped, so no kernel reads or writes out of bounds, but the
 *    outputs of a call whose status is non-zero are unspecified.
 *  - Empty reductions (a node without incoming edges, a graph without
 *    nodes) give 0 for every reducer.
 *  - Results are deterministic: the same inputs give bit-identical outputs.
 */
#ifndef TFG_H
#define TFG_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* cudaStream_t without pulling in the CUDA headers. */
typedef struct CUstream_st *tfg_stream_t;

typedef enum {
    TFG_OK = 0,
    TFG_ERR_INVALID_ARG = -1, /* null pointer, negative/zero size, bad enum    */
    TFG_ERR_TOO_LARGE = -2,   /* N or E >= 2^31 (CSR indices are int32)       */
    TFG_ERR_WORKSPACE = -3,   /* workspace missing or smaller than required   */
    TFG_ERR_CUDA = -4,        /* a CUDA runtime call or launch failed         */
    TFG_ERR_INDEX_RANGE = -5, /* (status word) an index outside its range     */
    TFG_ERR_UNSORTED = -6,    /* (status word) batch vector not non-decreasing */
    TFG_ERR_TIMEOUT = -7      /* reserved: a bounded device wait gave up      */
} tfg_status;

typedef enum { TFG_F32 = 0, TFG_BF16 = 1 } tfg_dtype;
typedef enum { TFG_SUM = 0, TFG_MEAN = 1, TFG_MAX = 2 } tfg_reduce;

/* Library version (major * 10000 + minor * 100 + patch). */
int tfg_version(void);

/* Description of the last host-side failure on this thread ("" if none). */
const char *tfg_last_error(void);

/* 1 in the bounds-checked debug build (compiled with TFG_CHECK_BOUNDS=1),
 * 0 in the default build.  The debug build checks, before every launch,
 * that each device buffer a call touches lies inside its allocation and
 * that caller-built index arrays are valid (rowptr[0] = 0, rowptr[N] = E,
 * rowptr non-decreasing, col ids in [0, N), perm ids in [0, E)); a
 * violation returns TFG_ERR_INDEX_RANGE (TFG_ERR_INVALID_ARG for a pointer
 * that is not device memory) and launches nothing.  Each check reads the
 * arrays once on the device and synchronises the stream: a debugging aid. */
int tfg_check_bounds_enabled(void);

/* ------------------------------------------------------------------------
 * Grouping by the reduce key: COO -> CSR by target.
 * Section 2.1.2 / Fig. 5b: a reducer gathers the elements that share a key
 * (here the target node) into one group.
 *
 *   edge_index (device) int64 [2, num_edges]: sources then targets.
 *   rowptr     (device) int32 [num_nodes + 1]: edges into node t are
 *                       positions rowptr[t] .. rowptr[t+1]-1.
 *   col        (device) int32 [num_edges]: source node of each position.
 *   perm       (device) int32 [num_edges]: original edge id of each position.
 *   in_degree  (device) int32 [num_nodes]: number of edges into each node.
 *   workspace  (device) >= tfg_build_csr_workspace_size() bytes, 256-byte
 *                       aligned; contents are scratch.
 *   status     (device) int32 [1]: 0, or TFG_ERR_INDEX_RANGE when an edge id
 *                       lies outside [0, num_nodes).
 * The grouping is stable: inside a row, edges keep their original order, so
 * (rowptr, col, perm) is unique.  num_edges may be 0; num_nodes >= 1 when
 * num_edges > 0.
 * ---------------------------------------------------------------------- */
int tfg_build_csr_workspace_size(int64_t num_nodes, int64_t num_edges, size_t *bytes);
int tfg_build_csr(const int64_t *edge_index, int64_t num_edges, int64_t num_nodes,
                  int32_t *rowptr, int32_t *col, int32_t *perm, int32_t *in_degree,
                  void *workspace, size_t workspace_bytes, int32_t *status,
                  tfg_stream_t stream);
/* The same grouping from an int32 edge list (edge_index int32 [2, E], the
 * same layout; ids are checked the same way).  Same outputs, workspace size
 * and errors as tfg_build_csr; the first sort pass reads half the bytes. */
int tfg_build_csr32(const int32_t *edge_index, int64_t num_edges, int64_t num_nodes,
                    int32_t *rowptr, int32_t *col, int32_t *perm, int32_t *in_degree,
                    void *workspace, size_t workspace_bytes, int32_t *status,
                    tfg_stream_t stream);
/* The same grouping by SOURCE (the CSR of the transposed graph, used by the
 * backward calls): rows are sources, col_src holds the targets, perm_src the
 * original edge ids (stable: original order within a row), out_degree the
 * number of edges leaving each node.  Same workspace size and errors. */
int tfg_build_csr_by_source(const int64_t *edge_index, int64_t num_edges, int64_t num_nodes,
                            int32_t *rowptr_src, int32_t *col_src, int32_t *perm_src,
                            int32_t *out_degree, void *workspace, size_t workspace_bytes,
                            int32_t *status, tfg_stream_t stream);
int tfg_build_csr32_by_source(const int32_t *edge_index, int64_t num_edges, int64_t num_nodes,
                              int32_t *rowptr_src, int32_t *col_src, int32_t *perm_src,
                              int32_t *out_degree, void *workspace, size_t workspace_bytes,
                              int32_t *status, tfg_stream_t stream);

/* ------------------------------------------------------------------------
 * GCN symmetric normalisation of A + I (the propagation rule of the GCN
 * model that Section 2.2 lists and Table 1 evaluates), computed once per
 * graph and cached by the caller (graph-level caching, Section 3).
 *
 *   deg[t]   = sum of the weights of the edges into t, + self_loop_fill
 *              when add_self_loops is non-zero (one implicit self-loop per
 *              node, added even when the edge list already has one)
 *   dinv[t]  = deg[t]^-1/2, or 0 when deg[t] == 0
 *   w_csr[k] = w_e * dinv[col[k]] * dinv[t] for position k of row t, where
 *              e = perm[k] and w_e = edge_weight[e] (1 when edge_weight is NULL)
 *
 *   rowptr, col, perm (device): the output of tfg_build_csr.
 *   edge_weight (device) fp32 [num_edges] in ORIGINAL edge order, or NULL.
 *   dinv (device) fp32 [num_nodes], written.
 *   w_csr (device) fp32 [num_edges] in CSR order, written; may be NULL when
 *              only dinv is wanted (tfg_gcn_aggregate_sum can form the
 *              weights on the fly for an unweighted graph).
 * The implicit self-loop weight self_loop_fill * dinv[t]^2 is not part of
 * w_csr; tfg_gcn_aggregate_sum adds it.
 * ---------------------------------------------------------------------- */
int tfg_gcn_norm(const int32_t *rowptr, const int32_t *col, const int32_t *perm,
                 const float *edge_weight, int64_t num_nodes, int64_t num_edges,
                 int add_self_loops, float self_loop_fill, float *dinv, float *w_csr,
                 tfg_stream_t stream);

/* ------------------------------------------------------------------------
 * Message aggregation (Fig. 1) with the reducer of Fig. 5b:
 *   out[t, :] = REDUCE over positions k of row t of  w_k * x[col[k], :]
 *   sum; mean = sum / (rowptr[t+1] - rowptr[t]); max.
 *
 *   rowptr, col (device): CSR by target (tfg_build_csr).  col may be NULL
 *        only for a graph without edges; every row is then empty.
 *   w_csr (device) fp32 [num_edges] in CSR order, or NULL for w = 1.
 *   x (device) [num_nodes, num_features] row-major, x_dtype TFG_F32 or
 *        TFG_BF16.  16-byte alignment of x and a feature count that is a
 *        multiple of 4 (fp32) or 8 (bf16) select the vectorised kernels;
 *        any other layout takes a scalar path with the same results.
 *   out (device) fp32 [num_nodes, num_features], written (not accumulated).
 * The sum and mean accumulate in fp32 in a fixed order (deterministic);
 * max is exact (the maximum of fp32 products w_k * x).
 * ---------------------------------------------------------------------- */
int tfg_aggregate_sum(const int32_t *rowptr, const int32_t *col, const float *w_csr,
                      const void *x, int x_dtype, int64_t num_nodes, int64_t num_features,
                      float *out, tfg_stream_t stream);
int tfg_aggregate_mean(const int32_t *rowptr, const int32_t *col, const float *w_csr,
                       const void *x, int x_dtype, int64_t num_nodes, int64_t num_features,
                       float *out, tfg_stream_t stream);
int tfg_aggregate_max(const int32_t *rowptr, const int32_t *col, const float *w_csr,
                      const void *x, int x_dtype, int64_t num_nodes, int64_t num_features,
                      float *out, tfg_stream_t stream);

/* ------------------------------------------------------------------------
 * GCN propagation  out = D^-1/2 (A + I) D^-1/2 x  in one pass (GCN, Section
 * 2.2 / Table 1; the weights are those of tfg_gcn_norm):
 *   out[t, :] = sum over positions k of row t of  w_k * x[col[k], :]
 *               + (add_self_loops ? self_loop_fill * dinv[t]^2 * x[t, :] : 0)
 * with w_k = w_csr[k] when w_csr is given, else dinv[col[k]] * dinv[t]
 * (an unweighted graph; no per-edge weight array is read).
 *   dinv (device) fp32 [num_nodes] from tfg_gcn_norm (same add_self_loops
 *        and self_loop_fill).
 *   Other arguments as for tfg_aggregate_sum.
 * ---------------------------------------------------------------------- */
int tfg_gcn_aggregate_sum(const int32_t *rowptr, const int32_t *col, const float *dinv,
                          const float *w_csr, const void *x, int x_dtype, int64_t num_nodes,
                          int64_t num_features, int add_self_loops, float self_loop_fill,
                          float *out, tfg_stream_t stream);

/* ------------------------------------------------------------------------
 * Backward of the aggregation (the gradient with respect to x; the paper
 * keeps graph construction and mini-batching differentiable, Sections 2.1.1
 * and 2.1.3, so gradients flow through the aggregation).  For
 *   out[t] = sum over edges e = (s -> t) of w_e x[s]
 * the gradient is the same sum over the transposed graph:
 *   grad_x[s] = sum over edges e = (s -> t) of w_e grad_out[t].
 * All backward calls take the CSR grouped by SOURCE (tfg_build_csr_by_source):
 * rowptr_src indexes sources, col_src holds targets, perm_src the original
 * edge ids.
 *
 * tfg_aggregate_backward: reduce TFG_SUM (w_e = edge_weight[e], or 1) or
 *   TFG_MEAN (w_e / in_degree[t], in_degree the forward CSR's, as written by
 *   tfg_build_csr).  edge_weight is in ORIGINAL edge order, or NULL.  A
 *   workspace of tfg_aggregate_backward_workspace_size() bytes holds the
 *   weights in source-grouped order when there are any (NULL allowed for an
 *   unweighted sum).
 * tfg_gcn_aggregate_backward: the backward of tfg_gcn_aggregate_sum with
 *   weights formed from dinv.  The symmetric normalisation is its own
 *   transpose, so this is the GCN propagation on the source-grouped CSR with
 *   the forward's dinv (add_self_loops / self_loop_fill as in the forward).
 * tfg_aggregate_max_argmax: tfg_aggregate_max plus, per (t, f), the ORIGINAL
 *   id of the first edge (in original order) whose product w_k * x attains the
 *   maximum, -1 for a row without edges; perm is the forward CSR's.
 *   argmax int32 [num_nodes, num_features].
 * tfg_aggregate_max_backward: grad_x[s, f] = sum over edges e = (s -> t)
 *   with argmax[t, f] == e of w_e grad_out[t, f], w_e = edge_weight[e] in
 *   ORIGINAL edge order (the weights of the forward, w_csr[k] =
 *   edge_weight[perm[k]]), or 1 when edge_weight is NULL.  num_edges =
 *   rowptr_src[num_nodes].  argmax values outside [0, num_edges) match no
 *   edge.  tfg_aggregate_max_backward_workspace_size() gives the workspace
 *   (16-byte aligned, overwritten) for win marks: on long rows (mean
 *   in-degree num_edges / num_nodes >= min(num_features, 128)), where most
 *   edges win nothing, the call first marks, in a byte per edge, which
 *   eighths of the features the edge is the argmax of, and then reads
 *   argmax and gradient slices for those alone.  0 bytes: the marks would
 *   not pay and no workspace is used.
 *   Workspace NULL reads the argmax and gradient rows of every out-edge.
 *   Both ways give the same bits.
 * grad_out, grad_x: fp32 [num_nodes, num_features]; grad_x is written.
 * Every sum runs in a fixed order: results are bitwise reproducible.
 * ---------------------------------------------------------------------- */
int tfg_aggregate_backward_workspace_size(int reduce, int64_t num_edges, size_t *bytes);
int tfg_aggregate_backward(int reduce, const int32_t *rowptr_src, const int32_t *col_src,
                           const int32_t *perm_src, const float *edge_weight,
                           const int32_t *in_degree, const float *grad_out, int64_t num_nodes,
                           int64_t num_edges, int64_t num_features, float *grad_x,
                           void *workspace, size_t workspace_bytes, tfg_stream_t stream);
int tfg_gcn_aggregate_backward(const int32_t *rowptr_src, const int32_t *col_src,
                               const float *dinv, const float *grad_out, int64_t num_nodes,
                               int64_t num_features, int add_self_loops, float self_loop_fill,
                               float *grad_x, tfg_stream_t stream);
int tfg_aggregate_max_argmax(const int32_t *rowptr, const int32_t *col, const int32_t *perm,
                             const float *w_csr, const void *x, int x_dtype, int64_t num_nodes,
                             int64_t num_features, float *out, int32_t *argmax,
                             tfg_stream_t stream);
int tfg_aggregate_max_backward_workspace_size(int64_t num_nodes, int64_t num_edges,
                                              int64_t num_features, size_t *bytes);
int tfg_aggregate_max_backward(const int32_t *rowptr_src, const int32_t *col_src,
                               const int32_t *perm_src, const int32_t *argmax,
                               const float *edge_weight, const float *grad_out,
                               int64_t num_nodes, int64_t num_edges, int64_t num_features,
                               float *grad_x, void *workspace, size_t workspace_bytes,
                               tfg_stream_t stream);

/* ------------------------------------------------------------------------
 * Multi-hop propagation: APPNP and SGC, node-level models the paper lists
 * beside GCN and GAT (Section 2.2) and evaluates in Table 1.  With Ahat the
 * GCN-normalised adjacency of tfg_gcn_aggregate_sum:
 *   h_0 = x0,   h_{k+1} = (1 - alpha) * Ahat h_k + alpha * x0,   out = h_K
 * (K = num_hops).  APPNP (Klicpera et al.) is the power iteration for
 * personalised PageRank with teleport probability alpha; alpha = 0 gives
 * SGC's Ahat^K x0 (Wu et al.), also offered as tfg_sgc_propagate.
 *
 *   rowptr, col, dinv, w_csr, add_self_loops, self_loop_fill: as for
 *        tfg_gcn_aggregate_sum (w_csr NULL forms the weights from dinv).
 *   x0 (device) [num_nodes, num_features] row-major, TFG_F32 or TFG_BF16;
 *        read by every hop (the teleport term), never written.
 *   num_hops K in [0, 1024]; K = 0 copies x0 (widened to fp32) into out.
 *   alpha in [0, 1] (finite).
 *   out (device) fp32 [num_nodes, num_features], written.
 *   workspace (device) >= tfg_propagate_workspace_size() bytes, 16-byte
 *        aligned (N * F fp32 values when K >= 2, else 0 bytes and it may be
 *        NULL); contents are scratch.
 * Each hop is one fused launch: GCN gather-sum, self-loop term and the
 * teleport epilogue  alpha * x0[t] + (1 - alpha) * (...)  (one fp32 fma),
 * accumulated in fp32 in a fixed order; iterates between hops are fp32.
 * out, workspace and x0 must not overlap.
 * ---------------------------------------------------------------------- */
int tfg_propagate_workspace_size(int64_t num_nodes, int64_t num_features, int64_t num_hops,
                                 size_t *bytes);
int tfg_appnp_propagate(const int32_t *rowptr, const int32_t *col, const float *dinv,
                        const float *w_csr, const void *x0, int x_dtype, int64_t num_nodes,
                        int64_t num_features, int64_t num_hops, float alpha, int add_self_loops,
                        float self_loop_fill, float *out, void *workspace,
                        size_t workspace_bytes, tfg_stream_t stream);
int tfg_sgc_propagate(const int32_t *rowptr, const int32_t *col, const float *dinv,
                      const float *w_csr, const void *x0, int x_dtype, int64_t num_nodes,
                      int64_t num_features, int64_t num_hops, int add_self_loops,
                      float self_loop_fill, float *out, void *workspace, size_t workspace_bytes,
                      tfg_stream_t stream);

/* ------------------------------------------------------------------------
 * Edge-softmax (GAT) aggregation -- the map-reduce workflow of Fig. 5a
 * (Section 2.1.2) fused with the weighted sum it feeds:
 *   s_src[n, h] = <x[n, h, :], a_src[h, :]>,  s_dst[n, h] likewise with a_dst
 *   map:    l[k, h] = LeakyReLU(s_src[col[k], h] + s_dst[t, h]; negative_slope)
 *   reduce: alpha[k, h] = exp(l[k, h]) / sum over row t of exp(l[., h])
 *           (evaluated with the row maximum subtracted; same value)
 *   out[t, h, :] = sum over row t of alpha[k, h] * x[col[k], h, :]
 *
 *   x (device) [num_nodes, heads * channels], x_dtype TFG_F32 or TFG_BF16,
 *          head h in columns h*channels .. h*channels+channels-1.
 *   num_edges: rowptr[num_nodes]; col may be NULL when it is 0.
 *   a_src, a_dst (device) fp32 [heads * channels], same layout.
 *   out (device) fp32 [num_nodes, heads * channels], written.
 *   alpha (device) fp32 [num_edges, heads] in CSR order, or NULL.
 *   workspace (device) >= tfg_edge_softmax_workspace_size() bytes (node
 *          scores); contents are scratch.
 * Rows without incoming edges give 0.  The row maximum is tracked as a
 * running maximum in one pass (rescaling the partial sums when it grows),
 * which gives the same alpha and out as the three-pass workflow.
 * ---------------------------------------------------------------------- */
int tfg_edge_softmax_workspace_size(int64_t num_nodes, int heads, size_t *bytes);
int tfg_edge_softmax_aggregate(const int32_t *rowptr, const int32_t *col, const void *x,
                               int x_dtype, int64_t num_nodes, int64_t num_edges, int heads,
                               int channels,
                               const float *a_src, const float *a_dst, float negative_slope,
                               float *out, float *alpha, void *workspace,
                               size_t workspace_bytes, tfg_stream_t stream);

/* ------------------------------------------------------------------------
 * Dot-product (Transformer-style) edge-softmax aggregation: the attention
 * form of tf_geometric's own GAT (Section 4.2 calls it Transformer-based), on
 * the map-reduce workflow of Fig. 5a:
 *   map:    l[k, h] = scale * <q[t, h, :], k[col[k], h, :]>  (position k of row t)
 *   reduce: alpha[k, h] = exp(l[k, h]) / sum over row t of exp(l[., h])
 *           (evaluated with the row maximum subtracted; same value)
 *   out[t, h, :] = sum over row t of alpha[k, h] * v[col[k], h, :]
 * An empty row gives out = 0.
 *
 *   rowptr, col (device): CSR by target (tfg_build_csr).
 *   q, k, v (device) [num_nodes, heads * channels] row-major, head-major
 *        within a row ([h0c0 .. h0c(C-1), h1c0, ...]), all three of type
 *        x_dtype (TFG_F32 or TFG_BF16).  q is read at targets, k and v at
 *        sources.
 *   channels <= 256.  scale: finite multiplier of the dot product
 *        (1 / sqrt(channels) for the Transformer form).
 *   out (device) fp32 [num_nodes, heads * channels], written.
 *   alpha (device) fp32 [num_edges, heads] in CSR order, or NULL.
 * One pass per row with the running-maximum softmax, fp32 accumulation in a
 * fixed order (deterministic).  16-byte aligned rows with channels a power
 * of two times 4 (fp32) or 8 (bf16), up to 128 / 256, take the vectorised
 * kernel; any other layout a general one with the same definition.
 * No workspace.
 * ---------------------------------------------------------------------- */
int tfg_dot_edge_softmax_aggregate(const int32_t *rowptr, const int32_t *col, const void *q,
                                   const void *k, const void *v, int x_dtype, int64_t num_nodes,
                                   int64_t num_edges, int heads, int channels, float scale,
                                   float *out, float *alpha, tfg_stream_t stream);

/* ------------------------------------------------------------------------
 * Edge-softmax aggregation that allocates nothing and takes no workspace.
 * This entry point has no counterpart in the paper; it is a library
 * convenience.
 *
 * Some callers cannot allocate device memory at the time of the call: code
 * being recorded into a CUDA graph (a cudaMalloc there breaks the capture),
 * plugins whose host application owns all device memory and hands out none,
 * and real-time pipelines whose memory budget is fixed before they start.
 * For them, the node-score scratch that tfg_edge_softmax_aggregate takes
 * as a workspace lives here in a fixed array inside the library: 16 MiB,
 * enough for num_nodes * heads <= 2,097,152 (node, head) pairs, held on
 * every GPU that loads the library until the process exits.  Larger inputs
 * return TFG_ERR_TOO_LARGE; use tfg_edge_softmax_aggregate for them.
 *
 * Arguments, layout and results are those of tfg_edge_softmax_aggregate
 * without the workspace.  Nothing is allocated or freed by any call.
 * The first call on each device looks up the array's device address (which
 * may load the library's GPU code), so make that first call outside any
 * stream capture.  The address is then cached per device for the life of
 * the process: a cudaDeviceReset (or anything else that destroys the
 * device's primary context) unloads the array and makes the cached address
 * stale, so after such a reset this entry point must not be called again in
 * that process.  All calls on a device share the one array, and each call
 * overwrites it: calls that may overlap on the GPU (different streams,
 * different host threads) race with each other and must be serialised by the
 * caller.
 * ---------------------------------------------------------------------- */
int tfg_edge_softmax_aggregate_noalloc(const int32_t *rowptr, const int32_t *col, const void *x,
                                       int x_dtype, int64_t num_nodes, int64_t num_edges,
                                       int heads, int channels, const float *a_src,
                                       const float *a_dst, float negative_slope, float *out,
                                       float *alpha, tfg_stream_t stream);

/* ------------------------------------------------------------------------
 * Backward of the GAT edge-softmax aggregation (tfg_edge_softmax_aggregate):
 * the gradients of the Fig. 5a workflow with respect to x, a_src and a_dst,
 * given grad_out = dL/dout (the paper keeps graph construction and
 * mini-batching differentiable, Sections 2.1.1 and 2.1.3).  With alpha the
 * forward's weights, e = (s -> t), z = s_src[s,h] + s_dst[t,h]:
 *   dalpha[e,h] = <grad_out[t,h,:], x[s,h,:]>
 *   beta[t,h]   = <grad_out[t,h,:], out[t,h,:]>  (= sum over e into t of alpha dalpha)
 *   dz[e,h]     = alpha (dalpha - beta[t,h]) (z > 0 ? 1 : negative_slope)
 *   grad_x[s,h,:]  = sum over e out of s of alpha grad_out[t,h,:]
 *                    + ds_src[s,h] a_src[h,:] + ds_dst[s,h] a_dst[h,:]
 *   ds_src[s,h] = sum over e out of s of dz;  ds_dst[t,h] = sum over e into t of dz
 *   grad_a_src[h,c] = sum_v ds_src[v,h] x[v,h,c];  grad_a_dst likewise.
 *
 *   rowptr, col: the CSR by target of the forward (tfg_build_csr).
 *   rowptr_src, col_src: the CSR by source (tfg_build_csr_by_source).
 *   x, x_dtype, num_nodes, num_edges, heads, channels, a_src, a_dst,
 *          negative_slope: the forward's arguments.
 *   out (device) fp32 [num_nodes, H*C]: the forward's output.
 *   grad_out (device) fp32 [num_nodes, H*C].
 *   grad_x (device) fp32 [num_nodes, H*C]; grad_a_src, grad_a_dst (device)
 *          fp32 [H*C]: written.
 *   workspace >= tfg_edge_softmax_backward_workspace_size() bytes.
 * Layouts: channels a power of two up to 32, or a multiple of 32; H*C <= 256.
 * Others return TFG_ERR_INVALID_ARG.  Deterministic (no atomics).
 * ---------------------------------------------------------------------- */
int tfg_edge_softmax_backward_workspace_size(int64_t num_nodes, int heads, int channels,
                                             size_t *bytes);
int tfg_edge_softmax_aggregate_backward(const int32_t *rowptr, const int32_t *col,
                                        const int32_t *rowptr_src, const int32_t *col_src,
                                        const void *x, int x_dtype, int64_t num_nodes,
                                        int64_t num_edges, int heads, int channels,
                                        const float *a_src, const float *a_dst,
                                        float negative_slope, const float *out,
                                        const float *grad_out, float *grad_x, float *grad_a_src,
                                        float *grad_a_dst, void *workspace,
                                        size_t workspace_bytes, tfg_stream_t stream);

/* ------------------------------------------------------------------------
 * Backward of the dot-product attention aggregation
 * (tfg_dot_edge_softmax_aggregate): the gradients with respect to q, k and v
 * given grad_out = dL/dout, on the same Fig. 5a workflow.  With alpha the
 * forward's weights and e = (s -> t):
 *   dalpha[e,h] = <grad_out[t,h,:], v[s,h,:]>
 *   beta[t,h]   = <grad_out[t,h,:], out[t,h,:]>  (= sum over e into t of alpha dalpha)
 *   dl[e,h]     = alpha (dalpha - beta[t,h])
 *   grad_q[t,h,:] = scale * sum over e into t of dl k[s,h,:]
 *   grad_k[s,h,:] = scale * sum over e out of s of dl q[t,h,:]
 *   grad_v[s,h,:] = sum over e out of s of alpha grad_out[t,h,:]
 *
 *   rowptr, col: the CSR by target of the forward (tfg_build_csr).
 *   rowptr_src, col_src: the CSR by source (tfg_build_csr_by_source).
 *   q, k, v, x_dtype, num_nodes, num_edges, heads, channels, scale: the
 *          forward's arguments.
 *   out (device) fp32 [num_nodes, H*C]: the forward's output.
 *   grad_out (device) fp32 [num_nodes, H*C].
 *   grad_q, grad_k, grad_v (device) fp32 [num_nodes, H*C]: written.
 *   workspace >= tfg_dot_edge_softmax_backward_workspace_size() bytes.
 * Layouts: channels a power of two up to 32, or a multiple of 32; H*C <= 256.
 * Others return TFG_ERR_INVALID_ARG.  Deterministic (no atomics).
 * ---------------------------------------------------------------------- */
int tfg_dot_edge_softmax_backward_workspace_size(int64_t num_nodes, int heads, int channels,
                                                 size_t *bytes);
int tfg_dot_edge_softmax_aggregate_backward(const int32_t *rowptr, const int32_t *col,
                                            const int32_t *rowptr_src, const int32_t *col_src,
                                            const void *q, const void *k, const void *v,
                                            int x_dtype, int64_t num_nodes, int64_t num_edges,
                                            int heads, int channels, float scale,
                                            const float *out, const float *grad_out,
                                            float *grad_q, float *grad_k, float *grad_v,
                                            void *workspace, size_t workspace_bytes,
                                            tfg_stream_t stream);

/* ------------------------------------------------------------------------
 * Graph pooling keyed by node_graph_index (Section 2.1.1 BatchGraph; Fig. 2a
 * common graph pooling):
 *   out[g, :] = REDUCE over nodes v with batch[v] == g of x[v, :]
 *   sum; mean = sum / node count; max.
 *
 *   x (device) [num_nodes, num_features], x_dtype TFG_F32 or TFG_BF16.
 *   batch (device) int64 [num_nodes], non-decreasing, values in
 *          [0, num_graphs) -- the order a BatchGraph's reindexing produces.
 *   out (device) fp32 [num_graphs, num_features], written.
 *   status (device) int32 [1]: 0, TFG_ERR_UNSORTED or TFG_ERR_INDEX_RANGE.
 * ---------------------------------------------------------------------- */
int tfg_segment_pool(const void *x, int x_dtype, const int64_t *batch, int64_t num_nodes,
                     int64_t num_graphs, int64_t num_features, int reduce, float *out,
                     int32_t *status, tfg_stream_t stream);

/* ------------------------------------------------------------------------
 * Mean-Max graph pooling in one pass: out[g, 0:F] = mean and out[g, F:2F] =
 * max over the nodes of graph g -- the concatenated readout of the Mean-Max
 * Pool model evaluated in Table 2 (Section 4.1), built from the common graph
 * pooling of Fig. 2a.  Arguments as for tfg_segment_pool, with out
 * (device) fp32 [num_graphs, 2 * num_features].  Empty graphs give 0 in
 * both halves.
 * ---------------------------------------------------------------------- */
int tfg_segment_pool_meanmax(const void *x, int x_dtype, const int64_t *batch,
                             int64_t num_nodes, int64_t num_graphs, int64_t num_features,
                             float *out, int32_t *status, tfg_stream_t stream);

/* ------------------------------------------------------------------------
 * BatchGraph construction on the device: the reindexing trick of Section
 * 2.1.1 (Fig. 4).  Graph g's j-th node becomes node node_offsets[g] + j,
 * where node_offsets[g] is the number of nodes in graphs 0 .. g-1; every
 * edge of graph g is shifted by node_offsets[g]; batch[v] (node_graph_index)
 * is the graph of node v.
 *
 *   node_counts, edge_counts (device) int64 [num_graphs]: nodes and edges of
 *          each graph.
 *   edge_index (device) int64 [2, total_edges]: the graphs' own edge lists
 *          (local node ids 0 .. n_g - 1), stacked in graph order, sources
 *          row then targets row.
 *   total_edges, total_nodes: the sums of the counts (sizes of the outputs).
 *   out_edge_index (device) int64 [2, total_edges]: the batched edge list.
 *   batch (device) int64 [total_nodes], non-decreasing graph ids.
 *   node_offsets (device) int64 [num_graphs + 1]; the last entry is the total.
 *   workspace (device) >= tfg_batch_graphs_workspace_size() bytes.
 *   status (device) int32 [1]: TFG_ERR_INDEX_RANGE when a count is negative,
 *          a local id lies outside its graph, or the counts do not sum to the
 *          declared totals (bad ids are replaced by 0 of their graph).
 * ---------------------------------------------------------------------- */
int tfg_batch_graphs_workspace_size(int64_t num_graphs, size_t *bytes);
int tfg_batch_graphs(int64_t num_graphs, const int64_t *node_counts, const int64_t *edge_counts,
                     const int64_t *edge_index, int64_t total_edges, int64_t total_nodes,
                     int64_t *out_edge_index, int64_t *batch, int64_t *node_offsets,
                     void *workspace, size_t workspace_bytes, int32_t *status,
                     tfg_stream_t stream);

/* ------------------------------------------------------------------------
 * Gather-only floor (a measurement call; the paper has no counterpart).
 * The aggregations above read, for every CSR edge, the whole feature row of
 * its source node (Fig. 1 message aggregation: gather, weight, reduce).  This
 * call performs only the gather, on the same column array and rows, with
 * nothing else to compute: every row x[col[k]] for k < num_edges is read
 * once as 16-byte vectors and the rows are folded with bitwise XOR,
 *   out[j] = XOR over k of the j-th 32-bit word of x[col[k]].
 * Its duration is the time the SMs need to pull the gathered rows out of
 * the memory system, the floor the aggregation kernels are measured
 * against.  The result is exact and independent of order.
 *
 *   col (device) int32 [num_edges], values in [0, num_nodes) (not checked:
 *        pass a column array from tfg_build_csr).
 *   x (device) [num_nodes, row_bytes] of any element type, 16-byte aligned.
 *   row_bytes: 16, 32, 64, 128, 256 or 512 (bytes per row).
 *   out (device) uint32 [row_bytes / 4], written (zeroed first on stream).
 * ---------------------------------------------------------------------- */
int tfg_gather_xor(const int32_t *col, int64_t num_edges, const void *x, int64_t num_nodes,
                   int64_t row_bytes, uint32_t *out, tfg_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* TFG_H */
