/*
 * tfg_oracle.c -- plain, slow, fp64 CPU oracle for graph message aggregation.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test-suite, the smoke check and the
 * benchmark's CPU-baseline leg may load this file's library.  It shares no
 * code, header or constant with the CUDA library and includes nothing of it.
 *
 * What it follows (tf_geometric, arXiv:2101.11552):
 *   - Graph data structure, Section 2.1.1: edge_index is [2, E] int64, row 0
 *     the source and row 1 the target of each edge; A_ij > 0 is an edge i -> j.
 *   - Graph map-reduce framework, Section 2.1.2 / Fig. 5: a reducer groups
 *     elements by a key (here the target node index) and reduces each group;
 *     the GAT workflow is map (edge -> unnormalised score), reduce (segment
 *     sum -> softmax denominator), map (divide).
 *   - BatchGraph / graph pooling, Section 2.1.1 and Fig. 2a: nodes are reduced
 *     per graph by node_graph_index.
 *   - GCN normalisation D^-1/2 (A+I) D^-1/2 and GAT additive attention come
 *     from the works the paper cites for those models (Section 2.2).
 *
 * Every function loops over edges (or nodes) in their original order and
 * accumulates in double precision.  Empty groups reduce to 0 for every
 * reducer (the paper does not fix this; it is the convention of this library).
 *
 * Planted-mistake switches (ORACLE_PLANT_*) exist only so that the pin tests
 * can demonstrate that a plausible bug is caught; the normal build defines
 * none of them.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OK 0
#define E_ARG (-1)
#define E_RANGE (-5)
#define E_UNSORTED (-6)

#define R_SUM 0
#define R_MEAN 1
#define R_MAX 2

/* The magnitude one term m adds to an error scale (absout): |m|.  The tests
 * multiply the fp32 tolerance by that scale, so a slip here would loosen or
 * tighten every comparison; the planted variant doubles it. */
#ifdef ORACLE_PLANT_SCALE_DOUBLED
#define SCALE_TERM(m) (2.0 * fabs(m))                    /* planted: inflated scale */
#else
#define SCALE_TERM(m) fabs(m)
#endif

/* ---------------------------------------------------------------------------
 * CSR grouped by target: a stable counting sort of the edges by edge_index[1].
 * The "reduce key" of Section 2.1.2 is the target node; grouping by it makes
 * each group a contiguous row.  Within a row, edges keep their original order,
 * which fixes a single canonical CSR.
 *   rowptr[N+1], col[E] (source of each edge), perm[E] (original edge id),
 *   in_degree[N].
 * ------------------------------------------------------------------------- */
int oracle_build_csr(int64_t n, int64_t e, const int64_t *edge_index,
                     int32_t *rowptr, int32_t *col, int32_t *perm, int32_t *in_degree)
{
    if (n < 0 || e < 0) return E_ARG;
    const int64_t *src = edge_index, *dst = edge_index + e;
    for (int64_t i = 0; i < e; ++i)
        if (src[i] < 0 || src[i] >= n || dst[i] < 0 || dst[i] >= n) return E_RANGE;
    for (int64_t t = 0; t < n; ++t) in_degree[t] = 0;
    for (int64_t i = 0; i < e; ++i) in_degree[dst[i]] += 1;
    rowptr[0] = 0;
    for (int64_t t = 0; t < n; ++t) rowptr[t + 1] = rowptr[t] + in_degree[t];
    int32_t *cursor = (int32_t *)malloc(sizeof(int32_t) * (size_t)(n > 0 ? n : 1));
    if (!cursor) return E_ARG;
    for (int64_t t = 0; t < n; ++t) cursor[t] = rowptr[t];
#ifdef ORACLE_PLANT_UNSTABLE_CSR
    /* planted mistake: place edges in reverse order inside each row */
    for (int64_t t = 0; t < n; ++t) cursor[t] = rowptr[t + 1];
    for (int64_t i = 0; i < e; ++i) {
        int32_t p = --cursor[dst[i]];
        col[p] = (int32_t)src[i];
        perm[p] = (int32_t)i;
    }
#else
    for (int64_t i = 0; i < e; ++i) {
        int32_t p = cursor[dst[i]]++;
        col[p] = (int32_t)src[i];
        perm[p] = (int32_t)i;
    }
#endif
    free(cursor);
    return OK;
}

/* ---------------------------------------------------------------------------
 * GCN symmetric normalisation of (A + I) (Kipf & Welling, cited in Sec. 2.2).
 *   deg[t]  = sum of the weights of the edges whose target is t
 *             (+ fill when an implicit self-loop is added to every node)
 *   dinv[t] = deg[t]^-1/2, or 0 when deg[t] == 0
 *   w_norm[e] = w_e * dinv[src_e] * dinv[dst_e]         (COO order)
 *   self_w[t] = fill * dinv[t]^2  when add_self_loops, else 0
 * edge_weight == NULL means every weight is 1.
 * ------------------------------------------------------------------------- */
int oracle_gcn_norm(int64_t n, int64_t e, const int64_t *edge_index,
                    const double *edge_weight, int add_self_loops, double fill,
                    double *deg, double *dinv, double *w_norm, double *self_w)
{
    if (n < 0 || e < 0) return E_ARG;
    const int64_t *src = edge_index, *dst = edge_index + e;
    for (int64_t i = 0; i < e; ++i)
        if (src[i] < 0 || src[i] >= n || dst[i] < 0 || dst[i] >= n) return E_RANGE;
    for (int64_t t = 0; t < n; ++t) deg[t] = add_self_loops ? fill : 0.0;
#ifdef ORACLE_PLANT_DROP_SELF_LOOP_DEGREE
    for (int64_t t = 0; t < n; ++t) deg[t] = 0.0;
#endif
    for (int64_t i = 0; i < e; ++i) {
#ifdef ORACLE_PLANT_OUT_DEGREE
        deg[src[i]] += edge_weight ? edge_weight[i] : 1.0;   /* planted: by source */
#else
        deg[dst[i]] += edge_weight ? edge_weight[i] : 1.0;
#endif
    }
    for (int64_t t = 0; t < n; ++t) dinv[t] = deg[t] > 0.0 ? 1.0 / sqrt(deg[t]) : 0.0;
    for (int64_t i = 0; i < e; ++i) {
        double w = edge_weight ? edge_weight[i] : 1.0;
        w_norm[i] = w * dinv[src[i]] * dinv[dst[i]];
    }
    if (self_w)
        for (int64_t t = 0; t < n; ++t) self_w[t] = add_self_loops ? fill * dinv[t] * dinv[t] : 0.0;
    return OK;
}

/* ---------------------------------------------------------------------------
 * Message aggregation (Fig. 1; reducer of Fig. 5b keyed by the target node):
 *   out[t, :] = REDUCE over edges e with dst_e == t of  w_e * x[src_e, :]
 * SUM, MEAN (= SUM / number of incoming edges) or MAX.  Empty rows give 0.
 * self_w (optional, SUM only) adds self_w[t] * x[t, :], the implicit
 * self-loop of GCN.  absout[t, f] = sum of |w_e * x[src_e, f]| (+ |self term|),
 * the scale that a floating-point tolerance is measured against.
 * ------------------------------------------------------------------------- */
int oracle_aggregate(int reduce, int64_t n, int64_t e, const int64_t *edge_index,
                     const double *w, const double *x, int64_t f,
                     const double *self_w, double *out, double *absout)
{
    if (n < 0 || e < 0 || f < 0) return E_ARG;
    if (reduce != R_SUM && reduce != R_MEAN && reduce != R_MAX) return E_ARG;
    const int64_t *src = edge_index, *dst = edge_index + e;
#ifdef ORACLE_PLANT_SWAP_DIRECTION
    src = edge_index + e; dst = edge_index;          /* planted: aggregate into sources */
#endif
    for (int64_t i = 0; i < e; ++i)
        if (src[i] < 0 || src[i] >= n || dst[i] < 0 || dst[i] >= n) return E_RANGE;
    int64_t *count = (int64_t *)calloc((size_t)(n > 0 ? n : 1), sizeof(int64_t));
    if (!count) return E_ARG;
    for (int64_t k = 0; k < n * f; ++k) { out[k] = 0.0; absout[k] = 0.0; }
    for (int64_t i = 0; i < e; ++i) {
        int64_t s = src[i], t = dst[i];
        double we = w ? w[i] : 1.0;
        for (int64_t c = 0; c < f; ++c) {
            double m = we * x[s * f + c];
            if (reduce == R_MAX) {
#ifdef ORACLE_PLANT_MAX_FROM_ZERO
                if (m > out[t * f + c]) out[t * f + c] = m;      /* planted: max starts at 0 */
#else
                if (count[t] == 0 || m > out[t * f + c]) out[t * f + c] = m;
#endif
            } else {
                out[t * f + c] += m;
            }
            absout[t * f + c] += SCALE_TERM(m);
        }
        count[t] += 1;
    }
    if (reduce == R_MEAN) {
        for (int64_t t = 0; t < n; ++t) {
            if (count[t] == 0) continue;
#ifdef ORACLE_PLANT_MEAN_PLUS_ONE
            double cnt = (double)(count[t] + 1);              /* planted: off-by-one count */
#else
            double cnt = (double)count[t];
#endif
            for (int64_t c = 0; c < f; ++c) { out[t * f + c] /= cnt; absout[t * f + c] /= cnt; }
        }
    }
    if (self_w && reduce == R_SUM) {
        for (int64_t t = 0; t < n; ++t)
            for (int64_t c = 0; c < f; ++c) {
                double m = self_w[t] * x[t * f + c];
                out[t * f + c] += m;
                absout[t * f + c] += SCALE_TERM(m);
            }
    }
    free(count);
    return OK;
}

/* Same definition, evaluated only for the listed target rows, walking the
 * oracle's own stable CSR (rowptr/col/perm from oracle_build_csr).  A row's
 * edges in that CSR are exactly the edges with that target, in original
 * order, so each value equals the one oracle_aggregate computes.  w (COO
 * order, NULL = 1) is indexed through perm.  out/absout are [nrows, f]. */
int oracle_aggregate_rows(int reduce, int64_t n, const int32_t *rowptr, const int32_t *col,
                          const int32_t *perm, const double *w, const double *x, int64_t f,
                          const double *self_w, const int64_t *rows, int64_t nrows,
                          double *out, double *absout)
{
    if (reduce != R_SUM && reduce != R_MEAN && reduce != R_MAX) return E_ARG;
    for (int64_t r = 0; r < nrows; ++r) {
        int64_t t = rows[r];
        if (t < 0 || t >= n) return E_RANGE;
        double *o = out + r * f, *a = absout + r * f;
        for (int64_t c = 0; c < f; ++c) { o[c] = 0.0; a[c] = 0.0; }
        int64_t cnt = 0;
        for (int64_t k = rowptr[t]; k < rowptr[t + 1]; ++k) {
            int64_t s = col[k];
            double we = w ? w[perm[k]] : 1.0;
            for (int64_t c = 0; c < f; ++c) {
                double m = we * x[s * f + c];
                if (reduce == R_MAX) {
                    if (cnt == 0 || m > o[c]) o[c] = m;
                } else {
                    o[c] += m;
                }
                a[c] += SCALE_TERM(m);
            }
            cnt += 1;
        }
        if (reduce == R_MEAN && cnt > 0)
            for (int64_t c = 0; c < f; ++c) { o[c] /= (double)cnt; a[c] /= (double)cnt; }
        if (self_w && reduce == R_SUM)
            for (int64_t c = 0; c < f; ++c) {
                double m = self_w[t] * x[t * f + c];
                o[c] += m;
                a[c] += SCALE_TERM(m);
            }
    }
    return OK;
}

/* ---------------------------------------------------------------------------
 * GAT edge-softmax aggregation, following the map-reduce workflow of Fig. 5a:
 *   node scores  s_src[n,h] = sum_c x[n,h,c] a_src[h,c];  s_dst likewise
 *   map          l[e,h] = LeakyReLU(s_src[src_e,h] + s_dst[dst_e,h])
 *   reduce       m[t,h] = max over edges into t of l[e,h]          (stability)
 *                den[t,h] = sum over edges into t of exp(l[e,h] - m[t,h])
 *   map          alpha[e,h] = exp(l[e,h] - m[dst_e,h]) / den[dst_e,h]
 *   aggregate    out[t,h,:] = sum over edges into t of alpha[e,h] x[src_e,h,:]
 * Subtracting the per-target max does not change alpha mathematically.
 * x is [n, H*C] with the channels of head h at columns h*C .. h*C+C-1.
 * alpha is [e, H] in COO order.  Targets without incoming edges give 0.
 * absout[t, h*C+c] = sum of alpha[e,h] |x[src_e,h,c]|.
 * ------------------------------------------------------------------------- */
static double leaky(double v, double slope)
{
#ifdef ORACLE_PLANT_NO_LEAKY
    (void)slope;
    return v;                                             /* planted: no LeakyReLU */
#else
    return v > 0.0 ? v : slope * v;
#endif
}

int oracle_edge_softmax(int64_t n, int64_t e, const int64_t *edge_index, const double *x,
                        int h, int c, const double *a_src, const double *a_dst, double slope,
                        double *out, double *alpha, double *absout)
{
    if (n < 0 || e < 0 || h <= 0 || c <= 0) return E_ARG;
    const int64_t *src = edge_index, *dst = edge_index + e;
    for (int64_t i = 0; i < e; ++i)
        if (src[i] < 0 || src[i] >= n || dst[i] < 0 || dst[i] >= n) return E_RANGE;
    int64_t f = (int64_t)h * c;
    size_t nh = (size_t)(n > 0 ? n : 1) * (size_t)h;
    double *s_src = (double *)calloc(nh, sizeof(double));
    double *s_dst = (double *)calloc(nh, sizeof(double));
    double *mx = (double *)calloc(nh, sizeof(double));
    double *den = (double *)calloc(nh, sizeof(double));
    char *seen = (char *)calloc(nh, 1);
    double *logit = (double *)calloc((size_t)(e > 0 ? e : 1) * (size_t)h, sizeof(double));
    if (!s_src || !s_dst || !mx || !den || !seen || !logit) {
        free(s_src); free(s_dst); free(mx); free(den); free(seen); free(logit);
        return E_ARG;
    }
    for (int64_t v = 0; v < n; ++v)
        for (int hh = 0; hh < h; ++hh) {
            double a = 0.0, b = 0.0;
            for (int cc = 0; cc < c; ++cc) {
                a += x[v * f + hh * c + cc] * a_src[hh * c + cc];
                b += x[v * f + hh * c + cc] * a_dst[hh * c + cc];
            }
            s_src[v * h + hh] = a;
            s_dst[v * h + hh] = b;
        }
    /* map: unnormalised scores; reduce: per-target max */
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh) {
            double l = leaky(s_src[src[i] * h + hh] + s_dst[dst[i] * h + hh], slope);
            logit[i * h + hh] = l;
            size_t k = (size_t)dst[i] * h + hh;
            if (!seen[k] || l > mx[k]) mx[k] = l;
            seen[k] = 1;
        }
    /* reduce: segment sum of exp -> softmax denominator */
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh)
            den[(size_t)dst[i] * h + hh] += exp(logit[i * h + hh] - mx[(size_t)dst[i] * h + hh]);
    /* map: divide; then the attention-weighted sum */
    for (int64_t k = 0; k < n * f; ++k) { out[k] = 0.0; absout[k] = 0.0; }
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh) {
            size_t k = (size_t)dst[i] * h + hh;
            double al = exp(logit[i * h + hh] - mx[k]) / den[k];
            if (alpha) alpha[i * h + hh] = al;
            for (int cc = 0; cc < c; ++cc) {
                double m = al * x[src[i] * f + hh * c + cc];
                out[dst[i] * f + hh * c + cc] += m;
                absout[dst[i] * f + hh * c + cc] += SCALE_TERM(m);
            }
        }
    free(s_src); free(s_dst); free(mx); free(den); free(seen); free(logit);
    return OK;
}

/* The same three passes, restricted to the in-edges of the listed target rows
 * (walked through the oracle's stable CSR).  alpha_rows, when given, receives
 * for each listed row its alpha values [deg, H] in CSR order, rows packed one
 * after another (the caller sizes it from rowptr). */
int oracle_edge_softmax_rows(int64_t n, const int32_t *rowptr, const int32_t *col,
                             const double *x, int h, int c, const double *a_src,
                             const double *a_dst, double slope, const int64_t *rows,
                             int64_t nrows, double *out, double *alpha_rows, double *absout)
{
    if (h <= 0 || c <= 0) return E_ARG;
    int64_t f = (int64_t)h * c;
    int64_t apos = 0;
    for (int64_t r = 0; r < nrows; ++r) {
        int64_t t = rows[r];
        if (t < 0 || t >= n) return E_RANGE;
        int64_t k0 = rowptr[t], k1 = rowptr[t + 1], deg = k1 - k0;
        double *o = out + r * f, *ab = absout + r * f;
        for (int64_t q = 0; q < f; ++q) { o[q] = 0.0; ab[q] = 0.0; }
        if (deg == 0) continue;
        double *lg = (double *)malloc(sizeof(double) * (size_t)deg * (size_t)h);
        if (!lg) return E_ARG;
        for (int hh = 0; hh < h; ++hh) {
            double sd = 0.0;
            for (int cc = 0; cc < c; ++cc) sd += x[t * f + hh * c + cc] * a_dst[hh * c + cc];
            double mx = 0.0, den = 0.0;
            for (int64_t k = k0; k < k1; ++k) {
                int64_t s = col[k];
                double ss = 0.0;
                for (int cc = 0; cc < c; ++cc) ss += x[s * f + hh * c + cc] * a_src[hh * c + cc];
                double l = leaky(ss + sd, slope);
                lg[(k - k0) * h + hh] = l;
                if (k == k0 || l > mx) mx = l;
            }
            for (int64_t k = k0; k < k1; ++k) den += exp(lg[(k - k0) * h + hh] - mx);
            for (int64_t k = k0; k < k1; ++k) {
                int64_t s = col[k];
                double al = exp(lg[(k - k0) * h + hh] - mx) / den;
                if (alpha_rows) alpha_rows[(apos + (k - k0)) * h + hh] = al;
                for (int cc = 0; cc < c; ++cc) {
                    double m = al * x[s * f + hh * c + cc];
                    o[hh * c + cc] += m;
                    ab[hh * c + cc] += SCALE_TERM(m);
                }
            }
        }
        apos += deg;
        free(lg);
    }
    return OK;
}

/* ---------------------------------------------------------------------------
 * Graph pooling keyed by node_graph_index (Fig. 2a; Section 2.1.1):
 *   out[g, :] = REDUCE over nodes v with batch[v] == g of x[v, :]
 * SUM, MEAN (divide by the node count) or MAX; empty graphs give 0.
 * batch must be non-decreasing (a BatchGraph stacks graphs in order) and
 * inside [0, G).
 * ------------------------------------------------------------------------- */
int oracle_segment_pool(int reduce, int64_t n, int64_t f, int64_t g, const int64_t *batch,
                        const double *x, double *out, double *absout)
{
    if (n < 0 || f < 0 || g < 0) return E_ARG;
    if (reduce != R_SUM && reduce != R_MEAN && reduce != R_MAX) return E_ARG;
    for (int64_t v = 0; v < n; ++v) {
        if (batch[v] < 0 || batch[v] >= g) return E_RANGE;
        if (v > 0 && batch[v] < batch[v - 1]) return E_UNSORTED;
    }
    int64_t *count = (int64_t *)calloc((size_t)(g > 0 ? g : 1), sizeof(int64_t));
    if (!count) return E_ARG;
    for (int64_t k = 0; k < g * f; ++k) { out[k] = 0.0; absout[k] = 0.0; }
#ifdef ORACLE_PLANT_POOL_SKIP_LAST
    n = n > 0 ? n - 1 : 0;                                /* planted: drops the last node */
#endif
    for (int64_t v = 0; v < n; ++v) {
        int64_t b = batch[v];
        for (int64_t c = 0; c < f; ++c) {
            double m = x[v * f + c];
            if (reduce == R_MAX) {
                if (count[b] == 0 || m > out[b * f + c]) out[b * f + c] = m;
            } else {
                out[b * f + c] += m;
            }
            absout[b * f + c] += SCALE_TERM(m);
        }
        count[b] += 1;
    }
    if (reduce == R_MEAN)
        for (int64_t b = 0; b < g; ++b) {
            if (count[b] == 0) continue;
            for (int64_t c = 0; c < f; ++c) {
                out[b * f + c] /= (double)count[b];
                absout[b * f + c] /= (double)count[b];
            }
        }
    free(count);
    return OK;
}

/* ---------------------------------------------------------------------------
 * Multi-hop propagation: APPNP and SGC, two of the node-level models the
 * paper lists (Section 2.2) and evaluates (Table 1).  APPNP (Klicpera et al.)
 * runs K steps of
 *     h_0 = x0,   h_{k+1}[t] = (1 - alpha) * (sum over edges e into t of
 *                   w_e * h_k[src_e]  +  self_w[t] * h_k[t])  +  alpha * x0[t]
 * with w, self_w the GCN-normalised weights of oracle_gcn_norm; SGC
 * (Wu et al.) is alpha = 0.  Each step loops over the edges in their
 * original order, fp64 throughout.  absout runs the same recursion on
 * absolute values (|w|, |self_w|, |x0|): the scale of the rounding error of
 * an fp32 evaluation.  out/absout are [n, f].
 * ------------------------------------------------------------------------- */
int oracle_appnp(int64_t n, int64_t e, const int64_t *edge_index, const double *w,
                 const double *self_w, const double *x0, int64_t f, int64_t hops, double alpha,
                 double *out, double *absout)
{
    if (n < 0 || e < 0 || f < 0 || hops < 0 || !w) return E_ARG;
    const int64_t *src = edge_index, *dst = edge_index + e;
    for (int64_t i = 0; i < e; ++i)
        if (src[i] < 0 || src[i] >= n || dst[i] < 0 || dst[i] >= n) return E_RANGE;
    const size_t cells = (size_t)(n * f > 0 ? n * f : 1);
    double *th = (double *)calloc(cells, sizeof(double));
    double *ta = (double *)calloc(cells, sizeof(double));
    if (!th || !ta) { free(th); free(ta); return E_ARG; }
    for (int64_t k = 0; k < n * f; ++k) { out[k] = x0[k]; absout[k] = fabs(x0[k]); }
    for (int64_t hop = 0; hop < hops; ++hop) {
        for (int64_t k = 0; k < n * f; ++k) { th[k] = 0.0; ta[k] = 0.0; }
        for (int64_t i = 0; i < e; ++i) {
            const int64_t s = src[i], t = dst[i];
            for (int64_t c = 0; c < f; ++c) {
                th[t * f + c] += w[i] * out[s * f + c];
                ta[t * f + c] += fabs(w[i]) * absout[s * f + c];
            }
        }
        if (self_w)
            for (int64_t t = 0; t < n; ++t)
                for (int64_t c = 0; c < f; ++c) {
                    th[t * f + c] += self_w[t] * out[t * f + c];
                    ta[t * f + c] += fabs(self_w[t]) * absout[t * f + c];
                }
        for (int64_t k = 0; k < n * f; ++k) {
#ifdef ORACLE_PLANT_APPNP_TELEPORT_FROM_H
            const double tele = out[k];                  /* planted: teleport to h_k, not x0 */
#else
            const double tele = x0[k];
#endif
            out[k] = (1.0 - alpha) * th[k] + alpha * tele;
            absout[k] = (1.0 - alpha) * ta[k] + alpha * fabs(x0[k]);
        }
    }
    free(th);
    free(ta);
    return OK;
}

/* ---------------------------------------------------------------------------
 * Dot-product (Transformer-style) attention, the GAT form the paper says
 * tf_geometric uses (Section 4.2), on the workflow of Fig. 5a:
 *   map        l[e,h] = scale * sum_c q[dst_e,h,c] k[src_e,h,c]
 *   reduce     m[t,h] = max over edges into t of l[e,h]          (stability)
 *              den[t,h] = sum over edges into t of exp(l[e,h] - m[t,h])
 *   map        alpha[e,h] = exp(l[e,h] - m[dst_e,h]) / den[dst_e,h]
 *   aggregate  out[t,h,:] = sum over edges into t of alpha[e,h] v[src_e,h,:]
 * q, k, v are [n, H*C], head-major within a row; alpha is [e, H] in COO
 * order; targets without incoming edges give 0.
 * absout[t, h*C+c] = sum of alpha[e,h] |v[src_e,h,c]|.
 * ------------------------------------------------------------------------- */
static double dot_logit(const double *q, const double *k, int64_t t, int64_t s, int64_t f,
                        int hh, int c, double scale)
{
    double d = 0.0;
    for (int cc = 0; cc < c; ++cc) {
#ifdef ORACLE_PLANT_DOT_KEY_AT_TARGET
        d += q[t * f + hh * c + cc] * k[t * f + hh * c + cc];   /* planted: key of the target */
        (void)s;
#else
        d += q[t * f + hh * c + cc] * k[s * f + hh * c + cc];
#endif
    }
    return scale * d;
}

int oracle_dot_softmax(int64_t n, int64_t e, const int64_t *edge_index, const double *q,
                       const double *k, const double *v, int h, int c, double scale,
                       double *out, double *alpha, double *absout)
{
    if (n < 0 || e < 0 || h <= 0 || c <= 0) return E_ARG;
    const int64_t *src = edge_index, *dst = edge_index + e;
    for (int64_t i = 0; i < e; ++i)
        if (src[i] < 0 || src[i] >= n || dst[i] < 0 || dst[i] >= n) return E_RANGE;
    int64_t f = (int64_t)h * c;
    size_t nh = (size_t)(n > 0 ? n : 1) * (size_t)h;
    double *mx = (double *)calloc(nh, sizeof(double));
    double *den = (double *)calloc(nh, sizeof(double));
    char *seen = (char *)calloc(nh, 1);
    double *logit = (double *)calloc((size_t)(e > 0 ? e : 1) * (size_t)h, sizeof(double));
    if (!mx || !den || !seen || !logit) {
        free(mx); free(den); free(seen); free(logit);
        return E_ARG;
    }
    /* map: scaled query-key products; reduce: per-target max */
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh) {
            double l = dot_logit(q, k, dst[i], src[i], f, hh, c, scale);
            logit[i * h + hh] = l;
            size_t kk = (size_t)dst[i] * h + hh;
            if (!seen[kk] || l > mx[kk]) mx[kk] = l;
            seen[kk] = 1;
        }
    /* reduce: segment sum of exp -> softmax denominator */
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh)
            den[(size_t)dst[i] * h + hh] += exp(logit[i * h + hh] - mx[(size_t)dst[i] * h + hh]);
    /* map: divide; then the attention-weighted sum of values */
    for (int64_t kk = 0; kk < n * f; ++kk) { out[kk] = 0.0; absout[kk] = 0.0; }
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh) {
            size_t kk = (size_t)dst[i] * h + hh;
            double al = exp(logit[i * h + hh] - mx[kk]) / den[kk];
            if (alpha) alpha[i * h + hh] = al;
            for (int cc = 0; cc < c; ++cc) {
                double m = al * v[src[i] * f + hh * c + cc];
                out[dst[i] * f + hh * c + cc] += m;
                absout[dst[i] * f + hh * c + cc] += SCALE_TERM(m);
            }
        }
    free(mx); free(den); free(seen); free(logit);
    return OK;
}

/* The same passes for the listed target rows only, through the oracle's
 * stable CSR; alpha_rows packs each listed row's [deg, H] block in CSR order. */
int oracle_dot_softmax_rows(int64_t n, const int32_t *rowptr, const int32_t *col,
                            const double *q, const double *k, const double *v, int h, int c,
                            double scale, const int64_t *rows, int64_t nrows, double *out,
                            double *alpha_rows, double *absout)
{
    if (h <= 0 || c <= 0) return E_ARG;
    int64_t f = (int64_t)h * c;
    int64_t apos = 0;
    for (int64_t r = 0; r < nrows; ++r) {
        int64_t t = rows[r];
        if (t < 0 || t >= n) return E_RANGE;
        int64_t k0 = rowptr[t], k1 = rowptr[t + 1], deg = k1 - k0;
        double *o = out + r * f, *ab = absout + r * f;
        for (int64_t x = 0; x < f; ++x) { o[x] = 0.0; ab[x] = 0.0; }
        if (deg == 0) continue;
        double *lg = (double *)malloc(sizeof(double) * (size_t)deg);
        if (!lg) return E_ARG;
        for (int hh = 0; hh < h; ++hh) {
            double mx = 0.0, den = 0.0;
            for (int64_t p = k0; p < k1; ++p) {
                double l = dot_logit(q, k, t, col[p], f, hh, c, scale);
                lg[p - k0] = l;
                if (p == k0 || l > mx) mx = l;
            }
            for (int64_t p = k0; p < k1; ++p) den += exp(lg[p - k0] - mx);
            for (int64_t p = k0; p < k1; ++p) {
                int64_t s = col[p];
                double al = exp(lg[p - k0] - mx) / den;
                if (alpha_rows) alpha_rows[(apos + (p - k0)) * h + hh] = al;
                for (int cc = 0; cc < c; ++cc) {
                    double m = al * v[s * f + hh * c + cc];
                    o[hh * c + cc] += m;
                    ab[hh * c + cc] += SCALE_TERM(m);
                }
            }
        }
        apos += deg;
        free(lg);
    }
    return OK;
}

/* ---------------------------------------------------------------------------
 * Backward of the GAT edge-softmax aggregation: gradients of the Fig. 5a
 * workflow with respect to x, a_src and a_dst, given grad_out = dL/dout.
 * The forward quantities (node scores, z = s_src[s] + s_dst[t], logits
 * l = LeakyReLU(z), per-target maximum and denominator, alpha) are
 * recomputed exactly as oracle_edge_softmax forms them.  Then, per edge
 * e = (s -> t) and head h:
 *   dalpha[e,h] = sum_c grad_out[t,h,c] x[s,h,c]
 *   beta[t,h]   = sum over edges e' into t of alpha[e',h] dalpha[e',h]
 *   dl[e,h]     = alpha[e,h] (dalpha[e,h] - beta[t,h])      (softmax Jacobian)
 *   dz[e,h]     = dl[e,h] * (z > 0 ? 1 : slope)             (LeakyReLU)
 *   grad_x[s,h,:]   += alpha[e,h] grad_out[t,h,:]           (weighted sum)
 *   ds_src[s,h] += dz[e,h];   ds_dst[t,h] += dz[e,h]
 * and per node v:  grad_x[v,h,c] += ds_src[v,h] a_src[h,c] + ds_dst[v,h] a_dst[h,c],
 * grad_a_src[h,c] = sum_v ds_src[v,h] x[v,h,c], grad_a_dst likewise.
 * absout_* run the same recursion on absolute values (|dalpha| = sum |g||x|,
 * |beta| = sum alpha |dalpha|, |dl| = alpha (|dalpha| + |beta|), ...): the
 * scale that a tolerance on each gradient is measured against.
 * ------------------------------------------------------------------------- */
int oracle_edge_softmax_backward(int64_t n, int64_t e, const int64_t *edge_index, const double *x,
                                 int h, int c, const double *a_src, const double *a_dst,
                                 double slope, const double *grad_out, double *grad_x,
                                 double *grad_a_src, double *grad_a_dst, double *abs_x,
                                 double *abs_a_src, double *abs_a_dst)
{
    if (n < 0 || e < 0 || h <= 0 || c <= 0) return E_ARG;
    const int64_t *src = edge_index, *dst = edge_index + e;
    for (int64_t i = 0; i < e; ++i)
        if (src[i] < 0 || src[i] >= n || dst[i] < 0 || dst[i] >= n) return E_RANGE;
    int64_t f = (int64_t)h * c;
    size_t nh = (size_t)(n > 0 ? n : 1) * (size_t)h, eh = (size_t)(e > 0 ? e : 1) * (size_t)h;
    double *s_src = (double *)calloc(nh, sizeof(double));
    double *s_dst = (double *)calloc(nh, sizeof(double));
    double *mx = (double *)calloc(nh, sizeof(double));
    double *den = (double *)calloc(nh, sizeof(double));
    double *beta = (double *)calloc(nh, sizeof(double));
    double *abeta = (double *)calloc(nh, sizeof(double));
    double *ds_src = (double *)calloc(nh, sizeof(double));
    double *ds_dst = (double *)calloc(nh, sizeof(double));
    double *as_src = (double *)calloc(nh, sizeof(double));
    double *as_dst = (double *)calloc(nh, sizeof(double));
    char *seen = (char *)calloc(nh, 1);
    double *z = (double *)calloc(eh, sizeof(double));
    double *alpha = (double *)calloc(eh, sizeof(double));
    double *dal = (double *)calloc(eh, sizeof(double));
    double *adal = (double *)calloc(eh, sizeof(double));
    int rc = OK;
    if (!s_src || !s_dst || !mx || !den || !beta || !abeta || !ds_src || !ds_dst || !as_src ||
        !as_dst || !seen || !z || !alpha || !dal || !adal) { rc = E_ARG; goto done; }
    /* forward: node scores, logits, per-target maximum and denominator, alpha */
    for (int64_t v = 0; v < n; ++v)
        for (int hh = 0; hh < h; ++hh) {
            double a = 0.0, b = 0.0;
            for (int cc = 0; cc < c; ++cc) {
                a += x[v * f + hh * c + cc] * a_src[hh * c + cc];
                b += x[v * f + hh * c + cc] * a_dst[hh * c + cc];
            }
            s_src[v * h + hh] = a;
            s_dst[v * h + hh] = b;
        }
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh) {
            double zz = s_src[src[i] * h + hh] + s_dst[dst[i] * h + hh];
            z[i * h + hh] = zz;
            double l = leaky(zz, slope);
            size_t k = (size_t)dst[i] * h + hh;
            if (!seen[k] || l > mx[k]) mx[k] = l;
            seen[k] = 1;
        }
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh) {
            size_t k = (size_t)dst[i] * h + hh;
            den[k] += exp(leaky(z[i * h + hh], slope) - mx[k]);
        }
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh) {
            size_t k = (size_t)dst[i] * h + hh;
            alpha[i * h + hh] = exp(leaky(z[i * h + hh], slope) - mx[k]) / den[k];
        }
    /* dalpha and beta */
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh) {
            double d = 0.0, ad = 0.0;
            for (int cc = 0; cc < c; ++cc) {
                double p = grad_out[dst[i] * f + hh * c + cc] * x[src[i] * f + hh * c + cc];
                d += p;
                ad += fabs(p);
            }
            dal[i * h + hh] = d;
            adal[i * h + hh] = ad;
            size_t k = (size_t)dst[i] * h + hh;
            beta[k] += alpha[i * h + hh] * d;
            abeta[k] += alpha[i * h + hh] * ad;
        }
    for (int64_t k = 0; k < n * f; ++k) { grad_x[k] = 0.0; abs_x[k] = 0.0; }
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh) {
            size_t kt = (size_t)dst[i] * h + hh;
            double al = alpha[i * h + hh];
#ifdef ORACLE_PLANT_BWD_NO_SOFTMAX_JACOBIAN
            double dl = al * dal[i * h + hh];                       /* planted: beta dropped */
#else
            double dl = al * (dal[i * h + hh] - beta[kt]);
#endif
            double adl = al * (adal[i * h + hh] + abeta[kt]);
            double lk = z[i * h + hh] > 0.0 ? 1.0 : slope;
            ds_src[src[i] * h + hh] += dl * lk;
            ds_dst[kt] += dl * lk;
            as_src[src[i] * h + hh] += adl * fabs(lk);
            as_dst[kt] += adl * fabs(lk);
            for (int cc = 0; cc < c; ++cc) {
                double m = al * grad_out[dst[i] * f + hh * c + cc];
                grad_x[src[i] * f + hh * c + cc] += m;
                abs_x[src[i] * f + hh * c + cc] += SCALE_TERM(m);
            }
        }
    for (int64_t v = 0; v < n; ++v)
        for (int hh = 0; hh < h; ++hh)
            for (int cc = 0; cc < c; ++cc) {
                size_t k = (size_t)v * h + hh;
                double m1 = ds_src[k] * a_src[hh * c + cc], m2 = ds_dst[k] * a_dst[hh * c + cc];
                grad_x[v * f + hh * c + cc] += m1 + m2;
                abs_x[v * f + hh * c + cc] += as_src[k] * fabs(a_src[hh * c + cc]) +
                                              as_dst[k] * fabs(a_dst[hh * c + cc]);
            }
    for (int64_t k = 0; k < f; ++k) {
        grad_a_src[k] = grad_a_dst[k] = 0.0;
        abs_a_src[k] = abs_a_dst[k] = 0.0;
    }
    for (int64_t v = 0; v < n; ++v)
        for (int hh = 0; hh < h; ++hh)
            for (int cc = 0; cc < c; ++cc) {
                size_t k = (size_t)v * h + hh;
                double xv = x[v * f + hh * c + cc];
                grad_a_src[hh * c + cc] += ds_src[k] * xv;
                grad_a_dst[hh * c + cc] += ds_dst[k] * xv;
                abs_a_src[hh * c + cc] += as_src[k] * fabs(xv);
                abs_a_dst[hh * c + cc] += as_dst[k] * fabs(xv);
            }
done:
    free(s_src); free(s_dst); free(mx); free(den); free(beta); free(abeta); free(ds_src);
    free(ds_dst); free(as_src); free(as_dst); free(seen); free(z); free(alpha); free(dal);
    free(adal);
    return rc;
}

/* ---------------------------------------------------------------------------
 * Backward of the dot-product (Transformer-style) attention aggregation:
 * gradients with respect to q, k and v given grad_out = dL/dout.  Forward
 * quantities are recomputed as oracle_dot_softmax forms them; then per edge
 * e = (s -> t) and head h:
 *   dalpha[e,h] = sum_c grad_out[t,h,c] v[s,h,c]
 *   beta[t,h]   = sum over edges e' into t of alpha[e',h] dalpha[e',h]
 *   dl[e,h]     = alpha[e,h] (dalpha[e,h] - beta[t,h])          (softmax Jacobian)
 *   grad_q[t,h,:] += scale dl[e,h] k[s,h,:]
 *   grad_k[s,h,:] += scale dl[e,h] q[t,h,:]
 *   grad_v[s,h,:] += alpha[e,h] grad_out[t,h,:]
 * abs_* run the same recursion on absolute values.
 * ------------------------------------------------------------------------- */
int oracle_dot_softmax_backward(int64_t n, int64_t e, const int64_t *edge_index, const double *q,
                                const double *k, const double *v, int h, int c, double scale,
                                const double *grad_out, double *grad_q, double *grad_k,
                                double *grad_v, double *abs_q, double *abs_k, double *abs_v)
{
    if (n < 0 || e < 0 || h <= 0 || c <= 0) return E_ARG;
    const int64_t *src = edge_index, *dst = edge_index + e;
    for (int64_t i = 0; i < e; ++i)
        if (src[i] < 0 || src[i] >= n || dst[i] < 0 || dst[i] >= n) return E_RANGE;
    int64_t f = (int64_t)h * c;
    size_t nh = (size_t)(n > 0 ? n : 1) * (size_t)h, eh = (size_t)(e > 0 ? e : 1) * (size_t)h;
    double *mx = (double *)calloc(nh, sizeof(double));
    double *den = (double *)calloc(nh, sizeof(double));
    double *beta = (double *)calloc(nh, sizeof(double));
    double *abeta = (double *)calloc(nh, sizeof(double));
    char *seen = (char *)calloc(nh, 1);
    double *logit = (double *)calloc(eh, sizeof(double));
    double *alpha = (double *)calloc(eh, sizeof(double));
    double *dal = (double *)calloc(eh, sizeof(double));
    double *adal = (double *)calloc(eh, sizeof(double));
    int rc = OK;
    if (!mx || !den || !beta || !abeta || !seen || !logit || !alpha || !dal || !adal) {
        rc = E_ARG;
        goto done;
    }
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh) {
            double l = dot_logit(q, k, dst[i], src[i], f, hh, c, scale);
            logit[i * h + hh] = l;
            size_t kk = (size_t)dst[i] * h + hh;
            if (!seen[kk] || l > mx[kk]) mx[kk] = l;
            seen[kk] = 1;
        }
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh)
            den[(size_t)dst[i] * h + hh] += exp(logit[i * h + hh] - mx[(size_t)dst[i] * h + hh]);
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh) {
            size_t kk = (size_t)dst[i] * h + hh;
            double al = exp(logit[i * h + hh] - mx[kk]) / den[kk];
            double d = 0.0, ad = 0.0;
            for (int cc = 0; cc < c; ++cc) {
                double pr = grad_out[dst[i] * f + hh * c + cc] * v[src[i] * f + hh * c + cc];
                d += pr;
                ad += fabs(pr);
            }
            alpha[i * h + hh] = al;
            dal[i * h + hh] = d;
            adal[i * h + hh] = ad;
            beta[kk] += al * d;
            abeta[kk] += al * ad;
        }
    for (int64_t kk = 0; kk < n * f; ++kk) {
        grad_q[kk] = grad_k[kk] = grad_v[kk] = 0.0;
        abs_q[kk] = abs_k[kk] = abs_v[kk] = 0.0;
    }
    for (int64_t i = 0; i < e; ++i)
        for (int hh = 0; hh < h; ++hh) {
            size_t kt = (size_t)dst[i] * h + hh;
            double al = alpha[i * h + hh];
#ifdef ORACLE_PLANT_BWD_NO_SOFTMAX_JACOBIAN
            double dl = al * dal[i * h + hh];                       /* planted: beta dropped */
#else
            double dl = al * (dal[i * h + hh] - beta[kt]);
#endif
            double adl = al * (adal[i * h + hh] + abeta[kt]);
            for (int cc = 0; cc < c; ++cc) {
                int64_t ot = dst[i] * f + hh * c + cc, os = src[i] * f + hh * c + cc;
                double mq = scale * dl * k[os], mk = scale * dl * q[ot], mv = al * grad_out[ot];
                grad_q[ot] += mq;
                grad_k[os] += mk;
                grad_v[os] += mv;
                abs_q[ot] += fabs(scale) * adl * fabs(k[os]);
                abs_k[os] += fabs(scale) * adl * fabs(q[ot]);
                abs_v[os] += SCALE_TERM(mv);
            }
        }
done:
    free(mx); free(den); free(beta); free(abeta); free(seen); free(logit); free(alpha);
    free(dal); free(adal);
    return rc;
}

/* ---------------------------------------------------------------------------
 * Backward of the aggregation: the gradient with respect to x of the
 * aggregation out[t] = sum over edges e = (s -> t) of w_e x[s] (sum), the
 * same divided by the number of edges into t (mean), or with the GCN weights
 * w_e = w_norm[e] plus the implicit self-loop term self_w[t] x[t].  With
 * grad_out = dL/dout, dL/dx[s] = sum over edges e = (s -> t) of
 * w_e grad_out[t] (/ count[t] for the mean) (+ self_w[s] grad_out[s]).
 * Loops over the edges in original order, fp64.  absout = same with |terms|.
 * ------------------------------------------------------------------------- */
int oracle_aggregate_backward(int reduce, int64_t n, int64_t e, const int64_t *edge_index,
                              const double *w, const double *self_w, const double *grad_out,
                              int64_t f, double *grad_x, double *absout)
{
    if (n < 0 || e < 0 || f < 0) return E_ARG;
    if (reduce != R_SUM && reduce != R_MEAN) return E_ARG;
    const int64_t *src = edge_index, *dst = edge_index + e;
    for (int64_t i = 0; i < e; ++i)
        if (src[i] < 0 || src[i] >= n || dst[i] < 0 || dst[i] >= n) return E_RANGE;
    int64_t *count = (int64_t *)calloc((size_t)(n > 0 ? n : 1), sizeof(int64_t));
    if (!count) return E_ARG;
    for (int64_t i = 0; i < e; ++i) count[dst[i]] += 1;
    for (int64_t k = 0; k < n * f; ++k) { grad_x[k] = 0.0; absout[k] = 0.0; }
    for (int64_t i = 0; i < e; ++i) {
#ifdef ORACLE_PLANT_BACKWARD_NO_TRANSPOSE
        int64_t s = dst[i], t = src[i];            /* planted: gradient sent along the edge */
#else
        int64_t s = src[i], t = dst[i];
#endif
        double we = w ? w[i] : 1.0;
        if (reduce == R_MEAN) we /= (double)count[dst[i]];
        for (int64_t c = 0; c < f; ++c) {
            double m = we * grad_out[t * f + c];
            grad_x[s * f + c] += m;
            absout[s * f + c] += SCALE_TERM(m);
        }
    }
    if (self_w && reduce == R_SUM)
        for (int64_t s = 0; s < n; ++s)
            for (int64_t c = 0; c < f; ++c) {
                double m = self_w[s] * grad_out[s * f + c];
                grad_x[s * f + c] += m;
                absout[s * f + c] += SCALE_TERM(m);
            }
    free(count);
    return OK;
}

/* Max with argmax: per (t, c) the original id of the FIRST edge into t (in
 * original order) whose product w_e x[s, c] is the largest, -1 without
 * edges.  The product is compared after rounding to fp32 (the precision in
 * which the CUDA kernel forms and compares it), so both sides make the same
 * choice; out holds the exact fp64 value of the chosen product. */
int oracle_max_argmax(int64_t n, int64_t e, const int64_t *edge_index, const float *w,
                      const double *x, int64_t f, double *out, int32_t *argmax)
{
    if (n < 0 || e < 0 || f < 0) return E_ARG;
    const int64_t *src = edge_index, *dst = edge_index + e;
    for (int64_t i = 0; i < e; ++i)
        if (src[i] < 0 || src[i] >= n || dst[i] < 0 || dst[i] >= n) return E_RANGE;
    float *best = (float *)malloc(sizeof(float) * (size_t)(n * f > 0 ? n * f : 1));
    if (!best) return E_ARG;
    for (int64_t k = 0; k < n * f; ++k) { out[k] = 0.0; argmax[k] = -1; }
    for (int64_t i = 0; i < e; ++i) {
        int64_t s = src[i], t = dst[i];
        double we = w ? (double)w[i] : 1.0;
        for (int64_t c = 0; c < f; ++c) {
            double m = we * x[s * f + c];
            float m32 = (float)m;
            if (argmax[t * f + c] < 0 || m32 > best[t * f + c]) {
                best[t * f + c] = m32;
                out[t * f + c] = m;
                argmax[t * f + c] = (int32_t)i;
            }
        }
    }
    free(best);
    return OK;
}

/* grad_x[s, c] = sum over edges e = (s -> t), in original order, with
 * argmax[t, c] == e of w_e grad_out[t, c] (w NULL: 1). */
int oracle_max_backward(int64_t n, int64_t e, const int64_t *edge_index, const int32_t *argmax,
                        const double *w, const double *grad_out, int64_t f, double *grad_x,
                        double *absout)
{
    if (n < 0 || e < 0 || f < 0) return E_ARG;
    const int64_t *src = edge_index, *dst = edge_index + e;
    for (int64_t k = 0; k < n * f; ++k) { grad_x[k] = 0.0; absout[k] = 0.0; }
    for (int64_t i = 0; i < e; ++i) {
        int64_t s = src[i], t = dst[i];
        if (s < 0 || s >= n || t < 0 || t >= n) return E_RANGE;
        for (int64_t c = 0; c < f; ++c)
            if (argmax[t * f + c] == (int32_t)i) {
                double m = (w ? w[i] : 1.0) * grad_out[t * f + c];
                grad_x[s * f + c] += m;
                absout[s * f + c] += SCALE_TERM(m);
            }
    }
    return OK;
}
