"""Pins of the fp64 oracle against facts fixed outside the oracle itself.

Each pin is a function of an oracle object so that the same check can be run
against a build with a planted mistake (``test_planted_mistakes_are_caught``):
every plausible slip planted in ``oracle/tfg_oracle.c`` must make at least
one pin fail.  No GPU is used here.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle
from paper_2101_11552_gb300 import graphgen as gg

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as fh:
        return json.load(fh)


def _undirected_random(n, m, seed, self_loops=False):
    rng = np.random.default_rng(seed)
    ei = gg.symmetrise(gg.er_pairs(n, m, rng))
    return gg.with_self_loops(ei, n) if self_loops else ei


# ---------------------------------------------------------------------------
# CSR by target: brute force with Python's (stable) sort
# ---------------------------------------------------------------------------
def pin_csr_is_stable_grouping(o):
    for seed, (n, e) in enumerate([(7, 40), (50, 300), (1, 5), (30, 0), (200, 2000)]):
        w = gg.random_edge_case_graph(n, e, 1, seed, hub=0 if n > 1 else -1, isolated=min(3, n - 1))
        ei = w.edge_index
        rowptr, col, perm, deg = o.build_csr(ei, n)
        order = sorted(range(e), key=lambda k: int(ei[1, k]))       # stable
        assert list(perm) == order
        assert list(col) == [int(ei[0, k]) for k in order]
        counts = [0] * n
        for k in range(e):
            counts[int(ei[1, k])] += 1
        assert list(deg) == counts
        acc = [0]
        for c in counts:
            acc.append(acc[-1] + c)
        assert list(rowptr) == acc


def test_csr_is_stable_grouping():
    pin_csr_is_stable_grouping(oracle.default)


def test_csr_rejects_out_of_range():
    ei = np.array([[0, 3], [1, 0]], dtype=np.int64)
    with pytest.raises(oracle.OracleError) as exc:
        oracle.build_csr(ei, 3)
    assert exc.value.code == -5


# ---------------------------------------------------------------------------
# GCN normalisation and sum: hand examples, eigenvector identity, dense form
# ---------------------------------------------------------------------------
def pin_gcn_p4(o):
    g = _golden("gcn_p4.json")
    ei = gg.symmetrise(np.array(g["edges_undirected"], dtype=np.int64))
    x = np.array(g["x"], dtype=np.float32)[:, None]
    out, _ = o.gcn_aggregate(ei, 4, x, add_self_loops=g["add_self_loops"])
    np.testing.assert_allclose(out[:, 0], g["out"], rtol=0, atol=g["abs_tol"])
    closed = [1 / 2 + 2 / math.sqrt(6), 1 / math.sqrt(6) + 2 / 3 + 1, 2 / 3 + 1 + 4 / math.sqrt(6),
              3 / math.sqrt(6) + 2]
    np.testing.assert_allclose(out[:, 0], closed, rtol=1e-14)
    nrm = o.gcn_norm(ei, 4, add_self_loops=1)
    np.testing.assert_allclose(nrm["deg"], g["degree"], rtol=0, atol=0)


def test_gcn_p4():
    pin_gcn_p4(oracle.default)


def pin_gcn_directed(o):
    g = _golden("gcn_directed3.json")
    ei = np.array(g["edge_index"], dtype=np.int64)
    x = np.array(g["x"], dtype=np.float32)[:, None]
    out, _ = o.gcn_aggregate(ei, 3, x, add_self_loops=1)
    np.testing.assert_allclose(out[:, 0], g["out"], rtol=0, atol=g["abs_tol"])
    nrm = o.gcn_norm(ei, 3, add_self_loops=1)
    np.testing.assert_array_equal(nrm["deg"], g["in_degree_with_self_loop"])


def test_gcn_directed_hand_example():
    pin_gcn_directed(oracle.default)


def pin_gcn_sqrt_degree_eigenvector(o):
    """For a symmetric graph, D^-1/2 A' D^-1/2 sqrt(d) = sqrt(d) exactly (math).

    (A' = A + fill I with weighted degrees d = row sums of A'.)  Holds with
    and without implicit self-loops and with symmetric edge weights.
    """
    for seed, (n, m, selfl, weighted) in enumerate(
            [(40, 90, 1, False), (300, 1200, 0, False), (120, 400, 1, True), (64, 64, 0, True)]):
        rng = np.random.default_rng(50 + seed)
        pairs = gg.er_pairs(n, m, rng)
        ei = gg.symmetrise(pairs)
        w = None
        if weighted:
            wp = rng.uniform(0.5, 2.0, size=m)
            w = np.concatenate([wp, wp])
        nrm = o.gcn_norm(ei, n, w, add_self_loops=selfl, fill=1.0)
        x = np.sqrt(nrm["deg"])[:, None]
        out, _ = o.aggregate(ei, n, x, "sum", w=nrm["w_norm"], self_w=nrm["self_w"])
        np.testing.assert_allclose(out[:, 0], x[:, 0], rtol=1e-12, atol=1e-14)


def test_gcn_sqrt_degree_eigenvector():
    pin_gcn_sqrt_degree_eigenvector(oracle.default)


def pin_dense_equivalence(o):
    """Per-edge loops == numpy dense matrices for tiny random multigraphs."""
    for seed in range(6):
        n = [1, 5, 17, 33, 64, 64][seed]
        e = [3, 12, 80, 200, 500, 0][seed]
        wl = gg.random_edge_case_graph(n, e, 7, seed, hub=0 if n > 2 else -1, isolated=min(2, n - 1))
        ei, x = wl.edge_index, wl.x
        rng = np.random.default_rng(seed)
        ew = rng.uniform(0.1, 3.0, size=e)
        xd = x.astype(np.float64)
        for selfl in (0, 1):
            out, _ = o.gcn_aggregate(ei, n, x, ew, add_self_loops=selfl, fill=1.5)
            ref = oracle.dense_gcn_matrix(ei, n, ew, selfl, 1.5) @ xd
            np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)
        m = oracle.dense_adjacency(ei, n, ew)
        cnt = oracle.dense_adjacency(ei, n, None).sum(axis=1)
        out, _ = o.aggregate(ei, n, x, "sum", w=ew)
        np.testing.assert_allclose(out, m @ xd, rtol=1e-12, atol=1e-12)
        out, _ = o.aggregate(ei, n, x, "mean", w=ew)
        ref = np.where(cnt[:, None] > 0, (m @ xd) / np.maximum(cnt, 1)[:, None], 0.0)
        np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)


def test_dense_equivalence():
    pin_dense_equivalence(oracle.default)


def pin_ones_give_in_degree(o):
    for seed in range(3):
        wl = gg.random_edge_case_graph(90, 700, 3, 10 + seed, hub=4, isolated=5)
        ones = np.ones((90, 3), np.float32)
        out, _ = o.aggregate(wl.edge_index, 90, ones, "sum")
        deg = np.bincount(wl.edge_index[1], minlength=90)
        np.testing.assert_array_equal(out, np.repeat(deg[:, None], 3, axis=1).astype(float))
        out, _ = o.aggregate(wl.edge_index, 90, ones * 2.5, "mean")
        np.testing.assert_array_equal(out, np.where(deg[:, None] > 0, 2.5, 0.0) * np.ones((1, 3)))


def test_ones_give_in_degree_and_mean_of_constant():
    pin_ones_give_in_degree(oracle.default)


def pin_max_brute_force(o):
    for seed in range(4):
        n, e = 40, 300
        wl = gg.random_edge_case_graph(n, e, 5, 20 + seed, hub=1, isolated=4)
        ei, x = wl.edge_index, wl.x
        rng = np.random.default_rng(seed)
        w = rng.uniform(-2, 2, size=e).astype(np.float32)
        for weights in (None, w):
            out, _ = o.aggregate(ei, n, x, "max", w=weights)
            for t in range(n):
                ks = [k for k in range(e) if ei[1, k] == t]
                for c in range(5):
                    if not ks:
                        assert out[t, c] == 0.0
                        continue
                    vals = [(1.0 if weights is None else float(weights[k])) * float(x[ei[0, k], c])
                            for k in ks]
                    assert out[t, c] == max(vals)


def test_max_brute_force():
    pin_max_brute_force(oracle.default)


def test_permutation_invariance():
    wl = gg.random_edge_case_graph(300, 4000, 9, 77, hub=3, isolated=10)
    ei, x = wl.edge_index, wl.x
    p = np.random.default_rng(1).permutation(ei.shape[1])
    a, _ = oracle.aggregate(ei, 300, x, "max")
    b, _ = oracle.aggregate(ei[:, p], 300, x, "max")
    np.testing.assert_array_equal(a, b)
    a, _ = oracle.gcn_aggregate(ei, 300, x, add_self_loops=1)
    b, _ = oracle.gcn_aggregate(ei[:, p], 300, x, add_self_loops=1)
    np.testing.assert_allclose(a, b, rtol=1e-12, atol=1e-13)
    rp, col, perm, _ = oracle.build_csr(ei[:, p], 300)
    # the permuted CSR holds the same multiset of sources per row
    r0, c0, _, _ = oracle.build_csr(ei, 300)
    np.testing.assert_array_equal(rp, r0)
    for t in range(300):
        assert sorted(col[rp[t]:rp[t + 1]]) == sorted(c0[r0[t]:r0[t + 1]])


# ---------------------------------------------------------------------------
# Edge softmax (GAT): hand values, normalisation, reduction to mean
# ---------------------------------------------------------------------------
def pin_star_softmax(o):
    g = _golden("gat_star.json")
    ei = np.array(g["edge_index"], dtype=np.int64)
    for case in g["cases"]:
        x = np.array([[case["x0"]], [1.0], [2.0], [3.0]], dtype=np.float32)
        out, alpha, _ = o.edge_softmax(ei, 4, x, 1, 1, g["a_src"], g["a_dst"], g["negative_slope"])
        np.testing.assert_allclose(alpha[:, 0], case["alpha"], rtol=0, atol=g["abs_tol"])
        np.testing.assert_allclose(out[0, 0], case["out0"], rtol=0, atol=g["abs_tol"])
        np.testing.assert_array_equal(out[1:, 0], 0.0)
        ex = np.exp(np.array(case["logits"]))
        np.testing.assert_allclose(alpha[:, 0], ex / ex.sum(), rtol=1e-13)


def test_star_softmax():
    pin_star_softmax(oracle.default)


def pin_softmax_normalised_and_mean_limit(o):
    for seed in range(3):
        n, e, h, c = 60, 500, 3, 4
        wl = gg.random_edge_case_graph(n, e, h * c, 30 + seed, hub=2, isolated=5)
        ei, x = wl.edge_index, wl.x
        rng = np.random.default_rng(seed)
        a_s = rng.standard_normal(h * c)
        a_d = rng.standard_normal(h * c)
        _, alpha, _ = o.edge_softmax(ei, n, x, h, c, a_s, a_d, 0.2)
        sums = np.zeros((n, h))
        np.add.at(sums, ei[1], alpha)
        deg = np.bincount(ei[1], minlength=n)
        np.testing.assert_allclose(sums[deg > 0], 1.0, rtol=1e-12)
        np.testing.assert_array_equal(sums[deg == 0], 0.0)
        # zero attention vectors: every logit is 0, alpha = 1/in-degree -> mean
        out, alpha, _ = o.edge_softmax(ei, n, x, h, c, np.zeros(h * c), np.zeros(h * c), 0.2)
        mean, _ = o.aggregate(ei, n, x, "mean")
        np.testing.assert_allclose(out, mean, rtol=1e-12, atol=1e-13)
        np.testing.assert_allclose(alpha[:, 0], 1.0 / deg[ei[1]], rtol=1e-13)


def test_softmax_normalised_and_mean_limit():
    pin_softmax_normalised_and_mean_limit(oracle.default)


def test_softmax_heads_are_independent():
    n, e, c = 50, 400, 5
    wl = gg.random_edge_case_graph(n, e, 2 * c, 41, hub=1)
    ei, x = wl.edge_index, wl.x
    rng = np.random.default_rng(3)
    a_s0, a_d0 = rng.standard_normal(c), rng.standard_normal(c)
    a_s = np.concatenate([a_s0, np.zeros(c)])
    a_d = np.concatenate([a_d0, np.zeros(c)])
    out, alpha, _ = oracle.edge_softmax(ei, n, x, 2, c, a_s, a_d, 0.2)
    one, alpha1, _ = oracle.edge_softmax(ei, n, x[:, :c].copy(), 1, c, a_s0, a_d0, 0.2)
    np.testing.assert_allclose(out[:, :c], one, rtol=1e-13, atol=1e-14)
    np.testing.assert_allclose(alpha[:, 0], alpha1[:, 0], rtol=1e-13)
    mean, _ = oracle.aggregate(ei, n, x[:, c:].copy(), "mean")
    np.testing.assert_allclose(out[:, c:], mean, rtol=1e-12, atol=1e-13)


def test_row_variants_match_full():
    wl = gg.random_edge_case_graph(120, 1500, 8, 5, hub=7, isolated=6)
    ei, x, n = wl.edge_index, wl.x, 120
    csr = oracle.build_csr(ei, n)
    rows = np.array([0, 7, 119, 118, 50, 3], dtype=np.int64)
    rng = np.random.default_rng(0)
    w = rng.uniform(-1, 1, ei.shape[1])
    for red in ("sum", "mean", "max"):
        full, fab = oracle.aggregate(ei, n, x, red, w=w)
        part, pab = oracle.aggregate_rows(csr, n, x, red, rows, w=w)
        np.testing.assert_array_equal(part, full[rows])
        np.testing.assert_allclose(pab, fab[rows], rtol=1e-15)
    a_s, a_d = rng.standard_normal(8), rng.standard_normal(8)
    full, alpha, _ = oracle.edge_softmax(ei, n, x, 2, 4, a_s, a_d, 0.2)
    part, alpha_r, _ = oracle.edge_softmax_rows(csr, n, x, 2, 4, a_s, a_d, 0.2, rows)
    np.testing.assert_allclose(part, full[rows], rtol=1e-13, atol=1e-14)
    rowptr, _, perm, _ = csr
    want = np.concatenate([alpha[perm[rowptr[r]:rowptr[r + 1]]] for r in rows])
    np.testing.assert_allclose(alpha_r, want, rtol=1e-13)


# ---------------------------------------------------------------------------
# BatchGraph: the paper's reindexing example and batched == per-graph
# ---------------------------------------------------------------------------
def test_batch_reindex_example():
    g = _golden("batch_reindex.json")
    sizes = g["graph_sizes"]
    parts = [np.zeros((2, 0), np.int64) for _ in sizes]
    _, batch, offsets = gg.batch_graphs(parts, sizes)
    assert list(offsets) == g["offsets"]
    for item in g["one_based"]:          # the paper counts from 1
        assert item["node"] + offsets[item["graph"] - 1] == item["index"]
    for item in g["zero_based"]:
        assert item["node"] + offsets[item["graph"]] == item["index"]
    assert list(batch) == [0, 0, 0, 0, 1, 1, 2, 2, 2]


def test_oracle_batch_graphs_worked_example():
    """The oracle's own reindexing reproduces the paper's example and agrees
    with the generator's stacking (two independent implementations)."""
    g = _golden("batch_reindex.json")
    sizes = g["graph_sizes"]
    rng = np.random.default_rng(2)
    parts = [gg.symmetrise(gg.er_pairs(s, s - 1, rng)) if s > 1 else np.zeros((2, 0), np.int64)
             for s in sizes]
    stacked = np.concatenate(parts, axis=1)
    ei, batch, offs = oracle.batch_graphs(sizes, [p.shape[1] for p in parts], stacked)
    assert list(offs[:-1]) == g["offsets"] and offs[-1] == sum(sizes)
    for item in g["one_based"]:
        assert item["node"] + offs[item["graph"] - 1] == item["index"]
    ref_ei, ref_batch, ref_offs = gg.batch_graphs(parts, sizes)
    assert np.array_equal(ei, ref_ei) and np.array_equal(batch, ref_batch)
    assert np.array_equal(offs[:-1], ref_offs)
    with pytest.raises(oracle.OracleError):
        oracle.batch_graphs([2, 2], [1, 0], np.array([[0], [2]]))   # node 2 outside graph 0


def pin_batched_equals_per_graph(o):
    """Applying the aggregation to a BatchGraph equals applying it per graph
    and concatenating (Section 2.1.1); pooling equals per-graph full reductions."""
    rng = np.random.default_rng(9)
    sizes = [int(s) for s in rng.integers(5, 30, size=12)] + [1]
    graphs = [gg.with_self_loops(gg.symmetrise(gg.er_pairs(s, min(2 * s, s * (s - 1) // 2), rng)), s)
              for s in sizes]
    ei, batch, offsets = gg.batch_graphs(graphs, sizes)
    n = sum(sizes)
    x = rng.standard_normal((n, 6)).astype(np.float32)
    full_gcn, _ = o.gcn_aggregate(ei, n, x)
    full_max, _ = o.aggregate(ei, n, x, "max")
    for g, (s, off) in enumerate(zip(sizes, offsets)):
        xs = x[off:off + s]
        part, _ = o.gcn_aggregate(graphs[g], s, xs)
        np.testing.assert_array_equal(part, full_gcn[off:off + s])
        part, _ = o.aggregate(graphs[g], s, xs, "max")
        np.testing.assert_array_equal(part, full_max[off:off + s])
    g_n = len(sizes)
    for red, fn in (("sum", np.sum), ("mean", np.mean), ("max", np.max)):
        pooled, _ = o.segment_pool(full_gcn, batch, g_n, red)
        for g, (s, off) in enumerate(zip(sizes, offsets)):
            np.testing.assert_allclose(pooled[g], fn(full_gcn[off:off + s], axis=0),
                                       rtol=1e-13, atol=1e-14)


def test_batched_equals_per_graph():
    pin_batched_equals_per_graph(oracle.default)


def pin_pool_counts(o):
    batch = np.array([0, 0, 0, 2, 2, 4, 4, 4, 4], dtype=np.int64)
    ones = np.ones((9, 2), np.float32)
    out, _ = o.segment_pool(ones, batch, 6, "sum")
    np.testing.assert_array_equal(out[:, 0], [3, 0, 2, 0, 4, 0])
    # x[v] = [2v - 10, 2v - 9]
    x = np.arange(18, dtype=np.float32).reshape(9, 2) - 10
    out, _ = o.segment_pool(x, batch, 6, "max")
    np.testing.assert_array_equal(out[:, 1], [-5, 0, -1, 0, 7, 0])
    out, _ = o.segment_pool(x, batch, 6, "mean")
    np.testing.assert_array_equal(out[:, 0], [-8, 0, -3, 0, 3, 0])


def test_pool_counts_and_empty_graphs():
    pin_pool_counts(oracle.default)


def test_pool_rejects_unsorted_and_out_of_range():
    x = np.ones((3, 1), np.float32)
    with pytest.raises(oracle.OracleError) as exc:
        oracle.segment_pool(x, np.array([0, 1, 0]), 2, "sum")
    assert exc.value.code == -6
    with pytest.raises(oracle.OracleError) as exc:
        oracle.segment_pool(x, np.array([0, 1, 2]), 2, "sum")
    assert exc.value.code == -5


def test_bf16_widening_is_exact():
    x = np.random.default_rng(0).standard_normal((10, 8)).astype(np.float32)
    bits = gg.bf16_bits_rne(x)
    wide = oracle.widen(bits)
    np.testing.assert_array_equal(wide, gg.bf16_bits_to_f32(bits).astype(np.float64))
    # RNE: at most half an ulp of bf16 (2^-8 relative) from the fp32 value
    assert np.all(np.abs(wide - x) <= np.abs(x) * 2.0 ** -8)


# ---------------------------------------------------------------------------
# Backward of the aggregation
# ---------------------------------------------------------------------------
def _fd_directional(forward, x, g, u, h):
    """(L(x + h u) - L(x - h u)) / 2h for L(x) = <g, forward(x)>."""
    return (np.sum(g * forward(x + h * u)) - np.sum(g * forward(x - h * u))) / (2 * h)


def pin_backward_finite_differences(o):
    """<grad_x, u> equals the central difference of <grad_out, forward(x)>
    along u: exact (to rounding) for the linear sum, mean and GCN
    aggregations, and for max away from ties (distinct random values)."""
    for seed in range(3):
        n, e, f = 40, 260, 3
        wl = gg.random_edge_case_graph(n, e, f, 80 + seed, hub=1, isolated=4)
        ei = wl.edge_index
        rng = np.random.default_rng(80 + seed)
        x = rng.standard_normal((n, f))
        g = rng.standard_normal((n, f))
        u = rng.standard_normal((n, f))
        ew = rng.uniform(0.2, 2.0, size=e)
        for reduce, w in (("sum", None), ("sum", ew), ("mean", None), ("mean", ew)):
            gx, _ = o.aggregate_backward(ei, n, g, reduce, w=w)
            fd = _fd_directional(lambda z: o.aggregate(ei, n, z, reduce, w=w)[0], x, g, u, 1e-3)
            assert abs(np.sum(gx * u) - fd) <= 1e-9 * (1 + abs(fd)), (reduce, w is None)
        for selfl in (0, 1):
            gx, _ = o.gcn_aggregate_backward(ei, n, g, ew, selfl, 1.5)
            fd = _fd_directional(lambda z: o.gcn_aggregate(ei, n, z, ew, selfl, 1.5)[0], x, g, u, 1e-3)
            assert abs(np.sum(gx * u) - fd) <= 1e-9 * (1 + abs(fd)), ("gcn", selfl)
        xm = x.astype(np.float32).astype(np.float64)
        for w in (None, ew.astype(np.float32)):
            _, arg = o.max_argmax(ei, n, xm, w)
            gx, _ = o.max_backward(ei, n, arg, g, None if w is None else w.astype(np.float64))
            fd = _fd_directional(lambda z: o.max_argmax(ei, n, z, w)[0], xm, g, u, 1e-7)
            assert abs(np.sum(gx * u) - fd) <= 1e-5 * (1 + abs(fd)), ("max", w is None)


def test_backward_finite_differences():
    pin_backward_finite_differences(oracle.default)


def pin_backward_dense_transpose(o):
    """grad_x = M^T grad_out with M the numpy dense aggregation matrix."""
    for seed in range(4):
        n = [1, 7, 25, 60][seed]
        e = [3, 20, 150, 400][seed]
        wl = gg.random_edge_case_graph(n, e, 4, 90 + seed, hub=0 if n > 2 else -1,
                                       isolated=min(2, n - 1))
        ei = wl.edge_index
        g = np.random.default_rng(seed).standard_normal((n, 4))
        ew = np.random.default_rng(seed + 1).uniform(0.1, 3.0, size=e)
        m = oracle.dense_adjacency(ei, n, ew)
        gx, _ = o.aggregate_backward(ei, n, g, "sum", w=ew)
        np.testing.assert_allclose(gx, m.T @ g, rtol=1e-12, atol=1e-12)
        cnt = oracle.dense_adjacency(ei, n, None).sum(axis=1)
        mm = m / np.maximum(cnt, 1)[:, None]
        gx, _ = o.aggregate_backward(ei, n, g, "mean", w=ew)
        np.testing.assert_allclose(gx, mm.T @ g, rtol=1e-12, atol=1e-12)
        a_hat = oracle.dense_gcn_matrix(ei, n, ew, 1, 1.0)
        gx, _ = o.gcn_aggregate_backward(ei, n, g, ew, 1, 1.0)
        np.testing.assert_allclose(gx, a_hat.T @ g, rtol=1e-12, atol=1e-12)


def test_backward_dense_transpose():
    pin_backward_dense_transpose(oracle.default)


def pin_max_argmax_first_of_ties(o):
    """Ties keep the first edge in original order; the argmax points at an
    edge into the row whose product equals the maximum; empty rows give -1."""
    ei = np.array([[1, 2, 3, 0], [0, 0, 0, 4]])
    x = np.array([[9.0], [2.0], [5.0], [5.0], [0.0]])
    out, arg = o.max_argmax(ei, 5, x)
    assert arg[0, 0] == 1 and out[0, 0] == 5.0           # edges 1 and 2 tie at 5: the first wins
    assert arg[4, 0] == 3 and out[4, 0] == 9.0
    assert np.all(arg[1:4] == -1) and np.all(out[1:4] == 0.0)
    g = np.array([[1.0], [0.0], [0.0], [0.0], [2.0]])
    gx, _ = o.max_backward(ei, 5, arg, g)
    np.testing.assert_array_equal(gx[:, 0], [2.0, 0.0, 1.0, 0.0, 0.0])


def test_max_argmax_first_of_ties():
    pin_max_argmax_first_of_ties(oracle.default)


# ---------------------------------------------------------------------------
# Dot-product (Transformer-style) attention
# ---------------------------------------------------------------------------
def pin_dot_star(o):
    g = _golden("dot_star.json")
    ei = np.array(g["edge_index"], dtype=np.int64)
    q = np.zeros((4, 2))
    q[0] = g["q0"]
    k = np.zeros((4, 2))
    for s, m in zip((1, 2, 3), g["key_logs"]):
        k[s, 0] = 2.0 * math.log(m)
    v = np.array(g["v"])
    out, alpha, _ = o.dot_softmax(ei, 4, q, k, v, g["heads"], g["channels"], g["scale"])
    np.testing.assert_allclose(alpha[:, 0], g["alpha"], rtol=0, atol=g["abs_tol"])
    np.testing.assert_allclose(out[0], g["out0"], rtol=0, atol=g["abs_tol"])
    np.testing.assert_array_equal(out[1:], 0.0)


def test_dot_star():
    pin_dot_star(oracle.default)


def pin_dot_limits(o):
    """q = 0 makes every logit 0, so the result is the mean of the value rows
    over in-edges (the dense row-normalised adjacency times v); a single
    in-edge gives its source's value row with weight 1; weights sum to 1 per
    (target, head); shifting every key of a head by one vector changes each
    target's logits by a constant and leaves the result unchanged; heads
    are independent."""
    n, e, h, c = 50, 400, 3, 4
    wl = gg.random_edge_case_graph(n, e, h * c, 71, hub=2, isolated=4)
    ei = wl.edge_index
    rng = np.random.default_rng(71)
    q = rng.standard_normal((n, h * c))
    k = rng.standard_normal((n, h * c))
    v = rng.standard_normal((n, h * c))
    out, _, _ = o.dot_softmax(ei, n, np.zeros_like(q), k, v, h, c)
    cnt = oracle.dense_adjacency(ei, n, None)
    deg = cnt.sum(axis=1)
    mean = np.where(deg[:, None] > 0, (cnt @ v) / np.maximum(deg, 1)[:, None], 0.0)
    np.testing.assert_allclose(out, mean, rtol=1e-12, atol=1e-12)
    out, alpha, _ = o.dot_softmax(ei, n, q, k, v, h, c)
    sums = np.zeros((n, h))
    np.add.at(sums, ei[1], alpha)
    np.testing.assert_allclose(sums[deg > 0], 1.0, rtol=1e-13)
    shift = np.tile(rng.standard_normal(c), h)
    out2, _, _ = o.dot_softmax(ei, n, q, k + shift[None, :], v, h, c)
    np.testing.assert_allclose(out2, out, rtol=1e-10, atol=1e-12)
    one = np.array([[3, 7], [5, 9]])       # 3 -> 5, 7 -> 9
    out1, al1, _ = o.dot_softmax(one, 10, q[:10], k[:10], v[:10], h, c)
    np.testing.assert_allclose(out1[5], v[3], rtol=1e-15)
    np.testing.assert_allclose(al1, 1.0, rtol=1e-15)
    # head 1 alone: the same numbers as a one-head problem on its columns
    cols = slice(c, 2 * c)
    out_h, al_h, _ = o.dot_softmax(ei, n, q[:, cols], k[:, cols], v[:, cols], 1, c)
    np.testing.assert_allclose(out[:, cols], out_h, rtol=1e-13, atol=1e-13)
    np.testing.assert_allclose(alpha[:, 1], al_h[:, 0], rtol=1e-13)


def test_dot_limits():
    pin_dot_limits(oracle.default)


def test_dot_rows_match_full():
    n, e, h, c = 80, 900, 2, 8
    wl = gg.random_edge_case_graph(n, e, h * c, 72, hub=1, isolated=6)
    rng = np.random.default_rng(72)
    q, k, v = (rng.standard_normal((n, h * c)) for _ in range(3))
    out, alpha, ab = oracle.dot_softmax(wl.edge_index, n, q, k, v, h, c, 0.3)
    csr = oracle.build_csr(wl.edge_index, n)
    rows = np.arange(n)
    out_r, alpha_r, ab_r = oracle.dot_softmax_rows(csr, n, q, k, v, h, c, 0.3, rows)
    np.testing.assert_allclose(out_r, out, rtol=1e-13, atol=1e-14)
    np.testing.assert_allclose(ab_r, ab, rtol=1e-13, atol=1e-14)
    np.testing.assert_allclose(alpha_r, alpha[csr[2]], rtol=1e-13)


# ---------------------------------------------------------------------------
# Multi-hop propagation (APPNP / SGC)
# ---------------------------------------------------------------------------
def pin_appnp_hand_example(o):
    """Path 0-1-2 with implicit self-loops: d = (2, 3, 2), so Ahat has 1/2 at
    the ends of the diagonal, 1/3 in the middle and 1/sqrt(6) off it.  Two
    APPNP steps from x0 = I with alpha = 0.1 give 0.81 Ahat^2 + 0.09 Ahat + 0.1 I;
    entry (0, 0) is 0.81 (1/4 + 1/6) + 0.09 / 2 + 0.1 = 0.4825 and entry (0, 2)
    is 0.81 / 6 = 0.135."""
    ei = np.array([[0, 1, 1, 2], [1, 0, 2, 1]])
    out, _ = o.appnp(ei, 3, np.eye(3), 2, 0.1, add_self_loops=1)
    assert abs(out[0, 0] - 0.4825) < 1e-15
    assert abs(out[0, 2] - 0.135) < 1e-15
    assert abs(out[1, 1] - (0.81 * (1 / 6 + 1 / 9 + 1 / 6) + 0.09 / 3 + 0.1)) < 1e-15
    assert abs(out[0, 1] - (0.81 * (1 / (2 * math.sqrt(6)) + 1 / (3 * math.sqrt(6)))
                            + 0.09 / math.sqrt(6))) < 1e-15


def test_appnp_hand_example():
    pin_appnp_hand_example(oracle.default)


def pin_appnp_dense_closed_form(o):
    """h_K = ((1-a) Ahat)^K x0 + a * sum_{j<K} ((1-a) Ahat)^j x0, with Ahat the
    numpy dense GCN matrix (an independent route); SGC is a = 0."""
    for seed in range(5):
        n = [1, 6, 20, 40, 64][seed]
        e = [2, 14, 90, 160, 0][seed]
        wl = gg.random_edge_case_graph(n, e, 5, 40 + seed, hub=0 if n > 2 else -1,
                                       isolated=min(2, n - 1))
        ew = np.random.default_rng(seed).uniform(0.2, 2.0, size=e)
        xd = wl.x.astype(np.float64)
        for selfl, alpha, k in ((1, 0.1, 4), (0, 0.25, 3), (1, 0.0, 3), (1, 1.0, 2), (0, 0.5, 0)):
            a_hat = oracle.dense_gcn_matrix(wl.edge_index, n, ew, selfl, 1.0)
            m = (1.0 - alpha) * a_hat
            ref = np.linalg.matrix_power(m, k) @ xd
            for j in range(k):
                ref = ref + alpha * (np.linalg.matrix_power(m, j) @ xd)
            out, _ = o.appnp(wl.edge_index, n, wl.x, k, alpha, ew, add_self_loops=selfl, fill=1.0)
            np.testing.assert_allclose(out, ref, rtol=1e-12, atol=1e-12)


def test_appnp_dense_closed_form():
    pin_appnp_dense_closed_form(oracle.default)


def pin_appnp_limits(o):
    """K = 0 and alpha = 1 return x0; many steps reach the personalised
    PageRank fixed point alpha (I - (1 - alpha) Ahat)^-1 x0 of APPNP; on a
    symmetric graph with self-loops x0 = sqrt(d) is a fixed point of every
    step (Ahat sqrt(d) = sqrt(d)); the error scale equals the value when all
    weights and features are non-negative."""
    ei = _undirected_random(30, 70, 3)
    x0 = np.random.default_rng(3).standard_normal((30, 4))
    for k, alpha in ((0, 0.3), (5, 1.0)):
        out, _ = o.appnp(ei, 30, x0, k, alpha, add_self_loops=1)
        np.testing.assert_array_equal(out, x0)
    alpha = 0.2
    out, _ = o.appnp(ei, 30, x0, 300, alpha, add_self_loops=1)
    a_hat = oracle.dense_gcn_matrix(ei, 30, None, 1, 1.0)
    ppr = alpha * np.linalg.solve(np.eye(30) - (1 - alpha) * a_hat, x0)
    np.testing.assert_allclose(out, ppr, rtol=1e-10, atol=1e-12)
    d = np.bincount(ei[1], minlength=30) + 1.0
    sq = np.sqrt(d)[:, None] * np.array([[1.0, -2.0]])
    out, _ = o.appnp(ei, 30, sq, 6, 0.15, add_self_loops=1)
    np.testing.assert_allclose(out, sq, rtol=1e-12)
    pos = np.abs(x0)
    out, ab = o.appnp(ei, 30, pos, 4, 0.1, add_self_loops=1)
    np.testing.assert_allclose(ab, out, rtol=1e-14)


def test_appnp_limits():
    pin_appnp_limits(oracle.default)


# ---------------------------------------------------------------------------
# Backward of the GAT edge softmax
# ---------------------------------------------------------------------------
def pin_gat_backward_finite_differences(o):
    """<grad, u> equals the central difference of <grad_out, forward> along u
    for each of x, a_src and a_dst, the forward being the independent
    forward oracle (edge_softmax)."""
    for seed in range(3):
        n, e, h, c = [(30, 220, 2, 3), (45, 400, 1, 5), (20, 90, 4, 2)][seed]
        f = h * c
        wl = gg.random_edge_case_graph(n, e, f, 150 + seed, hub=1, isolated=3)
        ei = wl.edge_index
        rng = np.random.default_rng(150 + seed)
        x = rng.standard_normal((n, f))
        a_s, a_d = rng.standard_normal(f), rng.standard_normal(f)
        g = rng.standard_normal((n, f))
        gx, gs, gd, _ = o.edge_softmax_backward(ei, n, x, h, c, a_s, a_d, 0.2, g)

        def loss(xx, aa, bb):
            out, _, _ = oracle.edge_softmax(ei, n, xx, h, c, aa, bb, 0.2)
            return float(np.sum(out * g))
        eps = 1e-6
        ux, ua = rng.standard_normal((n, f)), rng.standard_normal(f)
        fd = (loss(x + eps * ux, a_s, a_d) - loss(x - eps * ux, a_s, a_d)) / (2 * eps)
        assert abs(np.sum(gx * ux) - fd) <= 1e-6 * (1 + abs(fd)), ("x", seed)
        fd = (loss(x, a_s + eps * ua, a_d) - loss(x, a_s - eps * ua, a_d)) / (2 * eps)
        assert abs(np.sum(gs * ua) - fd) <= 1e-6 * (1 + abs(fd)), ("a_src", seed)
        fd = (loss(x, a_s, a_d + eps * ua) - loss(x, a_s, a_d - eps * ua)) / (2 * eps)
        assert abs(np.sum(gd * ua) - fd) <= 1e-6 * (1 + abs(fd)), ("a_dst", seed)


def test_gat_backward_finite_differences():
    pin_gat_backward_finite_differences(oracle.default)


def pin_gat_backward_limits(o):
    """Zero attention vectors make every weight 1/in-degree, so the gradient
    with respect to x is the mean aggregation's backward (and its scale the
    mean backward's scale); a single in-edge per target has weight 1 whatever
    the logits, so the softmax passes no gradient to a_src or a_dst and x's
    gradient is grad_out routed back along the edge."""
    n, e, h, c = 40, 300, 2, 4
    wl = gg.random_edge_case_graph(n, e, h * c, 160, hub=2, isolated=4)
    ei = wl.edge_index
    rng = np.random.default_rng(160)
    x, g = rng.standard_normal((n, h * c)), rng.standard_normal((n, h * c))
    z = np.zeros(h * c)
    gx, _, _, (ax, _, _) = o.edge_softmax_backward(ei, n, x, h, c, z, z, 0.2, g)
    mb, mab = oracle.aggregate_backward(ei, n, g, "mean")
    np.testing.assert_allclose(gx, mb, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(ax, mab, rtol=1e-12, atol=1e-12)
    one = np.array([[3, 7, 1], [5, 9, 2]])        # 3 -> 5, 7 -> 9, 1 -> 2
    a_s, a_d = rng.standard_normal(h * c), rng.standard_normal(h * c)
    gx, gs, gd, _ = o.edge_softmax_backward(one, 10, x[:10], h, c, a_s, a_d, 0.2, g[:10])
    np.testing.assert_allclose(gs, 0.0, atol=1e-13)
    np.testing.assert_allclose(gd, 0.0, atol=1e-13)
    want = np.zeros((10, h * c))
    for s_, t_ in zip(one[0], one[1]):
        want[s_] += g[t_]
    np.testing.assert_allclose(gx, want, rtol=1e-13, atol=1e-13)


def test_gat_backward_limits():
    pin_gat_backward_limits(oracle.default)


def pin_dot_backward_finite_differences(o):
    """<grad, u> equals the central difference of <grad_out, forward> along u
    for each of q, k and v (the forward oracle dot_softmax)."""
    for seed in range(3):
        n, e, h, c = [(30, 220, 2, 3), (40, 350, 1, 4), (20, 90, 4, 2)][seed]
        f = h * c
        wl = gg.random_edge_case_graph(n, e, f, 170 + seed, hub=1, isolated=3)
        ei = wl.edge_index
        rng = np.random.default_rng(170 + seed)
        q, k, v, g = (rng.standard_normal((n, f)) for _ in range(4))
        gq, gk, gv, _ = o.dot_softmax_backward(ei, n, q, k, v, h, c, 0.4, g)

        def loss(qq, kk, vv):
            out, _, _ = oracle.dot_softmax(ei, n, qq, kk, vv, h, c, 0.4)
            return float(np.sum(out * g))
        eps = 1e-6
        for name, grad, shift in (("q", gq, (1, 0, 0)), ("k", gk, (0, 1, 0)), ("v", gv, (0, 0, 1))):
            u = rng.standard_normal((n, f))
            plus = [t + eps * u * sh for t, sh in zip((q, k, v), shift)]
            minus = [t - eps * u * sh for t, sh in zip((q, k, v), shift)]
            fd = (loss(*plus) - loss(*minus)) / (2 * eps)
            assert abs(np.sum(grad * u) - fd) <= 1e-6 * (1 + abs(fd)), (name, seed)


def test_dot_backward_finite_differences():
    pin_dot_backward_finite_differences(oracle.default)


def pin_dot_backward_limits(o):
    """q = 0 makes every weight 1/in-degree, so v's gradient is the mean
    aggregation's backward; a single in-edge per target has weight 1, so q
    and k receive no gradient and v's gradient is grad_out routed back."""
    n, e, h, c = 40, 300, 2, 4
    wl = gg.random_edge_case_graph(n, e, h * c, 180, hub=2, isolated=4)
    ei = wl.edge_index
    rng = np.random.default_rng(180)
    k, v, g = (rng.standard_normal((n, h * c)) for _ in range(3))
    _, _, gv, (_, _, av) = o.dot_softmax_backward(ei, n, np.zeros((n, h * c)), k, v, h, c, 0.5, g)
    mb, mab = oracle.aggregate_backward(ei, n, g, "mean")
    np.testing.assert_allclose(gv, mb, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(av, mab, rtol=1e-12, atol=1e-12)
    one = np.array([[3, 7, 1], [5, 9, 2]])
    q = rng.standard_normal((10, h * c))
    gq, gk, gv, _ = o.dot_softmax_backward(one, 10, q, k[:10], v[:10], h, c, 0.5, g[:10])
    np.testing.assert_allclose(gq, 0.0, atol=1e-13)
    np.testing.assert_allclose(gk, 0.0, atol=1e-13)
    want = np.zeros((10, h * c))
    for s_, t_ in zip(one[0], one[1]):
        want[s_] += g[t_]
    np.testing.assert_allclose(gv, want, rtol=1e-13, atol=1e-13)


def test_dot_backward_limits():
    pin_dot_backward_limits(oracle.default)


# ---------------------------------------------------------------------------
# Error scales: every tolerance is a multiple of the oracle's absout, so it is
# pinned to an independent numpy form -- |M| |X| with dense matrices, and for
# attention the weights re-derived densely from their definition
# ---------------------------------------------------------------------------
def _np_softmax_weights(logit, dst, n, heads):
    """alpha[e, h] = exp(l[e, h]) / sum over the edges into dst_e of exp(l[., h])."""
    alpha = np.zeros_like(logit)
    for t in range(n):
        m = dst == t
        if m.any():
            ex = np.exp(logit[m] - logit[m].max(axis=0))
            alpha[m] = ex / ex.sum(axis=0)
    return alpha


def _np_attention_scale(alpha, ei, n, vals, heads, channels):
    """sum over the edges into t of alpha[e, h] |vals[src_e, h, :]|."""
    ab = np.zeros((n, heads * channels))
    for e in range(ei.shape[1]):
        s, t = ei[0, e], ei[1, e]
        ab[t] += np.repeat(alpha[e], channels) * np.abs(vals[s])
    return ab


def pin_error_scales(o):
    for seed in range(3):
        n, e, h, c = [(30, 200, 2, 3), (45, 380, 1, 4), (12, 60, 3, 2)][seed]
        f = h * c
        wl = gg.random_edge_case_graph(n, e, f, 140 + seed, hub=1, isolated=3)
        ei = wl.edge_index
        rng = np.random.default_rng(140 + seed)
        x = rng.standard_normal((n, f))
        w = rng.uniform(-2.0, 2.0, e)
        wpos = np.abs(w) + 0.1
        ax = np.abs(x)
        mabs = oracle.dense_adjacency(ei, n, np.abs(w))
        cnt = oracle.dense_adjacency(ei, n, None).sum(axis=1)
        for reduce in ("sum", "mean", "max"):
            _, ab = o.aggregate(ei, n, x, reduce, w=w)
            want = mabs @ ax
            if reduce == "mean":
                want = want / np.maximum(cnt, 1)[:, None]
            np.testing.assert_allclose(ab, want, rtol=1e-12, atol=1e-12)
        csr = o.build_csr(ei, n)
        rows = np.array([0, n - 1, 5, 2], np.int64)
        _, ab = o.aggregate_rows(csr, n, x, "mean", rows, w=w)
        np.testing.assert_allclose(ab, (mabs @ ax / np.maximum(cnt, 1)[:, None])[rows],
                                   rtol=1e-12, atol=1e-12)
        for selfl in (0, 1):
            _, ab = o.gcn_aggregate(ei, n, x, wpos, selfl, 1.5)
            want = oracle.dense_gcn_matrix(ei, n, wpos, selfl, 1.5) @ ax
            np.testing.assert_allclose(ab, want, rtol=1e-12, atol=1e-12)
        # additive attention: weights from the definition, then sum alpha |x|
        a_s, a_d = rng.standard_normal(f), rng.standard_normal(f)
        xs = x.reshape(n, h, c)
        s_src = np.einsum("nhc,hc->nh", xs, a_s.reshape(h, c))
        s_dst = np.einsum("nhc,hc->nh", xs, a_d.reshape(h, c))
        z = s_src[ei[0]] + s_dst[ei[1]]
        alpha = _np_softmax_weights(np.where(z > 0, z, 0.2 * z), ei[1], n, h)
        want = _np_attention_scale(alpha, ei, n, x, h, c)
        _, _, ab = o.edge_softmax(ei, n, x, h, c, a_s, a_d, 0.2)
        np.testing.assert_allclose(ab, want, rtol=1e-11, atol=1e-12)
        _, _, ab = o.edge_softmax_rows(csr, n, x, h, c, a_s, a_d, 0.2, rows)
        np.testing.assert_allclose(ab, want[rows], rtol=1e-11, atol=1e-12)
        # dot-product attention
        q, k, v = (rng.standard_normal((n, f)) for _ in range(3))
        lg = 0.3 * np.einsum("ehc,ehc->eh", q[ei[1]].reshape(-1, h, c), k[ei[0]].reshape(-1, h, c))
        alpha = _np_softmax_weights(lg, ei[1], n, h)
        want = _np_attention_scale(alpha, ei, n, v, h, c)
        _, _, ab = o.dot_softmax(ei, n, q, k, v, h, c, 0.3)
        np.testing.assert_allclose(ab, want, rtol=1e-11, atol=1e-12)
        _, _, ab = o.dot_softmax_rows(csr, n, q, k, v, h, c, 0.3, rows)
        np.testing.assert_allclose(ab, want[rows], rtol=1e-11, atol=1e-12)
        # pooling: sum of |x| per graph (divided by the count for mean)
        batch = np.sort(rng.integers(0, 4, n))
        pool_abs = np.zeros((5, f))
        np.add.at(pool_abs, batch, ax)
        counts = np.bincount(batch, minlength=5)
        for reduce in ("sum", "mean", "max"):
            _, ab = o.segment_pool(x, batch, 5, reduce)
            want = pool_abs / np.maximum(counts, 1)[:, None] if reduce == "mean" else pool_abs
            np.testing.assert_allclose(ab, want, rtol=1e-12, atol=1e-12)
        # backward: |M|^T |grad_out|
        g = rng.standard_normal((n, f))
        _, ab = o.aggregate_backward(ei, n, g, "sum", w=w)
        np.testing.assert_allclose(ab, mabs.T @ np.abs(g), rtol=1e-12, atol=1e-12)
        _, ab = o.aggregate_backward(ei, n, g, "mean", w=w)
        np.testing.assert_allclose(ab, (mabs / np.maximum(cnt, 1)[:, None]).T @ np.abs(g),
                                   rtol=1e-12, atol=1e-12)
        _, ab = o.gcn_aggregate_backward(ei, n, g, wpos, 1, 1.5)
        np.testing.assert_allclose(ab, oracle.dense_gcn_matrix(ei, n, wpos, 1, 1.5).T @ np.abs(g),
                                   rtol=1e-12, atol=1e-12)
        _, arg = o.max_argmax(ei, n, x.astype(np.float32), w.astype(np.float32))
        want = np.zeros((n, f))
        for t in range(n):
            for j in range(f):
                if arg[t, j] >= 0:
                    want[ei[0, arg[t, j]], j] += abs(w[arg[t, j]] * g[t, j])
        _, ab = o.max_backward(ei, n, arg, g, w)
        np.testing.assert_allclose(ab, want, rtol=1e-12, atol=1e-12)


def test_error_scales():
    pin_error_scales(oracle.default)


# ---------------------------------------------------------------------------
# Planted mistakes: each one must trip at least one pin
# ---------------------------------------------------------------------------
PLANTS = {
    "UNSTABLE_CSR": [pin_csr_is_stable_grouping],
    "DROP_SELF_LOOP_DEGREE": [pin_gcn_p4, pin_gcn_sqrt_degree_eigenvector],
    "OUT_DEGREE": [pin_gcn_directed],
    "SWAP_DIRECTION": [pin_gcn_directed, pin_ones_give_in_degree],
    "MAX_FROM_ZERO": [pin_max_brute_force],
    "MEAN_PLUS_ONE": [pin_ones_give_in_degree, pin_softmax_normalised_and_mean_limit],
    "NO_LEAKY": [pin_star_softmax],
    "POOL_SKIP_LAST": [pin_pool_counts],
    "APPNP_TELEPORT_FROM_H": [pin_appnp_hand_example, pin_appnp_dense_closed_form],
    "DOT_KEY_AT_TARGET": [pin_dot_star],
    "BACKWARD_NO_TRANSPOSE": [pin_backward_finite_differences, pin_backward_dense_transpose],
    "SCALE_DOUBLED": [pin_error_scales, pin_gat_backward_limits, pin_dot_backward_limits],
    "BWD_NO_SOFTMAX_JACOBIAN": [pin_gat_backward_finite_differences,
                                pin_dot_backward_finite_differences],
}


@pytest.mark.parametrize("plant", sorted(PLANTS))
def test_planted_mistakes_are_caught(plant):
    bad = oracle.planted(plant)
    for pin in PLANTS[plant]:
        with pytest.raises((AssertionError, oracle.OracleError)):
            pin(bad)


def test_all_cores_rows_equal_single_thread():
    """The OpenMP CPU baseline calls the same row functions on blocks of rows
    in parallel: its results equal the single-threaded oracle's exactly."""
    n = 2000
    wl = gg.random_edge_case_graph(n, 40000, 16, 9, hub=2, isolated=30)
    csr = oracle.build_csr(wl.edge_index, n)
    rows = np.arange(n, dtype=np.int64)
    nrm = oracle.gcn_norm(wl.edge_index, n, None, 1, 1.0)
    a, ab = oracle.aggregate_rows(csr, n, wl.x_bf16, "sum", rows, w=nrm["w_norm"],
                                  self_w=nrm["self_w"])
    b, bb = oracle.omp_rows.aggregate_all(csr, n, wl.x_bf16, "sum", w=nrm["w_norm"],
                                          self_w=nrm["self_w"])
    np.testing.assert_array_equal(a, b)
    np.testing.assert_array_equal(ab, bb)
    rng = np.random.default_rng(9)
    a_s, a_d = rng.standard_normal(16), rng.standard_normal(16)
    a, _, ab = oracle.edge_softmax_rows(csr, n, wl.x_bf16, 2, 8, a_s, a_d, 0.2, rows)
    b, bb = oracle.omp_rows.edge_softmax_all(csr, n, wl.x_bf16, 2, 8, a_s, a_d, 0.2)
    np.testing.assert_array_equal(a, b)
    np.testing.assert_array_equal(ab, bb)
    assert oracle.omp_rows.threads() >= 1
