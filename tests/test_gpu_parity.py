"""CUDA path vs fp64 oracle, element by element, through the C ABI.

Small and mid-size seeded graphs span several tiles of every kernel and a
ragged tail, plus the degenerate cases (no edges, one node, isolated nodes,
duplicate edges, self-loops, a single hub taking half of all edges, feature
counts that are not a multiple of the vector width).  The four smaller
workloads run at full size.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2101_11552_gb300 import graphgen as gg
from paper_2101_11552_gb300 import tfg
from _helpers import (KAPPA_GAT, TOL_F32, assert_alpha_close, assert_exact_f32, assert_scaled_close,
                      csr_rows, dev, dot_logit_mag, gat_logit_mag, kappa_dot,
                      features, host_features)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_11552_gb300 import build
    build.build_library()


def gpu_csr(ei: np.ndarray, n: int):
    csr = tfg.tfg_build_csr(dev(ei), n)
    tfg.check_status(csr.status)
    return csr


def np_(t):
    return t.cpu().numpy()


# ---------------------------------------------------------------------------
# CSR build: bit-exact
# ---------------------------------------------------------------------------
CSR_CASES = [
    # (n, e, hub, isolated, seed)
    (1, 5, -1, 0, 0), (5, 0, -1, 0, 1), (2, 1, -1, 0, 2), (7, 40, 0, 2, 3),
    (1000, 30000, 3, 10, 4),          # 10-bit keys: one radix pass
    (1025, 9000, -1, 0, 5),           # 11 bits: two passes
    (70000, 250000, 12, 100, 6),      # several tiles, ragged tail
    (1_500_000, 120_000, -1, 0, 7),   # 21 bits: three passes
    (300, 8192 * 3, 5, 0, 8),         # exact multiple of the tile
]


@pytest.mark.parametrize("n,e,hub,iso,seed", CSR_CASES)
def test_csr_bit_exact(n, e, hub, iso, seed):
    wl = gg.random_edge_case_graph(n, e, 1, seed, hub=hub, isolated=iso)
    want = oracle.build_csr(wl.edge_index, n)
    got = gpu_csr(wl.edge_index, n)
    for name, g, w in zip(("rowptr", "col", "perm", "in_degree"), got[:4], want):
        assert np.array_equal(np_(g), w), name


@pytest.mark.parametrize("by_source", [False, True])
def test_csr_from_int32_edges_equals_int64(by_source):
    """tfg_build_csr32 / _by_source: the same CSR from an int32 edge list, and
    out-of-range int32 ids reported the same way."""
    n = 50_000
    wl = gg.random_edge_case_graph(n, 700_000, 1, 83, hub=4, isolated=50)
    build = tfg.tfg_build_csr_by_source if by_source else tfg.tfg_build_csr
    a = build(dev(wl.edge_index), n)
    b = build(dev(wl.edge_index.astype(np.int32)), n)
    tfg.check_status(b.status)
    for name, u, v in zip(("rowptr", "col", "perm", "in_degree"), a[:4], b[:4]):
        assert torch.equal(u, v), name
    want = oracle.build_csr(np.ascontiguousarray(wl.edge_index[::-1]) if by_source else wl.edge_index, n)
    for name, g, w in zip(("rowptr", "col", "perm", "in_degree"), b[:4], want):
        assert np.array_equal(np_(g), w), name
    bad = np.array([[0, 1, 2, 7], [1, 2, -1, 0]], dtype=np.int32)
    got = build(dev(bad), 4)
    assert int(got.status.item()) == tfg.TFG_ERR_INDEX_RANGE


def test_csr_empty_graph():
    got = tfg.tfg_build_csr(torch.zeros(2, 0, dtype=torch.int64, device="cuda"), 0)
    tfg.check_status(got.status)
    assert np_(got.rowptr).tolist() == [0]


def test_csr_out_of_range_ids_set_status():
    ei = np.array([[0, 1, 2, 7], [1, 2, -1, 0]], dtype=np.int64)   # 7 >= N, -1 < 0
    got = tfg.tfg_build_csr(dev(ei), 4)
    assert int(got.status.item()) == tfg.TFG_ERR_INDEX_RANGE
    # the clamped ids keep every write in bounds: rowptr still partitions E
    rp = np_(got.rowptr)
    assert rp[0] == 0 and rp[-1] == 4 and np.all(np.diff(rp) >= 0)


def test_csr_many_tiles_bit_exact():
    """2.5M edges over 200,000 nodes: 611 tiles in each of the two passes."""
    n = 200_000
    wl = gg.random_edge_case_graph(n, 2_500_000, 1, 78, hub=5, isolated=100)
    want = oracle.build_csr(wl.edge_index, n)
    got = gpu_csr(wl.edge_index, n)
    for name, g, w in zip(("rowptr", "col", "perm", "in_degree"), got[:4], want):
        assert np.array_equal(np_(g), w), name


# ---------------------------------------------------------------------------
# GCN normalisation
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("weighted", [False, True])
@pytest.mark.parametrize("add_self", [0, 1])
def test_gcn_norm(weighted, add_self):
    n, e = 5000, 60000
    wl = gg.random_edge_case_graph(n, e, 1, 11, hub=4, isolated=30)
    ew = np.random.default_rng(0).uniform(0.1, 2.0, e).astype(np.float32) if weighted else None
    csr = gpu_csr(wl.edge_index, n)
    dinv, w_csr = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n,
                                   dev(ew) if weighted else None, add_self, 1.0)
    ref = oracle.gcn_norm(wl.edge_index, n, ew, add_self, 1.0)
    np.testing.assert_allclose(np_(dinv), ref["dinv"], rtol=2e-6, atol=0)
    _, _, perm, _ = oracle.build_csr(wl.edge_index, n)
    np.testing.assert_allclose(np_(w_csr), ref["w_norm"][perm], rtol=4e-6, atol=0)


# ---------------------------------------------------------------------------
# Aggregation: sum / mean / max, fp32 and bf16, weighted and unweighted
# ---------------------------------------------------------------------------
AGG_GRAPHS = [
    (1, 3, -1, 0),          # one node with self-loops
    (50, 0, -1, 0),         # no edges
    (300, 4000, 7, 20),     # a hub with ~2000 in-edges (CTA-cooperative path)
    (4000, 30000, -1, 50),
    (2000, 60000, 1, 0),    # hub with ~30000 in-edges
]


@pytest.mark.parametrize("reduce", ["sum", "mean", "max"])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("weighted", [False, True])
@pytest.mark.parametrize("f", [1, 3, 8, 20, 64, 128, 136, 256])
def test_aggregate(reduce, dtype, weighted, f):
    for gi, (n, e, hub, iso) in enumerate(AGG_GRAPHS):
        wl = gg.random_edge_case_graph(n, e, f, 100 + gi + f, hub=hub, isolated=iso)
        ocsr = oracle.build_csr(wl.edge_index, n)
        w_coo = (np.random.default_rng(gi).uniform(-1.5, 1.5, e).astype(np.float32)
                 if weighted else None)
        csr = gpu_csr(wl.edge_index, n)
        w_csr = dev(w_coo[ocsr[2]]) if weighted else None
        x = features(wl, dtype)
        fn = {"sum": tfg.tfg_aggregate_sum, "mean": tfg.tfg_aggregate_mean,
              "max": tfg.tfg_aggregate_max}[reduce]
        got = np_(fn(csr.rowptr, csr.col, x, w_csr))
        ref, scale = oracle.aggregate(wl.edge_index, n, host_features(wl, dtype), reduce, w=w_coo)
        what = f"{reduce} {dtype} w={weighted} F={f} graph={gi}"
        if reduce == "max":
            assert_exact_f32(got, ref, what)
        else:
            assert_scaled_close(got, ref, scale, TOL_F32, what)


@pytest.mark.parametrize("f", [8, 64, 128])
@pytest.mark.parametrize("n,e,hub", [(1000, 31999, -1), (1000, 32000, -1), (700, 35000, 2),
                                     (64, 32 * 64, 0)])
def test_fp32_sums_on_both_sides_of_the_degree_split(n, e, hub, f):
    """fp32 sums in 16-byte slices run the merge-path kernel below a mean
    in-degree of 32 and the row-per-warp kernel from 32 up (each kernel
    reads E on the device); E = 32 N - 1 and E = 32 N sit on the two sides."""
    wl = gg.random_edge_case_graph(n, e, f, 300 + e % 97 + f, hub=hub, isolated=3)
    csr = gpu_csr(wl.edge_index, n)
    x = features(wl, "f32")
    for reduce, fn in (("sum", tfg.tfg_aggregate_sum), ("mean", tfg.tfg_aggregate_mean),
                       ("max", tfg.tfg_aggregate_max)):
        got = np_(fn(csr.rowptr, csr.col, x))
        ref, scale = oracle.aggregate(wl.edge_index, n, wl.x, reduce)
        what = f"{reduce} n={n} e={e} F={f}"
        if reduce == "max":
            assert_exact_f32(got, ref, what)
        else:
            assert_scaled_close(got, ref, scale, TOL_F32, what)
    for add_self in (0, 1):
        dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, add_self, 1.0,
                                   want_w_csr=False)
        got = np_(tfg.tfg_gcn_aggregate_sum(csr.rowptr, csr.col, dinv, x, None, add_self, 1.0))
        ref, scale = oracle.gcn_aggregate(wl.edge_index, n, wl.x, None, add_self, 1.0)
        assert_scaled_close(got, ref, scale, TOL_F32, f"gcn self={add_self} n={n} e={e} F={f}")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("add_self", [0, 1])
@pytest.mark.parametrize("f", [5, 64, 128])
def test_gcn_aggregate_on_the_fly(dtype, add_self, f):
    n, e = 3000, 40000
    wl = gg.random_edge_case_graph(n, e, f, 7 + f, hub=2, isolated=10)
    csr = gpu_csr(wl.edge_index, n)
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, add_self, 1.0,
                               want_w_csr=False)
    got = np_(tfg.tfg_gcn_aggregate_sum(csr.rowptr, csr.col, dinv, features(wl, dtype), None,
                                        add_self, 1.0))
    ref, scale = oracle.gcn_aggregate(wl.edge_index, n, host_features(wl, dtype), None, add_self, 1.0)
    assert_scaled_close(got, ref, scale, TOL_F32, f"gcn {dtype} self={add_self} F={f}")


@pytest.mark.parametrize("add_self", [0, 1])
def test_gcn_aggregate_weighted(add_self):
    n, e, f = 2500, 30000, 32
    wl = gg.random_edge_case_graph(n, e, f, 19, hub=0, isolated=5)
    ew = np.random.default_rng(4).uniform(0.2, 3.0, e).astype(np.float32)
    csr = gpu_csr(wl.edge_index, n)
    dinv, w_csr = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, dev(ew), add_self, 2.0)
    got = np_(tfg.tfg_gcn_aggregate_sum(csr.rowptr, csr.col, dinv, features(wl, "f32"), w_csr,
                                        add_self, 2.0))
    ref, scale = oracle.gcn_aggregate(wl.edge_index, n, wl.x, ew, add_self, 2.0)
    assert_scaled_close(got, ref, scale, TOL_F32, f"weighted gcn self={add_self}")


# ---------------------------------------------------------------------------
# Edge softmax (GAT)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("heads,channels", [(1, 1), (2, 3), (4, 4), (8, 16), (3, 48), (1, 160),
                                            (2, 8), (16, 8),
                                            # head-per-lane kernel: C of one or two 16-byte vectors
                                            (1, 4), (8, 4), (1, 8), (4, 8), (8, 8), (1, 16),
                                            (2, 16), (4, 16)])
def test_edge_softmax(heads, channels, dtype):
    n, e = 3000, 25000
    f = heads * channels
    wl = gg.random_edge_case_graph(n, e, f, 31 + f, hub=9, isolated=40)
    rng = np.random.default_rng(heads * 100 + channels)
    a_s = rng.standard_normal(f).astype(np.float32)
    a_d = rng.standard_normal(f).astype(np.float32)
    csr = gpu_csr(wl.edge_index, n)
    out, alpha = tfg.tfg_edge_softmax_aggregate(csr.rowptr, csr.col, features(wl, dtype), heads,
                                                channels, dev(a_s), dev(a_d), 0.2, want_alpha=True)
    ref, ref_alpha, scale = oracle.edge_softmax(wl.edge_index, n, host_features(wl, dtype), heads,
                                                channels, a_s, a_d, 0.2)
    # the oracle reads the same bf16 values, so fp32 arithmetic is the only error
    assert_scaled_close(np_(out), ref, scale, TOL_F32, f"softmax {dtype} H={heads} C={channels}")
    rowptr, col, perm, _ = oracle.build_csr(wl.edge_index, n)
    row = csr_rows(rowptr)
    lam = gat_logit_mag(oracle.widen(host_features(wl, dtype)), col, row, heads, channels, a_s, a_d)
    assert_alpha_close(np_(alpha), ref_alpha[perm], lam, row, KAPPA_GAT,
                       f"alpha {dtype} H={heads} C={channels}")


# ---------------------------------------------------------------------------
# Segment pooling
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("reduce", ["sum", "mean", "max"])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("f", [1, 7, 128, 264])
def test_segment_pool(reduce, dtype, f):
    rng = np.random.default_rng(f)
    g = 300
    sizes = rng.integers(0, 40, size=g)
    sizes[[0, 17, 299]] = 0                    # empty graphs, including the last
    sizes[5] = 3000                            # one large graph
    batch = np.repeat(np.arange(g), sizes).astype(np.int64)
    n = batch.size
    wl = gg.Workload("pool", n, np.zeros((2, 0), np.int64),
                     rng.standard_normal((n, f)).astype(np.float32))
    out, status = tfg.tfg_segment_pool(features(wl, dtype), dev(batch), g, reduce)
    tfg.check_status(status)
    ref, scale = oracle.segment_pool(host_features(wl, dtype), batch, g, reduce)
    if reduce == "max":
        assert_exact_f32(np_(out), ref, f"pool max {dtype}")
    else:
        assert_scaled_close(np_(out), ref, scale, TOL_F32, f"pool {reduce} {dtype} F={f}")


@pytest.mark.parametrize("reduce", ["sum", "mean", "max"])
def test_segment_pool_large_graphs_cluster_path(reduce):
    """Graphs of thousands of nodes: several CTAs per graph combine through
    distributed shared memory."""
    rng = np.random.default_rng(3)
    sizes = rng.integers(6000, 12000, size=9)
    sizes[4] = 0
    batch = np.repeat(np.arange(9), sizes).astype(np.int64)
    n, f = batch.size, 128
    x = rng.standard_normal((n, f)).astype(np.float32)
    out, status = tfg.tfg_segment_pool(dev(x), dev(batch), 9, reduce)
    tfg.check_status(status)
    ref, scale = oracle.segment_pool(x, batch, 9, reduce)
    if reduce == "max":
        assert_exact_f32(np_(out), ref, "cluster pool max")
    else:
        assert_scaled_close(np_(out), ref, scale, TOL_F32, f"cluster pool {reduce}")


def test_segment_pool_bad_batch_sets_status():
    x = torch.ones(6, 4, device="cuda")
    _, status = tfg.tfg_segment_pool(x, dev(np.array([0, 0, 2, 1, 1, 2])), 3, "sum")
    assert int(status.item()) == tfg.TFG_ERR_UNSORTED
    _, status = tfg.tfg_segment_pool(x, dev(np.array([0, 0, 1, 1, 2, 3])), 3, "sum")
    assert int(status.item()) == tfg.TFG_ERR_INDEX_RANGE


# ---------------------------------------------------------------------------
# The four smaller workloads at full size
# ---------------------------------------------------------------------------
def test_er2708_gcn_full():
    wl = gg.make_er_2708()
    n = wl.num_nodes
    csr = gpu_csr(wl.edge_index, n)
    want = oracle.build_csr(wl.edge_index, n)
    assert all(np.array_equal(np_(a), b) for a, b in zip(csr[:4], want))
    dinv, w_csr = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, 0, 1.0)
    got = np_(tfg.tfg_aggregate_sum(csr.rowptr, csr.col, dev(wl.x), w_csr))
    ref, scale = oracle.gcn_aggregate(wl.edge_index, n, wl.x, None, 0)
    assert_scaled_close(got, ref, scale, TOL_F32, "er2708")
    got2 = np_(tfg.tfg_gcn_aggregate_sum(csr.rowptr, csr.col, dinv, dev(wl.x)))
    assert_scaled_close(got2, ref, scale, TOL_F32, "er2708 on the fly")


def test_ba19717_sum_mean_max_full():
    wl = gg.make_ba_19717()
    n = wl.num_nodes
    csr = gpu_csr(wl.edge_index, n)
    x = dev(wl.x)
    for reduce, fn in (("sum", tfg.tfg_aggregate_sum), ("mean", tfg.tfg_aggregate_mean),
                       ("max", tfg.tfg_aggregate_max)):
        got = np_(fn(csr.rowptr, csr.col, x))
        ref, scale = oracle.aggregate(wl.edge_index, n, wl.x, reduce)
        if reduce == "max":
            assert_exact_f32(got, ref, "ba19717 max")
        else:
            assert_scaled_close(got, ref, scale, TOL_F32, f"ba19717 {reduce}")


def test_gat169343_edge_softmax_full():
    wl = gg.make_gat_169343()
    n = wl.num_nodes
    csr = gpu_csr(wl.edge_index, n)
    out, alpha = tfg.tfg_edge_softmax_aggregate(csr.rowptr, csr.col, dev(wl.x), wl.heads,
                                                wl.channels, dev(wl.a_src), dev(wl.a_dst),
                                                wl.negative_slope, want_alpha=True)
    ref, ref_alpha, scale = oracle.edge_softmax(wl.edge_index, n, wl.x, wl.heads, wl.channels,
                                                wl.a_src, wl.a_dst, wl.negative_slope)
    assert_scaled_close(np_(out), ref, scale, TOL_F32, "gat169343 out")
    perm = np_(csr.perm)
    row = csr_rows(np_(csr.rowptr))
    lam = gat_logit_mag(wl.x, np_(csr.col), row, wl.heads, wl.channels, wl.a_src, wl.a_dst)
    assert_alpha_close(np_(alpha), ref_alpha[perm], lam, row, KAPPA_GAT, "gat169343 alpha")
    deg = np.bincount(wl.edge_index[1], minlength=n)
    assert np.all(np_(out)[deg == 0] == 0.0)


def test_molecules_batched_gcn_then_pool_full():
    wl = gg.make_molecules_1024()
    n = wl.num_nodes
    csr = gpu_csr(wl.edge_index, n)
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, 0, 1.0, want_w_csr=False)
    h = tfg.tfg_gcn_aggregate_sum(csr.rowptr, csr.col, dinv, dev(wl.x))
    ref_h, scale = oracle.gcn_aggregate(wl.edge_index, n, wl.x, None, 0)
    assert_scaled_close(np_(h), ref_h, scale, TOL_F32, "molecules gcn")
    batch = dev(wl.batch)
    h32 = np_(h)                      # the pooling oracle reads what the GPU pooled
    for reduce in ("sum", "mean", "max"):
        out, status = tfg.tfg_segment_pool(h, batch, wl.num_graphs, reduce)
        tfg.check_status(status)
        ref, pscale = oracle.segment_pool(h32, wl.batch, wl.num_graphs, reduce)
        if reduce == "max":
            assert_exact_f32(np_(out), ref, "molecules pool max")
        else:
            assert_scaled_close(np_(out), ref, pscale, TOL_F32, f"molecules pool {reduce}")
    # batched == per graph (Section 2.1.1): graph g's rows only see graph g
    offs = np.concatenate([[0], np.cumsum(wl.graph_sizes)])
    for g in (0, 511, 1023):
        s0, s1 = offs[g], offs[g + 1]
        m = (wl.edge_index[1] >= s0) & (wl.edge_index[1] < s1)
        sub = wl.edge_index[:, m] - s0
        ref_g, _ = oracle.gcn_aggregate(sub, s1 - s0, wl.x[s0:s1], None, 0)
        np.testing.assert_allclose(h32[s0:s1], ref_g, rtol=1e-5, atol=1e-5)


def test_er2708_appnp_and_sgc_full():
    """APPNP with the settings of its paper (K = 10, alpha = 0.1) and SGC with
    K = 2 on the 2,708-node citation-sized graph (explicit self-loops)."""
    wl = gg.make_er_2708()
    n = wl.num_nodes
    csr = gpu_csr(wl.edge_index, n)
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, 0, 1.0, want_w_csr=False)
    got = np_(tfg.tfg_appnp_propagate(csr.rowptr, csr.col, dinv, dev(wl.x), 10, 0.1))
    ref, scale = oracle.appnp(wl.edge_index, n, wl.x, 10, 0.1)
    assert_scaled_close(got, ref, scale, TOL_F32, "er2708 appnp")
    got = np_(tfg.tfg_sgc_propagate(csr.rowptr, csr.col, dinv, dev(wl.x), 2))
    ref, scale = oracle.sgc(wl.edge_index, n, wl.x, 2)
    assert_scaled_close(got, ref, scale, TOL_F32, "er2708 sgc")


def test_gat169343_dot_softmax_full():
    """Transformer-style attention on the GAT workload's graph (169,343 nodes,
    1,166,243 edges, 8 heads x 16): q from the features, k and v seeded."""
    wl = gg.make_gat_169343()
    n = wl.num_nodes
    csr = gpu_csr(wl.edge_index, n)
    rng = np.random.default_rng(1303)
    k = rng.standard_normal(wl.x.shape, dtype=np.float32)
    v = rng.standard_normal(wl.x.shape, dtype=np.float32)
    out, alpha = tfg.tfg_dot_edge_softmax_aggregate(csr.rowptr, csr.col, dev(wl.x), dev(k), dev(v),
                                                    wl.heads, wl.channels, want_alpha=True)
    ref, ref_alpha, scale = oracle.dot_softmax(wl.edge_index, n, wl.x, k, v, wl.heads, wl.channels,
                                               float(np.float32(1.0 / np.sqrt(wl.channels))))
    assert_scaled_close(np_(out), ref, scale, TOL_F32, "gat169343 dot out")
    perm = np_(csr.perm)
    row = csr_rows(np_(csr.rowptr))
    lam = dot_logit_mag(wl.x, k, np_(csr.col), row, wl.heads, wl.channels,
                        float(np.float32(1.0 / np.sqrt(wl.channels))))
    assert_alpha_close(np_(alpha), ref_alpha[perm], lam, row, kappa_dot(wl.channels),
                       "gat169343 dot alpha")


def test_molecules_device_batching_and_meanmax_full():
    """The 1,024 molecule graphs batched on the device equal the generator's
    BatchGraph; the Mean-Max readout of the GCN output equals the oracle."""
    wl = gg.make_molecules_1024()
    sizes = np.asarray(wl.graph_sizes, np.int64)
    offs = np.concatenate([[0], np.cumsum(sizes)[:-1]])
    src_graph = wl.batch[wl.edge_index[0]]
    local = np.ascontiguousarray(wl.edge_index - offs[src_graph][None, :])
    ecount = np.bincount(src_graph, minlength=len(sizes)).astype(np.int64)
    bg = tfg.tfg_batch_graphs(dev(sizes), dev(ecount), dev(local), wl.num_nodes)
    tfg.check_status(bg.status)
    ei, batch, node_offsets = oracle.batch_graphs(sizes, ecount, local)
    assert np.array_equal(np_(bg.edge_index), ei) and np.array_equal(ei, wl.edge_index)
    assert np.array_equal(np_(bg.batch), batch) and np.array_equal(batch, wl.batch)
    assert np.array_equal(np_(bg.node_offsets), node_offsets)
    n = wl.num_nodes
    csr = gpu_csr(wl.edge_index, n)
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, 0, 1.0, want_w_csr=False)
    h = tfg.tfg_gcn_aggregate_sum(csr.rowptr, csr.col, dinv, dev(wl.x))
    out, status = tfg.tfg_segment_pool_meanmax(h, bg.batch, wl.num_graphs)
    tfg.check_status(status)
    ref, scale = oracle.segment_pool_meanmax(np_(h), wl.batch, wl.num_graphs)
    f = wl.x.shape[1]
    assert_scaled_close(np_(out)[:, :f], ref[:, :f], scale[:, :f], TOL_F32, "molecules mean")
    assert_exact_f32(np_(out)[:, f:], ref[:, f:], "molecules max")


def test_deterministic_bitwise():
    wl = gg.random_edge_case_graph(20000, 400000, 128, 5, hub=3, isolated=100)
    n = wl.num_nodes
    runs = []
    for _ in range(2):
        csr = gpu_csr(wl.edge_index, n)
        dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, 1, 1.0, want_w_csr=False)
        a = tfg.tfg_gcn_aggregate_sum(csr.rowptr, csr.col, dinv, features(wl, "bf16"), None, 1, 1.0)
        b, al = tfg.tfg_edge_softmax_aggregate(csr.rowptr, csr.col, dev(wl.x), 8, 16,
                                               dev(np.ones(128, np.float32)),
                                               dev(np.ones(128, np.float32)), 0.2, want_alpha=True)
        runs.append([np_(t).tobytes() for t in (csr.col, csr.perm, dinv, a, b, al)])
    assert runs[0] == runs[1]
