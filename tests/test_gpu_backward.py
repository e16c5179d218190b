"""Backward of the aggregation against the oracle.

CSR by source and argmax indices are compared bit for bit; gradients within
TOL_F32 of the oracle's sum of absolute terms (the gradient sums are plain
fp32 sums of grad_out rows, in a fixed order).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2101_11552_gb300 import graphgen as gg
from paper_2101_11552_gb300 import tfg
from _helpers import TOL_F32, assert_exact_f32, assert_scaled_close, dev, features, host_features

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_11552_gb300 import build
    build.build_library()


def _graphs(n, e, seed, f=1, reverse=False):
    wl = gg.random_edge_case_graph(n, e, f, seed, hub=3, isolated=30)
    if reverse:
        wl.edge_index = np.ascontiguousarray(wl.edge_index[::-1])
    csr = tfg.tfg_build_csr(dev(wl.edge_index), n)
    csr_src = tfg.tfg_build_csr_by_source(dev(wl.edge_index), n)
    tfg.check_status(csr.status)
    tfg.check_status(csr_src.status)
    return wl, csr, csr_src


@pytest.mark.parametrize("n,e,seed", [(1, 0, 1), (500, 0, 2), (3000, 40000, 3), (20000, 300000, 4)])
def test_csr_by_source_bit_exact(n, e, seed):
    wl = gg.random_edge_case_graph(n, e, 1, seed, hub=3 if n > 4 else -1, isolated=min(30, n - 1))
    got = tfg.tfg_build_csr_by_source(dev(wl.edge_index), n)
    tfg.check_status(got.status)
    want = oracle.build_csr(wl.edge_index[::-1].copy(), n)
    for a, b, name in zip(got[:4], want, ("rowptr", "col", "perm", "out_degree")):
        assert np.array_equal(a.cpu().numpy(), b), name


@pytest.mark.parametrize("reduce", ["sum", "mean"])
@pytest.mark.parametrize("weighted", [False, True])
@pytest.mark.parametrize("f", [1, 7, 64, 128])
def test_aggregate_backward(reduce, weighted, f):
    n, e = 3000, 40000
    wl, csr, csr_src = _graphs(n, e, 30 + f)
    rng = np.random.default_rng(f)
    g = rng.standard_normal((n, f)).astype(np.float32)
    ew = rng.uniform(0.1, 3.0, size=e).astype(np.float32) if weighted else None
    got = tfg.tfg_aggregate_backward(reduce, csr_src, dev(g), None if ew is None else dev(ew),
                                     csr.in_degree)
    ref, scale = oracle.aggregate_backward(wl.edge_index, n, g, reduce,
                                           w=None if ew is None else ew.astype(np.float64))
    assert_scaled_close(got.cpu().numpy(), ref, scale, TOL_F32, f"{reduce} backward")


@pytest.mark.parametrize("add_self", [0, 1])
@pytest.mark.parametrize("f", [5, 128])
def test_gcn_aggregate_backward(add_self, f):
    n, e = 4000, 60000
    wl, csr, csr_src = _graphs(n, e, 50 + f)
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, add_self, 1.0,
                               want_w_csr=False)
    g = np.random.default_rng(f).standard_normal((n, f)).astype(np.float32)
    got = tfg.tfg_gcn_aggregate_backward(csr_src, dinv, dev(g), add_self, 1.0)
    ref, scale = oracle.gcn_aggregate_backward(wl.edge_index, n, g, None, add_self, 1.0)
    assert_scaled_close(got.cpu().numpy(), ref, scale, TOL_F32, "gcn backward")


@pytest.mark.parametrize("reverse", [False, True])
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("weighted", [False, True])
@pytest.mark.parametrize("f", [1, 33, 128])
def test_max_argmax_and_backward(dtype, weighted, f, reverse):
    """The hub (about 20,000 edges) is a target row, split over a CTA in the
    forward; reversed, it is a source row, split in the backward."""
    n, e = 3000, 40000
    wl, csr, csr_src = _graphs(n, e, 70 + f, f, reverse)
    rng = np.random.default_rng(f)
    ew = rng.uniform(0.1, 3.0, size=e).astype(np.float32) if weighted else None
    w_csr = None if ew is None else dev(ew[csr.perm.cpu().numpy()])
    out, arg = tfg.tfg_aggregate_max_argmax(csr, features(wl, dtype), w_csr)
    ref, ref_arg = oracle.max_argmax(wl.edge_index, n, host_features(wl, dtype), ew)
    assert np.array_equal(arg.cpu().numpy(), ref_arg), "argmax"
    assert_exact_f32(out.cpu().numpy(), ref, "max with argmax")
    plain = tfg.tfg_aggregate_max(csr.rowptr, csr.col, features(wl, dtype), w_csr)
    assert torch.equal(out, plain)                   # the same values as the forward max
    g = rng.standard_normal((n, f)).astype(np.float32)
    got = tfg.tfg_aggregate_max_backward(csr_src, arg, dev(g), None if ew is None else dev(ew))
    refg, scale = oracle.max_backward(wl.edge_index, n, ref_arg, g,
                                      None if ew is None else ew.astype(np.float64))
    assert_scaled_close(got.cpu().numpy(), refg, scale, TOL_F32, "max backward")
    # without the win marks every out-edge's rows are read: the same bits
    plain = tfg.tfg_aggregate_max_backward(csr_src, arg, dev(g), None if ew is None else dev(ew),
                                           marks=False)
    assert torch.equal(got, plain)


def test_max_backward_ignores_argmax_ids_outside_the_edges():
    """argmax values outside [0, E) (and ids of edges into another row) match
    no out-edge of the row, with and without the win marks."""
    n, e, f = 400, 60000, 32
    wl, csr, csr_src = _graphs(n, e, 41, f)
    assert tfg.tfg_aggregate_max_backward_workspace_size(n, e, f) > 0
    rng = np.random.default_rng(41)
    _, arg = tfg.tfg_aggregate_max_argmax(csr, features(wl, "f32"))
    bad = arg.cpu().numpy().copy()
    pick = rng.random(bad.shape)
    bad[pick < 0.05] = -7
    bad[(pick >= 0.05) & (pick < 0.1)] = e + 3
    bad[(pick >= 0.1) & (pick < 0.12)] = np.iinfo(np.int32).max
    other = (pick >= 0.12) & (pick < 0.2)
    bad[other] = rng.integers(0, e, size=int(other.sum()))    # mostly edges into other rows
    g = rng.standard_normal((n, f)).astype(np.float32)
    refg, scale = oracle.max_backward(wl.edge_index, n, bad, g, None)
    for marks in (True, False):
        got = tfg.tfg_aggregate_max_backward(csr_src, dev(bad), dev(g), marks=marks)
        assert_scaled_close(got.cpu().numpy(), refg, scale, TOL_F32, f"max backward marks={marks}")


@pytest.mark.parametrize("reverse", [False, True])
@pytest.mark.parametrize("weighted", [False, True])
@pytest.mark.parametrize("f", [4, 33, 36, 64])
def test_max_backward_with_win_marks(f, weighted, reverse):
    """Long rows (E >= min(F, 128) N): the call marks which eighths of the
    features each edge wins and reads argmax and gradient slices for those
    alone; the same bits as the walk over every out-edge.  Reversed, the hub (about half of the
    edges) is a source row split over a CTA."""
    n, e = 400, 60000
    wl, csr, csr_src = _graphs(n, e, 90 + f, f, reverse)
    assert tfg.tfg_aggregate_max_backward_workspace_size(n, e, f) > 0
    rng = np.random.default_rng(f)
    ew = rng.uniform(0.1, 3.0, size=e).astype(np.float32) if weighted else None
    w_csr = None if ew is None else dev(ew[csr.perm.cpu().numpy()])
    _, arg = tfg.tfg_aggregate_max_argmax(csr, features(wl, "bf16"), w_csr)
    g = rng.standard_normal((n, f)).astype(np.float32)
    got = tfg.tfg_aggregate_max_backward(csr_src, arg, dev(g), None if ew is None else dev(ew))
    plain = tfg.tfg_aggregate_max_backward(csr_src, arg, dev(g), None if ew is None else dev(ew),
                                           marks=False)
    assert torch.equal(got, plain)
    refg, scale = oracle.max_backward(wl.edge_index, n, arg.cpu().numpy(), g,
                                      None if ew is None else ew.astype(np.float64))
    assert_scaled_close(got.cpu().numpy(), refg, scale, TOL_F32, f"max backward with marks F={f}")


def test_max_backward_workspace_is_checked():
    n, e, f = 100, 4000, 4
    wl, csr, csr_src = _graphs(n, e, 43, f)
    _, arg = tfg.tfg_aggregate_max_argmax(csr, features(wl, "f32"))
    g = dev(np.ones((n, f), np.float32))
    out = torch.empty(n, f, device="cuda")
    assert tfg.tfg_aggregate_max_backward_workspace_size(n, e, f) > 100
    small = torch.empty(100, dtype=torch.uint8, device="cuda")
    rc = tfg.lib().tfg_aggregate_max_backward(
        tfg._ptr(csr_src.rowptr), tfg._ptr(csr_src.col), tfg._ptr(csr_src.perm), tfg._ptr(arg),
        None, tfg._ptr(g), n, e, f, tfg._ptr(out), tfg._ptr(small), small.numel(), None)
    assert rc == tfg.TFG_ERR_WORKSPACE


def test_backward_is_deterministic_and_validates():
    n, e, f = 20000, 400000, 64
    wl, csr, csr_src = _graphs(n, e, 99, f)
    g = dev(np.random.default_rng(9).standard_normal((n, f)).astype(np.float32))
    a = tfg.tfg_aggregate_backward("mean", csr_src, g, None, csr.in_degree)
    b = tfg.tfg_aggregate_backward("mean", csr_src, g, None, csr.in_degree)
    assert torch.equal(a, b)
    with pytest.raises(tfg.TfgError):
        tfg.tfg_aggregate_backward("max", csr_src, g)
    with pytest.raises(tfg.TfgError):                # the mean needs the forward in-degrees
        tfg.tfg_aggregate_backward("mean", csr_src, g, None, None)


@pytest.mark.parametrize("n", [1, 500])
def test_backward_without_edges(n):
    """No edges: every gradient is 0 (plus the self-loop term for GCN), the
    argmax is -1 everywhere."""
    f = 8
    ei = np.zeros((2, 0), np.int64)
    csr = tfg.tfg_build_csr(dev(ei), n)
    csr_src = tfg.tfg_build_csr_by_source(dev(ei), n)
    g = np.random.default_rng(n).standard_normal((n, f)).astype(np.float32)
    for reduce in ("sum", "mean"):
        got = tfg.tfg_aggregate_backward(reduce, csr_src, dev(g), None, csr.in_degree)
        assert torch.count_nonzero(got).item() == 0
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, 1, 1.0, want_w_csr=False)
    got = tfg.tfg_gcn_aggregate_backward(csr_src, dinv, dev(g), 1, 1.0)
    ref, scale = oracle.gcn_aggregate_backward(ei, n, g, None, 1, 1.0)
    assert_scaled_close(got.cpu().numpy(), ref, scale, TOL_F32, "gcn backward without edges")
    out, arg = tfg.tfg_aggregate_max_argmax(csr, dev(g))
    assert torch.count_nonzero(out).item() == 0 and bool((arg == -1).all())
    got = tfg.tfg_aggregate_max_backward(csr_src, arg, dev(g))
    assert torch.count_nonzero(got).item() == 0


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_max_argmax_ties_across_hub_segments(dtype):
    """Equal values everywhere: every argmax is the row's first edge in input
    order, also in hub rows that the kernel splits into segments, and the
    backward hands each gradient to that edge's source."""
    n, e, f = 3000, 40000, 64
    wl, csr, csr_src = _graphs(n, e, 5, f)
    x = np.ones((n, f), np.float32)
    xd = dev(x) if dtype == "f32" else dev(x).to(torch.bfloat16)
    out, arg = tfg.tfg_aggregate_max_argmax(csr, xd)
    rowptr, perm = csr.rowptr.cpu().numpy(), csr.perm.cpu().numpy()
    deg = np.diff(rowptr)
    assert deg.max() > 4096                          # the hub is split
    first = np.where(deg > 0, perm[np.minimum(rowptr[:-1], e - 1)], -1)
    assert np.array_equal(arg.cpu().numpy(), np.repeat(first[:, None], f, axis=1))
    ref, ref_arg = oracle.max_argmax(wl.edge_index, n, x, None)
    assert np.array_equal(arg.cpu().numpy(), ref_arg)
    assert_exact_f32(out.cpu().numpy(), ref, "max of ones")
    g = np.random.default_rng(6).standard_normal((n, f)).astype(np.float32)
    got = tfg.tfg_aggregate_max_backward(csr_src, arg, dev(g))
    refg, scale = oracle.max_backward(wl.edge_index, n, ref_arg, g, None)
    assert_scaled_close(got.cpu().numpy(), refg, scale, TOL_F32, "max backward, ties")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("weighted", [False, True])
def test_max_argmax_with_nan_and_inf(dtype, weighted):
    """NaN, +inf and -inf features (and 0 * inf = NaN products with zero
    weights): the first edge of a row is taken whatever its value, later
    edges only when strictly larger, as in one ordered pass -- also across
    the lane groups and the segments of the split hub row."""
    n, e, f = 3000, 40000, 16
    wl, csr, csr_src = _graphs(n, e, 11, f)
    rng = np.random.default_rng(12)
    x = rng.standard_normal((n, f)).astype(np.float32)
    for val, frac in ((np.nan, 0.02), (np.inf, 0.01), (-np.inf, 0.02)):
        x[rng.random((n, f)) < frac] = val
    xt = torch.from_numpy(x)
    if dtype == "bf16":
        xt = xt.to(torch.bfloat16)
        x = xt.float().numpy()                       # the values the kernel reads
    ew = None
    if weighted:
        ew = rng.uniform(0.5, 2.0, size=e).astype(np.float32)
        ew[rng.random(e) < 0.05] = 0.0
    w_csr = None if ew is None else dev(ew[csr.perm.cpu().numpy()])
    out, arg = tfg.tfg_aggregate_max_argmax(csr, xt.cuda(), w_csr)
    ref, ref_arg = oracle.max_argmax(wl.edge_index, n, x, ew)
    assert np.array_equal(arg.cpu().numpy(), ref_arg), "argmax"
    np.testing.assert_array_equal(out.cpu().numpy(), ref.astype(np.float32))   # NaN == NaN here
    g = rng.standard_normal((n, f)).astype(np.float32)
    got = tfg.tfg_aggregate_max_backward(csr_src, arg, dev(g), None if ew is None else dev(ew))
    refg, scale = oracle.max_backward(wl.edge_index, n, ref_arg, g,
                                      None if ew is None else ew.astype(np.float64))
    assert_scaled_close(got.cpu().numpy(), refg, scale, TOL_F32, "max backward, NaN and inf")
