"""Backward of the GAT edge-softmax aggregation against the fp64 oracle.

The oracle's backward is pinned by central finite differences of the forward
oracle (test_oracle_pins.py).  Tolerance: each gradient element within
tol * scale, scale the oracle's sum of absolute terms of the same recursion;
tol = 1e-5 + kappa * max(lam_e + lam_max): every term carries the attention
weight, whose fp32 relative error grows with the logit magnitude lam (the
attention-weight bound of the forward tests).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2101_11552_gb300 import graphgen as gg
from paper_2101_11552_gb300 import tfg
from _helpers import KAPPA_GAT, TOL_F32, assert_scaled_close, csr_rows, dev, gat_logit_mag

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_11552_gb300 import build
    build.build_library()


def _case(n, e, heads, channels, dtype, seed, hub=3, isolated=20):
    f = heads * channels
    wl = gg.random_edge_case_graph(n, e, f, seed, hub=hub, isolated=isolated)
    rng = np.random.default_rng(seed)
    a_s = (0.5 * rng.standard_normal(f)).astype(np.float32)
    a_d = (0.5 * rng.standard_normal(f)).astype(np.float32)
    g = rng.standard_normal((n, f)).astype(np.float32)
    if dtype == "bf16":
        xh = wl.x_bf16
        x = dev(xh.view(np.int16)).view(torch.bfloat16)
    else:
        xh = wl.x
        x = dev(xh)
    return wl, x, xh, a_s, a_d, g


def _run(wl, x, heads, channels, a_s, a_d, g, slope=0.2):
    n = wl.num_nodes
    ei = dev(wl.edge_index)
    csr = tfg.tfg_build_csr(ei, n)
    csr_src = tfg.tfg_build_csr_by_source(ei, n)
    tfg.check_status(csr.status)
    tfg.check_status(csr_src.status)
    out, _ = tfg.tfg_edge_softmax_aggregate(csr.rowptr, csr.col, x, heads, channels, dev(a_s),
                                            dev(a_d), slope)
    gx, ga, gd = tfg.tfg_edge_softmax_aggregate_backward(
        csr.rowptr, csr.col, csr_src.rowptr, csr_src.col, x, heads, channels, dev(a_s), dev(a_d),
        slope, out, dev(g))
    torch.cuda.synchronize()
    return gx.cpu().numpy(), ga.cpu().numpy(), gd.cpu().numpy(), csr


def _tol(wl, xh, heads, channels, a_s, a_d, csr):
    rowptr, col = csr.rowptr.cpu().numpy(), csr.col.cpu().numpy()
    if len(col) == 0:
        return TOL_F32
    row = csr_rows(rowptr)
    lam = gat_logit_mag(oracle.widen(xh), col, row, heads, channels, a_s, a_d)
    lam_max = np.zeros((wl.num_nodes, heads))
    np.maximum.at(lam_max, row, lam)
    return TOL_F32 + KAPPA_GAT * float(np.max(lam + lam_max[row]))


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("heads,channels", [(8, 16), (4, 8), (2, 32), (1, 64), (16, 2), (1, 1),
                                            (2, 128), (3, 4)])
def test_gat_backward_matches_oracle(heads, channels, dtype):
    n, e = 2500, 30000
    wl, x, xh, a_s, a_d, g = _case(n, e, heads, channels, dtype, 11 + heads * channels)
    gx, ga, gd, csr = _run(wl, x, heads, channels, a_s, a_d, g)
    rgx, rga, rgd, (sx, sa, sd) = oracle.edge_softmax_backward(wl.edge_index, n, xh, heads,
                                                               channels, a_s, a_d, 0.2, g)
    tol = _tol(wl, xh, heads, channels, a_s, a_d, csr)
    what = f"{dtype} H={heads} C={channels}"
    assert_scaled_close(gx, rgx, sx, tol, "grad_x " + what)
    assert_scaled_close(ga, rga, sa, tol, "grad_a_src " + what)
    assert_scaled_close(gd, rgd, sd, tol, "grad_a_dst " + what)


def test_gat_backward_hub_rows_and_degenerate_graphs():
    """A 20k-edge hub (sums blocked per 32 edges), then graphs with no edges
    and with a single node carrying self-loops."""
    heads, channels = 8, 16
    wl, x, xh, a_s, a_d, g = _case(3000, 40000, heads, channels, "f32", 5, hub=0, isolated=10)
    gx, ga, gd, csr = _run(wl, x, heads, channels, a_s, a_d, g)
    rgx, rga, rgd, (sx, sa, sd) = oracle.edge_softmax_backward(wl.edge_index, 3000, xh, heads,
                                                               channels, a_s, a_d, 0.2, g)
    tol = _tol(wl, xh, heads, channels, a_s, a_d, csr)
    assert_scaled_close(gx, rgx, sx, tol, "hub grad_x")
    assert_scaled_close(ga, rga, sa, tol, "hub grad_a_src")
    assert_scaled_close(gd, rgd, sd, tol, "hub grad_a_dst")
    rng = np.random.default_rng(3)
    for n, ei in ((40, np.zeros((2, 0), np.int64)), (1, np.zeros((2, 3), np.int64))):
        f = heads * channels
        xh = rng.standard_normal((n, f)).astype(np.float32)
        g = rng.standard_normal((n, f)).astype(np.float32)
        w = gg.Workload("degenerate", n, ei, xh)
        gx, ga, gd, _ = _run(w, dev(xh), heads, channels, a_s, a_d, g)
        rgx, rga, rgd, (sx, sa, sd) = oracle.edge_softmax_backward(ei, n, xh, heads, channels,
                                                                   a_s, a_d, 0.2, g)
        assert_scaled_close(gx, rgx, sx, TOL_F32, f"grad_x n={n}")
        assert_scaled_close(ga, rga, sa, TOL_F32, f"grad_a_src n={n}")
        assert_scaled_close(gd, rgd, sd, TOL_F32, f"grad_a_dst n={n}")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_gat_backward_unaligned_rows_take_the_general_kernels(dtype):
    """x shifted off 16-byte alignment runs the general kernels (the aligned
    8 x 16 layout runs the fast ones); both meet the oracle's bound."""
    heads, channels = 8, 16
    n, f = 2000, heads * channels
    wl, x, xh, a_s, a_d, g = _case(n, 25000, heads, channels, dtype, 41)
    buf = torch.empty(n * f + 1, dtype=x.dtype, device=x.device)
    buf[1:].copy_(x.reshape(-1))
    xu = buf[1:].view(n, f)
    rgx, rga, rgd, (sx, sa, sd) = oracle.edge_softmax_backward(wl.edge_index, n, xh, heads,
                                                               channels, a_s, a_d, 0.2, g)
    for xx, what in ((xu, "unaligned"), (x, "aligned")):
        gx, ga, gd, csr = _run(wl, xx, heads, channels, a_s, a_d, g)
        tol = _tol(wl, xh, heads, channels, a_s, a_d, csr)
        assert_scaled_close(gx, rgx, sx, tol, f"grad_x {what} {dtype}")
        assert_scaled_close(ga, rga, sa, tol, f"grad_a_src {what} {dtype}")
        assert_scaled_close(gd, rgd, sd, tol, f"grad_a_dst {what} {dtype}")


def test_gat_backward_is_deterministic_and_rejects_bad_layouts():
    heads, channels = 4, 16
    wl, x, _, a_s, a_d, g = _case(2000, 30000, heads, channels, "bf16", 9)
    a = _run(wl, x, heads, channels, a_s, a_d, g)
    b = _run(wl, x, heads, channels, a_s, a_d, g)
    for u, v in zip(a[:3], b[:3]):
        assert np.array_equal(u, v)
    with pytest.raises(tfg.TfgError):
        tfg.tfg_edge_softmax_backward_workspace_size(100, 2, 24)     # 24: not a power of two
    with pytest.raises(tfg.TfgError):
        tfg.tfg_edge_softmax_backward_workspace_size(100, 4, 128)    # F = 512 > 256
