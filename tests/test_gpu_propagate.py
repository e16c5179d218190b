"""APPNP / SGC multi-hop propagation against the oracle's K repeated hops.

Tolerance: per element |gpu - oracle| <= TOL_F32 * scale, with scale the
oracle's recursion on absolute values (|Ahat|^k |x0| mixed with alpha |x0|).
The iterates are fp32 for both storage types of x0 (the oracle reads the same
bf16 values), so TOL_F32 holds for bf16 x0 as well.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2101_11552_gb300 import graphgen as gg
from paper_2101_11552_gb300 import tfg
from _helpers import TOL_F32, assert_scaled_close, dev, features, host_features

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_11552_gb300 import build
    build.build_library()


def _graph(wl):
    csr = tfg.tfg_build_csr(dev(wl.edge_index), wl.num_nodes)
    tfg.check_status(csr.status)
    return csr


CASES = [  # (n, e, f, hub, isolated, seed)
    (1, 0, 8, -1, 0, 1),
    (300, 0, 16, -1, 0, 2),           # no edges: only self-loops and teleport
    (2000, 16000, 1, 3, 40, 3),
    (2000, 16000, 7, 3, 40, 4),       # scalar paths
    (5000, 60000, 64, 2, 100, 5),
    (5000, 60000, 128, 9, 100, 6),
    (3000, 90000, 136, 1, 20, 7),     # hub rows above the CTA-cooperative threshold
]


@pytest.mark.parametrize("case", CASES)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("hops,alpha", [(0, 0.1), (1, 0.1), (2, 0.0), (5, 0.2), (10, 0.1), (3, 1.0)])
def test_appnp_matches_oracle(case, dtype, hops, alpha):
    n, e, f, hub, iso, seed = case
    wl = gg.random_edge_case_graph(n, e, f, 500 + seed, hub=hub, isolated=min(iso, n - 1))
    csr = _graph(wl)
    selfl = 1 if seed % 2 == 0 or e == 0 else 0
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, selfl, 1.0,
                               want_w_csr=False)
    x0 = features(wl, dtype)
    out = tfg.tfg_appnp_propagate(csr.rowptr, csr.col, dinv, x0, hops, alpha,
                                  add_self_loops=selfl)
    ref, scale = oracle.appnp(wl.edge_index, n, host_features(wl, dtype), hops, alpha,
                              add_self_loops=selfl)
    assert_scaled_close(out.cpu().numpy(), ref, scale, TOL_F32, f"appnp K={hops}")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_appnp_weighted_graph(dtype):
    n, e, f = 4000, 50000, 32
    wl = gg.random_edge_case_graph(n, e, f, 77, hub=2, isolated=30)
    ew = np.random.default_rng(77).uniform(0.1, 3.0, size=e).astype(np.float32)
    csr = _graph(wl)
    dinv, w_csr = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, dev(ew), 1, 2.0)
    out = tfg.tfg_appnp_propagate(csr.rowptr, csr.col, dinv, features(wl, dtype), 4, 0.15,
                                  w_csr=w_csr, add_self_loops=1, self_loop_fill=2.0)
    ref, scale = oracle.appnp(wl.edge_index, n, host_features(wl, dtype), 4, 0.15,
                              edge_weight=ew.astype(np.float64), add_self_loops=1, fill=2.0)
    # w_csr carries the fp32 rounding of each normalised weight: a relative
    # 2^-24 per weight, inside the same bound
    assert_scaled_close(out.cpu().numpy(), ref, scale, TOL_F32, "appnp weighted")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_sgc_is_chained_gcn_bit_exact(dtype):
    """SGC's K hops are exactly K GCN aggregations: the same kernels, sums in
    the same order, and alpha = 0 leaves the epilogue an identity."""
    n, e, f = 6000, 80000, 128
    wl = gg.random_edge_case_graph(n, e, f, 91, hub=4, isolated=50)
    csr = _graph(wl)
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, 1, 1.0, want_w_csr=False)
    x0 = features(wl, dtype)
    got = tfg.tfg_sgc_propagate(csr.rowptr, csr.col, dinv, x0, 3, add_self_loops=1)
    h = x0
    for _ in range(3):
        h = tfg.tfg_gcn_aggregate_sum(csr.rowptr, csr.col, dinv, h, None, 1, 1.0)
    assert torch.equal(got, h)
    h0 = tfg.tfg_sgc_propagate(csr.rowptr, csr.col, dinv, x0, 0)
    assert torch.equal(h0, x0.float())


def test_propagate_workspace_and_buffers():
    n, e, f = 1000, 8000, 24
    wl = gg.random_edge_case_graph(n, e, f, 13, hub=1, isolated=10)
    csr = _graph(wl)
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, 1, 1.0, want_w_csr=False)
    assert tfg.tfg_propagate_workspace_size(n, f, 1) == 0
    assert tfg.tfg_propagate_workspace_size(n, f, 2) >= n * f * 4
    x0 = dev(wl.x)
    ws = torch.full((tfg.tfg_propagate_workspace_size(n, f, 7),), 255, dtype=torch.uint8,
                    device="cuda")
    out = torch.full((n, f), float("nan"), device="cuda")
    tfg.tfg_appnp_propagate(csr.rowptr, csr.col, dinv, x0, 7, 0.3, add_self_loops=1, out=out,
                            workspace=ws)
    again = tfg.tfg_appnp_propagate(csr.rowptr, csr.col, dinv, x0, 7, 0.3, add_self_loops=1)
    assert torch.equal(out, again)    # deterministic, and no stale workspace value is read
    ref, scale = oracle.appnp(wl.edge_index, n, wl.x, 7, 0.3, add_self_loops=1)
    assert_scaled_close(out.cpu().numpy(), ref, scale, TOL_F32, "appnp odd K")


def test_appnp_rejects_bad_arguments():
    n, f = 10, 4
    rowptr = torch.zeros(n + 1, dtype=torch.int32, device="cuda")
    col = torch.zeros(1, dtype=torch.int32, device="cuda")
    dinv = torch.ones(n, device="cuda")
    x0 = torch.zeros(n, f, device="cuda")
    for hops, alpha in ((-1, 0.1), (5000, 0.1), (2, 1.5), (2, float("nan"))):
        with pytest.raises(tfg.TfgError):
            tfg.tfg_appnp_propagate(rowptr, col, dinv, x0, hops, alpha)
