"""Largest sizes the ABI accepts: N = 2^31 - 1 nodes (int32 CSR ids, four
radix passes of 8 bits) and F = 2^24 features.

The CSR is compared whole against the oracle (chunk by chunk, to bound host
memory).  Aggregations at N = 2^31 - 1 are compared on sampled target rows:
the oracle runs on the sub-graph made of those rows' in-edges with the nodes
renumbered compactly, which defines the same sums, means and maxima (an
unweighted aggregate of row t reads only t's in-edges and their sources).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2101_11552_gb300 import tfg
from _helpers import TOL_F32, assert_exact_f32, assert_scaled_close, dev

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

N_MAX = (1 << 31) - 1
F_MAX = 1 << 24


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_11552_gb300 import build
    build.build_library()


def _equal_in_chunks(gpu: torch.Tensor, host: np.ndarray, what: str, chunk: int = 1 << 26):
    assert gpu.numel() == host.size, what
    for s in range(0, host.size, chunk):
        g = gpu[s:s + chunk].cpu().numpy()
        assert np.array_equal(g, host[s:s + chunk]), f"{what}: mismatch in [{s}, {s + chunk})"


@pytest.fixture(scope="module")
def huge_graph():
    rng = np.random.default_rng(2024)
    e = 1 << 20
    ei = rng.integers(0, N_MAX, size=(2, e), dtype=np.int64)
    ei[:, :4] = [[0, N_MAX - 1, N_MAX - 1, 0], [N_MAX - 1, 0, N_MAX - 1, 0]]
    ei[1, 4:4000] = N_MAX - 1                      # a hub at the last node
    ei[1, 4000:4100] = N_MAX - 2
    csr = tfg.tfg_build_csr(dev(ei), N_MAX)
    tfg.check_status(csr.status)
    torch.cuda.synchronize()
    return ei, csr


def test_csr_at_max_nodes(huge_graph):
    ei, csr = huge_graph
    rowptr, col, perm, deg = oracle.build_csr(ei, N_MAX)
    assert np.array_equal(csr.col.cpu().numpy(), col)
    assert np.array_equal(csr.perm.cpu().numpy(), perm)
    _equal_in_chunks(csr.rowptr, rowptr, "rowptr")
    del rowptr
    _equal_in_chunks(csr.in_degree, deg, "in_degree")


def test_csr_from_int32_edges_at_max_nodes(huge_graph):
    """tfg_build_csr32 with ids up to 2^31 - 2: the same CSR as the int64 build."""
    ei, csr = huge_graph
    c32 = tfg.tfg_build_csr(dev(ei.astype(np.int32)), N_MAX)
    tfg.check_status(c32.status)
    assert torch.equal(c32.col, csr.col) and torch.equal(c32.perm, csr.perm)
    assert torch.equal(c32.rowptr, csr.rowptr) and torch.equal(c32.in_degree, csr.in_degree)


@pytest.mark.parametrize("reduce", ["sum", "mean", "max"])
def test_aggregate_at_max_nodes(huge_graph, reduce):
    ei, csr = huge_graph
    rng = np.random.default_rng(7)
    x = torch.empty(N_MAX, 1, dtype=torch.float32, device="cuda")
    # values by node id (a hash of it, an integer below 2^20 times 2^-20, so
    # exact in fp32 on both sides) so that any row of x can be rebuilt on the host
    ids = torch.arange(N_MAX, dtype=torch.int64, device="cuda")
    x[:, 0] = (((ids * 2654435761) % 1000003) - 500001).float() * (2.0 ** -20)
    del ids
    fn = {"sum": tfg.tfg_aggregate_sum, "mean": tfg.tfg_aggregate_mean,
          "max": tfg.tfg_aggregate_max}[reduce]
    out = fn(csr.rowptr, csr.col, x)
    rows = np.unique(np.concatenate([[0, 1, N_MAX - 2, N_MAX - 1],
                                     rng.choice(ei[1], 2000, replace=False)]))
    got = out[dev(rows)][:, 0].cpu().numpy()
    # sub-graph of the sampled rows' in-edges, nodes renumbered compactly
    keep = np.isin(ei[1], rows)
    sub = ei[:, keep]
    nodes, inv = np.unique(sub, return_inverse=True)
    nodes = np.union1d(nodes, rows)
    remap = np.searchsorted(nodes, sub)
    xs = (((nodes * 2654435761) % 1000003) - 500001).astype(np.float32) * np.float32(2.0 ** -20)
    assert np.array_equal(x[dev(nodes)][:, 0].cpu().numpy(), xs)   # host copy of those rows
    ref, scale = oracle.aggregate(remap, len(nodes), xs[:, None], reduce)
    pos = np.searchsorted(nodes, rows)
    if reduce == "max":
        assert_exact_f32(got, ref[pos, 0], "max at 2^31 - 1 nodes")
    else:
        assert_scaled_close(got, ref[pos, 0], scale[pos, 0], TOL_F32, f"{reduce} at 2^31 - 1 nodes")
    del out, x


def test_max_features():
    """F = 2^24 on a four-node graph: sum, max, GCN, APPNP and a one-head edge
    softmax all walk 2^24 features per row."""
    n, f = 4, F_MAX
    ei = np.array([[0, 1, 2, 3, 3], [1, 2, 3, 0, 1]], np.int64)
    x = np.random.default_rng(3).standard_normal((n, f)).astype(np.float32)
    csr = tfg.tfg_build_csr(dev(ei), n)
    xd = dev(x)
    for reduce, fn in (("sum", tfg.tfg_aggregate_sum), ("max", tfg.tfg_aggregate_max)):
        got = fn(csr.rowptr, csr.col, xd).cpu().numpy()
        ref, scale = oracle.aggregate(ei, n, x, reduce)
        if reduce == "max":
            assert_exact_f32(got, ref, "max F = 2^24")
        else:
            assert_scaled_close(got, ref, scale, TOL_F32, "sum F = 2^24")
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, 1, 1.0, want_w_csr=False)
    got = tfg.tfg_appnp_propagate(csr.rowptr, csr.col, dinv, xd, 2, 0.1, add_self_loops=1)
    ref, scale = oracle.appnp(ei, n, x, 2, 0.1, add_self_loops=1)
    assert_scaled_close(got.cpu().numpy(), ref, scale, TOL_F32, "appnp F = 2^24")
    del got
    a = np.random.default_rng(4).standard_normal((2, f)).astype(np.float32) / 4096
    out, _ = tfg.tfg_edge_softmax_aggregate(csr.rowptr, csr.col, xd, 1, f, dev(a[0]), dev(a[1]), 0.2)
    ref, _, scale = oracle.edge_softmax(ei, n, x, 1, f, a[0], a[1], 0.2)
    assert_scaled_close(out.cpu().numpy(), ref, scale, TOL_F32, "edge softmax F = 2^24")


def test_pool_feature_limit():
    f_ok = 65535 * 8
    n, g = 6, 2
    x = torch.randn(n, f_ok, device="cuda")
    batch = dev(np.array([0, 0, 0, 1, 1, 1], np.int64))
    out, status = tfg.tfg_segment_pool_meanmax(x, batch, g)
    tfg.check_status(status)
    ref, scale = oracle.segment_pool_meanmax(x.cpu().numpy(), batch.cpu().numpy(), g)
    assert_scaled_close(out[:, :f_ok].cpu().numpy(), ref[:, :f_ok], scale[:, :f_ok], TOL_F32, "mean")
    assert_exact_f32(out[:, f_ok:].cpu().numpy(), ref[:, f_ok:], "max")
    with pytest.raises(tfg.TfgError):
        tfg.tfg_segment_pool_meanmax(torch.zeros(n, f_ok + 1, device="cuda"), batch, g)
