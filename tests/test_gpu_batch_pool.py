"""Device BatchGraph construction and the fused Mean-Max pool against the oracle.

BatchGraph (Section 2.1.1, reindexing trick): edge lists, batch vector and
offsets are integer outputs and must match bit for bit.  Mean-Max pool
(Table 2 readout): max halves bit-exact, mean halves within the fp32
tolerance, and both identical to two separate tfg_segment_pool calls.
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


def random_graphs(seed, g, max_nodes=50):
    rng = np.random.default_rng(seed)
    sizes = rng.integers(0, max_nodes, size=g)
    sizes[0] = 0                       # empty graphs, first and middle
    sizes[g // 2] = 0
    if g > 2:
        sizes[1] = 1                   # a single node, no edges
    parts = []
    for s in sizes:
        s = int(s)
        m = min(2 * s, s * (s - 1) // 2)
        ei = gg.symmetrise(gg.er_pairs(s, m, rng)) if m > 0 else np.zeros((2, 0), np.int64)
        if s > 0 and rng.random() < 0.5:
            ei = gg.with_self_loops(ei, s)
        parts.append(ei)
    stacked = np.ascontiguousarray(np.concatenate(parts, axis=1)) if parts else np.zeros((2, 0), np.int64)
    return sizes.astype(np.int64), np.array([p.shape[1] for p in parts], np.int64), stacked


@pytest.mark.parametrize("seed,g", [(0, 1), (1, 3), (2, 7), (3, 1024), (4, 5000)])
def test_batch_graphs_bit_exact(seed, g):
    sizes, ecounts, stacked = random_graphs(seed, g)
    n = int(sizes.sum())
    got = tfg.tfg_batch_graphs(dev(sizes), dev(ecounts), dev(stacked), n)
    tfg.check_status(got.status)
    ei, batch, offs = oracle.batch_graphs(sizes, ecounts, stacked)
    assert np.array_equal(got.edge_index.cpu().numpy(), ei)
    assert np.array_equal(got.batch.cpu().numpy(), batch)
    assert np.array_equal(got.node_offsets.cpu().numpy(), offs)


def test_batch_graphs_paper_example_on_device():
    sizes = np.array([4, 2, 3], np.int64)
    stacked = np.array([[0, 3, 1, 2], [1, 2, 0, 1]], np.int64)   # 2 edges in graph 0, 1 in 1 and 2
    ecounts = np.array([2, 1, 1], np.int64)
    got = tfg.tfg_batch_graphs(dev(sizes), dev(ecounts), dev(stacked), 9)
    tfg.check_status(got.status)
    offs = got.node_offsets.cpu().numpy()
    assert list(offs) == [0, 4, 6, 9]             # offsets of the 2nd and 3rd graph: 4 and 6
    assert list(got.batch.cpu().numpy()) == [0, 0, 0, 0, 1, 1, 2, 2, 2]
    assert got.edge_index.cpu().numpy().tolist() == [[0, 3, 5, 8], [1, 2, 4, 7]]


def test_batch_graphs_zero_graphs():
    empty = torch.zeros(0, dtype=torch.int64, device="cuda")
    bg = tfg.tfg_batch_graphs(empty, empty, torch.zeros(2, 0, dtype=torch.int64, device="cuda"), 0)
    tfg.check_status(bg.status)
    assert bg.node_offsets.cpu().tolist() == [0]
    assert bg.edge_index.shape == (2, 0) and bg.batch.numel() == 0


def test_batch_graphs_bad_input_sets_status():
    sizes = np.array([2, 2], np.int64)
    stacked = np.array([[0, 5], [1, 0]], np.int64)   # 5 is outside graph 1
    got = tfg.tfg_batch_graphs(dev(sizes), dev(np.array([1, 1])), dev(stacked), 4)
    assert int(got.status.item()) == tfg.TFG_ERR_INDEX_RANGE
    got = tfg.tfg_batch_graphs(dev(sizes), dev(np.array([1, 1])), dev(np.array([[0, 1], [1, 0]])), 5)
    assert int(got.status.item()) == tfg.TFG_ERR_INDEX_RANGE   # counts sum to 4, not 5


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("f", [1, 7, 128, 264])
@pytest.mark.parametrize("big", [False, True])
def test_meanmax_pool(dtype, f, big):
    rng = np.random.default_rng(f + big)
    g = 9 if big else 300
    sizes = rng.integers(6000, 12000, size=g) if big else rng.integers(0, 40, size=g)
    sizes[g // 2] = 0
    batch = np.repeat(np.arange(g), sizes).astype(np.int64)
    n = batch.size
    wl = gg.Workload("pool", n, np.zeros((2, 0), np.int64), rng.standard_normal((n, f)).astype(np.float32))
    x = features(wl, dtype)
    out, status = tfg.tfg_segment_pool_meanmax(x, dev(batch), g)
    tfg.check_status(status)
    got = out.cpu().numpy()
    ref, scale = oracle.segment_pool_meanmax(host_features(wl, dtype), batch, g)
    assert_scaled_close(got[:, :f], ref[:, :f], scale[:, :f], TOL_F32, "meanmax mean")
    assert_exact_f32(got[:, f:], ref[:, f:], "meanmax max")
    mean, _ = tfg.tfg_segment_pool(x, dev(batch), g, "mean")
    mx, _ = tfg.tfg_segment_pool(x, dev(batch), g, "max")
    assert np.array_equal(got[:, :f], mean.cpu().numpy())
    assert np.array_equal(got[:, f:], mx.cpu().numpy())


def test_batched_pipeline_on_device():
    """Graphs batched on the device, then CSR, GCN and Mean-Max pooling, against
    the oracle run on each graph separately (applying the model to a
    BatchGraph equals applying it graph by graph, Section 2.1.1)."""
    sizes, ecounts, stacked = random_graphs(11, 400, max_nodes=120)
    n = int(sizes.sum())
    bg = tfg.tfg_batch_graphs(dev(sizes), dev(ecounts), dev(stacked), n)
    tfg.check_status(bg.status)
    f = 64
    x = np.random.default_rng(5).standard_normal((n, f)).astype(np.float32)
    csr = tfg.tfg_build_csr(bg.edge_index, n)
    tfg.check_status(csr.status)
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, 1, 1.0, want_w_csr=False)
    h = tfg.tfg_gcn_aggregate_sum(csr.rowptr, csr.col, dinv, dev(x), None, 1, 1.0)
    pooled, status = tfg.tfg_segment_pool_meanmax(h, bg.batch, len(sizes))
    tfg.check_status(status)
    h_np, pooled = h.cpu().numpy(), pooled.cpu().numpy()
    offs = np.concatenate([[0], np.cumsum(sizes)])
    col = 0
    for g, (s, e_g) in enumerate(zip(sizes, ecounts)):
        s, e_g = int(s), int(e_g)
        sub = stacked[:, col:col + e_g]
        col += e_g
        if s == 0:
            assert np.all(pooled[g] == 0.0)
            continue
        ref, scale = oracle.gcn_aggregate(sub, s, x[offs[g]:offs[g] + s], None, 1, 1.0)
        assert_scaled_close(h_np[offs[g]:offs[g] + s], ref, scale, TOL_F32, f"graph {g}")
        ref_p, sc_p = oracle.segment_pool_meanmax(h_np[offs[g]:offs[g] + s], np.zeros(s, np.int64), 1)
        assert_scaled_close(pooled[g, :f], ref_p[0, :f], sc_p[0, :f], TOL_F32, f"mean {g}")
        assert_exact_f32(pooled[g, f:], ref_p[0, f:], f"max {g}")
