"""Full-size dense-community workload (232,965 nodes, 114.6M edges, bf16 F=128).

Exactly the calls and launch configuration the benchmark times.  The CSR,
in-degrees and dinv are compared whole; the aggregations on sampled rows
(every hub above the CTA-cooperative threshold that the sample reaches, the
highest-degree rows and a seeded random sample), which the oracle computes
one by one from its own stable CSR.  Pooling is compared whole.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2101_11552_gb300 import graphgen as gg
from paper_2101_11552_gb300 import tfg
from _helpers import (KAPPA_GAT, TOL_F32, assert_alpha_close, assert_exact_f32, assert_scaled_close,
                      dev, dot_logit_mag, gat_logit_mag, kappa_dot, row_edges)

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module")
def dcsbm():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_11552_gb300 import build
    build.build_library()
    wl = gg.make_dcsbm_232965()
    ocsr = oracle.build_csr(wl.edge_index, wl.num_nodes)
    ei = dev(wl.edge_index)
    csr = tfg.tfg_build_csr(ei, wl.num_nodes)
    tfg.check_status(csr.status)
    del ei
    deg = ocsr[3]
    rng = np.random.default_rng(7)
    top = np.argsort(deg)[-64:]
    low = np.argsort(deg)[:16]
    rows = np.unique(np.concatenate([top, low, rng.choice(wl.num_nodes, 1500, replace=False),
                                     [0, wl.num_nodes - 1]])).astype(np.int64)
    return wl, ocsr, csr, rows


def test_dcsbm_csr_bit_exact(dcsbm):
    wl, ocsr, csr, _ = dcsbm
    for name, g, w in zip(("rowptr", "col", "perm", "in_degree"), csr[:4], ocsr):
        assert np.array_equal(g.cpu().numpy(), w), name
    c32 = tfg.tfg_build_csr(dev(wl.edge_index.astype(np.int32)), wl.num_nodes)
    tfg.check_status(c32.status)
    for name, g, w in zip(("rowptr", "col", "perm", "in_degree"), c32[:4], csr[:4]):
        assert torch.equal(g, w), f"int32 edge list: {name}"


def test_dcsbm_gcn_bf16_sampled_rows(dcsbm):
    wl, ocsr, csr, rows = dcsbm
    n = wl.num_nodes
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, 1, 1.0, want_w_csr=False)
    ref_norm = oracle.gcn_norm(wl.edge_index, n, None, 1, 1.0)
    np.testing.assert_allclose(dinv.cpu().numpy(), ref_norm["dinv"], rtol=2e-6, atol=0)
    x = dev(wl.x_bf16.view(np.int16)).view(torch.bfloat16)
    out = tfg.tfg_gcn_aggregate_sum(csr.rowptr, csr.col, dinv, x, None, 1, 1.0)
    got = out[dev(rows)].cpu().numpy()
    w_norm = ref_norm["w_norm"]
    ref, scale = oracle.aggregate_rows(ocsr, n, wl.x_bf16, "sum", rows, w=w_norm,
                                       self_w=ref_norm["self_w"])
    # the oracle reads the same bf16 values: fp32 accumulation is the only error
    assert_scaled_close(got, ref, scale, TOL_F32, "dcsbm gcn bf16")


def test_dcsbm_edge_softmax_sampled_rows(dcsbm):
    wl, ocsr, csr, rows = dcsbm
    n = wl.num_nodes
    x = dev(wl.x_bf16.view(np.int16)).view(torch.bfloat16)
    out, alpha = tfg.tfg_edge_softmax_aggregate(csr.rowptr, csr.col, x, wl.heads,
                                                wl.channels, dev(wl.a_src), dev(wl.a_dst),
                                                wl.negative_slope, want_alpha=True)
    sub = rows[:400]
    ref, ref_alpha, scale = oracle.edge_softmax_rows(ocsr, n, wl.x_bf16, wl.heads, wl.channels,
                                                     wl.a_src, wl.a_dst, wl.negative_slope, sub)
    got = out[dev(sub)].cpu().numpy()
    assert_scaled_close(got, ref, scale, TOL_F32, "dcsbm softmax")
    rp = ocsr[0]
    got_alpha = np.concatenate([alpha[int(rp[r]):int(rp[r + 1])].cpu().numpy() for r in sub])
    src, dst, row = row_edges(ocsr, sub)
    lam = gat_logit_mag(oracle.widen(wl.x_bf16), src, dst, wl.heads, wl.channels, wl.a_src,
                        wl.a_dst)
    assert_alpha_close(got_alpha, ref_alpha, lam, row, KAPPA_GAT, "dcsbm alpha")


def test_dcsbm_max_and_mean_sampled_rows(dcsbm):
    wl, ocsr, csr, rows = dcsbm
    n = wl.num_nodes
    x = dev(wl.x_bf16.view(np.int16)).view(torch.bfloat16)
    for reduce, fn in (("max", tfg.tfg_aggregate_max), ("mean", tfg.tfg_aggregate_mean)):
        got = fn(csr.rowptr, csr.col, x)[dev(rows)].cpu().numpy()
        ref, scale = oracle.aggregate_rows(ocsr, n, wl.x_bf16, reduce, rows)
        if reduce == "max":
            assert_exact_f32(got, ref, "dcsbm max")
        else:
            assert_scaled_close(got, ref, scale, TOL_F32, "dcsbm mean")


def test_dcsbm_community_pool(dcsbm):
    wl, _, csr, _ = dcsbm
    x = dev(wl.x)
    for reduce in ("sum", "mean", "max"):
        out, status = tfg.tfg_segment_pool(x, dev(wl.batch), wl.num_graphs, reduce)
        tfg.check_status(status)
        ref, scale = oracle.segment_pool(wl.x, wl.batch, wl.num_graphs, reduce)
        if reduce == "max":
            assert_exact_f32(out.cpu().numpy(), ref, "dcsbm pool max")
        else:
            assert_scaled_close(out.cpu().numpy(), ref, scale, TOL_F32, f"dcsbm pool {reduce}")


def test_dcsbm_appnp_sqrt_degree_fixed_point(dcsbm):
    """On a symmetric graph with self-loops Ahat sqrt(d) = sqrt(d), so
    x0 = sqrt(d) v^T is a fixed point of every APPNP step; the error scale
    |Ahat|^k |x0| is |x0| itself."""
    wl, ocsr, csr, _ = dcsbm
    n = wl.num_nodes
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, 1, 1.0, want_w_csr=False)
    d = ocsr[3].astype(np.float64) + 1.0
    v = np.random.default_rng(21).standard_normal(128)
    x0 = (np.sqrt(d)[:, None] * v[None, :]).astype(np.float32)
    out = tfg.tfg_appnp_propagate(csr.rowptr, csr.col, dinv, dev(x0), 10, 0.1, add_self_loops=1)
    got = out.cpu().numpy()
    assert_scaled_close(got, x0.astype(np.float64), np.abs(x0).astype(np.float64), TOL_F32,
                        "dcsbm appnp fixed point")


def test_dcsbm_appnp_one_hop_sampled_rows_and_sgc_chain(dcsbm):
    wl, ocsr, csr, rows = dcsbm
    n = wl.num_nodes
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, 1, 1.0, want_w_csr=False)
    x = dev(wl.x_bf16.view(np.int16)).view(torch.bfloat16)
    alpha = 0.1
    out = tfg.tfg_appnp_propagate(csr.rowptr, csr.col, dinv, x, 1, alpha, add_self_loops=1)
    nrm = oracle.gcn_norm(wl.edge_index, n, None, 1, 1.0)
    agg, scale = oracle.aggregate_rows(ocsr, n, wl.x_bf16, "sum", rows, w=nrm["w_norm"],
                                       self_w=nrm["self_w"])
    x0 = oracle.widen(wl.x_bf16)[rows]
    ref = (1 - alpha) * agg + alpha * x0
    sc = (1 - alpha) * scale + alpha * np.abs(x0)
    assert_scaled_close(out[dev(rows)].cpu().numpy(), ref, sc, TOL_F32, "dcsbm appnp 1 hop")
    sgc = tfg.tfg_sgc_propagate(csr.rowptr, csr.col, dinv, x, 2, add_self_loops=1)
    h = tfg.tfg_gcn_aggregate_sum(csr.rowptr, csr.col, dinv, x, None, 1, 1.0)
    h = tfg.tfg_gcn_aggregate_sum(csr.rowptr, csr.col, dinv, h, None, 1, 1.0)
    assert torch.equal(sgc, h)


def test_dcsbm_dot_softmax_sampled_rows(dcsbm):
    """Transformer-style attention at full size: q, k, v bf16 [N, 8 x 16]."""
    wl, ocsr, csr, rows = dcsbm
    n = wl.num_nodes
    rng = np.random.default_rng(1305)
    bits = [gg.bf16_bits_rne(rng.standard_normal((n, 128), dtype=np.float32)) for _ in range(3)]
    q, k, v = (dev(b.view(np.int16)).view(torch.bfloat16) for b in bits)
    out, alpha = tfg.tfg_dot_edge_softmax_aggregate(csr.rowptr, csr.col, q, k, v, 8, 16,
                                                    want_alpha=True)
    sub = rows[:400]
    ref, ref_alpha, scale = oracle.dot_softmax_rows(ocsr, n, *bits, 8, 16, 0.25, sub)
    got = out[dev(sub)].cpu().numpy()
    assert_scaled_close(got, ref, scale, TOL_F32, "dcsbm dot softmax")
    rp = ocsr[0]
    got_alpha = np.concatenate([alpha[int(rp[r]):int(rp[r + 1])].cpu().numpy() for r in sub])
    src, dst, row = row_edges(ocsr, sub)
    lam = dot_logit_mag(oracle.widen(bits[0]), oracle.widen(bits[1]), src, dst, 8, 16, 0.25)
    assert_alpha_close(got_alpha, ref_alpha, lam, row, kappa_dot(16), "dcsbm dot alpha")


def test_dcsbm_gcn_backward_sampled_rows(dcsbm):
    """Backward of the GCN aggregation at full size: the CSR grouped by
    source, then the GCN kernel on it with the forward's dinv."""
    wl, ocsr, csr, rows = dcsbm
    n = wl.num_nodes
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, n, None, 1, 1.0, want_w_csr=False)
    ei = dev(wl.edge_index)
    csr_src = tfg.tfg_build_csr_by_source(ei, n)
    tfg.check_status(csr_src.status)
    del ei
    g = np.random.default_rng(31).standard_normal((n, 128)).astype(np.float32)
    got = tfg.tfg_gcn_aggregate_backward(csr_src, dinv, dev(g), 1, 1.0)[dev(rows)].cpu().numpy()
    ocsr_src = oracle.build_csr(np.ascontiguousarray(wl.edge_index[::-1]), n)
    assert np.array_equal(csr_src.rowptr.cpu().numpy(), ocsr_src[0])
    nrm = oracle.gcn_norm(wl.edge_index, n, None, 1, 1.0)
    # row s of the source-grouped CSR sums w_norm[e] * g[target]: the backward
    ref, scale = oracle.aggregate_rows(ocsr_src, n, g, "sum", rows, w=nrm["w_norm"],
                                       self_w=nrm["self_w"])
    assert_scaled_close(got, ref, scale, TOL_F32, "dcsbm gcn backward")


def _dependency_subgraph(wl, ocsr, sources):
    """Original ids (ascending) of every edge the backward rows of `sources`
    depend on: the in-edges of each source and of each target of its
    out-edges (the softmax of a target runs over all of its in-edges)."""
    ei = wl.edge_index
    out_targets = np.unique(ei[1][np.isin(ei[0], sources)])
    nodes = np.unique(np.concatenate([out_targets, sources]))
    rp, perm = np.asarray(ocsr[0], np.int64), np.asarray(ocsr[2], np.int64)
    ids = np.concatenate([perm[rp[t]:rp[t + 1]] for t in nodes])
    return np.sort(ids)


def _backward_sources(ocsr):
    deg = ocsr[3]
    rng = np.random.default_rng(41)
    hubs = np.argsort(deg)[-2:]
    low = np.argsort(deg)[:3]
    return np.unique(np.concatenate([hubs, low, rng.choice(len(deg), 10, replace=False)])).astype(np.int64)


def test_dcsbm_gat_backward_sampled_rows(dcsbm):
    """GAT backward at full size (the launch the benchmark's next-row times):
    grad_x of sampled nodes -- the two largest hubs, the lowest-degree nodes and a
    random sample -- against the oracle's backward on the exact sub-graph those
    rows depend on."""
    wl, ocsr, csr, _ = dcsbm
    n, h, c = wl.num_nodes, wl.heads, wl.channels
    ei = dev(wl.edge_index)
    csr_src = tfg.tfg_build_csr_by_source(ei, n)
    tfg.check_status(csr_src.status)
    del ei
    x = dev(wl.x_bf16.view(np.int16)).view(torch.bfloat16)
    a_s, a_d = dev(wl.a_src), dev(wl.a_dst)
    out, _ = tfg.tfg_edge_softmax_aggregate(csr.rowptr, csr.col, x, h, c, a_s, a_d,
                                            wl.negative_slope)
    g = np.random.default_rng(43).standard_normal((n, h * c)).astype(np.float32)
    gx, _, _ = tfg.tfg_edge_softmax_aggregate_backward(csr.rowptr, csr.col, csr_src.rowptr,
                                                       csr_src.col, x, h, c, a_s, a_d,
                                                       wl.negative_slope, out, dev(g))
    sources = _backward_sources(ocsr)
    got = gx[dev(sources)].cpu().numpy()
    ids = _dependency_subgraph(wl, ocsr, sources)
    sub = np.ascontiguousarray(wl.edge_index[:, ids])
    rgx, _, _, (sx, _, _) = oracle.edge_softmax_backward(sub, n, wl.x_bf16, h, c, wl.a_src,
                                                         wl.a_dst, wl.negative_slope, g)
    lam = gat_logit_mag(oracle.widen(wl.x_bf16), sub[0], sub[1], h, c, wl.a_src, wl.a_dst)
    lam_max = np.zeros((n, h))
    np.maximum.at(lam_max, sub[1], lam)
    tol = TOL_F32 + KAPPA_GAT * float(np.max(lam + lam_max[sub[1]]))
    assert_scaled_close(got, rgx[sources], sx[sources], tol, "dcsbm gat backward grad_x")


def test_dcsbm_dot_backward_sampled_rows(dcsbm):
    """Dot-product attention backward at full size: grad_q, grad_k and grad_v
    of the same sampled nodes against the oracle on their dependency
    sub-graph (q, k, v bf16 [N, 8 x 16] as in the forward test)."""
    wl, ocsr, csr, _ = dcsbm
    n = wl.num_nodes
    ei = dev(wl.edge_index)
    csr_src = tfg.tfg_build_csr_by_source(ei, n)
    tfg.check_status(csr_src.status)
    del ei
    rng = np.random.default_rng(1305)
    bits = [gg.bf16_bits_rne(rng.standard_normal((n, 128), dtype=np.float32)) for _ in range(3)]
    q, k, v = (dev(b.view(np.int16)).view(torch.bfloat16) for b in bits)
    out, _ = tfg.tfg_dot_edge_softmax_aggregate(csr.rowptr, csr.col, q, k, v, 8, 16, scale=0.25)
    g = np.random.default_rng(47).standard_normal((n, 128)).astype(np.float32)
    grads = tfg.tfg_dot_edge_softmax_aggregate_backward(csr.rowptr, csr.col, csr_src.rowptr,
                                                        csr_src.col, q, k, v, 8, 16, 0.25, out,
                                                        dev(g))
    sources = _backward_sources(ocsr)
    ids = _dependency_subgraph(wl, ocsr, sources)
    sub = np.ascontiguousarray(wl.edge_index[:, ids])
    rq, rk, rv, (sq, sk, sv) = oracle.dot_softmax_backward(sub, n, *bits, 8, 16, 0.25, g)
    lam = dot_logit_mag(oracle.widen(bits[0]), oracle.widen(bits[1]), sub[0], sub[1], 8, 16, 0.25)
    lam_max = np.zeros((n, 8))
    np.maximum.at(lam_max, sub[1], lam)
    tol = TOL_F32 + kappa_dot(16) * float(np.max(lam + lam_max[sub[1]]))
    for name, got, ref, sc in (("grad_q", grads[0], rq, sq), ("grad_k", grads[1], rk, sk),
                               ("grad_v", grads[2], rv, sv)):
        assert_scaled_close(got[dev(sources)].cpu().numpy(), ref[sources], sc[sources], tol,
                            f"dcsbm dot backward {name}")
