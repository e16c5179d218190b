"""Backward of the dot-product attention aggregation against the fp64 oracle.

The oracle's backward is pinned by central finite differences of the forward
oracle (test_oracle_pins.py).  Each gradient element must lie within
tol * scale, scale the oracle's sum of absolute terms of the same sums;
tol = 1e-5 + kappa_dot(C) * max(lam_e + lam_max), the attention-weight bound
of the forward tests (every term carries one weight, recomputed in fp32 from
the logits).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2101_11552_gb300 import graphgen as gg
from paper_2101_11552_gb300 import tfg
from _helpers import TOL_F32, assert_scaled_close, csr_rows, dev, dot_logit_mag, kappa_dot

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_11552_gb300 import build
    build.build_library()


def _qkv(n, f, seed, dtype):
    rng = np.random.default_rng(seed)
    host = [rng.standard_normal((n, f)).astype(np.float32) for _ in range(3)]
    if dtype == "bf16":
        bits = [gg.bf16_bits_rne(a) for a in host]
        return [dev(b.view(np.int16)).view(torch.bfloat16) for b in bits], bits
    return [dev(a) for a in host], host


def _run(ei, n, qkv, heads, channels, scale, g):
    e = dev(ei)
    csr = tfg.tfg_build_csr(e, n)
    csr_src = tfg.tfg_build_csr_by_source(e, n)
    tfg.check_status(csr.status)
    tfg.check_status(csr_src.status)
    out, _ = tfg.tfg_dot_edge_softmax_aggregate(csr.rowptr, csr.col, *qkv, heads, channels,
                                                scale=scale)
    grads = tfg.tfg_dot_edge_softmax_aggregate_backward(
        csr.rowptr, csr.col, csr_src.rowptr, csr_src.col, *qkv, heads, channels, scale, out,
        dev(g))
    torch.cuda.synchronize()
    return [t.cpu().numpy() for t in grads], csr


def _tol(host, heads, channels, scale, csr):
    rowptr, col = csr.rowptr.cpu().numpy(), csr.col.cpu().numpy()
    if len(col) == 0:
        return TOL_F32
    row = csr_rows(rowptr)
    lam = dot_logit_mag(oracle.widen(host[0]), oracle.widen(host[1]), col, row, heads, channels,
                        scale)
    lam_max = np.zeros((len(rowptr) - 1, heads))
    np.maximum.at(lam_max, row, lam)
    return TOL_F32 + kappa_dot(channels) * float(np.max(lam + lam_max[row]))


def _check(got, ref, tol, what):
    (gq, gk, gv), (rq, rk, rv, (sq, sk, sv)) = got, ref
    assert_scaled_close(gq, rq, sq, tol, "grad_q " + what)
    assert_scaled_close(gk, rk, sk, tol, "grad_k " + what)
    assert_scaled_close(gv, rv, sv, tol, "grad_v " + what)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("heads,channels", [(8, 16), (4, 8), (2, 32), (1, 64), (16, 2), (1, 1),
                                            (2, 128), (4, 4)])
def test_dot_backward_matches_oracle(heads, channels, dtype):
    n, e = 2500, 30000
    f = heads * channels
    wl = gg.random_edge_case_graph(n, e, 1, 23 + f, hub=3, isolated=20)
    qkv, host = _qkv(n, f, 7 * heads + channels, dtype)
    scale = float(np.float32(1.0 / np.sqrt(channels)))
    g = np.random.default_rng(f).standard_normal((n, f)).astype(np.float32)
    got, csr = _run(wl.edge_index, n, qkv, heads, channels, scale, g)
    ref = oracle.dot_softmax_backward(wl.edge_index, n, *host, heads, channels, scale, g)
    _check(got, ref, _tol(host, heads, channels, scale, csr), f"{dtype} H={heads} C={channels}")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_dot_backward_unaligned_rows_take_the_general_kernels(dtype):
    """q, k, v shifted off 16-byte alignment run the general kernels (the
    aligned 8 x 16 layout runs the fast ones); both meet the oracle's bound."""
    heads, channels = 8, 16
    n, f = 2000, heads * channels
    wl = gg.random_edge_case_graph(n, 25000, 1, 43, hub=2, isolated=20)
    qkv, host = _qkv(n, f, 44, dtype)
    shifted = []
    for t in qkv:
        buf = torch.empty(n * f + 1, dtype=t.dtype, device=t.device)
        buf[1:].copy_(t.reshape(-1))
        shifted.append(buf[1:].view(n, f))
    g = np.random.default_rng(45).standard_normal((n, f)).astype(np.float32)
    ref = oracle.dot_softmax_backward(wl.edge_index, n, *host, heads, channels, 0.25, g)
    for xs, what in ((shifted, "unaligned"), (qkv, "aligned")):
        got, csr = _run(wl.edge_index, n, xs, heads, channels, 0.25, g)
        _check(got, ref, _tol(host, heads, channels, 0.25, csr), f"{what} {dtype}")


def test_dot_backward_hub_rows_and_degenerate_graphs():
    """A 20k-edge hub, then graphs with no edges and one node with self-loops."""
    heads, channels = 8, 16
    f = heads * channels
    n = 3000
    wl = gg.random_edge_case_graph(n, 40000, 1, 5, hub=0, isolated=10)
    qkv, host = _qkv(n, f, 4, "f32")
    g = np.random.default_rng(1).standard_normal((n, f)).astype(np.float32)
    got, csr = _run(wl.edge_index, n, qkv, heads, channels, 0.25, g)
    ref = oracle.dot_softmax_backward(wl.edge_index, n, *host, heads, channels, 0.25, g)
    _check(got, ref, _tol(host, heads, channels, 0.25, csr), "hub")
    for n, ei in ((40, np.zeros((2, 0), np.int64)), (1, np.zeros((2, 3), np.int64))):
        qkv, host = _qkv(n, f, n, "f32")
        g = np.random.default_rng(n).standard_normal((n, f)).astype(np.float32)
        got, _ = _run(ei, n, qkv, heads, channels, 0.25, g)
        ref = oracle.dot_softmax_backward(ei, n, *host, heads, channels, 0.25, g)
        _check(got, ref, TOL_F32, f"n={n}")


def test_dot_backward_is_deterministic_and_rejects_bad_layouts():
    heads, channels = 4, 16
    n = 2000
    wl = gg.random_edge_case_graph(n, 30000, 1, 9, hub=2, isolated=10)
    qkv, _ = _qkv(n, heads * channels, 3, "bf16")
    g = np.random.default_rng(2).standard_normal((n, heads * channels)).astype(np.float32)
    a, _ = _run(wl.edge_index, n, qkv, heads, channels, 0.25, g)
    b, _ = _run(wl.edge_index, n, qkv, heads, channels, 0.25, g)
    for u, v in zip(a, b):
        assert np.array_equal(u, v)
    with pytest.raises(tfg.TfgError):
        tfg.tfg_dot_edge_softmax_backward_workspace_size(100, 2, 24)
    with pytest.raises(tfg.TfgError):
        tfg.tfg_dot_edge_softmax_backward_workspace_size(100, 4, 128)
