"""Dot-product (Transformer-style) edge-softmax aggregation against the oracle.

Tolerances as for the additive form: out within TOL_F32 of the oracle's
sum of alpha |v| (the oracle reads the same bf16 values, so fp32 arithmetic
is the only error); alpha within alpha * (TOL_F32 + kappa (lam_e + lam_max))
with lam = scale * sum |q k| the magnitude each logit is computed from.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2101_11552_gb300 import graphgen as gg
from paper_2101_11552_gb300 import tfg
from _helpers import TOL_F32, assert_alpha_close, assert_scaled_close, csr_rows, dev, dot_logit_mag, kappa_dot

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


LAYOUTS = [  # (heads, channels): which kernel runs is noted per dtype
    (8, 16),     # fast: 2 lanes per head (bf16), 4 (fp32)
    (1, 128),    # fast: 16 / 32 lanes per head
    (2, 256),    # bf16 fast over two row tiles; fp32 general (8 chunks of 32)
    (4, 64),     # fp32 fast over two row tiles
    (16, 4),     # fp32 fast with 1 lane per head; bf16 general
    (3, 7),      # general
    (2, 40),     # general (5 lanes per head is not a power of two)
]


@pytest.mark.parametrize("heads,channels", LAYOUTS)
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_dot_softmax_matches_oracle(heads, channels, dtype):
    n, e = 3000, 40000
    f = heads * channels
    wl = gg.random_edge_case_graph(n, e, 1, 61 + f, hub=3, isolated=40)
    (q, k, v), host = _qkv(n, f, heads * 1000 + channels, dtype)
    csr = tfg.tfg_build_csr(dev(wl.edge_index), n)
    tfg.check_status(csr.status)
    out, alpha = tfg.tfg_dot_edge_softmax_aggregate(csr.rowptr, csr.col, q, k, v, heads,
                                                    channels, want_alpha=True)
    scale = float(np.float32(1.0 / np.sqrt(channels)))
    ref, ref_alpha, sc = oracle.dot_softmax(wl.edge_index, n, *host, heads, channels, scale)
    assert_scaled_close(out.cpu().numpy(), ref, sc, TOL_F32, f"dot {dtype} H={heads} C={channels}")
    rowptr, col, perm, _ = oracle.build_csr(wl.edge_index, n)
    row = csr_rows(rowptr)
    lam = dot_logit_mag(oracle.widen(host[0]), oracle.widen(host[1]), col, row, heads, channels,
                        scale)
    assert_alpha_close(alpha.cpu().numpy(), ref_alpha[perm], lam, row, kappa_dot(channels),
                       f"dot alpha {dtype} H={heads} C={channels}")


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_dot_softmax_unaligned_rows_take_the_general_kernel(dtype):
    """Rows shifted off 16-byte alignment run the general kernel; it computes
    the same definition (checked against the oracle and the fast kernel)."""
    n, e, heads, channels = 2000, 30000, 8, 16
    f = heads * channels
    wl = gg.random_edge_case_graph(n, e, 1, 17, hub=2, isolated=20)
    (q, k, v), host = _qkv(n, f, 5, dtype)
    shifted = []
    for t in (q, k, v):
        buf = torch.empty(n * f + 1, dtype=t.dtype, device=t.device)
        buf[1:].copy_(t.reshape(-1))
        shifted.append(buf[1:].view(n, f))
    csr = tfg.tfg_build_csr(dev(wl.edge_index), n)
    out_u, _ = tfg.tfg_dot_edge_softmax_aggregate(csr.rowptr, csr.col, *shifted, heads, channels)
    out_a, _ = tfg.tfg_dot_edge_softmax_aggregate(csr.rowptr, csr.col, q, k, v, heads, channels)
    ref, _, sc = oracle.dot_softmax(wl.edge_index, n, *host, heads, channels,
                                    float(np.float32(0.25)))
    assert_scaled_close(out_u.cpu().numpy(), ref, sc, TOL_F32, "dot unaligned")
    assert_scaled_close(out_a.cpu().numpy(), out_u.cpu().numpy().astype(np.float64), sc,
                        2 * TOL_F32, "fast vs general")


def test_dot_softmax_degenerate_graphs():
    heads, channels = 2, 16
    f = heads * channels
    for n, e in ((1, 0), (50, 0), (1, 3)):
        ei = np.zeros((2, e), np.int64)        # (1, 3): three self-loops on node 0
        (q, k, v), host = _qkv(n, f, n + e, "f32")
        csr = tfg.tfg_build_csr(dev(ei), n)
        out, alpha = tfg.tfg_dot_edge_softmax_aggregate(csr.rowptr, csr.col, q, k, v, heads,
                                                        channels, want_alpha=e > 0)
        ref, ref_alpha, sc = oracle.dot_softmax(ei, n, *host, heads, channels,
                                                float(np.float32(0.25)))
        assert_scaled_close(out.cpu().numpy(), ref, sc, TOL_F32, f"dot n={n} e={e}")
        if e:
            np.testing.assert_allclose(alpha.cpu().numpy(), 1.0 / 3.0, rtol=1e-6)


def test_dot_softmax_is_deterministic_and_rejects_bad_args():
    n, e, heads, channels = 4000, 60000, 8, 16
    wl = gg.random_edge_case_graph(n, e, 1, 3, hub=2, isolated=10)
    (q, k, v), _ = _qkv(n, heads * channels, 9, "bf16")
    csr = tfg.tfg_build_csr(dev(wl.edge_index), n)
    a, _ = tfg.tfg_dot_edge_softmax_aggregate(csr.rowptr, csr.col, q, k, v, heads, channels)
    b, _ = tfg.tfg_dot_edge_softmax_aggregate(csr.rowptr, csr.col, q, k, v, heads, channels)
    assert torch.equal(a, b)
    with pytest.raises(tfg.TfgError):
        tfg.tfg_dot_edge_softmax_aggregate(csr.rowptr, csr.col, q, k, v, heads, channels,
                                           scale=float("inf"))
    big = torch.zeros(10, 300, dtype=torch.float32, device="cuda")
    r = torch.zeros(11, dtype=torch.int32, device="cuda")
    with pytest.raises(tfg.TfgError):
        tfg.tfg_dot_edge_softmax_aggregate(r, r[:0], big, big, big, 1, 300)
