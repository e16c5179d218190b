"""The allocation-free edge-softmax entry point against the regular one.

tfg_edge_softmax_aggregate_noalloc is for callers that cannot allocate
device memory during the call (graph capture, plugin hosts that own all
memory, fixed-budget real-time pipelines): its scratch is a fixed array
inside the library.  It must give the same results as
tfg_edge_softmax_aggregate on the same inputs, call after call, even though
every call reuses the same scratch.  This file is collected last on purpose.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2101_11552_gb300 import graphgen as gg
from paper_2101_11552_gb300 import tfg
from _helpers import TOL_F32, assert_scaled_close, dev

pytestmark = pytest.mark.gpu


def _case(seed, n, e, heads, channels, dtype):
    wl = gg.random_edge_case_graph(n, e, heads * channels, seed, hub=3, isolated=7)
    rng = np.random.default_rng(seed)
    a_s = rng.standard_normal(heads * channels).astype(np.float32)
    a_d = rng.standard_normal(heads * channels).astype(np.float32)
    if dtype == "bf16":
        x = dev(wl.x_bf16.view(np.int16)).view(torch.bfloat16)
        xh = wl.x_bf16
    else:
        x = dev(wl.x)
        xh = wl.x
    return wl, x, xh, a_s, a_d


def test_noalloc_matches_regular_entry_point_twice():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_11552_gb300 import build
    build.build_library()
    # two calls in a row with different graphs and shapes: the second must
    # not see anything the first left in the shared scratch
    for seed, (n, e, heads, channels, dtype) in enumerate(
            [(5000, 60000, 8, 16, "bf16"), (3000, 20000, 4, 8, "f32")]):
        wl, x, xh, a_s, a_d = _case(11 + seed, n, e, heads, channels, dtype)
        csr = tfg.tfg_build_csr(dev(wl.edge_index), n)
        tfg.check_status(csr.status)
        out_ref, al_ref = tfg.tfg_edge_softmax_aggregate(csr.rowptr, csr.col, x, heads, channels,
                                                         dev(a_s), dev(a_d), 0.2, want_alpha=True)
        out = torch.empty(n, heads * channels, dtype=torch.float32, device="cuda")
        alpha = torch.empty(e, heads, dtype=torch.float32, device="cuda")
        got, got_alpha = tfg.tfg_edge_softmax_aggregate_noalloc(
            csr.rowptr, csr.col, x, heads, channels, dev(a_s), dev(a_d), 0.2, out=out, alpha=alpha)
        torch.cuda.synchronize()
        ref, _, scale = oracle.edge_softmax(wl.edge_index, n, xh, heads, channels, a_s, a_d, 0.2)
        assert_scaled_close(got.cpu().numpy(), out_ref.cpu().numpy().astype(np.float64), scale,
                            TOL_F32, f"noalloc vs regular, call {seed + 1}")
        assert_scaled_close(got.cpu().numpy(), ref, scale, TOL_F32, f"noalloc vs oracle, call {seed + 1}")
        np.testing.assert_allclose(got_alpha.cpu().numpy(), al_ref.cpu().numpy(), rtol=TOL_F32,
                                   atol=1e-7)


def test_noalloc_rejects_inputs_beyond_its_scratch():
    from paper_2101_11552_gb300 import build
    build.build_library()
    fake = tfg.ctypes.c_void_p(0x1000)   # never dereferenced: the size check fails first
    rc = tfg.lib().tfg_edge_softmax_aggregate_noalloc(fake, fake, fake, 0, 300_000, 10, 8, 16, fake,
                                                      fake, 0.2, fake, None, None)
    assert rc == tfg.TFG_ERR_TOO_LARGE
    assert "scratch" in tfg.tfg_last_error()
