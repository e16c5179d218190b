"""The bounds-checked debug build (TFG_CHECK_BOUNDS=1).

Valid calls give the default build's results bit for bit; bad index arrays
and too-small buffers are refused with an error code before any launch.  Every planted fault here is also harmless if it were launched: bad
ids point into padding rows that exist, a decreasing rowptr stays inside
[0, E], and the too-small buffer is only ever read at ids below the rows it
holds -- so a missing check shows up as a failed assertion, never as a bad
memory access.
"""
import numpy as np
import pytest
import torch

from paper_2101_11552_gb300 import build
from paper_2101_11552_gb300 import graphgen as gg
from paper_2101_11552_gb300 import tfg
from _helpers import dev

pytestmark = pytest.mark.gpu

N, E, F = 2000, 30000, 64


@pytest.fixture(scope="module")
def checked():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build_library()
    path = build.build_library(defines=("TFG_CHECK_BOUNDS=1",),
                               lib_path=build.os.path.join(build.OBJ_DIR, "libtfg_checked.so"))
    wl = gg.random_edge_case_graph(N, E, F, 91, hub=2, isolated=10)
    yield path, wl
    tfg.use_library(build.LIB_PATH)


def _with(path, fn):
    tfg.use_library(path)
    try:
        return fn()
    finally:
        tfg.use_library(build.LIB_PATH)


def _expect(path, fn, code, words):
    with pytest.raises(tfg.TfgError) as ei:
        _with(path, fn)
    assert ei.value.code == code, str(ei.value)
    for w in words:
        assert w in str(ei.value), str(ei.value)


def test_checked_build_reports_itself(checked):
    path, _ = checked
    assert tfg.lib().tfg_check_bounds_enabled() == 0
    assert _with(path, lambda: tfg.lib().tfg_check_bounds_enabled()) == 1


def test_valid_calls_match_the_default_build(checked):
    path, wl = checked
    ei, x = dev(wl.edge_index), dev(wl.x)
    a_s = dev(np.linspace(-1, 1, F).astype(np.float32))

    def run():
        csr = tfg.tfg_build_csr(ei, N)
        dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, N, None, 1, 1.0, want_w_csr=False)
        h = tfg.tfg_gcn_aggregate_sum(csr.rowptr, csr.col, dinv, x, None, 1, 1.0)
        att, _ = tfg.tfg_edge_softmax_aggregate(csr.rowptr, csr.col, x, 4, 16, a_s, a_s, 0.2)
        mx = tfg.tfg_aggregate_max(csr.rowptr, csr.col, x)
        torch.cuda.synchronize()
        return [t.clone() for t in (csr.rowptr, csr.col, csr.perm, h, att, mx)]

    want = run()
    got = _with(path, run)
    for g, w in zip(got, want):
        assert torch.equal(g, w)


def test_col_id_outside_the_graph_is_refused(checked):
    path, wl = checked
    csr = tfg.tfg_build_csr(dev(wl.edge_index), N)
    col = torch.zeros(E + 64, dtype=torch.int32, device="cuda")
    col[:E] = csr.col
    col[E // 2] = N + 3                               # a row that the padding below holds
    xpad = torch.zeros(N + 64, F, device="cuda")
    xpad[:N] = dev(wl.x)
    _expect(path, lambda: tfg.tfg_aggregate_sum(csr.rowptr, col[:E], xpad[:N]),
            tfg.TFG_ERR_INDEX_RANGE, ["col", "outside [0, N)"])
    col[E // 2] = -1
    _expect(path, lambda: tfg.tfg_aggregate_sum(csr.rowptr, col[:E], xpad[:N]),
            tfg.TFG_ERR_INDEX_RANGE, ["outside [0, N)"])


def test_bad_rowptr_is_refused(checked):
    path, wl = checked
    csr = tfg.tfg_build_csr(dev(wl.edge_index), N)
    x = dev(wl.x)
    rp = csr.rowptr.clone()
    a, b = int(rp[100]), int(rp[101])
    if a == b:
        b = a + 1
    rp[100], rp[101] = b, a                          # a decrease, values still in [0, E]
    _expect(path, lambda: tfg.tfg_aggregate_sum(rp, csr.col, x), tfg.TFG_ERR_INDEX_RANGE,
            ["rowptr decreases"])
    # rowptr[N] must equal the E the call is given
    _expect(path, lambda: tfg.tfg_edge_softmax_aggregate(csr.rowptr, csr.col[:E - 5], x, 4, 16,
                                                         dev(np.ones(F, np.float32)),
                                                         dev(np.ones(F, np.float32)), 0.2),
            tfg.TFG_ERR_INDEX_RANGE, ["rowptr[N]"])


def test_feature_buffer_smaller_than_num_nodes_rows_is_refused(checked):
    path, _ = checked
    # x = the last k rows of an allocation of its own: the call says N rows
    k = 256
    torch.cuda.empty_cache()
    # 32 MiB: the caching allocator rounds requests of 10 MiB and more to 2 MiB and gives
    # them a segment of exactly that size
    buf = torch.zeros((32 << 20) // 4, device="cuda")
    seg = [s for s in torch.cuda.memory_snapshot()
           if s["address"] <= buf.data_ptr() < s["address"] + s["total_size"]]
    if not seg or seg[0]["address"] + seg[0]["total_size"] != buf.data_ptr() + buf.numel() * 4:
        pytest.skip("the caching allocator did not give the buffer a segment of its own")
    x = buf[-k * F:].view(k, F)
    # every id below k: even an unchecked launch would read inside the k rows
    n = 1000
    src = np.random.default_rng(3).integers(0, k, 4000)
    dst = np.random.default_rng(4).integers(0, n, 4000)
    csr = tfg.tfg_build_csr(dev(np.stack([src, dst]).astype(np.int64)), n)
    out = torch.empty(n, F, device="cuda")

    def call():   # the C entry point with N = n rows of x (the binding would refuse the shape)
        return tfg.lib().tfg_aggregate_sum(tfg._ptr(csr.rowptr), tfg._ptr(csr.col), None,
                                           tfg._ptr(x), tfg.TFG_F32, n, F, tfg._ptr(out),
                                           tfg._stream(torch.device("cuda")))

    tfg.use_library(path)
    try:
        rc = call()
        msg = tfg.tfg_last_error()
    finally:
        tfg.use_library(build.LIB_PATH)
    assert rc == tfg.TFG_ERR_INDEX_RANGE and "x must hold" in msg, (rc, msg)


def test_backward_index_arrays_are_checked(checked):
    """A bad id in the source-grouped CSR of a backward call, and a perm id
    outside [0, E), are refused (the padded buffers keep even a launch in
    bounds)."""
    path, wl = checked
    ei = dev(wl.edge_index)
    csr = tfg.tfg_build_csr(ei, N)
    src = tfg.tfg_build_csr_by_source(ei, N)
    g = torch.randn(N, F, device="cuda")
    dinv, _ = tfg.tfg_gcn_norm(csr.rowptr, csr.col, csr.perm, N, None, 1, 1.0, want_w_csr=False)
    colp = torch.zeros(E + 64, dtype=torch.int32, device="cuda")
    colp[:E] = src.col
    colp[7] = N + 1                                    # a row the padding of gpad holds
    gpad = torch.zeros(N + 64, F, device="cuda")
    gpad[:N] = g
    bad = src._replace(col=colp[:E])
    _expect(path, lambda: tfg.tfg_gcn_aggregate_backward(bad, dinv, gpad[:N], 1, 1.0),
            tfg.TFG_ERR_INDEX_RANGE, ["col", "outside [0, N)"])
    permp = csr.perm.clone()
    permp[11] = E + 2       # only ever copied into argmax, never used as an address
    x = dev(wl.x)
    _expect(path, lambda: tfg.tfg_aggregate_max_argmax(csr._replace(perm=permp), x),
            tfg.TFG_ERR_INDEX_RANGE, ["perm id lies outside [0, E)"])
