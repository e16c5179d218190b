"""The C ABI library loads, exports what include/tfg.h declares, and rejects
bad arguments on the host before enqueuing anything (no GPU needed)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "tfg.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2101_11552_gb300 import build, tfg
    build.build_library()
    return tfg.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(tfg_[a-z0-9_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for want in ["tfg_build_csr", "tfg_gcn_norm", "tfg_aggregate_sum", "tfg_aggregate_mean",
                 "tfg_aggregate_max", "tfg_gcn_aggregate_sum", "tfg_edge_softmax_aggregate",
                 "tfg_segment_pool", "tfg_last_error"]:
        assert want in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), f"{name} declared in tfg.h but not exported"


def test_version(lib):
    assert lib.tfg_version() == 300


def test_workspace_queries(lib):
    n = ctypes.c_size_t(0)
    assert lib.tfg_build_csr_workspace_size(232965, 114_600_000, ctypes.byref(n)) == 0
    # ping-pong (key, source, edge id) + final keys + digit histograms
    assert n.value >= 4 * 114_600_000 * 4
    assert lib.tfg_build_csr_workspace_size(10, 0, ctypes.byref(n)) == 0 and n.value > 0
    assert lib.tfg_edge_softmax_workspace_size(1000, 8, ctypes.byref(n)) == 0
    assert n.value >= 2 * 1000 * 8 * 4
    assert lib.tfg_build_csr_workspace_size(1 << 31, 5, ctypes.byref(n)) == -2
    assert lib.tfg_build_csr_workspace_size(-1, 5, ctypes.byref(n)) == -1


def err(lib):
    return lib.tfg_last_error().decode()


FAKE = ctypes.c_void_p(0x1000)   # never dereferenced: every call below fails validation first


def test_build_csr_rejects(lib):
    assert lib.tfg_build_csr(None, 10, 5, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, FAKE, None) == -1
    assert "edge_index" in err(lib)
    assert lib.tfg_build_csr(FAKE, 10, 1 << 31, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, FAKE, None) == -2
    assert lib.tfg_build_csr(FAKE, 10, 5, FAKE, FAKE, FAKE, FAKE, FAKE, 16, FAKE, None) == -3
    assert "workspace" in err(lib)
    assert lib.tfg_build_csr(FAKE, 10, 5, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, None, None) == -1
    assert lib.tfg_build_csr(FAKE, 10, 0, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, FAKE, None) == -1
    assert lib.tfg_build_csr(FAKE, -3, 5, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, FAKE, None) == -1
    unaligned = ctypes.c_void_p(0x1008)
    assert lib.tfg_build_csr(FAKE, 10, 5, FAKE, FAKE, FAKE, FAKE, unaligned, 1 << 20, FAKE, None) == -1


def test_aggregate_rejects(lib):
    for fn in (lib.tfg_aggregate_sum, lib.tfg_aggregate_mean, lib.tfg_aggregate_max):
        assert fn(FAKE, FAKE, None, FAKE, 0, 10, 0, FAKE, None) == -1       # F = 0
        assert fn(FAKE, FAKE, None, FAKE, 7, 10, 4, FAKE, None) == -1       # bad dtype
        assert fn(None, FAKE, None, FAKE, 0, 10, 4, FAKE, None) == -1       # rowptr
        assert fn(FAKE, FAKE, None, None, 0, 10, 4, FAKE, None) == -1       # x
        assert fn(FAKE, FAKE, None, FAKE, 0, 1 << 31, 4, FAKE, None) == -2  # N too large
    assert lib.tfg_gcn_aggregate_sum(FAKE, FAKE, None, None, FAKE, 0, 10, 4, 1, 1.0, FAKE, None) == -1
    assert "dinv" in err(lib)


def test_gcn_norm_rejects(lib):
    assert lib.tfg_gcn_norm(FAKE, FAKE, FAKE, None, 10, 20, 1, 1.0, None, None, None) == -1
    assert lib.tfg_gcn_norm(FAKE, None, FAKE, None, 10, 20, 1, 1.0, FAKE, FAKE, None) == -1


def test_edge_softmax_rejects(lib):
    f = lib.tfg_edge_softmax_aggregate
    assert f(FAKE, FAKE, FAKE, 0, 10, 20, 0, 4, FAKE, FAKE, 0.2, FAKE, None, FAKE, 1 << 20, None) == -1
    assert f(FAKE, FAKE, FAKE, 0, 10, 20, 2, 4, None, FAKE, 0.2, FAKE, None, FAKE, 1 << 20, None) == -1
    assert f(FAKE, FAKE, FAKE, 0, 10, 20, 2, 4, FAKE, FAKE, 0.2, FAKE, None, FAKE, 8, None) == -3
    assert f(FAKE, FAKE, FAKE, 9, 10, 20, 2, 4, FAKE, FAKE, 0.2, FAKE, None, FAKE, 1 << 20, None) == -1
    assert f(FAKE, None, FAKE, 0, 10, 20, 2, 4, FAKE, FAKE, 0.2, FAKE, None, FAKE, 1 << 20, None) == -1


def test_segment_pool_rejects(lib):
    f = lib.tfg_segment_pool
    assert f(FAKE, 0, FAKE, 10, 3, 4, 9, FAKE, FAKE, None) == -1        # reducer
    assert f(FAKE, 0, FAKE, 10, 3, 4, 0, FAKE, None, None) == -1        # status
    assert f(FAKE, 0, None, 10, 3, 4, 0, FAKE, FAKE, None) == -1        # batch
    assert f(FAKE, 0, FAKE, -1, 3, 4, 0, FAKE, FAKE, None) == -1
    assert f(FAKE, 5, FAKE, 10, 3, 4, 0, FAKE, FAKE, None) == -1        # dtype


def test_segment_pool_meanmax_rejects(lib):
    f = lib.tfg_segment_pool_meanmax
    assert f(FAKE, 0, FAKE, 10, 3, 4, FAKE, None, None) == -1            # status
    assert f(FAKE, 0, None, 10, 3, 4, FAKE, FAKE, None) == -1            # batch
    assert f(FAKE, 0, FAKE, 10, 3, 4, None, FAKE, None) == -1            # out
    assert f(FAKE, 5, FAKE, 10, 3, 4, FAKE, FAKE, None) == -1            # dtype
    assert f(FAKE, 0, FAKE, 10, -3, 4, FAKE, FAKE, None) == -1
    assert f(FAKE, 0, FAKE, 10, 3, 0, FAKE, FAKE, None) == -1            # F = 0


def test_batch_graphs_rejects(lib):
    n = ctypes.c_size_t(0)
    assert lib.tfg_batch_graphs_workspace_size(5, ctypes.byref(n)) == 0 and n.value >= 8 * 6
    assert lib.tfg_batch_graphs_workspace_size(-1, ctypes.byref(n)) == -1
    f = lib.tfg_batch_graphs
    ok = (FAKE, FAKE, FAKE, 10, 7, FAKE, FAKE, FAKE, FAKE, 1 << 12, FAKE, None)
    assert f(-1, *ok) == -1
    assert f(0, *ok) == -1                                               # nodes for zero graphs
    assert f(1 << 31, *ok) == -2
    assert f(3, FAKE, FAKE, FAKE, 10, 7, FAKE, FAKE, FAKE, FAKE, 16, FAKE, None) == -3
    assert "workspace" in err(lib)
    assert f(3, FAKE, FAKE, FAKE, 10, 7, FAKE, FAKE, FAKE, None, 1 << 12, FAKE, None) == -3
    assert f(3, None, FAKE, FAKE, 10, 7, FAKE, FAKE, FAKE, FAKE, 1 << 12, FAKE, None) == -1
    assert f(3, FAKE, FAKE, None, 10, 7, FAKE, FAKE, FAKE, FAKE, 1 << 12, FAKE, None) == -1
    assert f(3, FAKE, FAKE, FAKE, 10, 7, FAKE, FAKE, None, FAKE, 1 << 12, FAKE, None) == -1
    assert f(3, FAKE, FAKE, FAKE, 10, 7, FAKE, FAKE, FAKE, FAKE, 1 << 12, None, None) == -1
    assert f(3, FAKE, FAKE, FAKE, -10, 7, FAKE, FAKE, FAKE, FAKE, 1 << 12, FAKE, None) == -1


def test_propagate_rejects(lib):
    n = ctypes.c_size_t(0)
    assert lib.tfg_propagate_workspace_size(100, 8, 1, ctypes.byref(n)) == 0 and n.value == 0
    assert lib.tfg_propagate_workspace_size(100, 8, 3, ctypes.byref(n)) == 0 and n.value >= 3200
    assert lib.tfg_propagate_workspace_size(100, 8, -1, ctypes.byref(n)) == -1
    f = lib.tfg_appnp_propagate
    args = lambda **kw: [kw.get(k, v) for k, v in dict(
        rowptr=FAKE, col=FAKE, dinv=FAKE, w=None, x0=FAKE, dt=0, n=10, f=4, k=3, a=0.1, sl=1,
        fill=1.0, out=FAKE, ws=FAKE, wsb=1 << 12, st=None).items()]
    assert f(*args(k=-1)) == -1
    assert f(*args(k=1025)) == -1
    assert f(*args(a=1.5)) == -1
    assert f(*args(a=float("nan"))) == -1
    assert f(*args(dinv=None)) == -1
    assert f(*args(x0=None)) == -1
    assert f(*args(out=None)) == -1
    assert f(*args(dt=4)) == -1
    assert f(*args(f=0)) == -1
    assert f(*args(ws=None)) == -3
    assert f(*args(wsb=64)) == -3
    assert "workspace" in err(lib)
    assert f(*args(ws=ctypes.c_void_p(0x1004))) == -1           # unaligned workspace
    sgc = lib.tfg_sgc_propagate
    assert sgc(FAKE, FAKE, None, None, FAKE, 0, 10, 4, 2, 1, 1.0, FAKE, FAKE, 1 << 12, None) == -1


def test_dot_softmax_rejects(lib):
    f = lib.tfg_dot_edge_softmax_aggregate
    ok = dict(rp=FAKE, col=FAKE, q=FAKE, k=FAKE, v=FAKE, dt=0, n=10, e=20, h=2, c=8, s=0.25,
              out=FAKE, al=None, st=None)
    call = lambda **kw: f(*[kw.get(key, val) for key, val in ok.items()])  # noqa: E731
    assert call(h=0) == -1
    assert call(c=257) == -2
    assert call(dt=3) == -1
    assert call(s=float("inf")) == -1
    assert call(s=float("nan")) == -1
    assert call(q=None) == -1
    assert call(k=None) == -1
    assert call(v=None) == -1
    assert call(col=None) == -1
    assert call(out=None) == -1
    assert call(e=-1) == -1


def test_backward_rejects(lib):
    n = ctypes.c_size_t(0)
    assert lib.tfg_aggregate_backward_workspace_size(0, 100, ctypes.byref(n)) == 0 and n.value >= 400
    assert lib.tfg_aggregate_backward_workspace_size(2, 100, ctypes.byref(n)) == -1     # max
    f = lib.tfg_aggregate_backward
    ok = dict(r=0, rp=FAKE, col=FAKE, perm=FAKE, w=None, deg=None, g=FAKE, n=10, e=20, f=4,
              gx=FAKE, ws=FAKE, wsb=1 << 12, st=None)
    call = lambda **kw: f(*[kw.get(key, val) for key, val in ok.items()])  # noqa: E731
    assert call(r=2) == -1
    assert call(r=1) == -1               # the mean needs in_degree
    assert call(r=1, deg=FAKE, perm=None) == -1
    assert call(w=FAKE, perm=None) == -1
    assert call(w=FAKE, ws=None) == -3
    assert call(g=None) == -1
    assert call(gx=None) == -1
    assert call(f=0) == -1
    assert lib.tfg_gcn_aggregate_backward(FAKE, FAKE, None, FAKE, 10, 4, 1, 1.0, FAKE, None) == -1
    am = lib.tfg_aggregate_max_argmax
    assert am(FAKE, FAKE, None, None, FAKE, 0, 10, 4, FAKE, FAKE, None) == -1           # perm
    assert am(FAKE, FAKE, FAKE, None, FAKE, 0, 10, 4, FAKE, None, None) == -1           # argmax
    assert am(FAKE, FAKE, FAKE, None, FAKE, 3, 10, 4, FAKE, FAKE, None) == -1           # dtype
    mb = lib.tfg_aggregate_max_backward
    assert mb(FAKE, FAKE, None, FAKE, None, FAKE, 10, 30, 4, FAKE, None, 0, None) == -1   # perm_src
    assert mb(FAKE, FAKE, FAKE, None, None, FAKE, 10, 30, 4, FAKE, None, 0, None) == -1   # argmax
    assert mb(FAKE, None, FAKE, FAKE, None, FAKE, 10, 30, 4, FAKE, None, 0, None) == -1   # col_src
    assert mb(FAKE, FAKE, FAKE, FAKE, None, FAKE, 10, 320, 4, FAKE, FAKE, 256, None) == -3  # workspace
    assert mb(FAKE, FAKE, FAKE, FAKE, None, FAKE, 10, 320, 4, FAKE, ctypes.c_void_p(0x1004), 1 << 20, None) == -1
    nb = ctypes.c_size_t(0)
    ws = lib.tfg_aggregate_max_backward_workspace_size
    assert ws(10, 320, 4, ctypes.byref(nb)) == 0
    assert nb.value == 512                           # a mark byte per edge, 256-byte rounded
    assert ws(2, 300, 4000, ctypes.byref(nb)) == 0 and nb.value == 512
    assert ws(10, 39, 4, ctypes.byref(nb)) == 0 and nb.value == 0      # E < 4 N: no marks
    assert ws(100, 12799, 200, ctypes.byref(nb)) == 0 and nb.value == 0  # E < 128 N: no marks
    assert ws(100, 12800, 200, ctypes.byref(nb)) == 0 and nb.value == 12800
    assert ws(10, 0, 4, ctypes.byref(nb)) == 0 and nb.value == 0
    assert ws(10, -1, 4, ctypes.byref(nb)) == -1
    assert lib.tfg_build_csr_by_source(None, 10, 5, FAKE, FAKE, FAKE, FAKE, FAKE, 1 << 20, FAKE, None) == -1


def test_gather_xor_rejects(lib):
    g = lib.tfg_gather_xor
    assert g(FAKE, 10, FAKE, 5, 48, FAKE, None) == -1            # not a power of two
    assert "row_bytes" in lib.tfg_last_error().decode()
    assert g(FAKE, 10, FAKE, 5, 1024, FAKE, None) == -1          # above 512
    assert g(FAKE, 10, FAKE, 5, 8, FAKE, None) == -1             # below 16
    assert g(None, 10, FAKE, 5, 256, FAKE, None) == -1
    assert g(FAKE, 10, FAKE, 5, 256, None, None) == -1
    assert g(FAKE, 10, ctypes.c_void_p(0x1004), 5, 256, FAKE, None) == -1   # unaligned x
    assert g(FAKE, 10, FAKE, 1 << 31, 256, FAKE, None) == -2
