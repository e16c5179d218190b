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
    assert lib.tfg_version() == 100


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
