"""Gather-only floor (tfg_gather_xor): the XOR of every gathered row equals
numpy's XOR reduction of the same rows, bit for bit, for every supported
row width, ragged edge counts, an empty edge list and the dense-community
workload's own column array."""
import numpy as np
import pytest
import torch

from paper_2101_11552_gb300 import graphgen as gg
from paper_2101_11552_gb300 import tfg
from _helpers import dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2101_11552_gb300 import build
    build.build_library()


def _xor_rows(col: np.ndarray, words: np.ndarray) -> np.ndarray:
    if len(col) == 0:
        return np.zeros(words.shape[1], np.uint32)
    return np.bitwise_xor.reduce(words[col], axis=0)


@pytest.mark.parametrize("row_bytes", [16, 32, 64, 128, 256, 512])
@pytest.mark.parametrize("e", [0, 1, 31, 33, 4097, 250_001])
def test_gather_xor_matches_numpy(row_bytes, e):
    n = 5000
    rng = np.random.default_rng(row_bytes + e)
    words = rng.integers(0, 2 ** 32, size=(n, row_bytes // 4), dtype=np.uint32)
    col = rng.integers(0, n, size=e).astype(np.int32)
    got = tfg.tfg_gather_xor(dev(col), dev(words.view(np.int32))).cpu().numpy().view(np.uint32)
    np.testing.assert_array_equal(got, _xor_rows(col, words))


def test_gather_xor_on_a_csr_column_array():
    """The column array of a CSR with a hub and isolated nodes, bf16 rows of
    128 features (256 bytes, the benchmark's row width)."""
    n, e = 20000, 300_000
    wl = gg.random_edge_case_graph(n, e, 128, 77, hub=3, isolated=100)
    csr = tfg.tfg_build_csr(dev(wl.edge_index), n)
    tfg.check_status(csr.status)
    xb = dev(wl.x_bf16.view(np.int16)).view(torch.bfloat16)
    got = tfg.tfg_gather_xor(csr.col, xb).cpu().numpy().view(np.uint32)
    words = wl.x_bf16.view(np.uint32).reshape(n, 64)
    np.testing.assert_array_equal(got, _xor_rows(csr.col.cpu().numpy(), words))
