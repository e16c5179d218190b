"""The seeded workload generators produce the shapes the workloads call for."""
import numpy as np
import pytest

from paper_2101_11552_gb300 import graphgen as gg


def test_er2708_shape():
    w = gg.make_er_2708()
    assert (w.num_nodes, w.num_edges, w.num_features) == (2708, 10556 + 2708, 64)
    ei = w.edge_index
    # symmetric: every (i, j) has its (j, i); explicit self-loops at the end
    fwd = set(zip(ei[0, :10556].tolist(), ei[1, :10556].tolist()))
    assert all((j, i) in fwd for i, j in fwd)
    assert np.array_equal(ei[0, 10556:], np.arange(2708)) and np.array_equal(ei[1, 10556:], np.arange(2708))


def test_ba19717_shape():
    w = gg.make_ba_19717()
    assert (w.num_nodes, w.num_edges, w.num_features) == (19717, 78860 + 19717, 256)


def test_gat169343_shape():
    w = gg.make_gat_169343()
    assert (w.num_nodes, w.num_edges, w.heads, w.channels) == (169343, 1166243, 8, 16)
    assert w.num_features == 128
    assert not np.any(w.edge_index[0] == w.edge_index[1])


def test_molecules_shape_and_batch():
    w = gg.make_molecules_1024()
    assert w.num_graphs == 1024
    assert 20 <= w.graph_sizes.min() and w.graph_sizes.max() <= 200
    assert w.num_nodes == int(w.graph_sizes.sum())
    assert np.all(np.diff(w.batch) >= 0)
    # edges never cross graphs
    assert np.array_equal(w.batch[w.edge_index[0]], w.batch[w.edge_index[1]])
    # average degree 4 plus one self-loop per node
    assert w.num_edges == int((4 * w.graph_sizes + w.graph_sizes).sum())


def test_generators_are_deterministic():
    a, b = gg.make_er_2708(), gg.make_er_2708()
    assert np.array_equal(a.edge_index, b.edge_index) and np.array_equal(a.x, b.x)


def test_dcsbm_small():
    rng = np.random.default_rng(0)
    pairs, block_of, sizes = gg.dcsbm_pairs(5000, 41, 60000, rng)
    assert pairs.shape == (60000, 2) and sizes.sum() == 5000 and len(sizes) == 41
    key = np.minimum(pairs[:, 0], pairs[:, 1]) * 5000 + np.maximum(pairs[:, 0], pairs[:, 1])
    assert np.unique(key).size == 60000
    assert not np.any(pairs[:, 0] == pairs[:, 1])
    inblock = np.mean(block_of[pairs[:, 0]] == block_of[pairs[:, 1]])
    assert inblock > 0.85


def test_bf16_rne():
    x = np.array([1.0, 1.00390625, 1.01171875, -2.5, 3.0e-3], dtype=np.float32)
    bits = gg.bf16_bits_rne(x)
    back = gg.bf16_bits_to_f32(bits)
    # 1 + 2^-8 is a tie between 1 and 1 + 2^-7: rounds to even (1.0)
    assert back[0] == 1.0 and back[1] == 1.0 and back[2] == np.float32(1.015625)
    assert back[3] == -2.5
