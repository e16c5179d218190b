"""Host-side logic of bench.py: units, launch counts and the over-ranks
reduction of replicas (two gloo ranks on the CPU)."""
import os
import socket

import numpy as np
import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def test_units_and_launches():
    n, e, f = 232965, 114_600_000, 128
    assert bench.units_per_step(n, e, f) == (e + n) * f + e * f + 2 * n * f
    assert bench.csr_passes(232965) == 2 and bench.csr_passes(1000) == 1
    assert bench.csr_passes(1_500_000) == 3
    # build: 2 passes x 5 + rowptr + degree; norm 1; gcn 1; softmax 2; pools 4
    assert bench.launches_per_step(n, e) == 12 + 1 + 1 + 2 + 4


def test_algorithmic_bytes_gcn():
    n, e, f = 232965, 114_600_000, 128
    b = bench.algorithmic_bytes(n, e, f, 8, 41)["gcn_aggregate"]
    # col 4E + rowptr + dinv + x bf16 once + out fp32
    assert abs(b / 1e6 - 639.1) < 1.0


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    t, u = bench.combine_ranks(1.0 + rank, 100 * (rank + 1), world, dist)
    q.put((rank, t, u))
    dist.destroy_process_group()


def test_combine_ranks_two_gloo_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    # max time over ranks, sum of units over ranks, same on every rank
    assert res == [(0, 2.0, 300), (1, 2.0, 300)]


def test_single_rank_passthrough():
    assert bench.combine_ranks(1.5, 7, 1, None) == (1.5, 7)


def test_sample_nodes_is_the_smallest_prefix_with_enough_edges():
    from paper_2101_11552_gb300 import graphgen as gg
    wl = gg.make_ba_19717()
    for target in (1000, 20_000, 90_000, 10 ** 9):
        k = bench.sample_nodes(wl, target)
        ei = wl.edge_index
        inside = lambda m: int(((ei[0] < m) & (ei[1] < m)).sum())  # noqa: E731
        if target <= wl.num_edges:
            assert inside(k) >= target > inside(k - 1)
        else:
            assert k == wl.num_nodes
        if k < wl.num_nodes:
            wl.x_bf16 = np.zeros((wl.num_nodes, 1), np.uint16)
            wl.batch = np.zeros(wl.num_nodes, np.int64)
            s = bench.oracle_sample(wl, k)
            assert s["edge_index"].shape[1] == inside(k) and s["n"] == k
