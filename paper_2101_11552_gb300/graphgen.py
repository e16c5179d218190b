"""Seeded synthetic graph workloads.

This module only *draws inputs*: edge lists, node features, attention vectors
and batch vectors.  It holds none of the aggregation arithmetic, so both the
CUDA path and the fp64 oracle can consume what it produces without sharing
any of the method's code.

Conventions (tf_geometric, Section 2.1.1 "Graph Data Structure"):
  * ``edge_index`` is int64 ``[2, E]``; row 0 holds the source node of each
    edge and row 1 its target.  A positive entry A_ij is an edge i -> j, and
    messages flow from source to target.
  * Node features ``x`` are a dense ``[N, F]`` row-major matrix.

The five workloads stand in for the graphs the paper evaluates on (Cora- and
Pubmed-sized citation graphs, a large citation graph, mini-batched molecule
graphs and a large dense-community graph, Section 4).  None of those datasets
is available, so each is replaced by a random graph of the same shape.

Seeds (``numpy.random.default_rng``), graph / features: Erdos-Renyi 2,708
nodes 1001 / 1101; Barabasi-Albert 19,717 nodes 1002 / 1102; Barabasi-Albert
169,343 nodes with attention vectors 1003 / 1103; 1,024 molecule graphs
1004 / 1104; dense-community 232,965 nodes 1005 / 1105 (attention vectors
1205).
"""
from __future__ import annotations

import dataclasses
from typing import Optional

import numpy as np

__all__ = [
    "Workload", "er_pairs", "ba_pairs", "symmetrise", "with_self_loops",
    "batch_graphs", "dcsbm_pairs", "bf16_bits_rne", "bf16_bits_to_f32",
    "make_er_2708", "make_ba_19717", "make_gat_169343", "make_molecules_1024", "make_dcsbm_232965", "make_workload",
    "random_edge_case_graph", "WORKLOADS",
]


@dataclasses.dataclass
class Workload:
    """One synthetic input set.  Arrays are host numpy arrays."""
    name: str
    num_nodes: int
    edge_index: np.ndarray               # int64 [2, E]
    x: np.ndarray                        # float32 [N, F]
    x_bf16: Optional[np.ndarray] = None  # uint16 [N, F] (bf16 bit patterns, RNE of x)
    add_self_loops: int = 0              # GCN: add an implicit self-loop per node
    self_loop_fill: float = 1.0
    heads: int = 0                       # edge softmax: H
    channels: int = 0                    # edge softmax: C (F = H * C)
    a_src: Optional[np.ndarray] = None   # float32 [H * C]
    a_dst: Optional[np.ndarray] = None   # float32 [H * C]
    negative_slope: float = 0.2
    batch: Optional[np.ndarray] = None   # int64 [N], sorted graph id per node
    num_graphs: int = 0
    graph_sizes: Optional[np.ndarray] = None

    @property
    def num_edges(self) -> int:
        return int(self.edge_index.shape[1])

    @property
    def num_features(self) -> int:
        return int(self.x.shape[1])


# --------------------------------------------------------------------------
# bf16 storage format (round-to-nearest-even of the fp32 bit pattern)
# --------------------------------------------------------------------------
def bf16_bits_rne(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit patterns, round to nearest even (finite inputs)."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32).astype(np.uint64)
    bias = 0x7FFF + ((b >> 16) & 1)
    return ((b + bias) >> 16).astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns -> the fp32 values they denote (exact)."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


# --------------------------------------------------------------------------
# Random graph families
# --------------------------------------------------------------------------
def er_pairs(n: int, m: int, rng: np.random.Generator) -> np.ndarray:
    """G(n, M): M distinct unordered pairs i < j drawn uniformly.

    Returns int64 ``[M, 2]`` in draw order.
    """
    if m > n * (n - 1) // 2:
        raise ValueError("too many edges for a simple graph")
    out = np.empty((0, 2), dtype=np.int64)
    seen = np.empty(0, dtype=np.int64)
    while out.shape[0] < m:
        need = m - out.shape[0]
        k = int(need * 1.2) + 16
        i = rng.integers(0, n, size=k, dtype=np.int64)
        j = rng.integers(0, n, size=k, dtype=np.int64)
        keep = i != j
        i, j = i[keep], j[keep]
        lo, hi = np.minimum(i, j), np.maximum(i, j)
        key = lo * n + hi
        # first occurrence within this draw, in draw order
        _, first = np.unique(key, return_index=True)
        first.sort()
        key, lo, hi = key[first], lo[first], hi[first]
        fresh = ~np.isin(key, seen)
        key, lo, hi = key[fresh][:need], lo[fresh][:need], hi[fresh][:need]
        seen = np.concatenate([seen, key])
        out = np.concatenate([out, np.stack([lo, hi], axis=1)])
    return out


def ba_pairs(n: int, m: int, rng: np.random.Generator) -> np.ndarray:
    """Barabasi-Albert preferential attachment.

    Nodes 0..m-1 start without edges; node m links to all of them; every later
    node v links to m distinct earlier nodes drawn with probability proportional
    to their current degree.  Gives m * (n - m) undirected pairs ``[M, 2]``
    as (new node, existing node).
    """
    total = m * (n - m)
    pairs = np.empty((total, 2), dtype=np.int64)
    ends = np.empty(2 * total, dtype=np.int64)   # every edge endpoint, repeated
    n_ends = 0
    k = 0
    for t in range(m):
        pairs[k] = (m, t)
        k += 1
        ends[n_ends] = m
        ends[n_ends + 1] = t
        n_ends += 2
    # Vectorised draws with rejection of repeats inside one node's m choices.
    for v in range(m + 1, n):
        chosen: list[int] = []
        while len(chosen) < m:
            cand = ends[rng.integers(0, n_ends, size=2 * m)]
            for c in cand:
                c = int(c)
                if c not in chosen:
                    chosen.append(c)
                    if len(chosen) == m:
                        break
        for c in chosen:
            pairs[k] = (v, c)
            k += 1
            ends[n_ends] = v
            ends[n_ends + 1] = c
            n_ends += 2
    assert k == total
    return pairs


def symmetrise(pairs: np.ndarray) -> np.ndarray:
    """Unordered pairs -> directed edge_index [2, 2M]: every (i, j) then every (j, i)."""
    m = pairs.shape[0]
    out = np.empty((2, 2 * m), dtype=np.int64)
    out[0, :m] = pairs[:, 0]
    out[0, m:] = pairs[:, 1]
    out[1, :m] = pairs[:, 1]
    out[1, m:] = pairs[:, 0]
    return out


def with_self_loops(edge_index: np.ndarray, n: int) -> np.ndarray:
    """Append one explicit edge t -> t per node (after the existing edges)."""
    loops = np.arange(n, dtype=np.int64)
    return np.ascontiguousarray(np.concatenate([edge_index, np.stack([loops, loops])], axis=1))


def batch_graphs(edge_indices: list[np.ndarray], sizes: list[int]):
    """BatchGraph construction by the reindexing trick (Section 2.1.1).

    The j-th node of the i-th graph gets index offset_i + j, where offset_i is
    the number of nodes in all graphs before graph i; the reindexed edge lists
    are stacked in graph order.  Returns (edge_index [2, sum E], batch [N]
    int64 non-decreasing, offsets [G] int64).
    """
    sizes_arr = np.asarray(sizes, dtype=np.int64)
    offsets = np.zeros(len(sizes), dtype=np.int64)
    if len(sizes) > 1:
        offsets[1:] = np.cumsum(sizes_arr)[:-1]
    parts = [ei + off for ei, off in zip(edge_indices, offsets)]
    edge_index = np.concatenate(parts, axis=1) if parts else np.zeros((2, 0), np.int64)
    batch = np.repeat(np.arange(len(sizes), dtype=np.int64), sizes_arr)
    return np.ascontiguousarray(edge_index.astype(np.int64)), batch, offsets


def _alias_table(p: np.ndarray):
    """Walker/Vose alias table for sampling index k with probability p[k]."""
    k = p.shape[0]
    scaled = p / p.sum() * k
    prob = np.zeros(k)
    alias = np.zeros(k, dtype=np.int64)
    small = [i for i in range(k) if scaled[i] < 1.0]
    large = [i for i in range(k) if scaled[i] >= 1.0]
    while small and large:
        s, g = small.pop(), large.pop()
        prob[s] = scaled[s]
        alias[s] = g
        scaled[g] = scaled[g] + scaled[s] - 1.0
        (small if scaled[g] < 1.0 else large).append(g)
    for i in small + large:
        prob[i] = 1.0
        alias[i] = i
    return prob, alias


def dcsbm_pairs(n: int, blocks: int, m: int, rng: np.random.Generator,
                p_in: float = 0.9, theta_sigma: float = 1.0, size_sigma: float = 0.6):
    """Degree-corrected stochastic block model with heavy-tailed degrees.

    Block sizes are lognormal(0, size_sigma) scaled to sum to n; nodes are
    numbered block by block.  Each node has a propensity theta ~ lognormal(0,
    theta_sigma).  A pair is drawn as: endpoint i with probability proportional
    to theta; with probability p_in the other endpoint j is drawn from i's own
    block (proportional to theta), else from the whole graph.  Self pairs and
    repeated pairs are dropped; exactly m distinct unordered pairs are kept, in
    a seeded random order.

    Returns (pairs [m, 2] int64, block_of_node [n] int64, block_sizes [blocks]).
    """
    w = rng.lognormal(0.0, size_sigma, size=blocks)
    sizes = np.maximum(np.floor(w / w.sum() * n).astype(np.int64), 1)
    sizes[np.argmax(sizes)] += n - sizes.sum()
    starts = np.zeros(blocks + 1, dtype=np.int64)
    starts[1:] = np.cumsum(sizes)
    block_of = np.repeat(np.arange(blocks, dtype=np.int64), sizes)
    theta = rng.lognormal(0.0, theta_sigma, size=n)
    g_prob, g_alias = _alias_table(theta)
    b_prob = np.zeros(n)
    b_alias = np.zeros(n, dtype=np.int64)      # global node ids
    for b in range(blocks):
        s0, s1 = starts[b], starts[b + 1]
        pr, al = _alias_table(theta[s0:s1])
        b_prob[s0:s1] = pr
        b_alias[s0:s1] = al + s0

    sizes32 = sizes.astype(np.int32)
    starts32 = starts.astype(np.int32)
    block32 = block_of.astype(np.int32)
    b_alias32 = b_alias.astype(np.int32)
    g_alias32 = g_alias.astype(np.int32)
    chunk = 1 << 21          # draw in chunks: bounded temporaries, reused memory

    def draw_global(k):
        idx = rng.integers(0, n, size=k, dtype=np.int32)
        return np.where(rng.random(k, dtype=np.float32) < g_prob[idx], idx, g_alias32[idx])

    def draw_keys(k, out):
        """Fill out[:k] with the keys of k drawn pairs; return how many were kept."""
        kept = 0
        for c0 in range(0, k, chunk):
            c = min(chunk, k - c0)
            i = draw_global(c)
            b = block32[i]
            loc = starts32[b] + (rng.random(c, dtype=np.float32) * sizes32[b]).astype(np.int32)
            np.minimum(loc, starts32[b + 1] - 1, out=loc)
            j_in = np.where(rng.random(c, dtype=np.float32) < b_prob[loc], loc, b_alias32[loc])
            j = np.where(rng.random(c, dtype=np.float32) < p_in, j_in, draw_global(c))
            ok = i != j
            lo = np.minimum(i[ok], j[ok]).astype(np.int64)
            hi = np.maximum(i[ok], j[ok])
            out[kept:kept + lo.shape[0]] = lo * n + hi
            kept += lo.shape[0]
        return kept

    factor = 1.5
    while True:
        k = int(m * factor) + 1024
        key = np.empty(k, dtype=np.int64)
        key = key[:draw_keys(k, key)]
        key.sort()
        key = key[np.concatenate([[True], key[1:] != key[:-1]])]
        if key.shape[0] >= m:
            break
        factor *= 1.25
    key = key[rng.permutation(key.shape[0])[:m]]
    pairs = np.empty((m, 2), dtype=np.int64)
    np.floor_divide(key, n, out=pairs[:, 0])
    np.remainder(key, n, out=pairs[:, 1])
    return pairs, block_of, sizes


# --------------------------------------------------------------------------
# The five workloads
# --------------------------------------------------------------------------
def make_er_2708() -> Workload:
    """GCN on G(2708, 5278) symmetrised + 2708 explicit self-loops, F=64 fp32."""
    n = 2708
    rng = np.random.default_rng(1001)
    ei = with_self_loops(symmetrise(er_pairs(n, 5278, rng)), n)
    x = np.random.default_rng(1101).standard_normal((n, 64), dtype=np.float32)
    return Workload("er-gcn-2708", n, ei, x, add_self_loops=0)


def make_ba_19717() -> Workload:
    """BA(19717, m=2) symmetrised + self-loops, F=256 fp32, unweighted reducers."""
    n = 19717
    rng = np.random.default_rng(1002)
    ei = with_self_loops(symmetrise(ba_pairs(n, 2, rng)), n)
    x = np.random.default_rng(1102).standard_normal((n, 256), dtype=np.float32)
    return Workload("ba-19717-sum-mean-max", n, ei, x)


def make_gat_169343() -> Workload:
    """BA(169343, m=7), subsampled to 1,166,243 edges, each oriented by a coin.

    No self-loops.  8 heads x 16 channels fp32, a_src/a_dst ~ N(0, 1), slope 0.2.
    """
    n, e_target = 169343, 1166243
    rng = np.random.default_rng(1003)
    pairs = ba_pairs(n, 7, rng)
    keep = np.sort(rng.choice(pairs.shape[0], size=e_target, replace=False))
    pairs = pairs[keep]
    flip = rng.random(e_target) < 0.5
    src = np.where(flip, pairs[:, 1], pairs[:, 0])
    dst = np.where(flip, pairs[:, 0], pairs[:, 1])
    ei = np.ascontiguousarray(np.stack([src, dst]).astype(np.int64))
    frng = np.random.default_rng(1103)
    x = frng.standard_normal((n, 128), dtype=np.float32)
    a_src = frng.standard_normal(128, dtype=np.float32)
    a_dst = frng.standard_normal(128, dtype=np.float32)
    return Workload("gat-edge-softmax-169343", n, ei, x, heads=8, channels=16,
                    a_src=a_src, a_dst=a_dst, negative_slope=0.2)


def make_molecules_1024() -> Workload:
    """1,024 graphs of U{20..200} nodes, each G(n_g, 2 n_g) symmetrised + self-loops.

    Graphs are combined by the reindexing trick; batch is the sorted graph id.
    """
    rng = np.random.default_rng(1004)
    g = 1024
    sizes = rng.integers(20, 201, size=g)
    parts = []
    for ng in sizes:
        ng = int(ng)
        parts.append(with_self_loops(symmetrise(er_pairs(ng, 2 * ng, rng)), ng))
    ei, batch, _ = batch_graphs(parts, [int(s) for s in sizes])
    n = int(sizes.sum())
    x = np.random.default_rng(1104).standard_normal((n, 128), dtype=np.float32)
    return Workload("batched-1024-graphs-pool", n, ei, x, batch=batch, num_graphs=g,
                    graph_sizes=sizes.astype(np.int64))


def make_dcsbm_232965(num_pairs: int = 57_300_000, n: int = 232_965) -> Workload:
    """Degree-corrected SBM: 41 blocks, ~114.6M directed edges, bf16 F=128.

    GCN with implicit self-loops (fill 1).  ``batch`` is the block id of each
    node (blocks are contiguous), used as a pooling key over communities.
    """
    rng = np.random.default_rng(1005)
    pairs, block_of, sizes = dcsbm_pairs(n, 41, num_pairs, rng)
    ei = symmetrise(pairs)
    del pairs
    x = np.random.default_rng(1105).standard_normal((n, 128), dtype=np.float32)
    frng = np.random.default_rng(1205)
    a_src = frng.standard_normal(128, dtype=np.float32)
    a_dst = frng.standard_normal(128, dtype=np.float32)
    return Workload("dcsbm-232965-bf16-gcn", n, ei, x, x_bf16=bf16_bits_rne(x),
                    add_self_loops=1, self_loop_fill=1.0,
                    heads=8, channels=16, a_src=a_src, a_dst=a_dst,
                    batch=block_of, num_graphs=41, graph_sizes=sizes)


WORKLOADS = {
    "er-gcn-2708": make_er_2708,
    "ba-19717-sum-mean-max": make_ba_19717,
    "gat-edge-softmax-169343": make_gat_169343,
    "batched-1024-graphs-pool": make_molecules_1024,
    "dcsbm-232965-bf16-gcn": make_dcsbm_232965,
}


def make_workload(name: str, **kw) -> Workload:
    return WORKLOADS[name](**kw)


def random_edge_case_graph(n: int, e: int, f: int, seed: int, *, hub: int = -1,
                           isolated: int = 0, dup_frac: float = 0.1,
                           self_frac: float = 0.05) -> Workload:
    """Small random directed multigraph with the awkward cases on purpose.

    * ``isolated`` nodes at the end receive no edge and send none;
    * ``dup_frac`` of the edges repeat an earlier edge;
    * ``self_frac`` are self-loops;
    * ``hub`` >= 0 makes that node the target of about half of all edges.
    """
    rng = np.random.default_rng(seed)
    live = max(n - isolated, 1) if n > 0 else 0
    if e == 0 or live == 0:
        ei = np.zeros((2, 0), dtype=np.int64)
    else:
        src = rng.integers(0, live, size=e, dtype=np.int64)
        dst = rng.integers(0, live, size=e, dtype=np.int64)
        if hub >= 0:
            dst[rng.random(e) < 0.5] = hub
        nd = int(e * dup_frac)
        if nd and e > 1:
            at = rng.integers(1, e, size=nd)
            frm = (rng.random(nd) * at).astype(np.int64)
            src[at], dst[at] = src[frm], dst[frm]
        ns = int(e * self_frac)
        if ns:
            at = rng.integers(0, e, size=ns)
            src[at] = dst[at]
        ei = np.ascontiguousarray(np.stack([src, dst]))
    x = rng.standard_normal((n, f), dtype=np.float32)
    return Workload(f"edge-case-n{n}-e{e}-f{f}-s{seed}", n, ei, x,
                    x_bf16=bf16_bits_rne(x))
