"""fp64 CPU oracle for graph message aggregation -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  It never imports the CUDA library or
its Python binding, and the CUDA path never imports it.

Two independent forms of the same definitions:

* ``tfg_oracle.c`` -- per-edge / per-node loops in original order, fp64
  accumulation (compiled with gcc into ``_build/liboracle.so`` on first use).
* numpy dense matrices for tiny graphs (``dense_*``), used to cross-check the
  loops by brute force.

Inputs are widened to float64 here: fp32 values exactly, bf16 bit patterns by
placing the 16 bits in the high half of an fp32 word (the bf16 definition).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from typing import Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "tfg_oracle.c")
_BUILD = os.path.join(_HERE, "_build")

REDUCE = {"sum": 0, "mean": 1, "max": 2}
_ERRORS = {-1: "invalid argument", -5: "index out of range", -6: "batch not sorted"}

_lock = threading.Lock()
_libs: dict = {}


class OracleError(RuntimeError):
    def __init__(self, code: int):
        super().__init__(f"oracle error {code}: {_ERRORS.get(code, 'unknown')}")
        self.code = code


def build(plant: Optional[str] = None, out_dir: Optional[str] = None) -> str:
    """Compile tfg_oracle.c (optionally with one planted mistake) and return the .so path."""
    out_dir = out_dir or _BUILD
    os.makedirs(out_dir, exist_ok=True)
    name = "liboracle.so" if plant is None else f"liboracle_{plant.lower()}.so"
    path = os.path.join(out_dir, name)
    if (not os.path.exists(path)) or os.path.getmtime(path) < os.path.getmtime(_SRC):
        cmd = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-o", path + ".tmp", _SRC, "-lm"]
        if plant is not None:
            cmd.insert(1, f"-DORACLE_PLANT_{plant.upper()}")
        subprocess.run(cmd, check=True)
        os.replace(path + ".tmp", path)
    return path


_SRC_OMP = os.path.join(_HERE, "tfg_oracle_omp.c")


def build_omp(out_dir: Optional[str] = None) -> str:
    """Compile tfg_oracle.c with tfg_oracle_omp.c and -fopenmp (the all-cores
    CPU baseline: the oracle's row functions on blocks of rows in parallel)."""
    out_dir = out_dir or _BUILD
    os.makedirs(out_dir, exist_ok=True)
    path = os.path.join(out_dir, "liboracle_omp.so")
    newest = max(os.path.getmtime(_SRC), os.path.getmtime(_SRC_OMP))
    if (not os.path.exists(path)) or os.path.getmtime(path) < newest:
        cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-shared", "-fPIC", "-o", path + ".tmp",
               _SRC, _SRC_OMP, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(path + ".tmp", path)
    return path


def _load(plant: Optional[str] = None) -> ctypes.CDLL:
    with _lock:
        if plant not in _libs:
            lib = ctypes.CDLL(build(plant))
            P = ctypes.c_void_p
            I64 = ctypes.c_int64
            I = ctypes.c_int
            D = ctypes.c_double
            sigs = {
                "oracle_build_csr": [I64, I64, P, P, P, P, P],
                "oracle_gcn_norm": [I64, I64, P, P, I, D, P, P, P, P],
                "oracle_aggregate": [I, I64, I64, P, P, P, I64, P, P, P],
                "oracle_aggregate_rows": [I, I64, P, P, P, P, P, I64, P, P, I64, P, P],
                "oracle_edge_softmax": [I64, I64, P, P, I, I, P, P, D, P, P, P],
                "oracle_edge_softmax_rows": [I64, P, P, P, I, I, P, P, D, P, I64, P, P, P],
                "oracle_segment_pool": [I, I64, I64, I64, P, P, P, P],
                "oracle_appnp": [I64, I64, P, P, P, P, I64, I64, D, P, P],
                "oracle_dot_softmax": [I64, I64, P, P, P, P, I, I, D, P, P, P],
                "oracle_aggregate_backward": [I, I64, I64, P, P, P, P, I64, P, P],
                "oracle_max_argmax": [I64, I64, P, P, P, I64, P, P],
                "oracle_max_backward": [I64, I64, P, P, P, P, I64, P, P],
                "oracle_dot_softmax_rows": [I64, P, P, P, P, P, I, I, D, P, I64, P, P, P],
                "oracle_edge_softmax_backward": [I64, I64, P, P, I, I, P, P, D, P, P, P, P, P,
                                                 P, P],
                "oracle_dot_softmax_backward": [I64, I64, P, P, P, P, I, I, D, P, P, P, P, P, P,
                                                P],
            }
            for fn, args in sigs.items():
                getattr(lib, fn).argtypes = args
                getattr(lib, fn).restype = ctypes.c_int
            _libs[plant] = lib
        return _libs[plant]


class _Oracle:
    """All oracle entry points bound to one compiled variant of tfg_oracle.c."""

    def __init__(self, plant: Optional[str] = None):
        self.plant = plant

    @property
    def lib(self) -> ctypes.CDLL:
        return _load(self.plant)

    @staticmethod
    def _p(a: Optional[np.ndarray]):
        return None if a is None else a.ctypes.data_as(ctypes.c_void_p)

    @staticmethod
    def _check(code: int):
        if code != 0:
            raise OracleError(code)

    # -- CSR -------------------------------------------------------------
    def build_csr(self, edge_index: np.ndarray, n: int):
        ei = np.ascontiguousarray(edge_index, dtype=np.int64)
        e = ei.shape[1]
        rowptr = np.zeros(n + 1, np.int32)
        col = np.zeros(max(e, 1), np.int32)
        perm = np.zeros(max(e, 1), np.int32)
        deg = np.zeros(max(n, 1), np.int32)
        self._check(self.lib.oracle_build_csr(n, e, self._p(ei), self._p(rowptr), self._p(col),
                                              self._p(perm), self._p(deg)))
        return rowptr, col[:e], perm[:e], deg[:n]

    # -- GCN normalisation ----------------------------------------------
    def gcn_norm(self, edge_index, n, edge_weight=None, add_self_loops=0, fill=1.0):
        ei = np.ascontiguousarray(edge_index, dtype=np.int64)
        e = ei.shape[1]
        w = None if edge_weight is None else np.ascontiguousarray(edge_weight, np.float64)
        deg = np.zeros(max(n, 1))
        dinv = np.zeros(max(n, 1))
        wn = np.zeros(max(e, 1))
        sw = np.zeros(max(n, 1))
        self._check(self.lib.oracle_gcn_norm(n, e, self._p(ei), self._p(w), int(add_self_loops),
                                             float(fill), self._p(deg), self._p(dinv),
                                             self._p(wn), self._p(sw)))
        return {"deg": deg[:n], "dinv": dinv[:n], "w_norm": wn[:e],
                "self_w": sw[:n] if add_self_loops else None}

    # -- aggregation ----------------------------------------------------
    def aggregate(self, edge_index, n, x, reduce, w=None, self_w=None):
        ei = np.ascontiguousarray(edge_index, dtype=np.int64)
        e = ei.shape[1]
        x = widen(x)
        f = x.shape[1]
        w = None if w is None else np.ascontiguousarray(w, np.float64)
        sw = None if self_w is None else np.ascontiguousarray(self_w, np.float64)
        out = np.zeros((max(n, 1), f))
        ab = np.zeros((max(n, 1), f))
        self._check(self.lib.oracle_aggregate(REDUCE[reduce], n, e, self._p(ei), self._p(w),
                                              self._p(x), f, self._p(sw), self._p(out),
                                              self._p(ab)))
        return out[:n], ab[:n]

    def gcn_aggregate(self, edge_index, n, x, edge_weight=None, add_self_loops=0, fill=1.0):
        nrm = self.gcn_norm(edge_index, n, edge_weight, add_self_loops, fill)
        return self.aggregate(edge_index, n, x, "sum", w=nrm["w_norm"], self_w=nrm["self_w"])

    def aggregate_rows(self, csr, n, x, reduce, rows, w=None, self_w=None):
        rowptr, col, perm, _ = csr
        x = widen(x)
        f = x.shape[1]
        rows = np.ascontiguousarray(rows, np.int64)
        w = None if w is None else np.ascontiguousarray(w, np.float64)
        sw = None if self_w is None else np.ascontiguousarray(self_w, np.float64)
        out = np.zeros((max(len(rows), 1), f))
        ab = np.zeros((max(len(rows), 1), f))
        self._check(self.lib.oracle_aggregate_rows(
            REDUCE[reduce], n, self._p(rowptr), self._p(np.ascontiguousarray(col)),
            self._p(np.ascontiguousarray(perm)), self._p(w), self._p(x), f, self._p(sw),
            self._p(rows), len(rows), self._p(out), self._p(ab)))
        return out[:len(rows)], ab[:len(rows)]

    # -- edge softmax ---------------------------------------------------
    def edge_softmax(self, edge_index, n, x, heads, channels, a_src, a_dst, slope=0.2):
        ei = np.ascontiguousarray(edge_index, dtype=np.int64)
        e = ei.shape[1]
        x = widen(x)
        f = x.shape[1]
        assert f == heads * channels
        a_s = np.ascontiguousarray(a_src, np.float64)
        a_d = np.ascontiguousarray(a_dst, np.float64)
        out = np.zeros((max(n, 1), f))
        ab = np.zeros((max(n, 1), f))
        alpha = np.zeros((max(e, 1), heads))
        self._check(self.lib.oracle_edge_softmax(n, e, self._p(ei), self._p(x), heads, channels,
                                                 self._p(a_s), self._p(a_d), float(slope),
                                                 self._p(out), self._p(alpha), self._p(ab)))
        return out[:n], alpha[:e], ab[:n]

    def edge_softmax_rows(self, csr, n, x, heads, channels, a_src, a_dst, slope, rows):
        rowptr, col, _, _ = csr
        x = widen(x)
        f = x.shape[1]
        rows = np.ascontiguousarray(rows, np.int64)
        a_s = np.ascontiguousarray(a_src, np.float64)
        a_d = np.ascontiguousarray(a_dst, np.float64)
        total = int(sum(rowptr[r + 1] - rowptr[r] for r in rows))
        out = np.zeros((max(len(rows), 1), f))
        ab = np.zeros((max(len(rows), 1), f))
        alpha = np.zeros((max(total, 1), heads))
        self._check(self.lib.oracle_edge_softmax_rows(
            n, self._p(rowptr), self._p(np.ascontiguousarray(col)), self._p(x), heads, channels,
            self._p(a_s), self._p(a_d), float(slope), self._p(rows), len(rows), self._p(out),
            self._p(alpha), self._p(ab)))
        return out[:len(rows)], alpha[:total], ab[:len(rows)]

    def edge_softmax_backward(self, edge_index, n, x, heads, channels, a_src, a_dst, slope,
                              grad_out):
        """Gradients of edge_softmax's output with respect to x, a_src and a_dst
        for a given dL/dout.  Returns (grad_x [N, F], grad_a_src [F],
        grad_a_dst [F], (scale_x, scale_a_src, scale_a_dst))."""
        ei = np.ascontiguousarray(edge_index, dtype=np.int64)
        e = ei.shape[1]
        x = widen(x)
        g = widen(grad_out)
        f = x.shape[1]
        assert f == heads * channels and g.shape == x.shape
        a_s = np.ascontiguousarray(a_src, np.float64)
        a_d = np.ascontiguousarray(a_dst, np.float64)
        gx, ax = np.zeros((max(n, 1), f)), np.zeros((max(n, 1), f))
        gs, gd, as_, ad = (np.zeros(f) for _ in range(4))
        self._check(self.lib.oracle_edge_softmax_backward(
            n, e, self._p(ei), self._p(x), heads, channels, self._p(a_s), self._p(a_d),
            float(slope), self._p(g), self._p(gx), self._p(gs), self._p(gd), self._p(ax),
            self._p(as_), self._p(ad)))
        return gx[:n], gs, gd, (ax[:n], as_, ad)

    def dot_softmax_backward(self, edge_index, n, q, k, v, heads, channels, scale, grad_out):
        """Gradients of dot_softmax's output with respect to q, k and v for a
        given dL/dout.  Returns (grad_q, grad_k, grad_v, (scale_q, scale_k, scale_v))."""
        ei = np.ascontiguousarray(edge_index, dtype=np.int64)
        e = ei.shape[1]
        q, k, v, g = widen(q), widen(k), widen(v), widen(grad_out)
        f = q.shape[1]
        assert f == heads * channels and k.shape == q.shape and v.shape == q.shape
        outs = [np.zeros((max(n, 1), f)) for _ in range(6)]
        self._check(self.lib.oracle_dot_softmax_backward(
            n, e, self._p(ei), self._p(q), self._p(k), self._p(v), heads, channels, float(scale),
            self._p(g), *[self._p(o) for o in outs]))
        gq, gk, gv, aq, ak, av = (o[:n] for o in outs)
        return gq, gk, gv, (aq, ak, av)

    # -- backward of the aggregation ------------------------------------
    def aggregate_backward(self, edge_index, n, grad_out, reduce, w=None, self_w=None):
        """dL/dx of aggregate(edge_index, n, x, reduce, w, self_w) for a given
        dL/dout (sum or mean; GCN = sum with w_norm and self_w).  Returns
        (grad_x, error scale), both [N, F]."""
        ei = np.ascontiguousarray(edge_index, dtype=np.int64)
        e = ei.shape[1]
        g = widen(grad_out)
        f = g.shape[1]
        w = None if w is None else np.ascontiguousarray(w, np.float64)
        sw = None if self_w is None else np.ascontiguousarray(self_w, np.float64)
        out = np.zeros((max(n, 1), f))
        ab = np.zeros((max(n, 1), f))
        self._check(self.lib.oracle_aggregate_backward(REDUCE[reduce], n, e, self._p(ei), self._p(w),
                                                       self._p(sw), self._p(g), f, self._p(out),
                                                       self._p(ab)))
        return out[:n], ab[:n]

    def gcn_aggregate_backward(self, edge_index, n, grad_out, edge_weight=None, add_self_loops=0,
                               fill=1.0):
        nrm = self.gcn_norm(edge_index, n, edge_weight, add_self_loops, fill)
        return self.aggregate_backward(edge_index, n, grad_out, "sum", w=nrm["w_norm"],
                                       self_w=nrm["self_w"])

    def max_argmax(self, edge_index, n, x, w=None):
        """(out [N, F], argmax int32 [N, F]): first edge (original order) with
        the largest fp32 product per (target, feature), -1 without edges."""
        ei = np.ascontiguousarray(edge_index, dtype=np.int64)
        e = ei.shape[1]
        x = widen(x)
        f = x.shape[1]
        w32 = None if w is None else np.ascontiguousarray(w, np.float32)
        out = np.zeros((max(n, 1), f))
        arg = np.zeros((max(n, 1), f), np.int32)
        self._check(self.lib.oracle_max_argmax(n, e, self._p(ei), self._p(w32), self._p(x), f,
                                               self._p(out), self._p(arg)))
        return out[:n], arg[:n]

    def max_backward(self, edge_index, n, argmax, grad_out, w=None):
        """dL/dx of the max: w_e grad_out[t, c] to the source of edge argmax[t, c]."""
        ei = np.ascontiguousarray(edge_index, dtype=np.int64)
        w = None if w is None else np.ascontiguousarray(w, np.float64)
        e = ei.shape[1]
        g = widen(grad_out)
        f = g.shape[1]
        arg = np.ascontiguousarray(argmax, np.int32)
        out = np.zeros((max(n, 1), f))
        ab = np.zeros((max(n, 1), f))
        self._check(self.lib.oracle_max_backward(n, e, self._p(ei), self._p(arg), self._p(w),
                                                 self._p(g), f, self._p(out), self._p(ab)))
        return out[:n], ab[:n]

    # -- dot-product (Transformer-style) attention ----------------------
    def dot_softmax(self, edge_index, n, q, k, v, heads, channels, scale=None):
        """Scaled query-key logits, softmax over each target's in-edges per
        head, attention-weighted sum of values.  scale defaults to 1/sqrt(C).
        Returns (out [N, H*C], alpha [E, H] in COO order, error scale)."""
        ei = np.ascontiguousarray(edge_index, dtype=np.int64)
        e = ei.shape[1]
        q, k, v = widen(q), widen(k), widen(v)
        f = q.shape[1]
        assert f == heads * channels and k.shape == q.shape and v.shape == q.shape
        sc = 1.0 / np.sqrt(channels) if scale is None else float(scale)
        out = np.zeros((max(n, 1), f))
        ab = np.zeros((max(n, 1), f))
        alpha = np.zeros((max(e, 1), heads))
        self._check(self.lib.oracle_dot_softmax(n, e, self._p(ei), self._p(q), self._p(k),
                                                self._p(v), heads, channels, sc, self._p(out),
                                                self._p(alpha), self._p(ab)))
        return out[:n], alpha[:e], ab[:n]

    def dot_softmax_rows(self, csr, n, q, k, v, heads, channels, scale, rows):
        rowptr, col, _, _ = csr
        q, k, v = widen(q), widen(k), widen(v)
        f = q.shape[1]
        rows = np.ascontiguousarray(rows, np.int64)
        total = int(sum(rowptr[r + 1] - rowptr[r] for r in rows))
        out = np.zeros((max(len(rows), 1), f))
        ab = np.zeros((max(len(rows), 1), f))
        alpha = np.zeros((max(total, 1), heads))
        self._check(self.lib.oracle_dot_softmax_rows(
            n, self._p(rowptr), self._p(np.ascontiguousarray(col)), self._p(q), self._p(k),
            self._p(v), heads, channels, float(scale), self._p(rows), len(rows), self._p(out),
            self._p(alpha), self._p(ab)))
        return out[:len(rows)], alpha[:total], ab[:len(rows)]

    # -- multi-hop propagation (APPNP / SGC) ----------------------------
    def appnp(self, edge_index, n, x0, num_hops, alpha, edge_weight=None, add_self_loops=0,
              fill=1.0):
        """K steps of h <- (1 - alpha) Ahat h + alpha x0 from h = x0 (APPNP, the
        propagation model of Section 2.2 / Table 1; alpha = 0 is SGC).  Ahat is the
        GCN normalisation of gcn_norm.  Returns (h_K, error scale), both [N, F]."""
        ei = np.ascontiguousarray(edge_index, dtype=np.int64)
        e = ei.shape[1]
        nrm = self.gcn_norm(ei, n, edge_weight, add_self_loops, fill)
        x0 = widen(x0)
        f = x0.shape[1]
        w = np.ascontiguousarray(nrm["w_norm"], np.float64)
        sw = None if nrm["self_w"] is None else np.ascontiguousarray(nrm["self_w"], np.float64)
        out = np.zeros((max(n, 1), f))
        ab = np.zeros((max(n, 1), f))
        self._check(self.lib.oracle_appnp(n, e, self._p(ei), self._p(w), self._p(sw),
                                          self._p(x0), f, int(num_hops), float(alpha),
                                          self._p(out), self._p(ab)))
        return out[:n], ab[:n]

    def sgc(self, edge_index, n, x0, num_hops, edge_weight=None, add_self_loops=0, fill=1.0):
        """Ahat^K x0 (SGC propagation: APPNP with alpha = 0)."""
        return self.appnp(edge_index, n, x0, num_hops, 0.0, edge_weight, add_self_loops, fill)

    # -- pooling --------------------------------------------------------
    def segment_pool(self, x, batch, num_graphs, reduce):
        x = widen(x)
        n, f = x.shape
        b = np.ascontiguousarray(batch, np.int64)
        out = np.zeros((max(num_graphs, 1), f))
        ab = np.zeros((max(num_graphs, 1), f))
        self._check(self.lib.oracle_segment_pool(REDUCE[reduce], n, f, num_graphs, self._p(b),
                                                 self._p(x), self._p(out), self._p(ab)))
        return out[:num_graphs], ab[:num_graphs]


class _OmpRows:
    """The oracle's row functions over all rows, blocks of rows in parallel on
    every host core (OpenMP).  A CPU baseline for the benchmark; the values
    equal those of the single-threaded row functions."""

    def __init__(self):
        self._lib = None

    @property
    def lib(self) -> ctypes.CDLL:
        with _lock:
            if self._lib is None:
                lib = ctypes.CDLL(build_omp())
                P, I64, I, D = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_double
                lib.oracle_omp_threads.argtypes = []
                lib.oracle_omp_aggregate_all.argtypes = [I, I64, P, P, P, P, P, I64, P, P, P]
                lib.oracle_omp_edge_softmax_all.argtypes = [I64, P, P, P, I, I, P, P, D, P, P]
                for fn in ("oracle_omp_threads", "oracle_omp_aggregate_all",
                           "oracle_omp_edge_softmax_all"):
                    getattr(lib, fn).restype = ctypes.c_int
                self._lib = lib
            return self._lib

    def threads(self) -> int:
        return int(self.lib.oracle_omp_threads())

    def aggregate_all(self, csr, n, x, reduce, w=None, self_w=None):
        rowptr, col, perm, _ = csr
        x = widen(x)
        f = x.shape[1]
        w = None if w is None else np.ascontiguousarray(w, np.float64)
        sw = None if self_w is None else np.ascontiguousarray(self_w, np.float64)
        out = np.zeros((max(n, 1), f))
        ab = np.zeros((max(n, 1), f))
        p = _Oracle._p
        _Oracle._check(self.lib.oracle_omp_aggregate_all(
            REDUCE[reduce], n, p(rowptr), p(np.ascontiguousarray(col)),
            p(np.ascontiguousarray(perm)), p(w), p(x), f, p(sw), p(out), p(ab)))
        return out[:n], ab[:n]

    def edge_softmax_all(self, csr, n, x, heads, channels, a_src, a_dst, slope=0.2):
        rowptr, col, _, _ = csr
        x = widen(x)
        f = x.shape[1]
        a_s = np.ascontiguousarray(a_src, np.float64)
        a_d = np.ascontiguousarray(a_dst, np.float64)
        out = np.zeros((max(n, 1), f))
        ab = np.zeros((max(n, 1), f))
        p = _Oracle._p
        _Oracle._check(self.lib.oracle_omp_edge_softmax_all(
            n, p(rowptr), p(np.ascontiguousarray(col)), p(x), heads, channels, p(a_s), p(a_d),
            float(slope), p(out), p(ab)))
        return out[:n], ab[:n]


omp_rows = _OmpRows()


def batch_graphs(node_counts, edge_counts, edge_index):
    """BatchGraph by the reindexing trick (Section 2.1.1, Fig. 4), one graph
    at a time: node j of graph g becomes offset_g + j with offset_g the number
    of nodes in graphs 0 .. g-1; graph g's edges (the next edge_counts[g]
    columns of the stacked local edge list) are shifted by offset_g.
    Returns (edge_index [2, E], batch [N], offsets [G + 1])."""
    node_counts = [int(c) for c in node_counts]
    edge_counts = [int(c) for c in edge_counts]
    ei = np.asarray(edge_index, dtype=np.int64)
    out = np.empty_like(ei)
    batch = []
    offsets = [0]
    col = 0
    for g, (n_g, e_g) in enumerate(zip(node_counts, edge_counts)):
        off = offsets[-1]
        for k in range(col, col + e_g):
            s, d = int(ei[0, k]), int(ei[1, k])
            if not (0 <= s < n_g and 0 <= d < n_g):
                raise OracleError(-5)
            out[0, k], out[1, k] = off + s, off + d
        col += e_g
        batch.extend([g] * n_g)
        offsets.append(off + n_g)
    return out, np.asarray(batch, dtype=np.int64), np.asarray(offsets, dtype=np.int64)


def segment_pool_meanmax(x, batch, num_graphs):
    """Mean-Max Pool readout (Table 2): [mean | max] per graph."""
    mean, amean = default.segment_pool(x, batch, num_graphs, "mean")
    mx, amax = default.segment_pool(x, batch, num_graphs, "max")
    return np.concatenate([mean, mx], axis=1), np.concatenate([amean, amax], axis=1)


def widen(x: np.ndarray) -> np.ndarray:
    """fp32 -> float64 exactly; uint16 is read as bf16 bit patterns."""
    x = np.asarray(x)
    if x.dtype == np.uint16:
        x = (x.astype(np.uint32) << 16).view(np.float32)
    return np.ascontiguousarray(x, dtype=np.float64)


# ---------------------------------------------------------------------------
# numpy dense forms (tiny graphs only): an independent route to the same numbers
# ---------------------------------------------------------------------------
def dense_adjacency(edge_index, n, edge_weight=None) -> np.ndarray:
    """M[t, s] = total weight of the edges s -> t (messages flow source -> target)."""
    m = np.zeros((n, n))
    w = np.ones(edge_index.shape[1]) if edge_weight is None else np.asarray(edge_weight, float)
    for k in range(edge_index.shape[1]):
        m[edge_index[1, k], edge_index[0, k]] += w[k]
    return m


def dense_gcn_matrix(edge_index, n, edge_weight=None, add_self_loops=0, fill=1.0) -> np.ndarray:
    """D^-1/2 (A' + fill I) D^-1/2 with D the row sums (weighted in-degrees)."""
    m = dense_adjacency(edge_index, n, edge_weight)
    if add_self_loops:
        m = m + fill * np.eye(n)
    d = m.sum(axis=1)
    dinv = np.where(d > 0, 1.0 / np.sqrt(np.where(d > 0, d, 1.0)), 0.0)
    return dinv[:, None] * m * dinv[None, :]


default = _Oracle()
build_csr = default.build_csr
gcn_norm = default.gcn_norm
aggregate = default.aggregate
gcn_aggregate = default.gcn_aggregate
aggregate_rows = default.aggregate_rows
edge_softmax = default.edge_softmax
edge_softmax_rows = default.edge_softmax_rows
segment_pool = default.segment_pool
appnp = default.appnp
dot_softmax = default.dot_softmax
aggregate_backward = default.aggregate_backward
gcn_aggregate_backward = default.gcn_aggregate_backward
max_argmax = default.max_argmax
max_backward = default.max_backward
edge_softmax_backward = default.edge_softmax_backward
dot_softmax_backward = default.dot_softmax_backward
dot_softmax_rows = default.dot_softmax_rows
sgc = default.sgc


def planted(plant: str) -> _Oracle:
    """An oracle compiled with one ORACLE_PLANT_<plant> mistake (for pin tests)."""
    return _Oracle(plant)
