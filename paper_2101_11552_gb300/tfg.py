"""Thin Python binding of libtfg (the C ABI in include/tfg.h).

Argument marshalling only: it checks tensor devices, dtypes and shapes,
allocates output and workspace tensors with PyTorch (device memory), passes
raw pointers and the current CUDA stream, and turns error codes into
exceptions.  Every step of the computation runs in the CUDA kernels of
libtfg.so; there is no CPU fallback.  If the library has not been built, the
first call raises.

Function names follow the ABI (``tfg_build_csr`` ...).  All tensors must be
CUDA tensors on the same device; calls are asynchronous on the current stream.
"""
from __future__ import annotations

import ctypes
import math
import os
import threading
from typing import NamedTuple, Optional

import torch

LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libtfg.so")

TFG_OK = 0
TFG_ERR_INVALID_ARG = -1
TFG_ERR_TOO_LARGE = -2
TFG_ERR_WORKSPACE = -3
TFG_ERR_CUDA = -4
TFG_ERR_INDEX_RANGE = -5
TFG_ERR_UNSORTED = -6
TFG_ERR_TIMEOUT = -7
TFG_F32, TFG_BF16 = 0, 1
REDUCERS = {"sum": 0, "mean": 1, "max": 2}

_lock = threading.Lock()
_lib: Optional[ctypes.CDLL] = None


class TfgError(RuntimeError):
    def __init__(self, code: int, message: str):
        super().__init__(f"libtfg error {code}: {message}")
        self.code = code


def lib() -> ctypes.CDLL:
    """Load libtfg.so (once).  Raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is None:
            _lib = _load(LIB_PATH)
        return _lib


def use_library(path: str) -> ctypes.CDLL:
    """Switch every call of this module to another build of the library (for
    example the bounds-checked debug build, ``build.build_library(defines=
    ("TFG_CHECK_BOUNDS=1",), lib_path=...)``); returns the loaded library."""
    global _lib
    with _lock:
        _lib = _load(path)
        return _lib


def _load(path: str) -> ctypes.CDLL:
    if not os.path.exists(path):
        raise RuntimeError(
            f"{path} is missing: build it first (python -m paper_2101_11552_gb300.build "
            "or __graft_entry__.build()); there is no CPU fallback")
    L = ctypes.CDLL(path)
    P, I64, I, F, SZ = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_float,
                        ctypes.c_size_t)
    sigs = {
        "tfg_version": [],
        "tfg_check_bounds_enabled": [],
        "tfg_build_csr_workspace_size": [I64, I64, ctypes.POINTER(SZ)],
        "tfg_build_csr": [P, I64, I64, P, P, P, P, P, SZ, P, P],
        "tfg_build_csr_by_source": [P, I64, I64, P, P, P, P, P, SZ, P, P],
        "tfg_build_csr32": [P, I64, I64, P, P, P, P, P, SZ, P, P],
        "tfg_build_csr32_by_source": [P, I64, I64, P, P, P, P, P, SZ, P, P],
        "tfg_aggregate_backward_workspace_size": [I, I64, ctypes.POINTER(SZ)],
        "tfg_aggregate_backward": [I, P, P, P, P, P, P, I64, I64, I64, P, P, SZ, P],
        "tfg_gcn_aggregate_backward": [P, P, P, P, I64, I64, I, F, P, P],
        "tfg_aggregate_max_argmax": [P, P, P, P, P, I, I64, I64, P, P, P],
        "tfg_aggregate_max_backward_workspace_size": [I64, I64, I64, ctypes.POINTER(SZ)],
        "tfg_aggregate_max_backward": [P, P, P, P, P, P, I64, I64, I64, P, P, SZ, P],
        "tfg_gcn_norm": [P, P, P, P, I64, I64, I, F, P, P, P],
        "tfg_aggregate_sum": [P, P, P, P, I, I64, I64, P, P],
        "tfg_aggregate_mean": [P, P, P, P, I, I64, I64, P, P],
        "tfg_aggregate_max": [P, P, P, P, I, I64, I64, P, P],
        "tfg_gcn_aggregate_sum": [P, P, P, P, P, I, I64, I64, I, F, P, P],
        "tfg_propagate_workspace_size": [I64, I64, I64, ctypes.POINTER(SZ)],
        "tfg_appnp_propagate": [P, P, P, P, P, I, I64, I64, I64, F, I, F, P, P, SZ, P],
        "tfg_sgc_propagate": [P, P, P, P, P, I, I64, I64, I64, I, F, P, P, SZ, P],
        "tfg_edge_softmax_workspace_size": [I64, I, ctypes.POINTER(SZ)],
        "tfg_edge_softmax_aggregate": [P, P, P, I, I64, I64, I, I, P, P, F, P, P, P, SZ, P],
        "tfg_dot_edge_softmax_aggregate": [P, P, P, P, P, I, I64, I64, I, I, F, P, P, P],
        "tfg_edge_softmax_aggregate_noalloc": [P, P, P, I, I64, I64, I, I, P, P, F, P, P, P],
        "tfg_segment_pool": [P, I, P, I64, I64, I64, I, P, P, P],
        "tfg_segment_pool_meanmax": [P, I, P, I64, I64, I64, P, P, P],
        "tfg_batch_graphs_workspace_size": [I64, ctypes.POINTER(SZ)],
        "tfg_batch_graphs": [I64, P, P, P, I64, I64, P, P, P, P, SZ, P, P],
        "tfg_gather_xor": [P, I64, P, I64, I64, P, P],
        "tfg_edge_softmax_backward_workspace_size": [I64, I, I, ctypes.POINTER(SZ)],
        "tfg_edge_softmax_aggregate_backward": [P, P, P, P, P, I, I64, I64, I, I, P, P, F,
                                                P, P, P, P, P, P, SZ, P],
        "tfg_dot_edge_softmax_backward_workspace_size": [I64, I, I, ctypes.POINTER(SZ)],
        "tfg_dot_edge_softmax_aggregate_backward": [P, P, P, P, P, P, P, I, I64, I64, I, I,
                                                    F, P, P, P, P, P, P, SZ, P],
    }
    for name, args in sigs.items():
        fn = getattr(L, name)
        fn.argtypes = args
        fn.restype = ctypes.c_int
    L.tfg_last_error.argtypes = []
    L.tfg_last_error.restype = ctypes.c_char_p
    return L


def tfg_version() -> int:
    return lib().tfg_version()


def tfg_last_error() -> str:
    return lib().tfg_last_error().decode()


def _check(rc: int):
    if rc != TFG_OK:
        raise TfgError(rc, tfg_last_error())


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(device: torch.device):
    return ctypes.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def _need_cuda(name: str, t: torch.Tensor, dtype=None, device=None):
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if device is not None and t.device != device:
        raise ValueError(f"{name} is on {t.device}, expected {device}")


def _x_dtype(x: torch.Tensor) -> int:
    if x.dtype == torch.float32:
        return TFG_F32
    if x.dtype == torch.bfloat16:
        return TFG_BF16
    raise ValueError(f"features must be float32 or bfloat16, got {x.dtype}")


class CSR(NamedTuple):
    rowptr: torch.Tensor     # int32 [N + 1]
    col: torch.Tensor        # int32 [E]
    perm: torch.Tensor       # int32 [E]
    in_degree: torch.Tensor  # int32 [N]
    status: torch.Tensor     # int32 [1] (device)


def check_status(status: torch.Tensor):
    """Synchronise on the status word and raise if a kernel flagged bad input."""
    code = int(status.item())
    if code != 0:
        raise TfgError(code, "device-side validation failed "
                             f"({'index out of range' if code == TFG_ERR_INDEX_RANGE else 'unsorted batch'})")


def tfg_build_csr_workspace_size(num_nodes: int, num_edges: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().tfg_build_csr_workspace_size(num_nodes, num_edges, ctypes.byref(n)))
    return n.value


def tfg_build_csr(edge_index: torch.Tensor, num_nodes: int,
                  workspace: Optional[torch.Tensor] = None) -> CSR:
    """Group the edges of ``edge_index`` (int64 or int32 [2, E]) by target node."""
    _need_cuda("edge_index", edge_index, None)
    if edge_index.dtype not in (torch.int64, torch.int32):
        raise TypeError("edge_index must be int64 or int32")
    if edge_index.dim() != 2 or edge_index.shape[0] != 2:
        raise ValueError("edge_index must have shape [2, E]")
    dev = edge_index.device
    e = edge_index.shape[1]
    rowptr = torch.empty(num_nodes + 1, dtype=torch.int32, device=dev)
    col = torch.empty(e, dtype=torch.int32, device=dev)
    perm = torch.empty(e, dtype=torch.int32, device=dev)
    deg = torch.empty(num_nodes, dtype=torch.int32, device=dev)
    status = torch.empty(1, dtype=torch.int32, device=dev)
    need = tfg_build_csr_workspace_size(num_nodes, e)
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=dev)
    fn = lib().tfg_build_csr32 if edge_index.dtype == torch.int32 else lib().tfg_build_csr
    _check(fn(_ptr(edge_index), e, num_nodes, _ptr(rowptr), _ptr(col), _ptr(perm), _ptr(deg),
              _ptr(workspace), workspace.numel(), _ptr(status), _stream(dev)))
    return CSR(rowptr, col, perm, deg, status)


def tfg_build_csr_by_source(edge_index: torch.Tensor, num_nodes: int,
                            workspace: Optional[torch.Tensor] = None) -> CSR:
    """Group the edges by SOURCE (the transposed graph's CSR).  Returns the CSR
    tuple with rowptr over sources, col = targets, perm = original edge ids,
    in_degree = out-degrees."""
    _need_cuda("edge_index", edge_index, None)
    if edge_index.dtype not in (torch.int64, torch.int32):
        raise TypeError("edge_index must be int64 or int32")
    if edge_index.dim() != 2 or edge_index.shape[0] != 2:
        raise ValueError("edge_index must have shape [2, E]")
    dev = edge_index.device
    e = edge_index.shape[1]
    rowptr = torch.empty(num_nodes + 1, dtype=torch.int32, device=dev)
    col = torch.empty(e, dtype=torch.int32, device=dev)
    perm = torch.empty(e, dtype=torch.int32, device=dev)
    deg = torch.empty(num_nodes, dtype=torch.int32, device=dev)
    status = torch.empty(1, dtype=torch.int32, device=dev)
    need = tfg_build_csr_workspace_size(num_nodes, e)
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=dev)
    fn = (lib().tfg_build_csr32_by_source if edge_index.dtype == torch.int32
          else lib().tfg_build_csr_by_source)
    _check(fn(_ptr(edge_index), e, num_nodes, _ptr(rowptr), _ptr(col), _ptr(perm), _ptr(deg),
              _ptr(workspace), workspace.numel(), _ptr(status), _stream(dev)))
    return CSR(rowptr, col, perm, deg, status)


def tfg_aggregate_backward(reduce: str, csr_src: CSR, grad_out, edge_weight=None, in_degree=None,
                           out=None):
    """grad_x of tfg_aggregate_sum / _mean: the sum over the transposed graph
    (csr_src from tfg_build_csr_by_source; edge_weight in original order; the
    forward CSR's in_degree for the mean)."""
    _need_cuda("grad_out", grad_out, torch.float32)
    dev = grad_out.device
    n, f = grad_out.shape
    e = csr_src.col.numel()
    code = REDUCERS[reduce]
    nb = ctypes.c_size_t(0)
    _check(lib().tfg_aggregate_backward_workspace_size(code, e, ctypes.byref(nb)))
    ws = torch.empty(max(nb.value, 1), dtype=torch.uint8, device=dev)
    if out is None:
        out = torch.empty(n, f, dtype=torch.float32, device=dev)
    _check(lib().tfg_aggregate_backward(code, _ptr(csr_src.rowptr), _ptr(csr_src.col), _ptr(csr_src.perm),
                                        _ptr(edge_weight), _ptr(in_degree), _ptr(grad_out), n, e, f,
                                        _ptr(out), _ptr(ws), ws.numel(), _stream(dev)))
    return out


def tfg_gcn_aggregate_backward(csr_src: CSR, dinv, grad_out, add_self_loops: int = 0,
                               self_loop_fill: float = 1.0, out=None):
    """grad_x of tfg_gcn_aggregate_sum (on-the-fly weights), with the forward's dinv."""
    _need_cuda("grad_out", grad_out, torch.float32)
    dev = grad_out.device
    n, f = grad_out.shape
    if out is None:
        out = torch.empty(n, f, dtype=torch.float32, device=dev)
    _check(lib().tfg_gcn_aggregate_backward(_ptr(csr_src.rowptr), _ptr(csr_src.col), _ptr(dinv),
                                            _ptr(grad_out), n, f, int(add_self_loops),
                                            float(self_loop_fill), _ptr(out), _stream(dev)))
    return out


def tfg_aggregate_max_argmax(csr: CSR, x, w_csr=None):
    """(out, argmax): the max aggregation and, per (t, f), the original id of
    the first edge attaining it (-1 for a row without edges)."""
    _need_cuda("x", x)
    dev = x.device
    n, f = x.shape
    out = torch.empty(n, f, dtype=torch.float32, device=dev)
    arg = torch.empty(n, f, dtype=torch.int32, device=dev)
    _check(lib().tfg_aggregate_max_argmax(_ptr(csr.rowptr), _ptr(csr.col), _ptr(csr.perm), _ptr(w_csr),
                                          _ptr(x), _x_dtype(x), n, f, _ptr(out), _ptr(arg), _stream(dev)))
    return out, arg


def tfg_aggregate_max_backward_workspace_size(num_nodes: int, num_edges: int,
                                              num_features: int) -> int:
    nb = ctypes.c_size_t(0)
    _check(lib().tfg_aggregate_max_backward_workspace_size(num_nodes, num_edges, num_features,
                                                           ctypes.byref(nb)))
    return nb.value


def tfg_aggregate_max_backward(csr_src: CSR, argmax, grad_out, edge_weight=None, out=None,
                               marks: bool = True):
    """grad_x of the max: w_e grad_out[t, f] to the source of the edge argmax[t, f]
    (edge_weight in original edge order, or None).  marks=False runs without the
    win-mark workspace (every out-edge's rows read; the same result)."""
    _need_cuda("grad_out", grad_out, torch.float32)
    dev = grad_out.device
    n, f = grad_out.shape
    e = csr_src.col.numel()
    ws = None
    nb = tfg_aggregate_max_backward_workspace_size(n, e, f) if marks else 0
    if nb > 0:
        ws = torch.empty(nb, dtype=torch.uint8, device=dev)
    if out is None:
        out = torch.empty(n, f, dtype=torch.float32, device=dev)
    _check(lib().tfg_aggregate_max_backward(_ptr(csr_src.rowptr), _ptr(csr_src.col), _ptr(csr_src.perm),
                                            _ptr(argmax), _ptr(edge_weight), _ptr(grad_out), n, e, f,
                                            _ptr(out), _ptr(ws), ws.numel() if ws is not None else 0,
                                            _stream(dev)))
    return out


def tfg_gcn_norm(rowptr: torch.Tensor, col: torch.Tensor, perm: torch.Tensor, num_nodes: int,
                 edge_weight: Optional[torch.Tensor] = None, add_self_loops: int = 0,
                 self_loop_fill: float = 1.0, want_w_csr: bool = True):
    """Return (dinv [N], w_csr [E] or None) of the GCN normalisation of A + I."""
    _need_cuda("rowptr", rowptr, torch.int32)
    dev = rowptr.device
    e = col.numel()
    if edge_weight is not None:
        _need_cuda("edge_weight", edge_weight, torch.float32, dev)
    dinv = torch.empty(num_nodes, dtype=torch.float32, device=dev)
    w_csr = torch.empty(e, dtype=torch.float32, device=dev) if want_w_csr else None
    _check(lib().tfg_gcn_norm(_ptr(rowptr), _ptr(col), _ptr(perm), _ptr(edge_weight), num_nodes, e,
                              int(add_self_loops), float(self_loop_fill), _ptr(dinv), _ptr(w_csr),
                              _stream(dev)))
    return dinv, w_csr


def _aggregate(fn_name: str, rowptr, col, x, w_csr, out):
    _need_cuda("rowptr", rowptr, torch.int32)
    dev = rowptr.device
    _need_cuda("col", col, torch.int32, dev)
    _need_cuda("x", x, None, dev)
    n, f = x.shape
    if rowptr.numel() != n + 1:
        raise ValueError("rowptr must have N + 1 entries")
    if w_csr is not None:
        _need_cuda("w_csr", w_csr, torch.float32, dev)
    if out is None:
        out = torch.empty(n, f, dtype=torch.float32, device=dev)
    _need_cuda("out", out, torch.float32, dev)
    _check(getattr(lib(), fn_name)(_ptr(rowptr), _ptr(col), _ptr(w_csr), _ptr(x), _x_dtype(x), n, f,
                                   _ptr(out), _stream(dev)))
    return out


def tfg_aggregate_sum(rowptr, col, x, w_csr=None, out=None):
    return _aggregate("tfg_aggregate_sum", rowptr, col, x, w_csr, out)


def tfg_aggregate_mean(rowptr, col, x, w_csr=None, out=None):
    return _aggregate("tfg_aggregate_mean", rowptr, col, x, w_csr, out)


def tfg_aggregate_max(rowptr, col, x, w_csr=None, out=None):
    return _aggregate("tfg_aggregate_max", rowptr, col, x, w_csr, out)


def tfg_gcn_aggregate_sum(rowptr, col, dinv, x, w_csr=None, add_self_loops: int = 0,
                          self_loop_fill: float = 1.0, out=None):
    _need_cuda("rowptr", rowptr, torch.int32)
    dev = rowptr.device
    _need_cuda("col", col, torch.int32, dev)
    _need_cuda("dinv", dinv, torch.float32, dev)
    _need_cuda("x", x, None, dev)
    n, f = x.shape
    if rowptr.numel() != n + 1:
        raise ValueError("rowptr must have N + 1 entries")
    if w_csr is not None:
        _need_cuda("w_csr", w_csr, torch.float32, dev)
    if out is None:
        out = torch.empty(n, f, dtype=torch.float32, device=dev)
    _need_cuda("out", out, torch.float32, dev)
    _check(lib().tfg_gcn_aggregate_sum(_ptr(rowptr), _ptr(col), _ptr(dinv), _ptr(w_csr), _ptr(x),
                                       _x_dtype(x), n, f, int(add_self_loops),
                                       float(self_loop_fill), _ptr(out), _stream(dev)))
    return out


def tfg_propagate_workspace_size(num_nodes: int, num_features: int, num_hops: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().tfg_propagate_workspace_size(num_nodes, num_features, num_hops, ctypes.byref(n)))
    return n.value


def tfg_appnp_propagate(rowptr, col, dinv, x0, num_hops: int, alpha: float, w_csr=None,
                        add_self_loops: int = 0, self_loop_fill: float = 1.0, out=None,
                        workspace=None):
    """h_{k+1} = (1 - alpha) Ahat h_k + alpha x0, h_0 = x0; returns h_K (fp32)."""
    return _propagate("tfg_appnp_propagate", rowptr, col, dinv, x0, num_hops, alpha, w_csr,
                      add_self_loops, self_loop_fill, out, workspace)


def tfg_sgc_propagate(rowptr, col, dinv, x0, num_hops: int, w_csr=None, add_self_loops: int = 0,
                      self_loop_fill: float = 1.0, out=None, workspace=None):
    """Ahat^K x0 (fp32)."""
    return _propagate("tfg_sgc_propagate", rowptr, col, dinv, x0, num_hops, None, w_csr,
                      add_self_loops, self_loop_fill, out, workspace)


def _propagate(name, rowptr, col, dinv, x0, num_hops, alpha, w_csr, add_self_loops,
               self_loop_fill, out, workspace):
    _need_cuda("rowptr", rowptr, torch.int32)
    dev = rowptr.device
    _need_cuda("col", col, torch.int32, dev)
    _need_cuda("dinv", dinv, torch.float32, dev)
    _need_cuda("x0", x0, None, dev)
    n, f = x0.shape
    if rowptr.numel() != n + 1:
        raise ValueError("rowptr must have N + 1 entries")
    if w_csr is not None:
        _need_cuda("w_csr", w_csr, torch.float32, dev)
    if out is None:
        out = torch.empty(n, f, dtype=torch.float32, device=dev)
    _need_cuda("out", out, torch.float32, dev)
    nb = tfg_propagate_workspace_size(n, f, num_hops)
    if workspace is None or workspace.numel() < nb:
        workspace = torch.empty(max(nb, 1), dtype=torch.uint8, device=dev)
    head = [_ptr(rowptr), _ptr(col), _ptr(dinv), _ptr(w_csr), _ptr(x0), _x_dtype(x0), n, f,
            int(num_hops)]
    tail = [int(add_self_loops), float(self_loop_fill), _ptr(out), _ptr(workspace),
            workspace.numel(), _stream(dev)]
    fn = getattr(lib(), name)
    _check(fn(*head, *([] if alpha is None else [float(alpha)]), *tail))
    return out


def tfg_edge_softmax_workspace_size(num_nodes: int, heads: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().tfg_edge_softmax_workspace_size(num_nodes, heads, ctypes.byref(n)))
    return n.value


def tfg_edge_softmax_aggregate(rowptr, col, x, heads: int, channels: int, a_src, a_dst,
                               negative_slope: float = 0.2, want_alpha: bool = False,
                               out=None, workspace=None):
    """Return (out [N, H*C], alpha [E, H] in CSR order or None)."""
    _need_cuda("rowptr", rowptr, torch.int32)
    dev = rowptr.device
    _need_cuda("col", col, torch.int32, dev)
    _need_cuda("x", x, None, dev)
    _need_cuda("a_src", a_src, torch.float32, dev)
    _need_cuda("a_dst", a_dst, torch.float32, dev)
    n, f = x.shape
    if f != heads * channels:
        raise ValueError("x must have heads * channels columns")
    e = col.numel()
    if out is None:
        out = torch.empty(n, f, dtype=torch.float32, device=dev)
    alpha = torch.empty(e, heads, dtype=torch.float32, device=dev) if want_alpha else None
    need = tfg_edge_softmax_workspace_size(n, heads)
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=dev)
    _check(lib().tfg_edge_softmax_aggregate(_ptr(rowptr), _ptr(col), _ptr(x), _x_dtype(x), n, e,
                                            heads, channels,
                                            _ptr(a_src), _ptr(a_dst), float(negative_slope),
                                            _ptr(out), _ptr(alpha), _ptr(workspace),
                                            workspace.numel(), _stream(dev)))
    return out, alpha


def tfg_dot_edge_softmax_aggregate(rowptr, col, q, k, v, heads: int, channels: int,
                                   scale: Optional[float] = None, want_alpha: bool = False,
                                   out=None, alpha=None):
    """Transformer-style attention over in-edges; scale defaults to 1/sqrt(channels).
    Returns (out [N, H*C] fp32, alpha [E, H] or None)."""
    _need_cuda("rowptr", rowptr, torch.int32)
    dev = rowptr.device
    _need_cuda("col", col, torch.int32, dev)
    _need_cuda("q", q, None, dev)
    _need_cuda("k", k, q.dtype, dev)
    _need_cuda("v", v, q.dtype, dev)
    n, f = q.shape
    if k.shape != q.shape or v.shape != q.shape:
        raise ValueError("q, k and v must have the same shape")
    if f != heads * channels:
        raise ValueError("feature width must equal heads * channels")
    e = col.numel()
    if scale is None:
        scale = 1.0 / math.sqrt(channels)
    if out is None:
        out = torch.empty(n, f, dtype=torch.float32, device=dev)
    if want_alpha and alpha is None:
        alpha = torch.empty(e, heads, dtype=torch.float32, device=dev)
    _check(lib().tfg_dot_edge_softmax_aggregate(
        _ptr(rowptr), _ptr(col), _ptr(q), _ptr(k), _ptr(v), _x_dtype(q), n, e, heads, channels,
        float(scale), _ptr(out), _ptr(alpha), _stream(dev)))
    return out, alpha


def tfg_edge_softmax_aggregate_noalloc(rowptr, col, x, heads: int, channels: int, a_src, a_dst,
                                       negative_slope: float = 0.2, out=None, alpha=None):
    """Edge-softmax aggregation through the entry point that allocates nothing.

    The library keeps the node scores in its own fixed device array, so the
    C call takes no workspace; ``out`` (and ``alpha`` if wanted) may be passed
    in preallocated so that nothing at all is allocated.  Returns
    (out, alpha)."""
    _need_cuda("rowptr", rowptr, torch.int32)
    dev = rowptr.device
    _need_cuda("col", col, torch.int32, dev)
    _need_cuda("x", x, None, dev)
    _need_cuda("a_src", a_src, torch.float32, dev)
    _need_cuda("a_dst", a_dst, torch.float32, dev)
    n, f = x.shape
    if f != heads * channels:
        raise ValueError("x must have heads * channels columns")
    if out is None:
        out = torch.empty(n, f, dtype=torch.float32, device=dev)
    _check(lib().tfg_edge_softmax_aggregate_noalloc(
        _ptr(rowptr), _ptr(col), _ptr(x), _x_dtype(x), n, col.numel(), heads, channels,
        _ptr(a_src), _ptr(a_dst), float(negative_slope), _ptr(out), _ptr(alpha), _stream(dev)))
    return out, alpha


def tfg_segment_pool(x, batch, num_graphs: int, reduce: str = "sum", out=None):
    """Return (out [G, F], status) -- status is the device status word."""
    _need_cuda("x", x)
    dev = x.device
    _need_cuda("batch", batch, torch.int64, dev)
    n, f = x.shape
    if out is None:
        out = torch.empty(num_graphs, f, dtype=torch.float32, device=dev)
    status = torch.empty(1, dtype=torch.int32, device=dev)
    _check(lib().tfg_segment_pool(_ptr(x), _x_dtype(x), _ptr(batch), n, num_graphs, f,
                                  REDUCERS[reduce], _ptr(out), _ptr(status), _stream(dev)))
    return out, status


def tfg_segment_pool_meanmax(x, batch, num_graphs: int, out=None):
    """Return (out [G, 2F] = [mean | max], status)."""
    _need_cuda("x", x)
    dev = x.device
    _need_cuda("batch", batch, torch.int64, dev)
    n, f = x.shape
    if out is None:
        out = torch.empty(num_graphs, 2 * f, dtype=torch.float32, device=dev)
    status = torch.empty(1, dtype=torch.int32, device=dev)
    _check(lib().tfg_segment_pool_meanmax(_ptr(x), _x_dtype(x), _ptr(batch), n, num_graphs, f,
                                          _ptr(out), _ptr(status), _stream(dev)))
    return out, status


def tfg_batch_graphs_workspace_size(num_graphs: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().tfg_batch_graphs_workspace_size(num_graphs, ctypes.byref(n)))
    return n.value


class BatchGraph(NamedTuple):
    edge_index: torch.Tensor    # int64 [2, E]
    batch: torch.Tensor         # int64 [N]
    node_offsets: torch.Tensor  # int64 [G + 1]
    status: torch.Tensor        # int32 [1] (device)


def tfg_batch_graphs(node_counts: torch.Tensor, edge_counts: torch.Tensor,
                     edge_index: torch.Tensor, total_nodes: int) -> BatchGraph:
    """Combine graphs into one BatchGraph on the device (reindexing trick)."""
    _need_cuda("node_counts", node_counts, torch.int64)
    dev = node_counts.device
    _need_cuda("edge_counts", edge_counts, torch.int64, dev)
    _need_cuda("edge_index", edge_index, torch.int64, dev)
    g = node_counts.numel()
    e = edge_index.shape[1]
    out_ei = torch.empty(2, e, dtype=torch.int64, device=dev)
    batch = torch.empty(total_nodes, dtype=torch.int64, device=dev)
    offs = torch.empty(g + 1, dtype=torch.int64, device=dev)
    status = torch.empty(1, dtype=torch.int32, device=dev)
    ws = torch.empty(tfg_batch_graphs_workspace_size(g), dtype=torch.uint8, device=dev)
    _check(lib().tfg_batch_graphs(g, _ptr(node_counts), _ptr(edge_counts), _ptr(edge_index), e,
                                  total_nodes, _ptr(out_ei), _ptr(batch), _ptr(offs), _ptr(ws),
                                  ws.numel(), _ptr(status), _stream(dev)))
    return BatchGraph(out_ei, batch, offs, status)


def tfg_gather_xor(col: torch.Tensor, x: torch.Tensor, out=None) -> torch.Tensor:
    """Gather-only floor: every row x[col[k]] read once and XOR-folded.
    Returns uint32 words as an int32 tensor [row_bytes / 4]."""
    _need_cuda("col", col, torch.int32)
    _need_cuda("x", x)
    dev = x.device
    row_bytes = x[0].numel() * x.element_size() if x.shape[0] else 16
    if out is None:
        out = torch.empty(row_bytes // 4, dtype=torch.int32, device=dev)
    _check(lib().tfg_gather_xor(_ptr(col), col.numel(), _ptr(x), x.shape[0], row_bytes, _ptr(out),
                                _stream(dev)))
    return out


def tfg_edge_softmax_backward_workspace_size(num_nodes: int, heads: int, channels: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().tfg_edge_softmax_backward_workspace_size(num_nodes, heads, channels,
                                                          ctypes.byref(n)))
    return n.value


def tfg_edge_softmax_aggregate_backward(rowptr, col, rowptr_src, col_src, x, heads: int,
                                        channels: int, a_src, a_dst, negative_slope: float,
                                        out, grad_out):
    """Gradients of tfg_edge_softmax_aggregate with respect to x, a_src and
    a_dst.  Returns (grad_x [N, H*C], grad_a_src [H*C], grad_a_dst [H*C])."""
    _need_cuda("x", x)
    dev = x.device
    for name, t, dt in (("rowptr", rowptr, torch.int32), ("col", col, torch.int32),
                        ("rowptr_src", rowptr_src, torch.int32), ("col_src", col_src, torch.int32),
                        ("a_src", a_src, torch.float32), ("a_dst", a_dst, torch.float32),
                        ("out", out, torch.float32), ("grad_out", grad_out, torch.float32)):
        _need_cuda(name, t, dt, dev)
    n = x.shape[0]
    f = heads * channels
    grad_x = torch.empty(n, f, dtype=torch.float32, device=dev)
    ga_src = torch.empty(f, dtype=torch.float32, device=dev)
    ga_dst = torch.empty(f, dtype=torch.float32, device=dev)
    ws = torch.empty(max(tfg_edge_softmax_backward_workspace_size(n, heads, channels), 1),
                     dtype=torch.uint8, device=dev)
    _check(lib().tfg_edge_softmax_aggregate_backward(
        _ptr(rowptr), _ptr(col), _ptr(rowptr_src), _ptr(col_src), _ptr(x), _x_dtype(x), n,
        col.numel(), heads, channels, _ptr(a_src), _ptr(a_dst), negative_slope, _ptr(out),
        _ptr(grad_out), _ptr(grad_x), _ptr(ga_src), _ptr(ga_dst), _ptr(ws), ws.numel(),
        _stream(dev)))
    return grad_x, ga_src, ga_dst


def tfg_dot_edge_softmax_backward_workspace_size(num_nodes: int, heads: int, channels: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().tfg_dot_edge_softmax_backward_workspace_size(num_nodes, heads, channels,
                                                              ctypes.byref(n)))
    return n.value


def tfg_dot_edge_softmax_aggregate_backward(rowptr, col, rowptr_src, col_src, q, k, v,
                                            heads: int, channels: int, scale: float, out,
                                            grad_out):
    """Gradients of tfg_dot_edge_softmax_aggregate with respect to q, k and v.
    Returns (grad_q, grad_k, grad_v), each [N, H*C] fp32."""
    _need_cuda("q", q)
    dev = q.device
    _need_cuda("k", k, q.dtype, dev)
    _need_cuda("v", v, q.dtype, dev)
    for name, t, dt in (("rowptr", rowptr, torch.int32), ("col", col, torch.int32),
                        ("rowptr_src", rowptr_src, torch.int32), ("col_src", col_src, torch.int32),
                        ("out", out, torch.float32), ("grad_out", grad_out, torch.float32)):
        _need_cuda(name, t, dt, dev)
    n = q.shape[0]
    f = heads * channels
    grads = [torch.empty(n, f, dtype=torch.float32, device=dev) for _ in range(3)]
    ws = torch.empty(max(tfg_dot_edge_softmax_backward_workspace_size(n, heads, channels), 1),
                     dtype=torch.uint8, device=dev)
    _check(lib().tfg_dot_edge_softmax_aggregate_backward(
        _ptr(rowptr), _ptr(col), _ptr(rowptr_src), _ptr(col_src), _ptr(q), _ptr(k), _ptr(v),
        _x_dtype(q), n, col.numel(), heads, channels, float(scale), _ptr(out), _ptr(grad_out),
        _ptr(grads[0]), _ptr(grads[1]), _ptr(grads[2]), _ptr(ws), ws.numel(), _stream(dev)))
    return tuple(grads)
