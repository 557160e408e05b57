"""Python binding of liblast (GB300 / sm_103a) -- argument marshalling only.

Every step of the path runs in the CUDA kernels of liblast.so; this module
only turns torch tensors (and, for last_prune_host, host buffers) into pointers
and host offset arrays into the C problem struct.  There is no CPU fallback: if
the library is missing, every call raises.

Functions carry the names of the C entry points in include/last.h:
  last_workspace_size, last_scores, last_select, last_select_topk, last_gather,
  last_prune, last_host_workspace_size, last_prune_host, last_scores_rows,
  last_scores_rows_workspace_size, last_scores_noalloc, last_check_bounded_wait,
  last_poll, last_budget, last_status_string, last_error_message.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "liblast.so")

LAST_OK = 0
LAST_ERR_INVALID_ARG = 1
LAST_ERR_UNSUPPORTED = 2
LAST_ERR_WORKSPACE_TOO_SMALL = 3
LAST_ERR_CUDA = 4
LAST_ERR_DEVICE_INDEX = 5
LAST_ERR_TIMEOUT = 6

LAST_DTYPE_F32 = 0
LAST_DTYPE_BF16 = 1

EXPORTED = ("last_workspace_size", "last_scores", "last_select", "last_gather", "last_prune",
            "last_poll", "last_budget", "last_status_string", "last_error_message",
            "last_scores_noalloc", "last_select_topk", "last_scores_rows",
            "last_scores_rows_workspace_size", "last_check_bounded_wait",
            "last_host_workspace_size", "last_prune_host")


class LastError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{_status_name(status)}: {message}")
        self.status = status


class _Problem(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("num_layers", ctypes.c_int32),
                ("num_q_heads", ctypes.c_int32), ("num_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("feat_dim", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("softmax_scale", ctypes.c_float),
                ("cu_seqlens", ctypes.POINTER(ctypes.c_int32)),
                ("vis_start", ctypes.POINTER(ctypes.c_int32)),
                ("cu_vis", ctypes.POINTER(ctypes.c_int32)),
                ("cu_keep", ctypes.POINTER(ctypes.c_int32))]


_lib = None


def load_library(path: str = LIB_PATH):
    """Loads liblast.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with "
                          "`python -c 'import __graft_entry__ as g; g.build()'`")
    try:  # share the CUDA runtime that torch loads
        import torch  # noqa: F401
    except ImportError:
        pass
    lib = ctypes.CDLL(path)
    P = ctypes.c_void_p
    PP = ctypes.POINTER(_Problem)
    lib.last_workspace_size.argtypes = [PP, ctypes.POINTER(ctypes.c_size_t)]
    lib.last_scores.argtypes = [PP, P, P, P, P, ctypes.c_size_t, P]
    lib.last_select.argtypes = [PP, P, P, P, P, P, ctypes.c_size_t, P]
    lib.last_gather.argtypes = [PP, P, P, P, P, ctypes.c_size_t, P]
    lib.last_select_topk.argtypes = [PP, P, P, P, P, P, ctypes.c_size_t, P]
    PI = ctypes.POINTER(ctypes.c_int32)
    lib.last_scores_rows.argtypes = [PP, PI, PI, P, P, P, P, ctypes.c_size_t, P]
    lib.last_scores_rows_workspace_size.argtypes = [PP, PI, PI, ctypes.POINTER(ctypes.c_size_t)]
    lib.last_prune.argtypes = [PP, P, P, P, P, P, P, P, ctypes.c_size_t, P]
    lib.last_host_workspace_size.argtypes = [PP, ctypes.POINTER(ctypes.c_size_t)]
    lib.last_prune_host.argtypes = [PP, P, P, P, P, P, P, P, ctypes.c_size_t, P]
    lib.last_poll.argtypes = [P, P]
    lib.last_check_bounded_wait.argtypes = [P, P]
    lib.last_scores_noalloc.argtypes = [PP, P, P, P, P]
    lib.last_budget.argtypes = [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32]
    lib.last_budget.restype = ctypes.c_int32
    lib.last_status_string.argtypes = [ctypes.c_int]
    lib.last_status_string.restype = ctypes.c_char_p
    lib.last_error_message.argtypes = []
    lib.last_error_message.restype = ctypes.c_char_p
    for name in ("last_workspace_size", "last_scores", "last_select", "last_gather",
                 "last_prune", "last_poll", "last_scores_noalloc", "last_select_topk",
                 "last_scores_rows", "last_scores_rows_workspace_size",
                 "last_check_bounded_wait"):
        getattr(lib, name).restype = ctypes.c_int
    _lib = lib
    return lib


def _status_name(st: int) -> str:
    try:
        return load_library().last_status_string(st).decode()
    except ImportError:
        return f"status {st}"


def _check(st: int):
    if st != LAST_OK:
        msg = load_library().last_error_message().decode()
        raise LastError(st, msg)


class Problem:
    """Problem description (include/last.h `last_problem`); keeps its host arrays alive."""

    def __init__(self, *, batch: int, num_layers: int, num_q_heads: int, num_kv_heads: int,
                 head_dim: int, feat_dim: int, dtype: str, cu_seqlens: Optional[Sequence[int]],
                 vis_start: Optional[Sequence[int]], cu_vis: Sequence[int],
                 cu_keep: Sequence[int], softmax_scale: float = 0.0):
        def arr(a):
            return None if a is None else np.ascontiguousarray(np.asarray(a, dtype=np.int32))
        self.arrays = dict(cu_seqlens=arr(cu_seqlens), vis_start=arr(vis_start),
                           cu_vis=arr(cu_vis), cu_keep=arr(cu_keep))
        self.dtype = dtype
        code = {"f32": LAST_DTYPE_F32, "bf16": LAST_DTYPE_BF16}[dtype]

        def ptr(a):
            return None if a is None else a.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))
        self.c = _Problem(batch, num_layers, num_q_heads, num_kv_heads, head_dim, feat_dim, code,
                          float(softmax_scale), ptr(self.arrays["cu_seqlens"]),
                          ptr(self.arrays["vis_start"]), ptr(self.arrays["cu_vis"]),
                          ptr(self.arrays["cu_keep"]))
        self.batch = batch
        self.feat_dim = feat_dim
        self.total_vis = int(self.arrays["cu_vis"][-1])
        self.total_keep = int(self.arrays["cu_keep"][-1])

    @property
    def ref(self):
        return ctypes.byref(self.c)


def _ptr(t) -> Optional[int]:
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if not t.is_cuda:
        raise ValueError("liblast takes device tensors")
    if not t.is_contiguous():
        raise ValueError("liblast takes contiguous tensors")
    return t.data_ptr()


def _host_ptr(t) -> Optional[int]:
    """Address of a contiguous host buffer: a CPU torch tensor (pinned for
    asynchronous copies) or a numpy array."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if isinstance(t, np.ndarray):
        if not t.flags["C_CONTIGUOUS"]:
            raise ValueError("host buffers must be contiguous")
        return t.ctypes.data
    if t.is_cuda:
        raise ValueError("last_prune_host takes host buffers")
    if not t.is_contiguous():
        raise ValueError("host buffers must be contiguous")
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return stream if isinstance(stream, int) else stream.cuda_stream


def _ws(ws):
    if isinstance(ws, tuple):
        return ws
    return _ptr(ws), ws.numel() * ws.element_size()


def last_workspace_size(problem: Problem) -> int:
    n = ctypes.c_size_t(0)
    _check(load_library().last_workspace_size(problem.ref, ctypes.byref(n)))
    return n.value


def workspace(problem: Problem, device="cuda"):
    """A torch uint8 tensor of last_workspace_size bytes (torch allocations are 512-B aligned)."""
    import torch
    return torch.empty(max(last_workspace_size(problem), 256), dtype=torch.uint8, device=device)


def last_scores(problem: Problem, q, k, w_out, ws, stream=None):
    p, n = _ws(ws)
    _check(load_library().last_scores(problem.ref, _ptr(q), _ptr(k), _ptr(w_out), p, n,
                                      _stream(stream)))


def last_scores_noalloc(problem: Problem, q, k, w_out, stream=None):
    """last_scores with the library's fixed scratch array instead of a workspace
    (for callers that cannot allocate device memory at run time)."""
    _check(load_library().last_scores_noalloc(problem.ref, _ptr(q), _ptr(k), _ptr(w_out),
                                              _stream(stream)))


def last_select(problem: Problem, w, x, idx_out, ws, stream=None, x_out=None):
    p, n = _ws(ws)
    _check(load_library().last_select(problem.ref, _ptr(w), _ptr(x), _ptr(idx_out), _ptr(x_out),
                                      p, n, _stream(stream)))


def last_select_topk(problem: Problem, w, idx_out, ws, stream=None, x=None, x_out=None):
    p, n = _ws(ws)
    _check(load_library().last_select_topk(problem.ref, _ptr(w), _ptr(x), _ptr(idx_out),
                                           _ptr(x_out), p, n, _stream(stream)))


class QueryRows:
    """Query rows of Table 4's attention sources: per-request offsets cu_rows
    [batch + 1] and request-local positions row_pos (host int32 arrays)."""

    def __init__(self, cu_rows: Sequence[int], row_pos: Sequence[int]):
        self.cu_rows = np.ascontiguousarray(np.asarray(cu_rows, dtype=np.int32))
        self.row_pos = np.ascontiguousarray(np.asarray(row_pos, dtype=np.int32))
        I = ctypes.POINTER(ctypes.c_int32)
        self.c_cu = self.cu_rows.ctypes.data_as(I)
        self.c_pos = self.row_pos.ctypes.data_as(I)


def last_scores_rows_workspace_size(problem: Problem, rows: QueryRows) -> int:
    n = ctypes.c_size_t(0)
    _check(load_library().last_scores_rows_workspace_size(problem.ref, rows.c_cu, rows.c_pos,
                                                          ctypes.byref(n)))
    return n.value


def rows_workspace(problem: Problem, rows: QueryRows, device="cuda"):
    import torch
    return torch.empty(max(last_scores_rows_workspace_size(problem, rows), 256), dtype=torch.uint8,
                       device=device)


def last_scores_rows(problem: Problem, rows: QueryRows, q_rows, k, w_out, ws, stream=None):
    p, n = _ws(ws)
    _check(load_library().last_scores_rows(problem.ref, rows.c_cu, rows.c_pos, _ptr(q_rows),
                                           _ptr(k), _ptr(w_out), p, n, _stream(stream)))


def last_gather(problem: Problem, x, idx, x_out, ws, stream=None):
    p, n = _ws(ws)
    _check(load_library().last_gather(problem.ref, _ptr(x), _ptr(idx), _ptr(x_out), p, n,
                                      _stream(stream)))


def last_prune(problem: Problem, q, k, x, w_out, idx_out, x_out, ws, stream=None):
    p, n = _ws(ws)
    _check(load_library().last_prune(problem.ref, _ptr(q), _ptr(k), _ptr(x), _ptr(w_out),
                                     _ptr(idx_out), _ptr(x_out), p, n, _stream(stream)))


def last_host_workspace_size(problem: Problem) -> int:
    n = ctypes.c_size_t(0)
    _check(load_library().last_host_workspace_size(problem.ref, ctypes.byref(n)))
    return n.value


def host_workspace(problem: Problem, device="cuda"):
    """A torch uint8 device tensor of last_host_workspace_size bytes."""
    import torch
    return torch.empty(max(last_host_workspace_size(problem), 256), dtype=torch.uint8,
                       device=device)


def last_prune_host(problem: Problem, q, k, x, w_out, idx_out, x_out, ws, stream=None):
    """last_prune on host buffers (pinned CPU tensors or numpy arrays); the copies
    are enqueued on `stream` with the path, so the outputs are ready once the
    stream has passed the call."""
    p, n = _ws(ws)
    _check(load_library().last_prune_host(problem.ref, _host_ptr(q), _host_ptr(k), _host_ptr(x),
                                          _host_ptr(w_out), _host_ptr(idx_out),
                                          _host_ptr(x_out), p, n, _stream(stream)))


def last_check_bounded_wait(ws, stream=None):
    p, _ = _ws(ws)
    _check(load_library().last_check_bounded_wait(p, _stream(stream)))


def last_poll(ws, stream=None):
    p, _ = _ws(ws)
    _check(load_library().last_poll(p, _stream(stream)))


def last_budget(n_vis: int, num: int, den: int) -> int:
    return int(load_library().last_budget(n_vis, num, den))


def last_status_string(st: int) -> str:
    return load_library().last_status_string(st).decode()
