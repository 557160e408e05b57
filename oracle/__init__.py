"""Python access to the plain C oracle of LAST's token-selection path.

TEST INFRASTRUCTURE ONLY: imported by the tests, by the smoke check and by
the CPU-baseline leg of the benchmark.  The CUDA library never imports or
calls it, and it imports nothing from the CUDA library.

Functions mirror the paper's equations (Sec. 3.2-3.4):
  last_row      Eq. 6   one causal-softmax attention row at p* = P_b - 1
  scores        Eq. 6-8 summed over layers/heads, normalised over the visual span
  select_fp32   Eq. 9-11 in canonical fp32 arithmetic (selection sequence)
  select_fp64   Eq. 9-11 in fp64 arithmetic (selection sequence)
  restore_order Eq. 12  sort(S)
  gather        Eq. 12  X_S
  budget        Eq. 2   ceil(rho N)
  prune         the whole path for a batch, request by request
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "last_oracle.c")
_DEFAULT_LIB = os.path.join(_HERE, "liblast_oracle.so")
# A test may point the wrapper at a deliberately mutated build of the same source
# (tests/test_oracle_mutations.py) to show that the pins catch planted mistakes.
_LIB = os.environ.get("LAST_ORACLE_LIB") or _DEFAULT_LIB

DTYPE_F32 = 0
DTYPE_BF16 = 1

# Canonical fp32 dot order: 32 lanes, 8 consecutive coordinates per lane group.
CANON_LANES = 32
CANON_VEC = 8


def compile_source(src: str, out: str) -> str:
    """gcc with no fast-math and no FMA contraction (every fma is an explicit fmaf)."""
    tmp = out + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c99", "-ffp-contract=off", "-fno-fast-math",
           "-fPIC", "-shared", src, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, out)
    return out


def build(force: bool = False) -> str:
    """Compile the oracle library next to its source (skipped when up to date)."""
    if _LIB != _DEFAULT_LIB:
        return _LIB
    if (not force and os.path.exists(_LIB)
            and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC)):
        return _LIB
    return compile_source(_SRC, _LIB)


_lib = None


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB)
        P = ctypes.c_void_p
        i32 = ctypes.c_int
        lib.oracle_last_row.argtypes = [i32, i32, i32, i32, i32, i32, ctypes.c_double,
                                        P, P, P, i32, i32, i32, P]
        lib.oracle_last_row.restype = i32
        lib.oracle_scores.argtypes = [i32, i32, i32, i32, i32, i32, ctypes.c_double,
                                      P, P, P, P, P, P]
        lib.oracle_scores.restype = i32
        lib.oracle_select_fp32.argtypes = [i32, i32, i32, P, P, i32, i32, i32, P]
        lib.oracle_select_fp32.restype = i32
        lib.oracle_select_fp64.argtypes = [i32, i32, i32, P, P, i32, P]
        lib.oracle_select_fp64.restype = i32
        lib.oracle_scores_rows.argtypes = [i32, i32, i32, i32, i32, i32, ctypes.c_double,
                                           P, P, P, P, P, P, P, P]
        lib.oracle_scores_rows.restype = i32
        lib.oracle_select_topk.argtypes = [i32, P, i32, P]
        lib.oracle_select_topk.restype = i32
        lib.oracle_restore_order.argtypes = [i32, P, P]
        lib.oracle_restore_order.restype = None
        lib.oracle_gather.argtypes = [i32, i32, i32, P, i32, P, P]
        lib.oracle_gather.restype = i32
        lib.oracle_budget.argtypes = [ctypes.c_int32, ctypes.c_int32, ctypes.c_int32]
        lib.oracle_budget.restype = ctypes.c_int32
        lib.oracle_dot_canonical.argtypes = [P, P, i32, i32, i32]
        lib.oracle_dot_canonical.restype = ctypes.c_float
        _lib = lib
    return _lib


def _ptr(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"], "oracle inputs must be C-contiguous"
    return a.ctypes.data_as(ctypes.c_void_p)


def _dtype_code(a: np.ndarray) -> int:
    if a.dtype == np.float32:
        return DTYPE_F32
    if a.dtype == np.uint16:  # bf16 bit patterns
        return DTYPE_BF16
    raise TypeError(f"oracle takes float32 or bf16-as-uint16 arrays, got {a.dtype}")


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.int32))


def last_row(q, k, cu_seqlens, b, l, h, *, num_kv_heads, scale=0.0):
    """Eq. 6: the attention row of p* = P_b - 1 for (b, l, h); q [B][L][Hq][D], k [L][sumP][Hkv][D]."""
    B, L, Hq, D = q.shape
    cu = _i32(cu_seqlens)
    P = int(cu[b + 1] - cu[b])
    out = np.zeros(P, dtype=np.float64)
    rc = _load().oracle_last_row(B, L, Hq, num_kv_heads, D, _dtype_code(q), float(scale),
                                 _ptr(cu), _ptr(q), _ptr(k), b, l, h, _ptr(out))
    if rc:
        raise ValueError(f"oracle_last_row rejected its arguments (rc={rc})")
    return out


def scores(q, k, cu_seqlens, vis_start, cu_vis, *, num_kv_heads, scale=0.0):
    """Eq. 6-8 in fp64; returns w [sum N] float64."""
    B, L, Hq, D = q.shape
    assert k.ndim == 4 and k.shape[0] == L and k.shape[2] == num_kv_heads and k.shape[3] == D
    assert q.dtype == k.dtype
    cu, vs, cv = _i32(cu_seqlens), _i32(vis_start), _i32(cu_vis)
    out = np.zeros(int(cv[-1]), dtype=np.float64)
    rc = _load().oracle_scores(B, L, Hq, num_kv_heads, D, _dtype_code(q), float(scale),
                               _ptr(cu), _ptr(vs), _ptr(cv), _ptr(q), _ptr(k), _ptr(out))
    if rc:
        raise ValueError(f"oracle_scores rejected its arguments (rc={rc})")
    return out


def scores_rows(q_rows, k, cu_seqlens, vis_start, cu_vis, cu_rows, row_pos, *, num_kv_heads,
                scale=0.0):
    """Table 4's attention sources in fp64: q_rows [sum M][L][Hq][D] holds the query
    rows of every request (cu_rows offsets, request-local positions row_pos); returns
    w [sum N] float64."""
    R, L, Hq, D = q_rows.shape
    assert k.ndim == 4 and k.shape[0] == L and k.shape[2] == num_kv_heads and k.shape[3] == D
    assert q_rows.dtype == k.dtype
    cu, vs, cv = _i32(cu_seqlens), _i32(vis_start), _i32(cu_vis)
    cr, rp = _i32(cu_rows), _i32(row_pos)
    B = len(cu) - 1
    assert int(cr[-1]) == R and len(rp) == R
    out = np.zeros(int(cv[-1]), dtype=np.float64)
    rc = _load().oracle_scores_rows(B, L, Hq, num_kv_heads, D, _dtype_code(q_rows), float(scale),
                                    _ptr(cu), _ptr(vs), _ptr(cv), _ptr(cr), _ptr(rp),
                                    _ptr(np.ascontiguousarray(q_rows)), _ptr(k), _ptr(out))
    if rc:
        raise ValueError(f"oracle_scores_rows rejected its arguments (rc={rc})")
    return out


def select_fp32(x, w, k, *, lanes=CANON_LANES, vec=CANON_VEC):
    """Eq. 9-11 in canonical fp32; x [N][d] (float32 or bf16 bits), w [N] float32.
    Returns the selection sequence j_1..j_k (int32)."""
    x = np.ascontiguousarray(x)
    w = np.ascontiguousarray(np.asarray(w, dtype=np.float32))
    N, d = x.shape
    out = np.zeros(max(k, 1), dtype=np.int32)
    rc = _load().oracle_select_fp32(N, d, _dtype_code(x), _ptr(x), _ptr(w), int(k),
                                    lanes, vec, _ptr(out))
    if rc:
        raise ValueError(f"oracle_select_fp32 rejected its arguments (rc={rc})")
    return out[:k]


def select_fp64(x, w, k):
    """Eq. 9-11 in fp64; returns the selection sequence (int32)."""
    x = np.ascontiguousarray(x)
    w = np.ascontiguousarray(np.asarray(w, dtype=np.float64))
    N, d = x.shape
    out = np.zeros(max(k, 1), dtype=np.int32)
    rc = _load().oracle_select_fp64(N, d, _dtype_code(x), _ptr(x), _ptr(w), int(k), _ptr(out))
    if rc:
        raise ValueError(f"oracle_select_fp64 rejected its arguments (rc={rc})")
    return out[:k]


def select_topk(w, k):
    """Table 5's Top-k selection: the k highest scores, ties to the lowest index.
    Returns the selection order (descending score, int32)."""
    w = np.ascontiguousarray(np.asarray(w, dtype=np.float32))
    out = np.zeros(max(k, 1), dtype=np.int32)
    rc = _load().oracle_select_topk(len(w), _ptr(w), int(k), _ptr(out))
    if rc:
        raise ValueError(f"oracle_select_topk rejected its arguments (rc={rc})")
    return out[:k]


def restore_order(order):
    """Eq. 12: sort(S)."""
    order = _i32(order)
    out = np.zeros(max(len(order), 1), dtype=np.int32)
    _load().oracle_restore_order(len(order), _ptr(order), _ptr(out))
    return out[:len(order)]


def gather(x, idx):
    """Eq. 12: X_S rows, bitwise."""
    x = np.ascontiguousarray(x)
    idx = _i32(idx)
    N, d = x.shape
    out = np.zeros((len(idx), d), dtype=x.dtype)
    if len(idx):
        rc = _load().oracle_gather(N, d, x.itemsize, _ptr(x), len(idx), _ptr(idx), _ptr(out))
        if rc:
            raise ValueError("oracle_gather: index out of range")
    return out


def dot_canonical(a, b, *, lanes=CANON_LANES, vec=CANON_VEC):
    a = np.ascontiguousarray(a, dtype=np.float32)
    b = np.ascontiguousarray(b, dtype=np.float32)
    return float(_load().oracle_dot_canonical(_ptr(a), _ptr(b), len(a), lanes, vec))


def budget(n, num, den):
    """Eq. 2: ceil(num * n / den)."""
    return int(_load().oracle_budget(int(n), int(num), int(den)))


def prune_request(x, w32, k):
    """Selection + order restore + gather for one request, canonical fp32.
    Returns (order, idx_sorted, x_sel)."""
    order = select_fp32(x, w32, k)
    idx = restore_order(order)
    return order, idx, gather(x, idx)


def prune(wl, *, requests=None):
    """The whole path on a workload (see workloads.synth.Workload):
    fp64 scores, rounded to fp32, then canonical-fp32 selection and gather per
    request.  Returns dict(w64, w32, idx [sum k], x_sel, orders)."""
    w64 = scores(wl.q, wl.k, wl.cu_seqlens, wl.vis_start, wl.cu_vis,
                 num_kv_heads=wl.num_kv_heads, scale=wl.scale)
    w32 = w64.astype(np.float32)
    reqs = range(wl.batch) if requests is None else requests
    orders, idx_all, xs_all = {}, [], []
    for b in reqs:
        v0, v1 = int(wl.cu_vis[b]), int(wl.cu_vis[b + 1])
        kb = int(wl.cu_keep[b + 1] - wl.cu_keep[b])
        order, idx, xs = prune_request(wl.x[v0:v1], w32[v0:v1], kb)
        orders[b] = order
        idx_all.append(idx)
        xs_all.append(xs)
    return dict(w64=w64, w32=w32, orders=orders,
                idx=np.concatenate(idx_all) if idx_all else np.zeros(0, np.int32),
                x_sel=np.concatenate(xs_all) if xs_all else np.zeros((0, wl.feat_dim), wl.x.dtype))
