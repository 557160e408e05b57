"""Synthetic LAST workloads (input generation only).

Each request b is an image's visual tokens placed inside a text prompt of a
guidance model.  The generator produces, per request,

  q  [B][L][Hq][D]        the query vector of the last prompt position, per layer/head
  k  [L][sum P][Hkv][D]   packed variable-length keys of every position
  x  [sum N][d_v]         the encoder features of the visual tokens

plus the ragged offsets (cu_seqlens, vis_start, cu_vis) and the per-request
budgets (cu_keep).  bf16 tensors are returned as uint16 bit patterns (round to
nearest even from fp32); fp32 tensors as float32.

Random numbers come from numpy's Philox counter-based generator, with one
independent stream per (config seed, request, tensor), so any subset of
requests can be regenerated on its own.

Value models (stand-ins for the paper's image/query workloads):
  * q and K entries ~ N(0, 1)/sqrt(D).
  * "planted" relevant visual tokens: their key for kv-head g is moved by
    3 * (1/sqrt(D)) along the unit direction of the mean q of g's query
    heads, which raises their logits by three standard deviations of the
    logit distribution at that q.
  * features: a mixture of unit-norm Gaussian centres; a token is its centre
    plus isotropic noise of total norm about `noise` (per coordinate
    noise/sqrt(d_v)).
  * near-duplicates (high-resolution tiles): a copy of an earlier token plus
    noise of norm 0.1 of its norm (cosine > 0.99).
  * video: frame 0 ~ N(0, 1) per coordinate, frame f = frame f-1 + N(0, 0.05^2).
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import Optional, Sequence

import numpy as np

CONFIG_NAMES = ("c1", "c2", "c3", "c4", "c5")

_STREAM_Q, _STREAM_K, _STREAM_X, _STREAM_META, _STREAM_PLANT = 1, 2, 3, 4, 5


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (nearest, ties to even); returns uint16 bits."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32)
    rounding = np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    out = ((u + rounding) >> np.uint32(16)).astype(np.uint16)
    nan = np.isnan(a)
    if nan.any():
        out[nan] = np.uint16(0x7FC0)
    return out


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _rng(seed: int, *stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.Philox(np.random.SeedSequence([seed, *stream])))


@dataclass
class Workload:
    name: str
    batch: int
    num_layers: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    feat_dim: int
    dtype: str                      # "f32" or "bf16"
    cu_seqlens: np.ndarray          # [B+1] int32
    vis_start: np.ndarray           # [B]   int32
    cu_vis: np.ndarray              # [B+1] int32
    cu_keep: np.ndarray             # [B+1] int32
    q: np.ndarray                   # [B][L][Hq][D]
    k: np.ndarray                   # [L][sum P][Hkv][D]
    x: np.ndarray                   # [sum N][d_v]
    scale: float = 0.0              # <= 0 -> 1/sqrt(D)
    planted: dict = field(default_factory=dict)
    note: str = ""

    @property
    def n_vis(self) -> np.ndarray:
        return np.diff(self.cu_vis)

    @property
    def n_keep(self) -> np.ndarray:
        return np.diff(self.cu_keep)

    @property
    def seqlens(self) -> np.ndarray:
        return np.diff(self.cu_seqlens)

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2

    def nbytes(self) -> dict:
        return dict(q=self.q.nbytes, k=self.k.nbytes, x=self.x.nbytes)

    def describe(self) -> dict:
        return dict(workload=self.name, batch=self.batch, layers=self.num_layers,
                    q_heads=self.num_q_heads, kv_heads=self.num_kv_heads,
                    head_dim=self.head_dim, feat_dim=self.feat_dim, dtype=self.dtype,
                    visual_tokens=int(self.cu_vis[-1]), keys=int(self.cu_seqlens[-1]),
                    kept=int(self.cu_keep[-1]), note=self.note)


def _cast(a: np.ndarray, dtype: str) -> np.ndarray:
    return f32_to_bf16_bits(a) if dtype == "bf16" else np.ascontiguousarray(a, dtype=np.float32)


def _features_clusters(rng, n, d, n_clusters, noise, dup_frac=0.0):
    centres = rng.standard_normal((n_clusters, d), dtype=np.float32)
    centres /= np.linalg.norm(centres, axis=1, keepdims=True)
    assign = rng.integers(0, n_clusters, size=n)
    x = centres[assign]
    x += rng.standard_normal((n, d), dtype=np.float32) * np.float32(noise / math.sqrt(d))
    if dup_frac > 0.0 and n > 1:
        n_dup = int(round(dup_frac * n))
        dup = np.sort(rng.choice(np.arange(1, n), size=min(n_dup, n - 1), replace=False))
        is_dup = np.zeros(n, dtype=bool)
        is_dup[dup] = True
        for i in dup:
            # copy an earlier original token, perturbed by 10% of its norm
            cand = np.flatnonzero(~is_dup[:i])
            src = int(cand[rng.integers(0, len(cand))])
            e = rng.standard_normal(d, dtype=np.float32)
            e *= np.float32(0.1) * np.linalg.norm(x[src]) / np.linalg.norm(e)
            x[i] = x[src] + e
    return x


def _features_video(rng, n, d, frame_tokens, step_sigma):
    n_frames = -(-n // frame_tokens)
    x = np.empty((n_frames * frame_tokens, d), dtype=np.float32)
    x[:frame_tokens] = rng.standard_normal((frame_tokens, d), dtype=np.float32)
    for f in range(1, n_frames):
        x[f * frame_tokens:(f + 1) * frame_tokens] = (
            x[(f - 1) * frame_tokens:f * frame_tokens]
            + rng.standard_normal((frame_tokens, d), dtype=np.float32) * np.float32(step_sigma))
    return x[:n]


def custom(*, name="custom", seed=0, batch=1, n_vis=(16,), n_text=(4,), n_before=(0,),
           num_layers=1, num_q_heads=2, num_kv_heads=2, head_dim=64, feat_dim=256,
           dtype="bf16", keep: Optional[Sequence[int]] = None, keep_frac=None,
           n_clusters=8, noise=0.1, dup_frac=0.0, n_planted=0, video_frame=0,
           video_sigma=0.05, scale=0.0, note="") -> Workload:
    """General builder.  Per-request sequences are [n_before text][n_vis visual][n_text text];
    the last text token is the query position p*.  n_text >= 1."""
    def per_req(v):
        v = list(v) if isinstance(v, (list, tuple, np.ndarray)) else [v]
        return [int(v[b % len(v)]) for b in range(batch)]
    N, T, V0 = per_req(n_vis), per_req(n_text), per_req(n_before)
    assert all(t >= 1 for t in T), "the query token is the last text token: n_text >= 1"
    if keep is None:
        num, den = keep_frac if keep_frac is not None else (1, 8)
        keep = [(num * n + den - 1) // den for n in N]
    Kp = per_req(keep)
    assert all(0 <= kb <= nb for kb, nb in zip(Kp, N))
    P = [v0 + n + t for v0, n, t in zip(V0, N, T)]
    cu_seqlens = np.zeros(batch + 1, np.int32)
    cu_seqlens[1:] = np.cumsum(P)
    cu_vis = np.zeros(batch + 1, np.int32)
    cu_vis[1:] = np.cumsum(N)
    cu_keep = np.zeros(batch + 1, np.int32)
    cu_keep[1:] = np.cumsum(Kp)
    vis_start = np.asarray(V0, np.int32)

    L, Hq, Hkv, D, dv = num_layers, num_q_heads, num_kv_heads, head_dim, feat_dim
    assert Hq % Hkv == 0
    G = Hq // Hkv
    inv = np.float32(1.0 / math.sqrt(D))
    q = np.empty((batch, L, Hq, D), np.float32)
    k = np.empty((L, int(cu_seqlens[-1]), Hkv, D), np.float32)
    x = np.empty((int(cu_vis[-1]), dv), np.float32)
    planted = {}
    for b in range(batch):
        q[b] = _rng(seed, b, _STREAM_Q).standard_normal((L, Hq, D), dtype=np.float32) * inv
        s0, s1 = int(cu_seqlens[b]), int(cu_seqlens[b + 1])
        k[:, s0:s1] = _rng(seed, b, _STREAM_K).standard_normal((L, s1 - s0, Hkv, D),
                                                                 dtype=np.float32) * inv
        if n_planted and N[b]:
            pr = _rng(seed, b, _STREAM_PLANT)
            idx = np.sort(pr.choice(N[b], size=min(n_planted, N[b]), replace=False))
            planted[b] = idx
            for l in range(L):
                for g in range(Hkv):
                    qg = q[b, l, g * G:(g + 1) * G].mean(axis=0)
                    qg = qg / np.float32(np.linalg.norm(qg))
                    k[l, s0 + V0[b] + idx, g] += np.float32(3.0) * inv * qg
        xr = _rng(seed, b, _STREAM_X)
        v0, v1 = int(cu_vis[b]), int(cu_vis[b + 1])
        if N[b]:
            if video_frame:
                x[v0:v1] = _features_video(xr, N[b], dv, video_frame, video_sigma)
            else:
                x[v0:v1] = _features_clusters(xr, N[b], dv, n_clusters, noise, dup_frac)
    return Workload(name=name, batch=batch, num_layers=L, num_q_heads=Hq, num_kv_heads=Hkv,
                    head_dim=D, feat_dim=dv, dtype=dtype, cu_seqlens=cu_seqlens,
                    vis_start=vis_start, cu_vis=cu_vis, cu_keep=cu_keep,
                    q=_cast(q, dtype), k=_cast(k, dtype), x=_cast(x, dtype), scale=scale,
                    planted=planted, note=note)


def _uniform_ints(seed, stream, lo, hi, n):
    return _rng(seed, 10_000 + stream, _STREAM_META).integers(lo, hi + 1, size=n).tolist()


def config(name: str, *, budget=None, batch=None, n_vis=None, seed=None) -> Workload:
    """The five workload presets (full size by default).

    c1  1 request, 576 visual + 32 text, L=1, 16x64 heads, fp32, d_v=1024, 24 clusters,
        20 planted, k=72.
    c2  64 requests, 576 visual + U[16,128] text, L=1, 16/16 heads x 128, bf16, d_v=2048,
        64 clusters, 10 planted; budget 64, 128, 192 or "mixed" (request b keeps
        64*(1 + b mod 3)).
    c3  32 requests, 2880 visual (5 tiles x 576, one pool) + 64 text, L=4, 16/4 x 128,
        bf16, d_v=2048, 128 clusters, 30% near-duplicates, k=360.
    c4  128 requests, U[256,4096] visual + U[8,256] text, L=1, 12/2 x 128, bf16,
        d_v=1536, 64 clusters, 10 planted, k=ceil(N/8).
    c5  8 requests, 16384 visual (32 frames x 512) + 128 text, L=1, 16/4 x 128, bf16,
        d_v=2048, inter-frame random walk, 10 planted; budget 5, 12.5 or 25 (% of N).

    `batch`/`n_vis` shrink a preset (same per-request distributions) for oracle-sized runs.
    """
    if name == "c1":
        return custom(name="c1", seed=0 if seed is None else seed, batch=batch or 1,
                      n_vis=n_vis or 576, n_text=32, num_layers=1, num_q_heads=16,
                      num_kv_heads=16, head_dim=64, feat_dim=1024, dtype="f32",
                      keep=[budget or 72], n_clusters=24, noise=0.1, n_planted=20,
                      note="fp32, 1 request")
    if name == "c2":
        s = 1 if seed is None else seed
        B = batch or 64
        budget = 128 if budget is None else budget
        keep = [64 * (1 + b % 3) for b in range(B)] if budget == "mixed" else [int(budget)]
        return custom(name=f"c2(k={budget})", seed=s, batch=B, n_vis=n_vis or 576,
                      n_text=_uniform_ints(s, 0, 16, 128, B), num_layers=1, num_q_heads=16,
                      num_kv_heads=16, head_dim=128, feat_dim=2048, dtype="bf16", keep=keep,
                      n_clusters=64, noise=0.1, n_planted=10, note="LLaVA-1.5 shape")
    if name == "c3":
        s = 2 if seed is None else seed
        nv = n_vis or 2880
        return custom(name="c3", seed=s, batch=batch or 32, n_vis=nv, n_text=64, num_layers=4,
                      num_q_heads=16, num_kv_heads=4, head_dim=128, feat_dim=2048,
                      dtype="bf16", keep=[budget or (nv + 7) // 8], n_clusters=128,
                      noise=0.1, dup_frac=0.3, n_planted=10,
                      note="5 tiles x 576 in one pool, 4 layers summed")
    if name == "c4":
        s = 3 if seed is None else seed
        B = batch or 128
        nv = n_vis or _uniform_ints(s, 0, 256, 4096, B)
        return custom(name="c4", seed=s, batch=B, n_vis=nv,
                      n_text=_uniform_ints(s, 1, 8, 256, B), num_layers=1, num_q_heads=12,
                      num_kv_heads=2, head_dim=128, feat_dim=1536, dtype="bf16",
                      keep_frac=(1, 8), n_clusters=64, noise=0.1, n_planted=10,
                      note="ragged dynamic resolution, k=ceil(N/8)")
    if name == "c5":
        s = 4 if seed is None else seed
        pct = {5: (1, 20), 12.5: (1, 8), 25: (1, 4)}[budget if budget is not None else 12.5]
        return custom(name=f"c5(k/N={budget if budget is not None else 12.5}%)", seed=s,
                      batch=batch or 8, n_vis=n_vis or 16384, n_text=128, num_layers=1,
                      num_q_heads=16, num_kv_heads=4, head_dim=128, feat_dim=2048,
                      dtype="bf16", keep_frac=pct, n_planted=10, video_frame=512,
                      video_sigma=0.05, note="32 frames x 512, random-walk frames")
    raise ValueError(f"unknown workload {name!r}")


def query_rows(wl: Workload, source: str, m_rows: int = 32, seed: int = 7):
    """Query rows for Table 4's attention sources: positions after each request's
    visual span (its text rows) -- the first ("first"), the middle ("middle"), the
    last ("last", p* = P_b - 1) or up to m_rows spread evenly over them ("all") --
    and one query vector per row, layer and q-head drawn like the workload's q (a
    row at p* takes the request's own p* query).  Returns (cu_rows, row_pos, q_rows)
    with q_rows [sum M][L][Hq][D] in the workload's dtype."""
    cu, pos = [0], []
    for b in range(wl.batch):
        P = int(wl.cu_seqlens[b + 1] - wl.cu_seqlens[b])
        first = int(wl.vis_start[b] + (wl.cu_vis[b + 1] - wl.cu_vis[b]))
        text = np.arange(first, P)
        if source == "first":
            sel = text[:1]
        elif source == "middle":
            sel = text[(len(text) - 1) // 2:][:1]
        elif source == "last":
            sel = text[-1:]
        elif source == "all":
            sel = np.unique(text[np.linspace(0, len(text) - 1, min(m_rows, len(text)))
                                 .round().astype(int)])
        else:
            raise ValueError(f"unknown attention source {source!r}")
        pos += sel.tolist()
        cu.append(len(pos))
    rng = _rng(seed, 99)
    q = rng.standard_normal((len(pos), wl.num_layers, wl.num_q_heads, wl.head_dim)).astype(np.float32)
    q = _cast(q * np.float32(1.0 / math.sqrt(wl.head_dim)), wl.dtype)   # q ~ N(0, 1)/sqrt(D)
    for b in range(wl.batch):
        for r in range(cu[b], cu[b + 1]):
            if pos[r] == int(wl.cu_seqlens[b + 1] - wl.cu_seqlens[b]) - 1:
                q[r] = wl.q[b]
    return np.array(cu, np.int32), np.array(pos, np.int32), np.ascontiguousarray(q)
