"""Helpers for the GPU parity tests: device copies of a workload, calls through
the C ABI, and the comparison rules against the oracle."""
from __future__ import annotations

import numpy as np

import oracle
import paper_2607_27952_gb300 as last

SCORE_RTOL = 1e-3      # scores: relative tolerance (fp32 accumulation from bf16/fp32 inputs)
SCORE_ATOL = 1e-30     # only matters for values below the fp32 normal range
POISON_IDX = -7


def to_dev(a: np.ndarray, dev):
    import torch
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).to(dev).view(torch.bfloat16)
    return torch.from_numpy(a).to(dev)


def to_host_bits(t) -> np.ndarray:
    import torch
    if t.dtype == torch.bfloat16:
        return t.view(torch.int16).cpu().numpy().view(np.uint16)
    return t.cpu().numpy()


def problem_of(wl, cu_keep=None) -> last.Problem:
    return last.Problem(batch=wl.batch, num_layers=wl.num_layers, num_q_heads=wl.num_q_heads,
                        num_kv_heads=wl.num_kv_heads, head_dim=wl.head_dim,
                        feat_dim=wl.feat_dim, dtype=wl.dtype, cu_seqlens=wl.cu_seqlens,
                        vis_start=wl.vis_start, cu_vis=wl.cu_vis,
                        cu_keep=wl.cu_keep if cu_keep is None else cu_keep,
                        softmax_scale=wl.scale)


class DeviceWorkload:
    def __init__(self, wl, dev="cuda:0"):
        import torch
        self.wl, self.dev = wl, torch.device(dev)
        self.q, self.k, self.x = to_dev(wl.q, self.dev), to_dev(wl.k, self.dev), to_dev(wl.x, self.dev)

    def outputs(self, cu_keep=None):
        import torch
        nkeep = int((self.wl.cu_keep if cu_keep is None else cu_keep)[-1])
        w = torch.full((int(self.wl.cu_vis[-1]),), float("nan"), dtype=torch.float32, device=self.dev)
        idx = torch.full((nkeep,), POISON_IDX, dtype=torch.int32, device=self.dev)
        xs = torch.empty((nkeep, self.wl.feat_dim), dtype=self.x.dtype, device=self.dev)
        xs.view(torch.uint8).fill_(0xFF)
        return w, idx, xs

    def prune(self, cu_keep=None, gather=True):
        prob = problem_of(self.wl, cu_keep)
        w, idx, xs = self.outputs(cu_keep)
        ws = last.workspace(prob, self.dev)
        last.last_prune(prob, self.q, self.k, self.x, w, idx, xs if gather else None, ws)
        last.last_poll(ws)
        return w.cpu().numpy(), idx.cpu().numpy(), to_host_bits(xs)

    def scores(self):
        prob = problem_of(self.wl)
        w, _, _ = self.outputs()
        ws = last.workspace(prob, self.dev)
        last.last_scores(prob, self.q, self.k, w, ws)
        last.last_poll(ws)
        return w.cpu().numpy()

    def select(self, w32: np.ndarray, cu_keep=None):
        import torch
        prob = problem_of(self.wl, cu_keep)
        _, idx, _ = self.outputs(cu_keep)
        ws = last.workspace(prob, self.dev)
        wt = torch.from_numpy(np.ascontiguousarray(w32, dtype=np.float32)).to(self.dev)
        last.last_select(prob, wt, self.x, idx, ws)
        last.last_poll(ws)
        return idx.cpu().numpy()


def assert_scores_close(w_gpu, w_ref, wl):
    assert np.isfinite(w_gpu).all(), "unwritten or non-finite scores"
    err = np.abs(w_gpu.astype(np.float64) - w_ref)
    bad = err > SCORE_RTOL * np.abs(w_ref) + SCORE_ATOL
    assert not bad.any(), (f"{bad.sum()} scores outside rtol {SCORE_RTOL}; worst rel "
                           f"{(err / np.abs(w_ref)).max():.3e}")
    for b in range(wl.batch):
        seg = w_gpu[wl.cu_vis[b]:wl.cu_vis[b + 1]]
        if len(seg):
            assert abs(seg.astype(np.float64).sum() - 1.0) < 1e-4


def oracle_selection(wl, w32, b, k=None):
    v0, v1 = int(wl.cu_vis[b]), int(wl.cu_vis[b + 1])
    kb = int(wl.cu_keep[b + 1] - wl.cu_keep[b]) if k is None else k
    return oracle.select_fp32(wl.x[v0:v1], w32[v0:v1], kb)


def assert_selection_equal(wl, w32, idx_gpu, requests, cu_keep=None):
    """Bit-exact rule: on identical scores the kept indices equal the oracle's."""
    cu_keep = wl.cu_keep if cu_keep is None else cu_keep
    for b in requests:
        k0, k1 = int(cu_keep[b]), int(cu_keep[b + 1])
        order = oracle_selection(wl, w32, b, k1 - k0)
        want = oracle.restore_order(order)
        got = idx_gpu[k0:k1]
        assert np.array_equal(got, want), (
            f"request {b}: {np.setdiff1d(got, want).tolist()[:8]} kept by GPU only, "
            f"{np.setdiff1d(want, got).tolist()[:8]} by oracle only")


def assert_gather_equal(wl, idx_gpu, xs_gpu, requests, cu_keep=None):
    cu_keep = wl.cu_keep if cu_keep is None else cu_keep
    for b in requests:
        k0, k1 = int(cu_keep[b]), int(cu_keep[b + 1])
        rows = oracle.gather(wl.x[wl.cu_vis[b]:wl.cu_vis[b + 1]], idx_gpu[k0:k1])
        assert np.array_equal(xs_gpu[k0:k1], rows), f"request {b}: gathered rows differ"


def assert_valid_selection(wl, idx_gpu, cu_keep=None):
    cu_keep = wl.cu_keep if cu_keep is None else cu_keep
    for b in range(wl.batch):
        k0, k1 = int(cu_keep[b]), int(cu_keep[b + 1])
        n = int(wl.cu_vis[b + 1] - wl.cu_vis[b])
        got = idx_gpu[k0:k1]
        assert len(got) == k1 - k0
        if len(got):
            assert got.min() >= 0 and got.max() < n, f"request {b}: index out of range"
            assert (np.diff(got) > 0).all(), f"request {b}: not strictly ascending"


# Two scores each within SCORE_RTOL of the oracle's can swap an argmax only when the
# two products w~ * delta differ by at most about 2 * SCORE_RTOL; the fp64 replay adds
# the fp32 rounding of delta on top, hence the margin below.
PRODUCT_TIE_RTOL = 2.5e-3


def near_tie_divergence(x, w_ref, seq_ref, seq_alt):
    """End-to-end rule.  Greedy sequences on the oracle's scores (seq_ref) and on the
    GPU's scores (seq_alt) may part only where the two candidates' products (under the
    oracle's scores, fp64 cosine distances of the bf16/fp32 features) are within
    PRODUCT_TIE_RTOL of each other.  Returns None when the sequences agree, else
    (step, relative gap)."""
    for t, (a, c) in enumerate(zip(seq_ref, seq_alt)):
        if a != c:
            break
    else:
        return None
    if t == 0:
        pa, pc = w_ref[a], w_ref[c]
    else:
        from workloads import bf16_bits_to_f32
        xf = (bf16_bits_to_f32(x) if x.dtype == np.uint16 else x).astype(np.float64)
        xb = xf / np.maximum(np.linalg.norm(xf, axis=1, keepdims=True), 1e-300)
        S = list(seq_ref[:t])
        da = (1.0 - xb[a] @ xb[S].T).min()
        dc = (1.0 - xb[c] @ xb[S].T).min()
        pa, pc = w_ref[a] * da, w_ref[c] * dc
    return t, abs(pa - pc) / max(abs(pa), abs(pc), 1e-300)
