"""Long greedy runs checked in full against the oracle (Eq. 9-11, every step).

The batched rounds, the tensor-core certificate and the triangle-inequality row
skipping all act at every step of a long greedy run, so the full-budget kept sets
of the longest configurations are compared bit for bit with the canonical-fp32
oracle on the GPU's own scores (the selection-on-identical-scores rule):

  * video batch (8 x 16384 tokens, k/N = 5%: k = 820) on all 8 requests, and
    k = 2048 (12.5%) on two of them;
  * 5-tile high-resolution batch (2880 tokens, k = 360) on 8 requests;
  * ragged dynamic-resolution batch (k = ceil(N/8)) on 16 requests, the 4
    longest among them.

The greedy sequence does not depend on k, so one oracle run at k = 2048 also gives
the k = 820 sequence of the same request (its prefix).  The oracle runs one
request per host thread (it is reentrant and its C calls release the GIL); the
pool is made of threads, not forked processes.
"""
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest

import oracle
from workloads import config

from gpu_util import DeviceWorkload, assert_gather_equal, assert_valid_selection

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module", autouse=True)
def _built():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2607_27952_gb300.build import build
    import paper_2607_27952_gb300 as last
    build()
    last.load_library()
    oracle.build()


def _threads():
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:
        return max(1, os.cpu_count() or 1)


def _oracle_sequences(wl, w32, tasks):
    """tasks: [(request, k)] -> {request: selection sequence of length k}."""
    def run(task):
        b, k = task
        v0, v1 = int(wl.cu_vis[b]), int(wl.cu_vis[b + 1])
        return b, oracle.select_fp32(wl.x[v0:v1], w32[v0:v1], k)
    # longest first, so that the pool ends as early as it can
    order = sorted(tasks, key=lambda t: -t[1] * int(wl.cu_vis[t[0] + 1] - wl.cu_vis[t[0]]))
    with ThreadPoolExecutor(max_workers=_threads()) as pool:
        return dict(pool.map(run, order))


def _check(idx_gpu, cu_keep, b, seq):
    k0, k1 = int(cu_keep[b]), int(cu_keep[b + 1])
    want = oracle.restore_order(np.asarray(seq[:k1 - k0], dtype=np.int32))
    got = idx_gpu[k0:k1]
    assert np.array_equal(got, want), (
        f"request {b} (k={k1 - k0}): {np.setdiff1d(got, want).tolist()[:8]} kept by GPU only, "
        f"{np.setdiff1d(want, got).tolist()[:8]} by oracle only")


def test_video_full_budget_every_request():
    wl = config("c5", budget=5)                       # k = 820 for N = 16384
    dw = DeviceWorkload(wl)
    w_gpu, idx, xs = dw.prune()
    assert_valid_selection(wl, idx)
    assert_gather_equal(wl, idx, xs, range(wl.batch))
    long_reqs = (0, 5)
    big = np.arange(wl.batch + 1, dtype=np.int32) * 2048  # k = 2048 (12.5%) for every request
    idx_big = dw.select(w_gpu, cu_keep=big)
    assert_valid_selection(wl, idx_big, cu_keep=big)
    tasks = [(b, 2048 if b in long_reqs else 820) for b in range(wl.batch)]
    seqs = _oracle_sequences(wl, w_gpu, tasks)
    for b in range(wl.batch):
        _check(idx, wl.cu_keep, b, seqs[b])            # k = 820: a prefix for 0 and 5
    for b in long_reqs:
        _check(idx_big, big, b, seqs[b])


def test_high_resolution_eight_requests():
    wl = config("c3")
    dw = DeviceWorkload(wl)
    w_gpu, idx, xs = dw.prune()
    assert_valid_selection(wl, idx)
    reqs = list(range(8))
    seqs = _oracle_sequences(wl, w_gpu, [(b, int(wl.cu_keep[b + 1] - wl.cu_keep[b])) for b in reqs])
    for b in reqs:
        _check(idx, wl.cu_keep, b, seqs[b])
    assert_gather_equal(wl, idx, xs, reqs)


def test_dynamic_resolution_sixteen_requests():
    wl = config("c4")
    dw = DeviceWorkload(wl)
    w_gpu, idx, xs = dw.prune()
    assert_valid_selection(wl, idx)
    n = np.diff(wl.cu_vis)
    longest = [int(b) for b in np.argsort(-n, kind="stable")[:4]]
    rest = [b for b in range(0, wl.batch, 7) if b not in longest][:12]
    reqs = longest + rest
    assert len(reqs) == 16
    seqs = _oracle_sequences(wl, w_gpu, [(b, int(wl.cu_keep[b + 1] - wl.cu_keep[b])) for b in reqs])
    for b in reqs:
        _check(idx, wl.cu_keep, b, seqs[b])
    assert_gather_equal(wl, idx, xs, reqs)
