"""GPU parity of the whole-GPU selection (requests too long for any cluster).

A request longer than the clustered selection's shared memory holds (16 CTAs of
a thread-block cluster: about 126K tokens at d_v = 128 bf16, 120K at d_v = 64
fp32, 72K at d_v = 2048) runs, with up to three others, on every SM: one
cooperative launch, a grid barrier per round through global memory (Eq. 9-11 in
exact batched rounds).  The kept indices must stay bit-identical to the
canonical-fp32 oracle on identical scores, and the gathered rows (Eq. 12)
bitwise equal:

  * one request of 250 000 tokens (d_v = 128);
  * three requests of 130 000 / 200 000 / 140 000 tokens (d_v = 128);
  * fp32 features, 125 000 tokens (d_v = 64);
  * 80 000 tokens of 2048 features;
  * the edges k = N and k = 1 on this path, end to end through last_prune.

The oracle runs one request per host thread (reentrant; threads, not forked
processes).
"""
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest

import oracle
from workloads import custom

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


def _check(wl, w32, idx, requests=None):
    assert_valid_selection(wl, idx)

    def run(b):
        v0, v1 = int(wl.cu_vis[b]), int(wl.cu_vis[b + 1])
        k = int(wl.cu_keep[b + 1] - wl.cu_keep[b])
        return b, oracle.restore_order(oracle.select_fp32(wl.x[v0:v1], w32[v0:v1], k))

    with ThreadPoolExecutor(max_workers=_threads()) as pool:
        for b, want in pool.map(run, range(wl.batch) if requests is None else requests):
            got = idx[wl.cu_keep[b]:wl.cu_keep[b + 1]]
            assert np.array_equal(got, want), (
                f"request {b}: {np.setdiff1d(got, want).tolist()[:8]} kept by GPU only, "
                f"{np.setdiff1d(want, got).tolist()[:8]} by oracle only")


def _weights(wl, seed):
    rng = np.random.default_rng(seed)
    n = np.diff(wl.cu_vis)
    return np.concatenate([rng.dirichlet(np.ones(int(m))) for m in n]).astype(np.float32)


def _long(name, seed, n_vis, keep, dv, dtype="bf16", **kw):
    return custom(name=name, seed=seed, batch=len(n_vis), n_vis=n_vis, n_text=[2], num_layers=1,
                  num_q_heads=2, num_kv_heads=2, head_dim=64, feat_dim=dv, dtype=dtype, keep=keep,
                  **({"n_clusters": 500, "noise": 0.1} | kw))


def test_grid_single_request():
    wl = _long("grid-one", 84, [250000], [64], 128)
    w32 = _weights(wl, 8401)
    _check(wl, w32, DeviceWorkload(wl).select(w32))


def test_grid_three_requests():
    wl = _long("grid-three", 82, [130000, 200000, 140000], [40, 60, 30], 128)
    w32 = _weights(wl, 8201)
    _check(wl, w32, DeviceWorkload(wl).select(w32))


def test_grid_fp32():
    wl = _long("grid-f32", 83, [125000], [50], 64, dtype="f32", n_clusters=200)
    w32 = _weights(wl, 8301)
    _check(wl, w32, DeviceWorkload(wl).select(w32))


def test_grid_wide_rows():
    wl = _long("grid-wide", 85, [80000], [30], 2048, video_frame=500, video_sigma=0.05)
    w32 = _weights(wl, 8501)
    _check(wl, w32, DeviceWorkload(wl).select(w32))


def test_grid_edges_end_to_end():
    # k = N keeps every token (no greedy to replay); k = 1 is the seed alone (Eq. 9)
    wl = custom(name="grid-edges", seed=86, batch=2, n_vis=[130000, 128000], n_text=[6, 3],
                num_layers=1, num_q_heads=4, num_kv_heads=2, head_dim=64, feat_dim=128,
                dtype="bf16", keep=[130000, 1], n_clusters=30, noise=0.1, n_planted=4)
    w_gpu, idx, xs = DeviceWorkload(wl).prune()
    assert_valid_selection(wl, idx)
    assert np.array_equal(idx[:130000], np.arange(130000))
    _check(wl, w_gpu, idx, requests=[1])
    assert_gather_equal(wl, idx, xs, range(wl.batch))
