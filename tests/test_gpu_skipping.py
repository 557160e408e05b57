"""GPU parity of the selection's row skipping on inputs chosen against its bounds.

The bf16 greedy skips a (token, new centre) pair when the triangle inequality on
the unit sphere proves that the centre cannot lower the token's delta (Eq. 10):
the bound goes through the token's nearest centre and that centre's root, with
every computed distance widened by its rounding bound and evaluated with directed
rounding.  A skipped pair must be one whose canonical fminf would have left delta
unchanged, so the kept indices stay bit-identical to the oracle's.  The library
uses the skipping only where a CTA's dense update streams at least 2 MB of rows;
requests of 8192 tokens at d_v = 2048 take it for every cluster size (at most 16
CTAs of 512 tokens, 2 MB each).

  * adversarial features: near-duplicate clusters (cosine distances of 1e-6 inside
    a cluster), per-row scales of 2^-20 .. 2^20, rows scaled by 2^55 or 2^-60
    (outside the norm range where the bound is used, so never skipped), exact
    duplicate rows and zero rows;
  * root capacity: 1500 tight clusters and k = 1200, so that the roots of a request
    (at most 1024) run out while new clusters are still being opened, and centres
    without a root leave their tokens unskippable.

The oracle runs one request per host thread (reentrant; threads, not forked
processes).
"""
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest

import oracle
from workloads import custom, f32_to_bf16_bits

from gpu_util import DeviceWorkload, assert_valid_selection

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


def _workload(batch, n, keep, seed):
    return custom(name="skip", seed=seed, batch=batch, n_vis=[n], n_text=[2], num_layers=1,
                  num_q_heads=2, num_kv_heads=2, head_dim=64, feat_dim=2048, dtype="bf16",
                  keep=[keep])


def _check_all(wl, w32, idx):
    assert_valid_selection(wl, idx)

    def run(b):
        v0, v1 = int(wl.cu_vis[b]), int(wl.cu_vis[b + 1])
        k = int(wl.cu_keep[b + 1] - wl.cu_keep[b])
        return b, oracle.restore_order(oracle.select_fp32(wl.x[v0:v1], w32[v0:v1], k))

    with ThreadPoolExecutor(max_workers=_threads()) as pool:
        for b, want in pool.map(run, range(wl.batch)):
            got = idx[wl.cu_keep[b]:wl.cu_keep[b + 1]]
            assert np.array_equal(got, want), (
                f"request {b}: {np.setdiff1d(got, want).tolist()[:8]} kept by GPU only, "
                f"{np.setdiff1d(want, got).tolist()[:8]} by oracle only")


def test_skipping_adversarial_features():
    batch, n, dv = 8, 8192, 2048
    wl = _workload(batch, n, 600, seed=71)
    rng = np.random.default_rng(7101)
    rows = []
    for _ in range(batch):
        proto = rng.standard_normal((200, dv))
        x = proto[rng.integers(0, 200, n)] * (1 + 1e-3 * rng.standard_normal((n, dv)))
        scale = np.exp2(rng.integers(-20, 21, n).astype(np.float64))   # per-row scales
        # rows whose 1/|x| lies outside [2^-50, 2^50] (never skipped); their squared
        # norms (about 2^121 and 2^-109) stay finite and normal in fp32
        far = rng.choice(n, n // 50, replace=False)
        scale[far] = np.where(rng.random(len(far)) < 0.5, 2.0 ** 55, 2.0 ** -60)
        x *= scale[:, None]
        src, dst = rng.choice(n, (2, n // 50), replace=False)       # exact duplicates
        x[dst] = x[src]
        x[rng.choice(n, n // 200, replace=False)] = 0.0             # zero rows
        rows.append(x)
    wl.x = f32_to_bf16_bits(np.concatenate(rows).astype(np.float32))
    w32 = np.concatenate([rng.dirichlet(np.ones(n)) for _ in range(batch)]).astype(np.float32)
    idx = DeviceWorkload(wl).select(w32)
    _check_all(wl, w32, idx)


def test_skipping_root_capacity():
    batch, n, dv = 4, 8192, 2048
    wl = _workload(batch, n, 1200, seed=72)
    rng = np.random.default_rng(7201)
    rows = []
    for _ in range(batch):
        proto = rng.standard_normal((1500, dv))
        rows.append(proto[rng.integers(0, 1500, n)] + 0.02 * rng.standard_normal((n, dv)))
    wl.x = f32_to_bf16_bits(np.concatenate(rows).astype(np.float32))
    w32 = np.concatenate([rng.dirichlet(np.ones(n)) for _ in range(batch)]).astype(np.float32)
    idx = DeviceWorkload(wl).select(w32)
    _check_all(wl, w32, idx)
