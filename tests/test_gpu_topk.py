"""GPU parity of the Top-k selection variant (Table 5) against the oracle,
through the C ABI: kept indices and gathered rows bit-exact on identical scores."""
import numpy as np
import pytest

import oracle
from workloads import config, custom

from gpu_util import POISON_IDX, problem_of, to_dev, to_host_bits

pytestmark = pytest.mark.gpu


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


def run_topk(wl, w32, cu_keep=None, gather=True):
    import torch
    import paper_2607_27952_gb300 as last
    dev = torch.device("cuda:0")
    cu_keep = wl.cu_keep if cu_keep is None else np.asarray(cu_keep, np.int32)
    prob = problem_of(wl, cu_keep)
    nkeep = int(cu_keep[-1])
    idx = torch.full((nkeep,), POISON_IDX, dtype=torch.int32, device=dev)
    x = to_dev(wl.x, dev)
    xs = torch.empty((nkeep, wl.feat_dim), dtype=x.dtype, device=dev)
    xs.view(torch.uint8).fill_(0xFF)
    ws = last.workspace(prob, dev)
    wt = torch.from_numpy(np.ascontiguousarray(w32, dtype=np.float32)).to(dev)
    last.last_select_topk(prob, wt, idx, ws, x=x if gather else None,
                          x_out=xs if gather else None)
    last.last_poll(ws)
    return idx.cpu().numpy(), to_host_bits(xs)


def check(wl, w32, idx, xs, cu_keep=None, gather=True):
    cu_keep = wl.cu_keep if cu_keep is None else cu_keep
    for b in range(wl.batch):
        v0, v1 = int(wl.cu_vis[b]), int(wl.cu_vis[b + 1])
        k0, k1 = int(cu_keep[b]), int(cu_keep[b + 1])
        want = oracle.restore_order(oracle.select_topk(w32[v0:v1], k1 - k0))
        assert np.array_equal(idx[k0:k1], want), f"request {b}"
        if gather:
            assert np.array_equal(xs[k0:k1], oracle.gather(wl.x[v0:v1], want)), f"request {b} rows"


def oracle_w32(wl):
    w = oracle.scores(wl.q, wl.k, wl.cu_seqlens, wl.vis_start, wl.cu_vis,
                      num_kv_heads=wl.num_kv_heads, scale=wl.scale)
    return w.astype(np.float32)


CASES = {
    "c1": lambda: config("c1"),
    "c2": lambda: config("c2", batch=6, budget="mixed"),
    "c3": lambda: config("c3", batch=2, n_vis=1152),
    "c4": lambda: config("c4", batch=8, n_vis=[300, 1024, 257, 777, 513, 260, 999, 640]),
    "c5": lambda: config("c5", batch=2, n_vis=2048, budget=12.5),
}


@pytest.mark.parametrize("name", list(CASES))
def test_topk_on_oracle_scores(name):
    wl = CASES[name]()
    w32 = oracle_w32(wl)
    idx, xs = run_topk(wl, w32)
    check(wl, w32, idx, xs)


def _edge_workload():
    return custom(name="topk-edges", seed=81, batch=7, n_vis=[0, 5, 40, 1, 300, 16, 33],
                  n_text=[1, 2, 3, 1, 4, 2, 1], num_layers=1, num_q_heads=2, num_kv_heads=2,
                  head_dim=64, feat_dim=264, dtype="bf16", keep=[0, 5, 0, 1, 299, 16, 1])


def test_budget_edges_and_ties():
    """k = 0, k = N, N = 0, N = 1, and scores full of exact ties (including -0/+0)."""
    wl = _edge_workload()
    rng = np.random.default_rng(82)
    w32 = rng.integers(0, 5, int(wl.cu_vis[-1])).astype(np.float32) / 8
    w32[w32 == 0] = -0.0                              # every zero a negative zero
    w32[wl.cu_vis[4]:wl.cu_vis[4] + 100:2] = 0.0      # mixed with positive zeros
    idx, xs = run_topk(wl, w32)
    check(wl, w32, idx, xs)


def test_all_equal_scores_take_first_indices():
    wl = custom(name="flat", seed=83, batch=2, n_vis=[700, 129], n_text=[2, 2], num_layers=1,
                num_q_heads=2, num_kv_heads=2, head_dim=64, feat_dim=256, dtype="f32",
                keep=[350, 100])
    w32 = np.full(int(wl.cu_vis[-1]), 1.0 / 700, np.float32)
    idx, xs = run_topk(wl, w32)
    check(wl, w32, idx, xs)
    assert idx[:350].tolist() == list(range(350))


def test_indices_only_without_features():
    wl = CASES["c4"]()
    w32 = oracle_w32(wl)
    idx, _ = run_topk(wl, w32, gather=False)
    check(wl, w32, idx, None, gather=False)


def test_long_request_many_radix_passes():
    """One request far longer than a CTA pass (70 000 tokens), scores with long
    runs of equal values so the select descends into the index digits."""
    n = 70000
    wl = custom(name="long", seed=84, batch=2, n_vis=[n, 3], n_text=[1, 1], num_layers=1,
                num_q_heads=2, num_kv_heads=2, head_dim=64, feat_dim=8, dtype="bf16",
                keep=[5003, 2])
    rng = np.random.default_rng(85)
    w32 = (rng.integers(0, 50, n + 3) / 64).astype(np.float32)
    idx, xs = run_topk(wl, w32)
    check(wl, w32, idx, xs)


def test_full_size_c5_scores():
    wl = config("c5", budget=12.5)
    w32 = oracle_w32(wl)
    idx, xs = run_topk(wl, w32)
    check(wl, w32, idx, xs)


def test_nan_scores_still_give_valid_indices():
    """NaN scores are outside the contract; the call must still return k_b distinct
    in-range ascending indices."""
    wl = _edge_workload()
    w32 = np.linspace(0, 1, int(wl.cu_vis[-1]), dtype=np.float32)
    w32[::7] = np.nan
    idx, _ = run_topk(wl, w32, gather=False)
    for b in range(wl.batch):
        k0, k1 = int(wl.cu_keep[b]), int(wl.cu_keep[b + 1])
        n = int(wl.cu_vis[b + 1] - wl.cu_vis[b])
        got = idx[k0:k1]
        assert len(got) == k1 - k0
        if len(got):
            assert got.min() >= 0 and got.max() < n and (np.diff(got) > 0).all()


def test_deterministic():
    wl = CASES["c2"]()
    w32 = oracle_w32(wl)
    a, xa = run_topk(wl, w32)
    b, xb = run_topk(wl, w32)
    assert np.array_equal(a, b) and np.array_equal(xa, xb)
