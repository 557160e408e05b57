"""GPU parity of the multi-row attention sources (Table 4: First, Middle, All Mean)
against the oracle, through the C ABI: scores within rtol 1e-3."""
import numpy as np
import pytest

import oracle
from workloads import config, custom, query_rows

from gpu_util import SCORE_ATOL, SCORE_RTOL, problem_of, to_dev

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


def make_rows(wl, source, rng, m_rows=8):
    """Query rows of the given source (First, Middle, Last or All Mean over up to
    m_rows text rows), seeded from rng."""
    return query_rows(wl, source, m_rows=m_rows, seed=int(rng.integers(1 << 30)))


def run_rows(wl, cu, pos, q):
    import torch
    import paper_2607_27952_gb300 as last
    dev = torch.device("cuda:0")
    prob = problem_of(wl)
    rows = last.QueryRows(cu, pos)
    w = torch.full((int(wl.cu_vis[-1]),), float("nan"), dtype=torch.float32, device=dev)
    ws = last.rows_workspace(prob, rows, dev)
    last.last_scores_rows(prob, rows, to_dev(q, dev), to_dev(wl.k, dev), w, ws)
    last.last_poll(ws)
    return w.cpu().numpy()


def check(wl, cu, pos, q):
    w_gpu = run_rows(wl, cu, pos, q)
    w_ref = oracle.scores_rows(q, wl.k, wl.cu_seqlens, wl.vis_start, wl.cu_vis, cu, pos,
                               num_kv_heads=wl.num_kv_heads, scale=wl.scale)
    assert np.isfinite(w_gpu).all()
    err = np.abs(w_gpu.astype(np.float64) - w_ref)
    bad = err > SCORE_RTOL * np.abs(w_ref) + SCORE_ATOL
    assert not bad.any(), f"{bad.sum()} scores outside rtol; worst {(err / w_ref).max():.2e}"
    return w_gpu


CASES = {
    "c2": lambda: config("c2", batch=4, budget="mixed"),
    "c3": lambda: config("c3", batch=2, n_vis=1152),
    "c5": lambda: config("c5", batch=2, n_vis=1024, budget=12.5),
    "gqa8_d64": lambda: custom(name="g8d64", seed=61, batch=3, n_vis=[200, 77, 300],
                               n_text=[40, 12, 3], n_before=[5, 0, 17], num_layers=2,
                               num_q_heads=16, num_kv_heads=2, head_dim=64, feat_dim=64,
                               dtype="bf16"),
    "mha_d256": lambda: custom(name="d256", seed=62, batch=2, n_vis=[130, 260], n_text=[9, 70],
                               num_layers=1, num_q_heads=4, num_kv_heads=4, head_dim=256,
                               feat_dim=64, dtype="bf16"),
}


@pytest.mark.parametrize("source", ["first", "middle", "last", "all"])
@pytest.mark.parametrize("name", list(CASES))
def test_rows_match_oracle(name, source):
    wl = CASES[name]()
    cu, pos, q = make_rows(wl, source, np.random.default_rng(7))
    check(wl, cu, pos, q)


def test_last_row_equals_single_row_scoring():
    """The Last source is the method's own Eq. 6-8: one row per request runs the
    last-row scoring kernels (cut after the row), so it equals last_scores bit for
    bit."""
    from gpu_util import DeviceWorkload
    wl = CASES["c3"]()
    cu, pos, q = make_rows(wl, "last", np.random.default_rng(8))
    w_rows = check(wl, cu, pos, q)
    w_one = DeviceWorkload(wl).scores()
    assert np.array_equal(w_rows.view(np.uint32), w_one.view(np.uint32))


def test_single_row_beyond_the_last_row_kernels():
    """G = 16 q-heads per kv-head is past the last-row kernels (G <= 8): one row per
    request then runs on the multi-row kernels, still within tolerance."""
    wl = custom(name="g16", seed=64, batch=3, n_vis=[120, 40, 260], n_text=[30, 5, 64],
                num_layers=1, num_q_heads=32, num_kv_heads=2, head_dim=64, feat_dim=64,
                dtype="bf16")
    for source in ("first", "middle"):
        cu, pos, q = make_rows(wl, source, np.random.default_rng(10))
        check(wl, cu, pos, q)


def test_many_rows_full_width():
    """64 rows x G = 4 = 256 MMA columns (the limit), ragged row counts."""
    wl = custom(name="wide", seed=63, batch=3, n_vis=[300, 500, 64], n_text=[80, 64, 200],
                num_layers=1, num_q_heads=8, num_kv_heads=2, head_dim=128, feat_dim=64,
                dtype="bf16")
    cu, pos, q = make_rows(wl, "all", np.random.default_rng(9), m_rows=64)
    assert int(np.diff(cu).max()) == 64
    check(wl, cu, pos, q)
