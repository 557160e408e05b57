"""GPU parity of the selection on inputs chosen against the tensor-core update's
certificate: the update decides from tensor-core distances only when they are
provably on one side of delta, and recomputes every other pair in the canonical
fp32 order, so the kept indices must stay bit-identical to the oracle's even when
distances are tiny, scores tie, or products cancel."""
import numpy as np
import pytest

from workloads import custom, f32_to_bf16_bits

from gpu_util import DeviceWorkload, assert_selection_equal, assert_valid_selection

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2607_27952_gb300.build import build
    import paper_2607_27952_gb300 as last
    import oracle
    build()
    last.load_library()
    oracle.build()


def _workload(dv, n_vis, keep, seed):
    return custom(name=f"cert-d{dv}", seed=seed, batch=len(n_vis), n_vis=n_vis,
                  n_text=[2] * len(n_vis), num_layers=1, num_q_heads=2, num_kv_heads=2,
                  head_dim=64, feat_dim=dv, dtype="bf16", keep=keep)


def _features(kind, n, dv, rng):
    if kind == "near_duplicates":
        # 24 prototypes, every token within ~1e-3 (relative) of one: cosine distances
        # of 1e-6..1e-5 between tokens of a prototype, far below the certificate's bound
        base = rng.standard_normal((24, dv))
        return base[rng.integers(0, 24, n)] * (1 + 1e-3 * rng.standard_normal((n, dv)))
    if kind == "dynamic_range":
        # magnitudes spread over 2^-20..2^20: sum |x_i x_j| far above |x_i . x_j|
        return rng.standard_normal((n, dv)) * np.exp2(rng.integers(-20, 21, (n, dv)))
    if kind == "exact_duplicates":
        base = rng.standard_normal((40, dv))
        return base[rng.integers(0, 40, n)]
    raise ValueError(kind)


@pytest.mark.parametrize("dv", [64, 512, 2048])
@pytest.mark.parametrize("kind", ["near_duplicates", "dynamic_range", "exact_duplicates"])
def test_certified_update_is_exact(kind, dv):
    wl = _workload(dv, [700, 250, 1300], [90, 249, 160], seed=90 + dv)
    rng = np.random.default_rng({"near_duplicates": 1, "dynamic_range": 2,
                                 "exact_duplicates": 3}[kind] * 10000 + dv)
    n = int(wl.cu_vis[-1])
    wl.x = f32_to_bf16_bits(_features(kind, n, dv, rng).astype(np.float32))
    if kind == "near_duplicates":
        w32 = np.full(n, 1.0 / 700, np.float32)            # products tie wherever delta ties
    else:
        w32 = rng.dirichlet(np.ones(n)).astype(np.float32)
    idx = DeviceWorkload(wl).select(w32)
    assert_valid_selection(wl, idx)
    assert_selection_equal(wl, w32, idx, range(wl.batch))
