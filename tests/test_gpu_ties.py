"""GPU parity of the selection where keys tie exactly and the lowest index decides.

Equal weights on mutually orthogonal features give every unselected token the same
key w~ delta (delta = 1 exactly), so the greedy of Eq. 10-11 takes the tokens in
index order; weight-zero tokens do the same once every positive weight is taken.
Under such ties one warp of a CTA owns that CTA's best keys, and the CTA's
candidate list holds only the published count after a rebuild: the round's bound
must then come from the list's own bound, or a round takes another CTA's
candidate ahead of this CTA's next one.  The kept indices must equal the oracle's
(single requests, so the launch uses large clusters, and a batch of several).
"""
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


def _workload(name, n_vis, keep, dv, seed):
    return custom(name=name, seed=seed, batch=len(n_vis), n_vis=n_vis, n_text=[2] * len(n_vis),
                  num_layers=1, num_q_heads=2, num_kv_heads=2, head_dim=64, feat_dim=dv,
                  dtype="bf16", keep=keep)


def _one_hot(n, dv, offset=0):
    x = np.zeros((n, dv), np.float32)
    x[np.arange(n), (np.arange(n) + offset) % dv] = 1.0
    return x


@pytest.mark.parametrize("n,k", [(2048, 64), (2048, 300), (1200, 100)])
def test_equal_weights_on_orthogonal_features(n, k):
    wl = _workload(f"ties-onehot-{n}", [n], [k], 2048, seed=11)
    wl.x = f32_to_bf16_bits(_one_hot(n, 2048))
    w32 = np.full(n, 1.0 / 4096, np.float32)        # exact: every key is the same product
    idx = DeviceWorkload(wl).select(w32)
    assert_valid_selection(wl, idx)
    assert np.array_equal(idx, np.arange(k))        # the greedy takes the lowest indices
    assert_selection_equal(wl, w32, idx, [0])


def test_weight_zero_tokens_after_the_positive_ones():
    rng = np.random.default_rng(12)
    n, k, npos = 3000, 400, 150
    wl = _workload("ties-zero-w", [n], [k], 256, seed=12)
    wl.x = f32_to_bf16_bits(rng.standard_normal((n, 256)).astype(np.float32))
    w32 = np.zeros(n, np.float32)
    w32[rng.choice(n, npos, replace=False)] = rng.dirichlet(np.ones(npos)).astype(np.float32)
    idx = DeviceWorkload(wl).select(w32)
    assert_valid_selection(wl, idx)
    assert_selection_equal(wl, w32, idx, [0])


def test_tied_batch():
    # several requests: orthogonal rows with equal weights, and one with weight-zero tails
    rng = np.random.default_rng(13)
    n_vis, keep = [900, 1500, 640, 2000], [120, 90, 200, 40]
    wl = _workload("ties-batch", n_vis, keep, 2048, seed=13)
    xs, ws = [], []
    for b, n in enumerate(n_vis):
        xs.append(_one_hot(n, 2048, offset=37 * b))
        w = np.full(n, 1.0 / 2048, np.float32)
        if b == 2:
            w[rng.random(n) < 0.8] = 0.0
        ws.append(w)
    wl.x = f32_to_bf16_bits(np.concatenate(xs))
    w32 = np.concatenate(ws)
    idx = DeviceWorkload(wl).select(w32)
    assert_valid_selection(wl, idx)
    assert_selection_equal(wl, w32, idx, range(wl.batch))
