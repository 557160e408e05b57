"""GPU parity of the greedy selection (Eq. 9-12) on the longest requests its
shared-memory plan takes: the tensor-core update at its TMEM limit (16 CTAs of
28 row tiles), a bf16 request past that limit (costed again for the CUDA-core
update), and fp32 rows of 2048 features near the plan's bound on N_b.  Kept
indices must equal the oracle's bit for bit."""
import numpy as np
import pytest

from workloads import custom

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


@pytest.mark.parametrize("n,dv,dtype,keep", [
    (16 * 28 * 128, 256, "bf16", 72),     # tensor cores, every TMEM column in use
    (70000, 256, "bf16", 72),             # past the tensor-core limit: CUDA-core update
    (12900, 2048, "f32", 40),             # fp32 rows of 8 KB near the N_b bound
])
def test_longest_requests(n, dv, dtype, keep):
    wl = custom(name=f"long-{dtype}-d{dv}", seed=n % 1000 + dv, batch=2, n_vis=[n, 37],
                n_text=[1, 1], num_layers=1, num_q_heads=2, num_kv_heads=2, head_dim=64,
                feat_dim=dv, dtype=dtype, keep=[keep, 9], n_clusters=64)
    rng = np.random.default_rng(n + dv)
    total = int(wl.cu_vis[-1])
    w32 = rng.gamma(0.3, size=total).astype(np.float32)
    for b in range(wl.batch):
        v0, v1 = int(wl.cu_vis[b]), int(wl.cu_vis[b + 1])
        w32[v0:v1] /= np.float32(w32[v0:v1].sum())
    idx = DeviceWorkload(wl).select(w32)
    assert_valid_selection(wl, idx)
    assert_selection_equal(wl, w32, idx, range(wl.batch))
