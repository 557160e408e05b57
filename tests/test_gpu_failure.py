"""Failure detection without a GPU fault: a device wait that expires is reported
through the workspace error word as LAST_ERR_TIMEOUT, the context stays usable, and
the next call on the same workspace starts clean."""
import numpy as np
import pytest

from gpu_util import DeviceWorkload
from workloads import config

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


def test_expired_wait_is_reported_and_the_context_survives():
    import torch
    import paper_2607_27952_gb300 as last
    ws = torch.zeros(256, dtype=torch.uint8, device="cuda:0")
    last.last_check_bounded_wait(ws)
    with pytest.raises(last.LastError) as e:
        last.last_poll(ws)
    assert e.value.status == last.LAST_ERR_TIMEOUT
    # the context is intact: a real call on a fresh workspace succeeds
    wl = config("c2", batch=2, budget="mixed")
    w, idx, _ = DeviceWorkload(wl).prune()
    assert np.isfinite(w).all() and len(idx) == int(wl.cu_keep[-1])
