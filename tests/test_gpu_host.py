"""last_prune_host (the whole path on host buffers, copies included) against
last_prune on device buffers: scores, kept indices and gathered rows identical bit
for bit, from pinned CPU tensors and from pageable numpy arrays, and back to
back on two streams with two workspaces (the overlapped form)."""
import numpy as np
import pytest

from workloads import config, custom

from gpu_util import DeviceWorkload, problem_of, to_host_bits

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


def _host(a, pinned):
    import torch
    if not pinned:
        return np.ascontiguousarray(a)
    t = torch.from_numpy(np.ascontiguousarray(a.view(np.int16) if a.dtype == np.uint16 else a))
    return t.pin_memory()


def _run_host(wl, pinned, stream=None):
    import torch
    import paper_2607_27952_gb300 as last
    prob = problem_of(wl)
    nkeep, nvis = int(wl.cu_keep[-1]), int(wl.cu_vis[-1])
    xs_dtype = np.uint16 if wl.x.dtype == np.uint16 else np.float32
    w = _host(np.full(nvis, np.nan, np.float32), pinned)
    idx = _host(np.full(nkeep, -7, np.int32), pinned)
    xs = _host(np.full((nkeep, wl.feat_dim), 0xFFFF if xs_dtype == np.uint16 else np.nan,
                       xs_dtype), pinned)
    ws = last.host_workspace(prob, "cuda:0")
    last.last_prune_host(prob, _host(wl.q, pinned), _host(wl.k, pinned), _host(wl.x, pinned),
                         w, idx, xs, ws, stream)
    (stream or torch.cuda.current_stream()).synchronize()
    last.last_poll(ws, stream)
    as_np = (lambda t: t if isinstance(t, np.ndarray) else t.numpy())
    xs_np = as_np(xs)
    if xs_np.dtype == np.int16:
        xs_np = xs_np.view(np.uint16)
    return as_np(w), as_np(idx), xs_np


@pytest.mark.parametrize("name", ["c1", "mixed"])
@pytest.mark.parametrize("pinned", [True, False])
def test_host_path_equals_device_path(name, pinned):
    if name == "c1":
        wl = config("c1")
    else:
        wl = custom(name="host-mixed", seed=31, batch=5, n_vis=[200, 1, 576, 0, 333],
                    n_text=[9, 3, 40, 2, 17], num_layers=2, num_q_heads=8, num_kv_heads=2,
                    head_dim=64, feat_dim=320, dtype="bf16", keep=[20, 1, 64, 0, 333])
    w_d, idx_d, xs_d = DeviceWorkload(wl).prune()
    w_h, idx_h, xs_h = _run_host(wl, pinned)
    assert np.array_equal(w_h.view(np.uint32), w_d.view(np.uint32))
    assert np.array_equal(idx_h, idx_d)
    assert np.array_equal(xs_h, xs_d)


def test_two_streams_two_workspaces():
    """The overlapped form a server uses: consecutive calls alternate between two
    workspaces on two streams; every call's outputs equal the device path's."""
    import torch
    import paper_2607_27952_gb300 as last
    wl = custom(name="host-streams", seed=32, batch=6, n_vis=[576], n_text=[20],
                num_layers=1, num_q_heads=16, num_kv_heads=16, head_dim=128, feat_dim=512,
                dtype="bf16", keep=[64, 128, 192])
    _, idx_d, xs_d = DeviceWorkload(wl).prune()
    prob = problem_of(wl)
    nkeep = int(wl.cu_keep[-1])
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    wss = [last.host_workspace(prob, "cuda:0") for _ in streams]
    q, k, x = _host(wl.q, True), _host(wl.k, True), _host(wl.x, True)
    outs = []
    for i in range(4):
        idx = torch.full((nkeep,), -7, dtype=torch.int32).pin_memory()
        xs = torch.empty((nkeep, wl.feat_dim), dtype=torch.int16).pin_memory()
        last.last_prune_host(prob, q, k, x, None, idx, xs, wss[i % 2], streams[i % 2])
        outs.append((idx, xs))
    torch.cuda.synchronize()
    for ws in wss:
        last.last_poll(ws)
    for idx, xs in outs:
        assert np.array_equal(idx.numpy(), idx_d)
        assert np.array_equal(xs.numpy().view(np.uint16), xs_d)
