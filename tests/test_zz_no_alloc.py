"""last_scores_noalloc: the scoring entry point that allocates nothing.

It serves callers that cannot allocate device memory at run time (for example a
service that reserves all of its device memory at start-up).  Its scratch is a
fixed array inside the library, so this test checks that two calls in a row give
the oracle's scores and those of last_scores with a caller workspace, within the
score tolerance of the parity tests, on problems of alternating size and dtype,
and that an oversized problem is rejected.
This file is collected last so that a stop-at-first-failure run has already run
every other test.
"""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    from paper_2607_27952_gb300.build import build
    import paper_2607_27952_gb300 as last
    build()
    last.load_library()
    return last


def _problem(last, wl):
    return last.Problem(batch=wl.batch, num_layers=wl.num_layers, num_q_heads=wl.num_q_heads,
                        num_kv_heads=wl.num_kv_heads, head_dim=wl.head_dim,
                        feat_dim=wl.feat_dim, dtype=wl.dtype, cu_seqlens=wl.cu_seqlens,
                        vis_start=wl.vis_start, cu_vis=wl.cu_vis, cu_keep=wl.cu_keep)


def _dev(a, dev):
    import torch
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).to(dev).view(torch.bfloat16)
    return torch.from_numpy(a).to(dev)


def test_noalloc_scores_match_workspace_path_twice(lib):
    """Large, small, large again (bf16, GQA, fp32 in between): every call must ignore
    the statistics and logits a previous, differently sized call left in the shared
    scratch.  Each call is checked against the fp64 oracle (rtol 1e-3, the parity
    tolerance) and against last_scores with a workspace, two calls in a row."""
    import torch
    import oracle
    from workloads import config, custom
    oracle.build()
    dev = torch.device("cuda:0")
    large = config("c2", batch=6, budget="mixed")
    small = custom(name="gqa7", seed=5, batch=3, n_vis=[120, 33, 300], n_text=[7, 2, 19],
                   n_before=[4, 0, 9], num_layers=2, num_q_heads=14, num_kv_heads=2,
                   head_dim=64, feat_dim=64, dtype="bf16", keep=[8, 3, 30])
    fp32 = config("c1")
    for wl in (large, small, fp32, large, small):
        prob = _problem(lib, wl)
        q, k = _dev(wl.q, dev), _dev(wl.k, dev)
        want = oracle.scores(wl.q, wl.k, wl.cu_seqlens, wl.vis_start, wl.cu_vis,
                             num_kv_heads=wl.num_kv_heads, scale=wl.scale)
        ref = torch.full((prob.total_vis,), float("nan"), device=dev)
        ws = lib.workspace(prob, dev)
        lib.last_scores(prob, q, k, ref, ws)
        lib.last_poll(ws)
        ref = ref.cpu().numpy().astype(np.float64)
        for _ in range(2):                      # two calls in a row share the scratch
            out = torch.full((prob.total_vis,), float("nan"), device=dev)
            lib.last_scores_noalloc(prob, q, k, out)
            torch.cuda.synchronize()
            got = out.cpu().numpy().astype(np.float64)
            assert np.isfinite(got).all()
            assert np.allclose(got, want, rtol=1e-3, atol=1e-30), wl.name
            assert np.allclose(got, ref, rtol=1e-3, atol=1e-30), wl.name


def test_noalloc_rejects_oversized_problem(lib):
    import torch
    # 4 layers x 16 heads x 70000 visual tokens of fp32 logits alone exceed 16 MiB
    B, N = 1, 70000
    prob = lib.Problem(batch=B, num_layers=4, num_q_heads=16, num_kv_heads=4, head_dim=128,
                       feat_dim=256, dtype="bf16", cu_seqlens=[0, N + 2], vis_start=[0],
                       cu_vis=[0, N], cu_keep=[0, 1])
    dev = torch.device("cuda:0")
    dummy = torch.empty(16, dtype=torch.float32, device=dev)
    with pytest.raises(lib.LastError) as e:
        lib.last_scores_noalloc(prob, dummy, dummy, dummy)
    assert e.value.status == lib.LAST_ERR_UNSUPPORTED
    assert "16777216" in str(e.value)
