"""CPU-side checks of the C ABI: the library loads, exports every function the
public header declares, and rejects bad problems on the host before touching
the GPU (no compute call runs here)."""
import ctypes
import os
import re

import numpy as np
import pytest

import paper_2607_27952_gb300 as last

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "last.h")


@pytest.fixture(scope="module")
def lib():
    from paper_2607_27952_gb300.build import build
    build()
    return last.load_library()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(last_[a-z_]+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 9
    for n in names:
        assert hasattr(lib, n), f"{n} declared in include/last.h but not exported"
    assert set(names) == set(last.EXPORTED)


def _problem(**kw):
    base = dict(batch=2, num_layers=1, num_q_heads=4, num_kv_heads=2, head_dim=64, feat_dim=256,
                dtype="bf16", cu_seqlens=[0, 10, 30], vis_start=[0, 2], cu_vis=[0, 6, 14],
                cu_keep=[0, 2, 5])
    base.update(kw)
    return last.Problem(**base)


def test_workspace_size_is_host_only(lib):
    n = last.last_workspace_size(_problem())
    assert n > 0 and n % 256 == 0
    bigger = last.last_workspace_size(_problem(cu_seqlens=[0, 3000, 7000]))
    assert bigger > n


@pytest.mark.parametrize("kw,status", [
    (dict(num_q_heads=6, num_kv_heads=4), last.LAST_ERR_INVALID_ARG),       # Hq % Hkv
    (dict(vis_start=[4, 2]), last.LAST_ERR_INVALID_ARG),                     # span reaches p*
    (dict(cu_keep=[0, 7, 9]), last.LAST_ERR_INVALID_ARG),                    # k_b > N_b
    (dict(cu_keep=[0, 3, 2]), last.LAST_ERR_INVALID_ARG),                    # k_b < 0
    (dict(cu_seqlens=[0, 0, 30], vis_start=[0, 2], cu_vis=[0, 0, 14],
          cu_keep=[0, 0, 5]), last.LAST_ERR_INVALID_ARG),                    # P_b = 0
    (dict(num_q_heads=18, num_kv_heads=2), last.LAST_ERR_UNSUPPORTED),       # G = 9 > 8
    (dict(head_dim=12), last.LAST_ERR_UNSUPPORTED),                          # 24 B rows
    (dict(num_q_heads=256, num_kv_heads=32, head_dim=128),
     last.LAST_ERR_UNSUPPORTED),                                             # q > smem
])
def test_scores_rejects_bad_problems_before_launch(lib, kw, status):
    prob = _problem(**kw)
    with pytest.raises(last.LastError) as e:
        last.last_scores(prob, 16, 16, 16, (256, 1 << 30), stream=0)
    assert e.value.status == status


@pytest.mark.parametrize("kw,status", [
    (dict(feat_dim=100), last.LAST_ERR_INVALID_ARG),
    (dict(feat_dim=4096), last.LAST_ERR_UNSUPPORTED),
    (dict(cu_vis=[0, 6, 5]), last.LAST_ERR_INVALID_ARG),
    # N_b past the clustered plan's shared memory, in a launch of five requests (the
    # whole-GPU selection takes at most four)
    (dict(dtype="f32", feat_dim=2048, batch=5, cu_seqlens=[0, 10, 20020, 20030, 20040, 20050],
          vis_start=[0, 2, 0, 0, 0], cu_vis=[0, 6, 20006, 20007, 20008, 20009],
          cu_keep=[0, 2, 5, 6, 7, 8]), last.LAST_ERR_UNSUPPORTED),
    (dict(feat_dim=64, batch=5, cu_seqlens=[0, 10, 140020, 140030, 140040, 140050],
          vis_start=[0, 2, 0, 0, 0], cu_vis=[0, 6, 140006, 140007, 140008, 140009],
          cu_keep=[0, 2, 5, 6, 7, 8]), last.LAST_ERR_UNSUPPORTED),
])
def test_select_rejects_bad_problems_before_launch(lib, kw, status):
    prob = _problem(**kw)
    with pytest.raises(last.LastError) as e:
        last.last_select(prob, 16, 16, 16, (256, 1 << 30), stream=0, x_out=None)
    assert e.value.status == status


@pytest.mark.parametrize("kw,args,status", [
    (dict(cu_keep=[0, 7, 9]), dict(x=16, x_out=16), last.LAST_ERR_INVALID_ARG),     # k_b > N_b
    (dict(feat_dim=100), dict(x=16, x_out=16), last.LAST_ERR_INVALID_ARG),          # gather width
    (dict(), dict(x=None, x_out=16), last.LAST_ERR_INVALID_ARG),                    # x missing
    (dict(), dict(x=24, x_out=16), last.LAST_ERR_INVALID_ARG),                      # misaligned x
])
def test_topk_rejects_bad_arguments_before_launch(lib, kw, args, status):
    prob = _problem(**kw)
    with pytest.raises(last.LastError) as e:
        last.last_select_topk(prob, 16, 16, (256, 1 << 30), stream=0, **args)
    assert e.value.status == status


def test_long_requests_pass_topk_and_gather_validation(lib):
    """The greedy's shared-memory bound on N_b applies to last_select alone: Top-k
    and the gather take the same request up to their pointer checks."""
    prob = _problem(dtype="f32", feat_dim=2048, cu_seqlens=[0, 10, 20020], cu_vis=[0, 6, 20006])
    with pytest.raises(last.LastError) as e:
        last.last_select_topk(prob, 16, 16, (256, 1 << 30), stream=0, x=24, x_out=16)
    assert e.value.status == last.LAST_ERR_INVALID_ARG and "align" in str(e.value)
    with pytest.raises(last.LastError) as e:
        last.last_gather(prob, 24, 16, 16, (256, 1 << 30), stream=0)
    assert e.value.status == last.LAST_ERR_INVALID_ARG and "align" in str(e.value)


def test_host_workspace_holds_the_device_copies(lib):
    prob = _problem()
    n_ws = last.last_workspace_size(prob)
    n_host = last.last_host_workspace_size(prob)
    # q [2][1][4][64], K [1][30][2][64], X [14][256] bf16; w [14], idx [5], rows [5][256]
    payload = (2 * 4 * 64 + 30 * 2 * 64 + 14 * 256) * 2 + 14 * 4 + 5 * 4 + 5 * 256 * 2
    assert n_host >= n_ws + payload and n_host % 256 == 0


@pytest.mark.parametrize("args,status", [
    (dict(ws=(256, 1024)), last.LAST_ERR_WORKSPACE_TOO_SMALL),
    (dict(ws=(300, 1 << 30)), last.LAST_ERR_INVALID_ARG),          # not 256-byte aligned
    (dict(ws=(256, 1 << 30), idx_out=None), last.LAST_ERR_INVALID_ARG),
    (dict(ws=(256, 1 << 30), k=None), last.LAST_ERR_INVALID_ARG),
])
def test_prune_host_rejects_bad_arguments_before_any_copy(lib, args, status):
    call = dict(q=16, k=16, x=16, w_out=None, idx_out=16, x_out=None)
    call.update(args)
    ws = call.pop("ws")
    with pytest.raises(last.LastError) as e:
        last.last_prune_host(_problem(), ws=ws, stream=0, **call)
    assert e.value.status == status


def test_topk_needs_no_sequence_fields(lib):
    # scores-only fields may be absent; validation then fails only on the workspace
    prob = last.Problem(batch=1, num_layers=0, num_q_heads=0, num_kv_heads=0, head_dim=0,
                        feat_dim=8, dtype="bf16", cu_seqlens=None, vis_start=None,
                        cu_vis=[0, 5], cu_keep=[0, 2])
    with pytest.raises(last.LastError) as e:
        last.last_select_topk(prob, 16, 16, (256, 1), stream=0)
    assert e.value.status == last.LAST_ERR_WORKSPACE_TOO_SMALL


@pytest.mark.parametrize("kw,rows,status", [
    (dict(dtype="f32"), ([0, 1, 2], [8, 20]), last.LAST_ERR_UNSUPPORTED),          # bf16 only
    (dict(), ([0, 1, 2], [5, 20]), last.LAST_ERR_INVALID_ARG),                     # inside span
    (dict(), ([0, 1, 2], [8, 20]), last.LAST_ERR_INVALID_ARG),                     # past P_b - 1
    (dict(), ([0, 0, 2], [20, 21]), last.LAST_ERR_INVALID_ARG),                    # no row
    (dict(head_dim=80), ([0, 1, 2], [8, 20]), last.LAST_ERR_UNSUPPORTED),          # head_dim
    (dict(num_q_heads=16, num_kv_heads=2), ([0, 33, 34], list(range(6, 10)) * 8 + [9, 19]),
     last.LAST_ERR_UNSUPPORTED),                                                 # 33 x 8 > 256
])
def test_scores_rows_rejects_bad_arguments(lib, kw, rows, status):
    prob = _problem(**kw)
    qr = last.QueryRows(*rows)
    with pytest.raises(last.LastError) as e:
        last.last_scores_rows(prob, qr, 16, 16, 16, (256, 1 << 30), stream=0)
    assert e.value.status == status


def test_scores_rows_workspace_grows_with_rows(lib):
    prob = _problem()
    one = last.last_scores_rows_workspace_size(prob, last.QueryRows([0, 1, 2], [9, 19]))
    many = last.last_scores_rows_workspace_size(prob, last.QueryRows([0, 3, 6], [6, 7, 9, 10, 15, 19]))
    assert many > one > 0
    # one row per request runs the last-row kernels: the workspace holds their plan
    # (the scoring part of last_workspace_size: with no budgets the selection's
    # root-row scratch is empty)
    assert one >= last.last_workspace_size(_problem(cu_keep=[0, 0, 0]))


def test_workspace_holds_selection_root_rows(lib):
    """bf16 problems carry the greedy's root rows: min(k_b, 1024) feature rows and a
    32-column bound table per request, on top of the scoring scratch."""
    base = last.last_workspace_size(_problem(cu_keep=[0, 0, 0]))
    full = last.last_workspace_size(_problem())
    assert full - base >= 5 * (256 * 2 + 32 * 4)
    assert last.last_workspace_size(_problem(dtype="f32")) < full + 4096


def test_workspace_checks(lib):
    prob = _problem()
    need = last.last_workspace_size(prob)
    with pytest.raises(last.LastError) as e:
        last.last_prune(prob, 16, 16, 16, None, 16, None, (256, need - 1), stream=0)
    assert e.value.status == last.LAST_ERR_WORKSPACE_TOO_SMALL
    with pytest.raises(last.LastError) as e:
        last.last_prune(prob, 16, 16, 16, None, 16, None, (8, need), stream=0)
    assert e.value.status == last.LAST_ERR_INVALID_ARG      # not 256-byte aligned
    with pytest.raises(last.LastError) as e:
        last.last_prune(prob, 16, 24, 16, None, 16, None, (256, need), stream=0)
    assert e.value.status == last.LAST_ERR_INVALID_ARG      # k not 16-byte aligned


@pytest.mark.parametrize("n,num,den", [(576, 1, 8), (16384, 1, 20), (16384, 1, 4), (257, 1, 8),
                                       (0, 1, 8), (2880, 1, 8), (4095, 1, 8), (7, 3, 3)])
def test_budget_matches_ceil(lib, n, num, den):
    import math
    from fractions import Fraction
    assert last.last_budget(n, num, den) == math.ceil(Fraction(num * n, den))


def test_budget_rejects_bad_ratio(lib):
    assert last.last_budget(-1, 1, 8) == -1
    assert last.last_budget(10, 1, 0) == -1


def test_status_strings(lib):
    for st in range(7):
        assert last.last_status_string(st).startswith("LAST_")


def test_library_path_is_in_tree(lib):
    assert os.path.dirname(last.LIB_PATH) == os.path.join(ROOT, "paper_2607_27952_gb300")
