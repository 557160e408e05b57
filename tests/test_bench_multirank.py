"""The multi-GPU path of bench.py is replicas only: every rank prunes its own batch,
the job time is the slowest rank's, and the request / token counts add up.  Two
gloo ranks on the CPU check that host-side logic (no GPU, no collective in the
data path)."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms, reqs, toks = bench.combine_over_ranks(10.0 + 5.0 * rank, 64 * 3, 36864 * 3)
    out[rank] = (ms, reqs, toks, bench.rank_seed(rank))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_combine_max_time_and_sum_work():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    for r in range(world):
        ms, reqs, toks, seed = res[r]
        assert ms == 15.0                      # the slowest rank
        assert reqs == 2 * 64 * 3 and toks == 2 * 36864 * 3
    assert res[0][3] != res[1][3]              # independent batches per rank


def test_single_process_is_identity():
    import bench
    assert bench.combine_over_ranks(3.5, 10, 20) == (3.5, 10, 20)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    import bench

    class A:
        gpus, steps, warmup, budget = 2, 1, 0, "mixed"
    bench.run_reference(A, rank=1, world=2)
    assert capsys.readouterr().out == ""


def test_reference_arm_runs_one_request_per_host_thread(capsys):
    """The oracle arm runs whole requests concurrently, one per host thread, and
    reports those threads as its cores."""
    import json
    import bench

    class A:
        gpus, steps, warmup, budget, workload = 1, 1, 0, "mixed", "c1"
        source, rows, selector = "last", 32, "greedy"
    bench.run_reference(A, rank=0, world=1)
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    threads = bench.host_threads()
    assert line["impl"] == "reference" and line["cpu_baseline"]["cores"] == threads
    assert line["value"] > 0 and line["e2e"]["h2d_bytes_per_step"] == 0
    # visual tokens per step: one 576-token request per thread
    assert abs(line["visual_tokens_scored_per_s"] / line["value"] - 576) < 1e-6


def test_scoring_kernel_count_per_source():
    """gpu_launches counts the scoring kernels of each attention source: two for
    the last row and for one row per request (G <= 8), four for several rows."""
    import bench
    from workloads import config, query_rows
    wl = config("c2", batch=3, budget="mixed")
    assert bench.scoring_kernels(wl) == 2
    assert bench.scoring_kernels(wl, query_rows(wl, "first")[0]) == 2
    assert bench.scoring_kernels(wl, query_rows(wl, "middle")[0]) == 2
    assert bench.scoring_kernels(wl, query_rows(wl, "all", m_rows=8)[0]) == 4
