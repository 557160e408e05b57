"""Throughput of LAST's edge-side token-selection path on GB300.

One step = one pass of the whole path over one batch: last-query-token
scores (Eq. 6-8), greedy k-center selection (Eq. 9-11) and the ordered gather
(Eq. 12), through the C ABI (last_scores, then last_select with the fused
gather), with the inputs already resident in device memory.

Default workload (the headline line): the long-context video batch, 8 requests
x 16384 visual tokens (32 frames x 512) + 128 text tokens, GQA 16/4 heads x 128,
bf16, 2048-d random-walk frame features, budget k/N = 12.5% (k = 2048).  Inputs
are 672 MB, larger than the 129 MB L2, so no flush is needed between steps.
The same JSON line carries `per_config`: every other workload preset (c1, c2
with budgets 64/128/192, c3, c4, the video batch at 5% and 25%) timed the same
way with fewer steps.

Prints one JSON line (rank 0).  `--impl reference` times the plain C oracle
(as it stands) on the host cores instead.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "pruned requests/sec and visual tokens scored/sec per GB300; % of HBM roofline"
UNIT = "requests/s"
PEAKS_FILE = os.path.join(ROOT, "MEASURED_PEAKS.json")
FALLBACK_HBM_GBS = 6800.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--budget", default=None,
                    help="c2: mixed (default), 64, 128 or 192; c5: 5, 12.5 (default) or 25 (%% of N)")
    ap.add_argument("--workload", default="c5", choices=["c1", "c2", "c3", "c4", "c5"],
                    help="c5 (default, the largest single-GPU configuration) is the headline line")
    ap.add_argument("--selector", default="greedy", choices=["greedy", "topk"],
                    help="greedy: importance-weighted k-center (Eq. 9-11, the method); "
                         "topk: the Top-k variant of Table 5")
    ap.add_argument("--source", default="last", choices=["last", "first", "middle", "all"],
                    help="attention source of the importance scores (Table 4): the last query "
                         "row (the method), the first or middle text row, or the mean of up "
                         "to --rows text rows")
    ap.add_argument("--rows", type=int, default=32, help="rows per request for --source all")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-per-config", action="store_true",
                    help="skip the per_config lines of the other workload presets")
    ap.add_argument("--per-config-seconds", type=float, default=1.0,
                    help="timed device seconds per per_config entry (at least 3 steps)")
    args = ap.parse_args()
    if args.budget is None:
        args.budget = {"c2": "mixed", "c5": "12.5"}.get(args.workload, "default")
    return args


def rank_seed(rank: int) -> int:
    """Each rank prunes its own batch of independent requests (weak scaling)."""
    return 1 + 1000 * rank


def workload(budget, rank, name="c5"):
    from workloads import config
    if name == "c2":
        b = budget if budget in ("mixed", "default") else int(budget)
        return config("c2", budget="mixed" if b == "default" else b, seed=rank_seed(rank))
    if name == "c5":
        return config("c5", budget=12.5 if budget in ("mixed", "default") else float(budget),
                      seed=4 + 1000 * rank)
    base = {"c1": 0, "c3": 2, "c4": 3}[name]
    return config(name, seed=base + 1000 * rank)


def combine_over_ranks(total_ms: float, requests: int, tokens: int, device=None):
    """Whole-job figures: the slowest rank's time and the requests / visual tokens of
    all ranks (replicas only: no data-path collective, just this reduction of
    timings).  Returns (max_ms, total_requests, total_tokens)."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return total_ms, requests, tokens
    t = torch.tensor([total_ms], dtype=torch.float64, device=device)
    n = torch.tensor([requests, tokens], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.all_reduce(n, op=dist.ReduceOp.SUM)
    return float(t.item()), int(n[0].item()), int(n[1].item())


WORKLOAD_DATA = {
    "c1": "synthetic (seeded; 1 request, 576 visual + 32 text tokens, 24-cluster features, "
          "20 planted relevant tokens)",
    "c2": "synthetic (seeded; shapes of the paper's LLaVA-1.5 workload: 576 visual tokens, "
          "64-cluster features, 10 planted relevant tokens)",
    "c3": "synthetic (seeded; 5 high-resolution tiles x 576 tokens in one pool, 128-cluster "
          "features with 30% near-duplicates, 4 guidance layers)",
    "c4": "synthetic (seeded; dynamic-resolution ragged batch, 256..4096 visual tokens, "
          "varlen packed keys)",
    "c5": "synthetic (seeded; video-like: 32 frames x 512 tokens, each frame the previous "
          "one plus N(0, 0.05^2) noise)",
}


def workload_dtype(wl) -> str:
    """The arithmetic the path computes in: inputs as stored, fp32 accumulation and
    fp32 scores; the selection decides in canonical fp32."""
    return "bf16 in, f32 accumulate" if wl.dtype == "bf16" else "f32"


def workload_desc(wl, budget, name="c5"):
    n = np.diff(wl.cu_vis)
    k = np.diff(wl.cu_keep)
    if name == "c2":
        title = (f"c2: {wl.batch} requests x {int(n[0])} visual tokens (LLaVA-1.5 shape), "
                 f"budgets {'64/128/192 round-robin' if budget in ('mixed', 'default') else budget}")
    elif name == "c5":
        title = (f"c5: {wl.batch} requests x {int(n[0])} visual tokens (32 frames x 512, video), "
                 f"k/N = {wl.name.split('=')[1].rstrip(')')} (k = {int(k[0])})")
    else:
        title = f"{wl.name}: {wl.batch} requests, {wl.note}"
    in_bytes = int(wl.q.nbytes + wl.k.nbytes + wl.x.nbytes)
    return {"workload": title,
            "batch": wl.batch, "visual_tokens": int(n.sum()), "kept_tokens": int(k.sum()),
            "keys": int(wl.cu_seqlens[-1]), "layers": wl.num_layers, "q_heads": wl.num_q_heads,
            "kv_heads": wl.num_kv_heads, "head_dim": wl.head_dim, "feat_dim": wl.feat_dim,
            "input_dtype": wl.dtype, "input_bytes": in_bytes,
            "l2": (f"inputs ({in_bytes / 1e6:.0f} MB) larger than L2 (129 MB); no flush"
                   if in_bytes > 129e6 else
                   f"inputs ({in_bytes / 1e6:.1f} MB) fit in L2: steady-state, L2-warm figure")}


def prune_bytes_moved(wl):
    """Bytes of the fused prune under a "bytes moved" accounting:
    compulsory bytes (K, q and X read once, w~ written, X_S written and its rows
    read) plus the greedy's notional feature reads, k_b * N_b * d_v elements per
    request (the O(K N d_v) distance work of Sec. 3.4).  The notional reads never
    all cross HBM (rows are reused on chip and most pairs are skipped), so this is
    reported as an effective bandwidth, never as a roofline fraction."""
    e = wl.elem_bytes
    keep = int(wl.cu_keep[-1])
    comp = wl.k.nbytes + wl.q.nbytes + wl.x.nbytes + 4 * int(wl.cu_vis[-1]) + 2 * keep * wl.feat_dim * e
    greedy = sum(int(wl.cu_keep[b + 1] - wl.cu_keep[b]) * int(wl.cu_vis[b + 1] - wl.cu_vis[b])
                 for b in range(wl.batch)) * wl.feat_dim * e
    return comp, greedy


def select_compulsory_bytes(wl):
    """Bytes the selection cannot avoid: X and w~ read once, the kept indices written,
    the kept rows read and written (Eq. 12)."""
    keep = int(wl.cu_keep[-1])
    return (wl.x.nbytes + 4 * int(wl.cu_vis[-1]) + 4 * keep
            + 2 * keep * wl.feat_dim * wl.elem_bytes)


def greedy_flops(wl):
    """2 k_b N_b d_v: the distance contraction of Eq. 10 if every (token, centre) pair
    were evaluated (the paper's O(K N d_v), Sec. 3.4)."""
    return 2.0 * sum(int(wl.cu_keep[b + 1] - wl.cu_keep[b]) * int(wl.cu_vis[b + 1] - wl.cu_vis[b])
                     for b in range(wl.batch)) * wl.feat_dim


def score_bytes(wl):
    """Compulsory bytes of the scoring kernels: every key once, q once, w written."""
    return wl.k.nbytes + wl.q.nbytes + 4 * int(wl.cu_vis[-1])


class ClockSampler:
    """nvidia-smi clocks/throttle reasons sampled every 100 ms while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self):
        if self.proc is None or not self.path or not os.path.exists(self.path):
            return None
        rows = []
        for line in open(self.path):
            p = [s.strip() for s in line.split(",")]
            if len(p) < 9:
                continue
            try:
                rows.append(dict(sm=float(p[1]), smax=float(p[2]), power=float(p[3]),
                                 hw=p[5], hwt=p[6], swt=p[7], pcap=p[8]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return None
        reasons = set()
        for r in rows:
            for key, name in (("hw", "hw_slowdown"), ("hwt", "hw_thermal_slowdown"),
                              ("swt", "sw_thermal_slowdown"), ("pcap", "sw_power_cap")):
                if r[key].lower() == "active":
                    reasons.add(name)
        loaded = [r for r in rows if r["power"] > 0.25 * max(x["power"] for x in rows)] or rows
        return {"sm_mhz": statistics.median(r["sm"] for r in loaded),
                "sm_max_mhz": max(r["smax"] for r in rows), "reasons": sorted(reasons),
                "samples": len(rows), "power_w_max": max(r["power"] for r in rows)}


TRAFFIC_FILE = os.path.join(ROOT, "profiles", "select_kernel_traffic.txt")


def traffic_record(kernel_source: str, workload: str):
    """The ncu record of this workload: (DRAM bytes per launch, whether the kernel
    source still has the SHA-256 recorded with the counters), or None.
    The record is `key value` lines; a `workload` line starts each entry."""
    import hashlib
    rec, cur = {}, None
    try:
        with open(TRAFFIC_FILE) as f:
            for line in f:
                parts = line.split()
                if len(parts) != 2 or line.startswith("#"):
                    continue
                if parts[0] == "workload":
                    cur = rec.setdefault(parts[1], {})
                elif cur is not None:
                    cur[parts[0]] = parts[1]
        src = os.path.join(ROOT, "paper_2607_27952_gb300", "csrc", kernel_source)
        with open(src, "rb") as f:
            digest = hashlib.sha256(f.read()).hexdigest()
    except OSError:
        return None
    r = rec.get(workload)
    if not r or "dram_bytes_per_launch" not in r:
        return None
    return int(r["dram_bytes_per_launch"]), r.get("source_sha256") == digest


def measured_traffic(kernel_source: str, workload: str):
    """DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) recorded
    from an ncu capture of this workload, or None when the kernel source has changed
    since (its SHA-256 no longer matches the one recorded with the counters)."""
    r = traffic_record(kernel_source, workload)
    return r[0] if r is not None and r[1] else None


def peaks():
    try:
        with open(PEAKS_FILE) as f:
            return json.load(f), "measured"
    except (OSError, ValueError):
        return {"hbm_gbs": FALLBACK_HBM_GBS, "sm_max_mhz": 2070.0}, "fallback"


def oracle_request(oracle, wl, b, selector="greedy", rows=None, picks=None):
    """One request through the oracle: fp64 scores of the request (from its last
    query row, or from the query rows `rows` = (cu_rows, row_pos, q_rows) of another
    attention source), then the canonical-fp32 greedy (or Top-k), order restore and
    gather.  `picks` < k_b runs only the first `picks` greedy steps (the sequence
    does not depend on k, so this is a prefix of the request's own run).
    Returns (N_b, seconds of scoring, seconds of selection, picks run, k_b)."""
    v0, v1 = int(wl.cu_vis[b]), int(wl.cu_vis[b + 1])
    s0, s1 = int(wl.cu_seqlens[b]), int(wl.cu_seqlens[b + 1])
    kb = int(wl.cu_keep[b + 1] - wl.cu_keep[b])
    ks = kb if picks is None else min(kb, int(picks))
    kreq = np.ascontiguousarray(wl.k[:, s0:s1])
    t0 = time.perf_counter()
    if rows is None:
        w = oracle.scores(wl.q[b:b + 1], kreq, [0, s1 - s0], [int(wl.vis_start[b])], [0, v1 - v0],
                          num_kv_heads=wl.num_kv_heads)
    else:
        cu, pos, qr = rows
        r0, r1 = int(cu[b]), int(cu[b + 1])
        w = oracle.scores_rows(np.ascontiguousarray(qr[r0:r1]), kreq, [0, s1 - s0],
                               [int(wl.vis_start[b])], [0, v1 - v0], [0, r1 - r0], pos[r0:r1],
                               num_kv_heads=wl.num_kv_heads)
    w32 = w.astype(np.float32)
    t1 = time.perf_counter()
    if selector == "topk":
        ks = kb
        oracle.gather(wl.x[v0:v1], oracle.restore_order(oracle.select_topk(w32, kb)))
    else:
        oracle.prune_request(wl.x[v0:v1], w32, ks)
    t2 = time.perf_counter()
    return v1 - v0, t1 - t0, t2 - t1, ks, kb


def request_seconds(r) -> float:
    """A request's whole oracle time from a (possibly prefix) run: scoring plus the
    greedy scaled to k_b picks.  The canonical greedy makes one pass over the
    request's N_b x d_v features for the norms and one per later pick, so its time
    is linear in the picks through the origin."""
    _, t_sc, t_sel, ks, kb = r
    return t_sc + (t_sel * kb / ks if ks > 0 else t_sel)


def oracle_picks_for(oracle, wl, target_s, selector="greedy", rows=None):
    """Greedy picks per sampled request so that one request's oracle run takes about
    target_s seconds (whole requests when they fit)."""
    if selector == "topk":
        return None
    b = int(np.argmax(np.diff(wl.cu_keep) * np.diff(wl.cu_vis)))
    r = oracle_request(oracle, wl, b, selector, rows, picks=4)
    per_pick = r[2] / max(r[3], 1)
    full = r[1] + per_pick * r[4]
    if full <= target_s:
        return None
    return max(4, int((target_s - r[1]) / max(per_pick, 1e-9)))


def scoring_kernels(wl, cu_rows=None):
    """Kernels one scoring call launches: logits + tokens for the last row, and for
    one query row per request (last_scores_rows runs those kernels when G <= 8);
    stats, merge, probs and final for several rows."""
    if cu_rows is None:
        return 2
    single = int(cu_rows[-1]) == wl.batch and wl.num_q_heads // wl.num_kv_heads <= 8
    return 2 if single else 4


def host_threads():
    """Host cores this process may run on (the oracle's harness uses one thread each)."""
    try:
        return max(1, len(os.sched_getaffinity(0)))
    except AttributeError:
        return max(1, os.cpu_count() or 1)


def oracle_requests_parallel(oracle, wl, ids, threads, selector="greedy", rows=None,
                             picks=None):
    """Requests `ids` through the oracle, one request per thread on `threads` host
    threads (the oracle is reentrant and its C calls run without the GIL; the oracle
    itself is unchanged: the parallelism is over independent requests).  Returns the
    per-request results of oracle_request."""
    from concurrent.futures import ThreadPoolExecutor
    with ThreadPoolExecutor(max_workers=threads) as pool:
        return list(pool.map(lambda b: oracle_request(oracle, wl, b, selector, rows, picks), ids))


def sample_note(picks, wl):
    if picks is None:
        return "whole requests"
    return (f"the first {picks} greedy picks of each request (of k_b up to "
            f"{int(np.diff(wl.cu_keep).max())}), scaled to whole requests: the oracle's greedy "
            "time is linear in the picks (one pass over N_b x d_v per pick)")


def cpu_baseline(wl, budget_s=10.0, selector="greedy", rows=None):
    """The oracle as it stands on a bounded sample of the same batch: (i) one thread,
    requests in batch order until about budget_s seconds have passed; (ii) every
    host core, one request per thread, about budget_s seconds.  Requests whose whole
    oracle run would take more than a few seconds run a prefix of their greedy and
    are scaled to whole requests (request_seconds).  The all-cores figure is the
    baseline; the single-thread one rides along."""
    import oracle
    oracle.build()
    picks = oracle_picks_for(oracle, wl, 2.0, selector, rows)
    t0 = time.perf_counter()
    res = []
    for b in range(wl.batch):
        res.append(oracle_request(oracle, wl, b, selector, rows, picks))
        if time.perf_counter() - t0 > budget_s:
            break
    dt1 = time.perf_counter() - t0
    per_req = sum(request_seconds(r) for r in res) / len(res)
    single = {"value": 1.0 / per_req, "unit": UNIT, "cores": 1, "kind": "oracle",
              "sample": f"{len(res)} requests of the same batch in batch order ({selector}; "
                        f"{sample_note(picks, wl)}), single-threaded C oracle, {dt1:.1f} s"}
    threads = host_threads()
    sample_s = sum(r[1] + r[2] for r in res) / len(res)   # wall time of one sampled request
    n_par = max(threads, int(budget_s * threads / max(sample_s, 1e-9)))
    n_par = min(n_par, 8 * max(threads, wl.batch))
    n_par = (n_par + threads - 1) // threads * threads
    t0 = time.perf_counter()
    res = oracle_requests_parallel(oracle, wl, [i % wl.batch for i in range(n_par)], threads,
                                   selector, rows, picks)
    dt = time.perf_counter() - t0
    if picks is None:
        value = n_par / dt
    else:   # wall time of the sample scaled by the ratio of whole to sampled request time
        scale = sum(request_seconds(r) for r in res) / sum(r[1] + r[2] for r in res)
        value = n_par / (dt * scale)
    return {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
            "sample": f"{n_par} requests of the same batch in batch order, repeated ({selector}; "
                      f"{sample_note(picks, wl)}), one request per thread on {threads} host "
                      f"threads, {dt:.1f} s",
            "single_core": single}


def run_reference(args, rank, world):
    """--impl reference: the oracle, as it stands, on the host cores (rank 0 only).
    A step is one request per host core, run concurrently (requests of the batch in
    turn); long requests run a prefix of their greedy and are scaled to whole
    requests (request_seconds)."""
    if rank != 0:
        return
    wl = workload(args.budget, 0, args.workload)
    rows = None
    if args.source != "last":
        from workloads import query_rows
        rows = query_rows(wl, args.source, args.rows)
    import oracle
    oracle.build()
    threads = host_threads()
    total_steps = args.warmup + args.steps
    # about three minutes for the whole run at most
    picks = oracle_picks_for(oracle, wl, min(5.0, 150.0 / max(total_steps, 1)), args.selector, rows)

    def requests(first_step, nsteps):
        return [(i * threads + j) % wl.batch
                for i in range(first_step, first_step + nsteps) for j in range(threads)]

    # the steps' requests go through one pool without a barrier between steps, so
    # that no core waits for a step's slowest request
    oracle_requests_parallel(oracle, wl, requests(0, args.warmup), threads, args.selector, rows,
                             picks)
    t0 = time.perf_counter()
    res = oracle_requests_parallel(oracle, wl, requests(args.warmup, args.steps), threads,
                                   args.selector, rows, picks)
    dt = time.perf_counter() - t0
    scale = 1.0 if picks is None else (sum(request_seconds(r) for r in res)
                                       / sum(r[1] + r[2] for r in res))
    dt_whole = dt * scale
    value = args.steps * threads / dt_whole
    toks = sum(r[0] for r in res)
    sample = (f"{threads} requests of the {args.workload} batch per step, one per host thread, "
              f"requests in turn, steps not separated; {sample_note(picks, wl)}")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1000 * dt_whole / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64 scores / f32 selection",
            "data": WORKLOAD_DATA[args.workload],
            "config": workload_desc(wl, args.budget, args.workload)
                      | {"per_step": f"{threads} requests (oracle, one per host thread)",
                         "selector": args.selector, "source": args.source},
            "visual_tokens_scored_per_s": toks / dt_whole,
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": threads, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


PAPER_CONTEXT = {
    "source": "Table 2 (efficiency on ChartQA), Sec. 4.4",
    "hardware": "1x NVIDIA A800 80GB; edge model InternVL2-1B components with a Qwen2-0.5B "
                "proxy LLM; precision not stated",
    "agg_ms": {"value": 2.51, "note": "token-importance aggregation per inference at 62.5% and "
                                      "12.5% retention; whether it includes the greedy "
                                      "selection is not stated"},
    "edge_stage_ms": {"retain_62.5": 237.92, "retain_12.5": 236.43, "full_tokens": 118.55,
                      "note": "vision encoder + proxy prefill + selection"},
    "relation": "context only: one request of 256 visual tokens per image tile on another "
                "GPU; not the same metric or workload as this line",
}


def earlier_capture(kernel_source, workload, select_ms, hbm):
    """The ncu DRAM bytes recorded for this workload on an earlier source of the
    kernel, when the current source has none: reported beside the roofline, never
    used for its `traffic` or `frac`."""
    r = traffic_record(kernel_source, workload)
    if r is None or r[1]:
        return {}
    return {"traffic_earlier_source": {
        "dram_bytes_per_launch": r[0],
        "frac_at_this_time": r[0] / (select_ms / 1e3) / 1e9 / hbm,
        "note": "ncu capture of an earlier source of the kernel (the record's SHA-256 no "
                "longer matches); for context only"}}


def selection_roofline(wl, select_ms, hbm, bf16_peak, traffic):
    """Roofline of select_kernel against real resources.  `achieved` is the DRAM
    rate: bytes per launch recorded by ncu for this workload and kernel source
    (`traffic`), else the compulsory bytes (a lower bound on what crosses DRAM),
    over the event time; `tensor_frac` is the greedy's full distance contraction
    (2 k N d_v FLOPs) over the event time against the bf16 tensor peak."""
    sec = select_ms / 1e3
    comp = select_compulsory_bytes(wl)
    dram = traffic if traffic is not None else comp
    achieved = dram / sec / 1e9
    return {"bound": "hbm", "kernel": "select_kernel", "achieved": achieved, "peak": hbm,
            "unit": "GB/s", "frac": achieved / hbm, "traffic": traffic,
            "achieved_basis": ("ncu dram__bytes_read.sum + dram__bytes_write.sum per launch"
                               if traffic is not None else
                               "compulsory bytes (X, w~ read once; indices and kept rows); no "
                               "ncu record matches this kernel source"),
            "compulsory_bytes": comp, "compulsory_frac": comp / sec / 1e9 / hbm,
            "tensor_frac": greedy_flops(wl) / sec / 1e12 / bf16_peak,
            "tensor_peak_TFLOPs": bf16_peak}


def dev_tensor(a, dev):
    import torch
    if a.dtype == np.uint16:
        return torch.from_numpy(a.view(np.int16)).to(dev).view(torch.bfloat16)
    return torch.from_numpy(a).to(dev)


def problem_for(last, wl):
    return last.Problem(batch=wl.batch, num_layers=wl.num_layers, num_q_heads=wl.num_q_heads,
                        num_kv_heads=wl.num_kv_heads, head_dim=wl.head_dim, feat_dim=wl.feat_dim,
                        dtype=wl.dtype, cu_seqlens=wl.cu_seqlens, vis_start=wl.vis_start,
                        cu_vis=wl.cu_vis, cu_keep=wl.cu_keep)


def measure_config(name, budget, rank, dev, last, seconds, hbm, bf16_peak):
    """One workload preset timed like the headline (resident inputs, CUDA events on
    the launching stream around last_scores and last_select), with as many steps as
    fill about `seconds` of device time (at least 3, after 2 warm-up steps)."""
    import torch
    wl = workload(budget, rank, name)
    prob = problem_for(last, wl)
    q, k, x = dev_tensor(wl.q, dev), dev_tensor(wl.k, dev), dev_tensor(wl.x, dev)
    nvis, nkeep = int(wl.cu_vis[-1]), int(wl.cu_keep[-1])
    w = torch.empty(nvis, dtype=torch.float32, device=dev)
    idx = torch.empty(nkeep, dtype=torch.int32, device=dev)
    xs = torch.empty((nkeep, wl.feat_dim), dtype=x.dtype, device=dev)
    ws = last.workspace(prob, dev)
    stream = torch.cuda.current_stream(dev)
    for _ in range(2):
        last.last_scores(prob, q, k, w, ws, stream)
        last.last_select(prob, w, x, idx, ws, stream, x_out=xs)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    last.last_scores(prob, q, k, w, ws, stream)
    last.last_select(prob, w, x, idx, ws, stream, x_out=xs)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    steps = int(max(3, min(500, seconds * 1e3 / max(e0.elapsed_time(e1), 1e-3))))
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(steps)]
    torch.cuda.synchronize(dev)
    for i in range(steps):
        ev[i][0].record(stream)
        last.last_scores(prob, q, k, w, ws, stream)
        ev[i][1].record(stream)
        last.last_select(prob, w, x, idx, ws, stream, x_out=xs)
        ev[i][2].record(stream)
    torch.cuda.synchronize(dev)
    last.last_poll(ws, stream)
    total = ev[0][0].elapsed_time(ev[-1][2])
    sc = statistics.mean(e[0].elapsed_time(e[1]) for e in ev)
    se = statistics.mean(e[1].elapsed_time(e[2]) for e in ev)
    key = f"{name}-{budget}"
    traffic = measured_traffic("select_impl.cuh", key)
    rl = selection_roofline(wl, se, hbm, bf16_peak, traffic)
    sc_gbs = score_bytes(wl) / (sc / 1e3) / 1e9
    out = {"workload": workload_desc(wl, budget, name)["workload"], "dtype": workload_dtype(wl),
           "steps": steps, "requests_per_s": wl.batch * steps / (total / 1e3),
           "ms_per_step": total / steps, "scores_ms": sc, "select_ms": se,
           "visual_tokens_scored_per_s": nvis / (sc / 1e3),
           "scores_hbm_frac": sc_gbs / hbm,
           "select_dram_frac": rl["frac"] if traffic is not None else None,
           "select_compulsory_frac": rl["compulsory_frac"],
           "select_tensor_frac": rl["tensor_frac"], "select_dram_bytes": traffic}
    out |= earlier_capture("select_impl.cuh", key, se, hbm)
    del q, k, x, w, idx, xs, ws
    torch.cuda.empty_cache()
    return out


PER_CONFIG = (("c1", "default"), ("c2", "mixed"), ("c3", "default"), ("c4", "default"),
              ("c5", "5"), ("c5", "12.5"), ("c5", "25"))


def main():
    args = parse()
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    local = int(os.environ.get("LOCAL_RANK", 0))
    if args.impl == "reference":
        run_reference(args, rank, world)
        return

    import torch
    import paper_2607_27952_gb300 as last

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    last.load_library()

    wl = workload(args.budget, rank, args.workload)
    prob = problem_for(last, wl)
    q, k, x = dev_tensor(wl.q, dev), dev_tensor(wl.k, dev), dev_tensor(wl.x, dev)
    nvis, nkeep = int(wl.cu_vis[-1]), int(wl.cu_keep[-1])
    w = torch.empty(nvis, dtype=torch.float32, device=dev)
    idx = torch.empty(nkeep, dtype=torch.int32, device=dev)
    xs = torch.empty((nkeep, wl.feat_dim), dtype=x.dtype, device=dev)
    ws = last.workspace(prob, dev)
    stream = torch.cuda.current_stream(dev)

    topk = args.selector == "topk"
    rows = rows_host = None
    if args.source != "last":
        from workloads import query_rows
        rows_host = query_rows(wl, args.source, args.rows)
        rows = last.QueryRows(rows_host[0], rows_host[1])
        q_rows = dev_tensor(rows_host[2], dev)
        ws_rows = last.rows_workspace(prob, rows, dev)

    def score():
        if rows is None:
            last.last_scores(prob, q, k, w, ws, stream)
        else:
            last.last_scores_rows(prob, rows, q_rows, k, w, ws_rows, stream)

    def select():
        if topk:
            last.last_select_topk(prob, w, idx, ws, stream, x=x, x_out=xs)
        else:
            last.last_select(prob, w, x, idx, ws, stream, x_out=xs)

    def step():
        score()
        select()

    for _ in range(args.warmup):
        step()
    last.last_poll(ws, stream)

    def barrier():
        if world > 1:
            torch.distributed.barrier()

    K = args.steps
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(K)]
    with ClockSampler(local) as clk:
        barrier()
        torch.cuda.synchronize(dev)
        for i in range(K):
            ev[i][0].record(stream)
            score()
            ev[i][1].record(stream)
            select()
            ev[i][2].record(stream)
        torch.cuda.synchronize(dev)
        barrier()
    clocks = clk.summary()
    last.last_poll(ws, stream)
    total_ms = ev[0][0].elapsed_time(ev[-1][2])
    scores_all = [e[0].elapsed_time(e[1]) for e in ev]
    select_all = [e[1].elapsed_time(e[2]) for e in ev]
    scores_ms, select_ms = statistics.mean(scores_all), statistics.mean(select_all)
    total_ms, reqs, toks = combine_over_ranks(total_ms, wl.batch * K, nvis * K, device=dev)
    value = reqs / (total_ms / 1e3)
    tokens_per_s = toks / (scores_ms * K / 1e3)   # visual tokens scored per second of scoring

    pk, pk_kind = peaks()
    hbm = float(pk.get("hbm_gbs", FALLBACK_HBM_GBS))
    bf16_peak = float(pk.get("bf16_tflops", 1900.0))
    sc_bytes = score_bytes(wl) if rows is None else (
        wl.k.nbytes + rows_host[2].nbytes + 4 * int(wl.cu_vis[-1]))
    sc_gbs = sc_bytes / (scores_ms / 1e3) / 1e9

    e2e = None
    if not args.no_e2e:
        if rows is None and not topk:
            e2e = measure_e2e_host(args, wl, prob, dev, last)
        else:
            e2e = measure_e2e(args, wl, prob, dev, stream, last, q, k, x,
                              None if rows is None else (rows, rows_host[2], q_rows, ws_rows))

    comp, greedy = prune_bytes_moved(wl)
    if topk:   # Top-k reads only the kept rows of X, and has no greedy reads
        comp, greedy = comp - wl.x.nbytes, 0
    key = f"{args.workload}-{args.budget}"
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": total_ms / K, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": workload_dtype(wl),
        "data": WORKLOAD_DATA[args.workload],
        "config": workload_desc(wl, args.budget, args.workload) | {"parallelism": f"replicas x{world}"},
        "visual_tokens_scored_per_s": tokens_per_s,
        # per step: scoring (logits + tokens, or the four multi-row passes) and the
        # selection (select_kernel, or topk_kernel + gather_kernel)
        "gpu_launches": (scoring_kernels(wl, None if rows is None else rows_host[0]) +
                         (2 if topk else 1)) * K,
        "kernels": {"scores_ms": scores_ms, "select_ms": select_ms,
                    "scores_ms_median": statistics.median(scores_all),
                    "select_ms_median": statistics.median(select_all),
                    "scores_GBps": sc_gbs, "scores_hbm_frac": sc_gbs / hbm},
        "roofline": selection_roofline(wl, select_ms, hbm, bf16_peak,
                                       measured_traffic("select_impl.cuh", key))
                    | {"peak_note": f"{pk_kind} HBM copy bandwidth (of {pk_kind}); tensor peak: "
                                    f"{pk_kind} cuBLAS bf16 burst"}
                    | earlier_capture("select_impl.cuh", key, select_ms, hbm),
        "clocks": clocks,
        "prune_bytes_moved": {"compulsory_bytes": comp, "greedy_feature_bytes": greedy,
                              "compulsory_frac": comp / (total_ms / K / 1e3) / 1e9 / hbm,
                              "greedy_effective_TBps": (comp + greedy) / (total_ms / K / 1e3) / 1e12,
                              "note": "compulsory_frac = the step's unavoidable HBM bytes (K, q, "
                                      "X once, w~, kept rows) over the step time, of measured "
                                      "HBM; greedy_effective_TBps values the greedy's notional "
                                      "k N d_v feature reads at HBM rate (bytes-moved accounting) "
                                      "and is not a fraction of any roof: most of those pairs "
                                      "are skipped or served on chip"},
        "paper_context": PAPER_CONTEXT,
    }
    if topk:
        # the selection is a few microseconds; the scoring pair dominates the step
        line["config"]["selector"] = "topk (Table 5)"
        line["roofline"] = {"bound": "hbm", "kernel": "score_logits_kernel+score_tokens_kernel",
                            "achieved": sc_gbs, "peak": hbm, "unit": "GB/s", "frac": sc_gbs / hbm,
                            "traffic": None,
                            "peak_note": f"{pk_kind} HBM copy bandwidth; achieved = compulsory "
                                         "scoring bytes / event time of last_scores"}
        line["kernels"]["topk_gather_ms"] = line["kernels"].pop("select_ms")
        line["kernels"]["topk_gather_ms_median"] = line["kernels"].pop("select_ms_median")
    if rows is not None:
        # Table 4's attention source: the logits are a bf16 tensor-core contraction of
        # every key with the request's query rows
        cu = rows_host[0]
        flops = 2.0 * sum(int(wl.cu_seqlens[b + 1] - wl.cu_seqlens[b]) * int(cu[b + 1] - cu[b])
                          for b in range(wl.batch)) * wl.num_q_heads * wl.head_dim * wl.num_layers
        line["config"]["source"] = f"{args.source} ({int(cu[-1])} query rows, Table 4)"
        line["kernels"]["scores_tensor_TFLOPs"] = flops / (scores_ms / 1e3) / 1e12
        if topk and scoring_kernels(wl, cu) == 4:
            line["roofline"]["kernel"] = ("rows_stats_kernel+rows_merge_kernel+"
                                          "rows_probs_kernel+rows_final_kernel")
    if e2e is not None:
        line["e2e"] = e2e
    if rank == 0 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl, selector=args.selector, rows=rows_host)
    if not args.no_per_config and rows is None and not topk:
        del q, k, x, w, idx, xs, ws
        torch.cuda.empty_cache()
        per = {}
        for name, bud in PER_CONFIG:
            if name == args.workload and bud == args.budget:
                continue
            per[f"{name}-{bud}"] = measure_config(name, bud, rank, dev, last,
                                                  args.per_config_seconds, hbm, bf16_peak)
        line["per_config"] = per
        line["gpu_launches"] += 3 * sum(v["steps"] for v in per.values())
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def measure_e2e_host(args, wl, prob, dev, last):
    """The same metric through the user call last_prune_host on pinned host buffers:
    every step copies q, K and X to the device, prunes, and copies the kept indices and
    rows back.  Steps alternate between two workspaces on two streams, as a server
    would run them, so one step's copies overlap the previous step's kernels; the
    timed region spans every step's copies and kernels."""
    import torch
    def pin(a):
        if a.dtype == np.uint16:
            return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).pin_memory()
        return torch.from_numpy(a).pin_memory()
    qh, kh, xh = pin(wl.q), pin(wl.k), pin(wl.x)
    nkeep = int(wl.cu_keep[-1])
    streams = [torch.cuda.Stream(dev), torch.cuda.Stream(dev)]
    wss = [last.host_workspace(prob, dev) for _ in streams]
    outs = [(torch.empty(nkeep, dtype=torch.int32).pin_memory(),
             torch.empty((nkeep, wl.feat_dim), dtype=xh.dtype).pin_memory()) for _ in streams]

    def step(i):
        j = i % 2
        last.last_prune_host(prob, qh, kh, xh, None, outs[j][0], outs[j][1], wss[j], streams[j])

    for i in range(max(2, args.warmup // 2)):
        step(i)
    torch.cuda.synchronize(dev)
    steps = max(4, args.steps // 2)
    e0, e1, join = (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True),
                    torch.cuda.Event())
    e0.record(streams[0])
    streams[1].wait_event(e0)
    for i in range(steps):
        step(i)
    join.record(streams[1])
    streams[0].wait_event(join)
    e1.record(streams[0])
    torch.cuda.synchronize(dev)
    for ws in wss:
        last.last_poll(ws, streams[0])
    ms = e0.elapsed_time(e1)
    h2d = int(qh.numel() + kh.numel() + xh.numel()) * xh.element_size()
    d2h = int(outs[0][0].numel() * 4 + outs[0][1].numel() * outs[0][1].element_size())
    return {"value": wl.batch * steps / (ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "steps": steps,
            "call": "last_prune_host, pinned host buffers, two streams and workspaces alternating"}


def measure_e2e(args, wl, prob, dev, stream, last, q_d, k_d, x_d, rows=None):
    """The same metric with host buffers for the variants: each step copies q (or the
    query rows), K and X from pinned host memory, scores and selects through the
    variant's calls, and reads back the kept indices and rows, on one stream."""
    import torch
    def pin(a):
        if a.dtype == np.uint16:
            return torch.from_numpy(a.view(np.int16)).view(torch.bfloat16).pin_memory()
        return torch.from_numpy(a).pin_memory()
    qh, kh, xh = pin(wl.q if rows is None else rows[1]), pin(wl.k), pin(wl.x)
    if rows is not None:
        q_d = rows[2]
    nkeep = int(wl.cu_keep[-1])
    idx_h = torch.empty(nkeep, dtype=torch.int32).pin_memory()
    xs_h = torch.empty((nkeep, wl.feat_dim), dtype=xh.dtype).pin_memory()
    idx_d = torch.empty(nkeep, dtype=torch.int32, device=dev)
    xs_d = torch.empty((nkeep, wl.feat_dim), dtype=xh.dtype, device=dev)
    ws = last.workspace(prob, dev)

    w_d = torch.empty(int(wl.cu_vis[-1]), dtype=torch.float32, device=dev)

    def step():
        q_d.copy_(qh, non_blocking=True)
        k_d.copy_(kh, non_blocking=True)
        x_d.copy_(xh, non_blocking=True)
        if rows is not None:
            last.last_scores_rows(prob, rows[0], q_d, k_d, w_d, rows[3], stream)
            if args.selector == "topk":
                last.last_select_topk(prob, w_d, idx_d, ws, stream, x=x_d, x_out=xs_d)
            else:
                last.last_select(prob, w_d, x_d, idx_d, ws, stream, x_out=xs_d)
        else:
            last.last_scores(prob, q_d, k_d, w_d, ws, stream)
            last.last_select_topk(prob, w_d, idx_d, ws, stream, x=x_d, x_out=xs_d)
        idx_h.copy_(idx_d, non_blocking=True)
        xs_h.copy_(xs_d, non_blocking=True)

    for _ in range(max(1, args.warmup // 2)):
        step()
    torch.cuda.synchronize(dev)
    steps = max(3, args.steps // 2)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize(dev)
    ms = e0.elapsed_time(e1)
    h2d = int(qh.numel() + kh.numel() + xh.numel()) * xh.element_size()
    d2h = int(idx_h.numel() * 4 + xs_h.numel() * xs_h.element_size())
    return {"value": wl.batch * steps / (ms / 1e3), "unit": UNIT, "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "steps": steps}


if __name__ == "__main__":
    main()
