"""bench.py's use of recorded ncu DRAM traffic.

A capture counts for the roofline only while the kernel source still has the
SHA-256 recorded with it; a capture of an earlier source is reported beside the
roofline (`traffic_earlier_source`) and never as its `traffic` or `frac`.
"""
import hashlib
import os

import bench


def _record(path, workload, sha, nbytes):
    with open(path, "w") as f:
        f.write("# header lines are ignored\n")
        f.write(f"workload {workload}\nsource_sha256 {sha}\ndram_bytes_per_launch {nbytes}\n")


def _current_sha():
    src = os.path.join(bench.ROOT, "paper_2607_27952_gb300", "csrc", "select_impl.cuh")
    with open(src, "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()


def test_matching_source_is_used(tmp_path, monkeypatch):
    path = tmp_path / "traffic.txt"
    _record(path, "c5-12.5", _current_sha(), 123456789)
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(path))
    assert bench.measured_traffic("select_impl.cuh", "c5-12.5") == 123456789
    assert bench.earlier_capture("select_impl.cuh", "c5-12.5", 10.0, 6780.7) == {}
    assert bench.measured_traffic("select_impl.cuh", "c2-mixed") is None


def test_changed_source_is_only_context(tmp_path, monkeypatch):
    path = tmp_path / "traffic.txt"
    _record(path, "c5-12.5", "0" * 64, 2_000_000_000)
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(path))
    assert bench.measured_traffic("select_impl.cuh", "c5-12.5") is None
    ctx = bench.earlier_capture("select_impl.cuh", "c5-12.5", 10.0, 6780.7)
    e = ctx["traffic_earlier_source"]
    assert e["dram_bytes_per_launch"] == 2_000_000_000
    assert abs(e["frac_at_this_time"] - 2e9 / 1e-2 / 1e9 / 6780.7) < 1e-12


def test_missing_record_gives_nothing(tmp_path, monkeypatch):
    monkeypatch.setattr(bench, "TRAFFIC_FILE", str(tmp_path / "absent.txt"))
    assert bench.measured_traffic("select_impl.cuh", "c5-12.5") is None
    assert bench.earlier_capture("select_impl.cuh", "c5-12.5", 10.0, 6780.7) == {}
