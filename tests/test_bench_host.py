"""Host-side logic of the benchmark on the CPU: the clock summary read from
nvidia-smi samples (median SM clock, throttle reasons), the traffic figure keyed
to the kernel sources' hash, and the whole-job throughput."""
import os
import shutil

import pytest

import bench


def _clocks_from(tmp_path, lines):
    p = tmp_path / "clocks.csv"
    p.write_text("\n".join(lines) + "\n")
    c = bench.Clocks(0)
    c.path = str(p)
    return c.summary()


def test_clock_summary_median_max_and_reasons(tmp_path):
    rows = [
        "0, 2070, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active",
        "0, 1980, 2070, 1395.0, 0x4, Not Active, Not Active, Not Active, Active",
        "0, 2070, 2070, 1010.0, 0x0, Not Active, Not Active, Not Active, Not Active",
        "garbage line",
        "0, [N/A], 2070, 0, 0x0, Not Active, Not Active, Not Active, Not Active",
    ]
    s = _clocks_from(tmp_path, rows)
    assert s["samples"] == 3 and s["sm_mhz"] == 2070.0 and s["sm_max_mhz"] == 2070.0
    assert s["reasons"] == ["sw_power_cap"]
    assert not os.path.exists(tmp_path / "clocks.csv")  # the sample file is removed


def test_clock_summary_flags_hardware_slowdown(tmp_path):
    s = _clocks_from(tmp_path, ["0, 1500, 2070, 1300, 0x8, Active, Not Active, Active, Not Active"])
    assert s["reasons"] == ["hw_slowdown", "sw_thermal_slowdown"]


def test_clock_summary_without_samples(tmp_path):
    assert _clocks_from(tmp_path, ["only noise"]) is None


def test_stored_traffic_is_keyed_to_the_kernel_sources(tmp_path, monkeypatch):
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "ncu_traffic.txt").write_text("dense_store_x abc123 51022336\nother def 1\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    monkeypatch.setattr(bench, "kernel_source_hash", lambda: "abc123")
    assert bench.stored_traffic("dense_store_x") == 51022336.0
    assert bench.stored_traffic("missing") is None
    monkeypatch.setattr(bench, "kernel_source_hash", lambda: "changed")
    assert bench.stored_traffic("dense_store_x") is None  # stale once the sources change


def test_kernel_source_hash_covers_every_library_source(tmp_path, monkeypatch):
    # a stored ncu traffic figure stays valid only while no source of the
    # library changed: the hash covers every file under csrc/ and the C header
    h = bench.kernel_source_hash()
    assert len(h) == 16 and h == bench.kernel_source_hash()
    src = os.path.join(bench.ROOT, "paper_2606_02963_gb300", "csrc")
    dst = tmp_path / "paper_2606_02963_gb300" / "csrc"
    shutil.copytree(src, dst, ignore=shutil.ignore_patterns("*.o", "*.so"))
    (tmp_path / "include").mkdir()
    shutil.copy(os.path.join(bench.ROOT, "include", "kf.h"), tmp_path / "include" / "kf.h")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.kernel_source_hash() == h
    for f in sorted(os.listdir(dst)) + ["../../include/kf.h"]:
        fp = dst / f
        old = fp.read_bytes()
        fp.write_bytes(old + b"\n")
        assert bench.kernel_source_hash() != h, f
        fp.write_bytes(old)
    assert bench.kernel_source_hash() == h


def test_whole_job_throughput_and_single_rank_max():
    assert bench.whole_job_tflops(2e12, 1.0, 1) == pytest.approx(2000.0)
    assert bench.whole_job_tflops(2e12, 1.0, 4) == pytest.approx(8000.0)
    assert bench.reduce_max_over_ranks([1.0, 2.0], None, 1) == [1.0, 2.0]
