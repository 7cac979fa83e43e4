"""Host logic of bench.py that needs no GPU: the clock and throttle-reason
sampler that runs beside the timed region, driven by a fake nvidia-smi."""
import os
import stat
import sys
import time

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _fake_smi(tmp_path, lines, period=0.03):
    """An executable named nvidia-smi that prints the given CSV rows in a loop,
    one every `period` seconds, as `nvidia-smi --query-gpu=... -lms` does."""
    body = "\n".join(f"    echo '{ln}'; sleep {period}" for ln in lines)
    script = tmp_path / "nvidia-smi"
    script.write_text("#!/bin/sh\nwhile true; do\n" + body + "\ndone\n")
    script.chmod(script.stat().st_mode | stat.S_IXUSR | stat.S_IXGRP | stat.S_IXOTH)
    return str(tmp_path)


@pytest.fixture
def bench_mod():
    if ROOT not in sys.path:
        sys.path.insert(0, ROOT)
    import bench
    return bench


def _sample(bench, monkeypatch, path_dir, seconds=0.4):
    monkeypatch.setenv("PATH", path_dir + os.pathsep + os.environ.get("PATH", ""))
    s = bench.ClockSampler(0)
    s.start()
    time.sleep(seconds)
    return s.stop()


def test_clock_sampler_reports_median_clock_and_power_cap(bench_mod, monkeypatch, tmp_path):
    rows = ["0, 1490, 2070, 1390.00, 0x0000000000000004, Not Active, Not Active, Not Active, Active",
            "0, 1510, 2070, 1395.00, 0x0000000000000004, Not Active, Not Active, Not Active, Active"]
    r = _sample(bench_mod, monkeypatch, _fake_smi(tmp_path, rows))
    assert r["samples"] >= 3
    assert 1490.0 <= r["sm_mhz"] <= 1510.0
    assert r["sm_max_mhz"] == 2070.0
    assert r["reasons"] == ["sw_power_cap"]


def test_clock_sampler_flags_thermal_and_hardware_slowdown(bench_mod, monkeypatch, tmp_path):
    rows = ["0, 900, 2070, 800.00, 0x0000000000000048, Active, Not Active, Not Active, Not Active",
            "0, 905, 2070, 805.00, 0x0000000000000048, Not Active, Active, Active, Not Active"]
    r = _sample(bench_mod, monkeypatch, _fake_smi(tmp_path, rows))
    assert r["reasons"] == ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"]


def test_clock_sampler_without_nvidia_smi_reports_nothing(bench_mod, monkeypatch, tmp_path):
    # An empty directory first on PATH and nothing else: the sampler cannot
    # start and the timed region goes on without clock records.
    monkeypatch.setenv("PATH", str(tmp_path))
    s = bench_mod.ClockSampler(0)
    s.start()
    assert s.stop() is None


def test_cpu_model_names_the_host(bench_mod):
    import platform
    name = bench_mod.cpu_model()
    assert isinstance(name, str) and platform.machine() in name
