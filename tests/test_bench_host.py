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


def test_gpus_flag_must_match_world_size(bench_mod, monkeypatch):
    """Under torchrun, --gpus N must equal WORLD_SIZE; without torchrun, N = 1
    runs in this process."""
    monkeypatch.setenv("WORLD_SIZE", "1")
    assert bench_mod.main(["--gpus", "2", "--steps", "1"]) == 2
    args = type("A", (), {"gpus": 1})()
    monkeypatch.delenv("WORLD_SIZE")
    assert bench_mod.launch_ranks(args, []) is None


def _fake_stats(**over):
    st = dict(ms_gemm_up=10.0, flops_gemm_up=1.5e13, n_gemm_up=2, bytes_gemm_up=4e9,
              ms_gemm_down=5.0, flops_gemm_down=7.5e12, n_gemm_down=2, bytes_gemm_down=2e9,
              gemm_flops=2.25e13, bytes_expert_weights=3e9, layer_tokens=2000, layer_calls=2,
              flops_attn=0.0, flops_attn_gemm=0.0)
    st.update(over)
    return st


def test_rooflines_use_burst_peak_and_report_sustained(bench_mod):
    from paper_2608_00573_gb300 import workload as W
    cfg = W.CONFIGS["mixtral"].replace(N=2, T=1000)
    peaks = dict(hbm=6790.7, bf16=1889.4, bf16_sus=1687.0, source="measured")
    roof, fwd = bench_mod.rooflines(cfg, _fake_stats(), 1, 20.0, peaks, None)
    assert roof["kernel"] == "grouped_gemm_gate_up" and roof["bound"] == "tensor"
    assert abs(roof["achieved"] - 1500.0) < 1e-9                       # 1.5e13 FLOP in 10 ms
    assert abs(roof["frac"] - 1500.0 / 1889.4) < 1e-12
    assert abs(roof["frac_sustained"] - 1500.0 / 1687.0) < 1e-12
    # forward: F_alg = GEMM FLOPs + router/exit-head dot products of the live tokens
    f = 2.25e13 + 2000 * 2.0 * cfg.d * (cfg.E + cfg.C)
    b = 3e9 + 2 * 2.0 * cfg.d * (cfg.E + cfg.C + 1) + 2000 * (4.0 * cfg.d + bench_mod.STATE_BYTES_PER_TOKEN_LAYER)
    assert abs(fwd["flops_per_forward"] - f) < 1 and abs(fwd["bytes_per_forward"] - b) < 1
    t = max(f / 1889.4e12, b / 6790.7e9) * 1e3
    assert abs(fwd["frac"] - t / 20.0) < 1e-12
    assert fwd["frac_sustained"] > fwd["frac"]


def test_rooflines_hbm_bound_for_decode_sized_launches(bench_mod):
    from paper_2608_00573_gb300 import workload as W
    cfg = W.CONFIGS["mixtral_decode"].replace(T=1)
    peaks = dict(hbm=6790.7, bf16=1889.4, bf16_sus=1687.0, source="measured")
    st = _fake_stats(ms_gemm_up=1.0, flops_gemm_up=1e9, bytes_gemm_up=3.7e9, gemm_flops=1.5e9,
                     ms_gemm_down=0.5, flops_gemm_down=5e8, bytes_gemm_down=1.9e9, layer_tokens=20,
                     bytes_expert_weights=5.6e9)
    roof, fwd = bench_mod.rooflines(cfg, st, 1, 2.0, peaks, None)
    assert roof["bound"] == "hbm" and roof["unit"] == "GB/s"
    assert abs(roof["achieved"] - 3700.0) < 1e-9
    assert fwd["bound"] == "hbm"


def test_both_arms_print_the_same_config(bench_mod):
    from paper_2608_00573_gb300 import workload as W
    cfg = W.CONFIGS["mixtral"]
    a = bench_mod.config_dict(cfg, 1)
    assert a == bench_mod.config_dict(cfg, 1)
    assert a["workload"] == "mixtral" and a["T"] == 16384 and a["parallelism"] == "replicas1"
