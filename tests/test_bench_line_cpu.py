"""CPU: the host logic of the benchmark's JSON line -- the clock record
(samples reduced over the window of the timed steps only) and the figures
derived from one device-resident run (step GB/s, phase GB/s, the roofline of
the dominant phase) -- on synthetic inputs with hand-computed results."""
import argparse

import pytest

import bench


def _sampler(samples, marks):
    c = bench.ClockSampler(0)
    c.source = "test"
    c.samples = list(samples)
    c.marks = dict(marks)
    return c


def test_clock_summary_covers_the_timed_window_only():
    # (host time, SM MHz, max MHz, power W, active reasons)
    samples = [(0.5, 1200.0, 2070.0, 150.0, []),                 # warm-up
               (1.1, 2070.0, 2070.0, 900.0, []),
               (1.2, 2040.0, 2070.0, 1100.0, ["sw_power_cap"]),
               (1.3, 2070.0, 2070.0, 1000.0, []),
               (2.5, 900.0, 2070.0, 200.0, ["hw_slowdown"])]     # after the timed steps
    c = _sampler(samples, {"start": 0.0, "timed_start": 1.0, "timed_end": 2.0, "end": 3.0})
    s = c.summary("timed_start", "timed_end")
    assert s["samples"] == 3
    assert s["sm_mhz"] == 2070.0 and s["sm_min_mhz"] == 2040.0 and s["sm_max_mhz"] == 2070.0
    assert s["reasons"] == ["sw_power_cap"]
    assert s["power_w_max"] == 1100.0
    whole = c.summary()
    assert whole["samples"] == 5 and whole["reasons"] == ["hw_slowdown", "sw_power_cap"]


def test_clock_summary_without_samples_says_why():
    c = _sampler([], {"timed_start": 1.0, "timed_end": 2.0})
    c.error = "nvml: no library"
    s = c.summary("timed_start", "timed_end")
    assert s["samples"] == 0 and s["sm_mhz"] is None and s["reasons"] == ["unavailable"]
    assert s["error"] == "nvml: no library"


def _run(n_elem, total_ms, phase_ms, ntensors=1):
    return dict(n_elem=n_elem, esz=2, total_ms=total_ms, phase_ms=phase_ms, phase_reps=8,
                clocks={"samples": 3}, l2_flushed=False, l2_resident_ms=None, ntensors=ntensors,
                grouped=False, launches_per_step=5)


def test_device_line_figures():
    case = bench.Case()                                # 2 GiB activations, NVFP4
    assert case.workload == "act_262144x4096" and case.fmt == "nvfp4"
    n = 262144 * 4096
    K = 10
    # per step: alpha 0.3 ms, fwd 0.75, bwd 1.2, pack 0.55; whole step 2.9 ms
    r = _run(n, 2.9 * K, {"alpha": 0.3 * K, "fwd": 0.75 * K, "bwd": 1.2 * K, "pack": 0.55 * K})
    args = argparse.Namespace(steps=K, warmup=5, staged=False)
    out = bench.device_line(case, r, args, 1, True)
    assert out["value"] == pytest.approx(n * 17.5625 / 2.9e-3 / 1e9, rel=1e-6)
    assert out["ms_per_step"] == pytest.approx(2.9)
    assert out["phase_gbs"]["bwd"] == pytest.approx(n * 7.5 / 1.2e-3 / 1e9, rel=1e-6)
    assert out["phase_gbs"]["alpha"] == pytest.approx(n * 2.0 / 0.3e-3 / 1e9, rel=1e-6)
    rf = out["roofline"]
    assert rf["kernel"] == "fq_bwd" and rf["bound"] == "hbm"
    assert rf["algorithmic_bytes"] == round(n * 7.5)
    assert rf["frac"] == pytest.approx(rf["achieved"] / rf["peak"], abs=1e-4)
    assert out["dtype"] == "f32" and out["config"]["io_dtype"] == "bf16"
    assert out["gpu_launches"] == K * 5
    assert out["config"]["workload"] == "act_262144x4096"


def test_traffic_only_on_matching_sources(monkeypatch):
    case = bench.Case()
    n = 1 << 20
    r = _run(n, 10.0, {"alpha": 1.0, "fwd": 2.0, "bwd": 4.0, "pack": 3.0})
    args = argparse.Namespace(steps=1, warmup=5, staged=False)
    key = (case.workload, case.fmt, "bwd")
    monkeypatch.setitem(bench.TRAFFIC, key, {"sources": "nope", "bytes_per_elem": 7.0})
    assert bench.device_line(case, r, args, 1, True)["roofline"]["traffic"] is None
    monkeypatch.setitem(bench.TRAFFIC, key, {"sources": bench.kernel_sources_sha(), "bytes_per_elem": 7.0})
    assert bench.device_line(case, r, args, 1, True)["roofline"]["traffic"] == 7 * n
    # never for a non-default case
    assert bench.device_line(case, r, args, 1, False)["roofline"]["traffic"] is None
