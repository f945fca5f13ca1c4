"""Host-side roofline logic of bench.py (no GPU): the whole-step roofline and the source-hash gate on the
DRAM traffic figures."""
import pytest

import bench


def test_step_roofline_is_flops_over_tensor_peak_plus_bytes_over_hbm():
    pk, _ = bench.peaks()
    steps = 4
    # one step's worth: 2 ms of tensor work and 1 ms of memory work at the measured peaks
    prof = {
        "gemm_layer": {"flops": 2e-3 * pk["bf16_tflops_sustained"] * 1e12 * steps, "bytes": 1.0, "ms": 9.0, "launches": 8},
        "local_loss": {"flops": 0.0, "bytes": 1e-3 * pk["hbm_gbs"] * 1e9 * steps, "ms": 5.0, "launches": 4},
        "adamw": {"flops": 0.0, "bytes": 0.0, "ms": 0.0, "launches": 0},
    }
    r = bench.step_roofline(prof, steps, ms_per_step=6.0)
    assert r["tensor_ms"] == pytest.approx(2.0)
    assert r["hbm_ms"] == pytest.approx(1.0)   # bytes of tensor classes are not counted twice
    assert r["ideal_ms"] == pytest.approx(3.0)
    assert r["frac"] == pytest.approx(0.5)


def test_traffic_figures_are_tied_to_the_kernel_sources(monkeypatch):
    sha = bench.sources_sha(bench.GEMM_SOURCES)
    monkeypatch.setitem(bench.TRAFFIC, "w", {"gemm_layer": {"sources": bench.GEMM_SOURCES, "sha256": sha,
                                                           "bytes_per_launch": 123.0}})
    assert bench.measured_traffic("gemm_layer", "w") == 123.0
    assert bench.measured_traffic("gemm_layer", "other") is None       # figures belong to one workload
    monkeypatch.setitem(bench.TRAFFIC, "w", {"gemm_layer": {"sources": bench.GEMM_SOURCES, "sha256": "0" * 16,
                                                           "bytes_per_launch": 123.0}})
    assert bench.measured_traffic("gemm_layer", "w") is None
    assert bench.measured_traffic("no_such_class", "w") is None


def test_clock_summary_keeps_the_median_the_max_and_every_active_reason():
    text = ("0, 1980, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active\n"
            "0, 2040, 2070, 1390.5, 0x4, Not Active, Not Active, Not Active, Active\n"
            "0, 1500, 2070, 1380.0, 0x8, Active, Not Active, Not Active, Not Active\n"
            "garbage line\n")
    c = bench.parse_clocks(text)
    assert c == {"sm_mhz": 1980.0, "sm_max_mhz": 2070.0, "reasons": ["hw_slowdown", "sw_power_cap"], "samples": 3}
    assert bench.parse_clocks("") is None


def test_fused_update_class_is_bound_by_its_bytes():
    """A class with both FLOPs and bytes (the dW product with the optimizer step in its epilogue) counts the
    larger of its compute time and its memory time, and the roofline entry names the memory bound then."""
    pk, _ = bench.peaks()
    prof = {"gemm_update": {"flops": 1e-3 * pk["bf16_tflops_sustained"] * 1e12,
                            "bytes": 3e-3 * pk["hbm_gbs"] * 1e9, "ms": 4.0, "launches": 2}}
    r = bench.step_roofline(prof, 1, ms_per_step=4.0)
    assert r["hbm_ms"] == pytest.approx(3.0) and r["tensor_ms"] == pytest.approx(0.0)
    e = bench.roofline_of(prof)
    assert e["bound"] == "hbm" and e["unit"] == "GB/s"
    assert e["achieved"] == pytest.approx(3e-3 * pk["hbm_gbs"] / 4e-3)
