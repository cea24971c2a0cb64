"""bench.py's bookkeeping, on the CPU: the algorithmic flops and bytes the
roofline divides by (against the figures worked out by hand for the
ResNet-50 3x3 layer), the roofline arithmetic and its bound selection, the
clock summary taken from nvidia-smi samples, and the rule that DRAM traffic
from a committed ncu summary is reported only while the kernel source is the
one it was measured on."""
import hashlib
import json
import os

import pytest

import bench
from paper_2105_14713_gb300 import workloads as wl


def _cfg2(dtype):
    return wl.ConvLayer("r50_3x3", 64, 28, 28, 128, 128, 3, 3, 1, 1, 1, N=8, rate=0.5, dtype=dtype)


def test_kept_flops_and_bytes_of_the_resnet50_3x3_layer():
    t = 9216                                    # half of 16 groups x 1152 kept indices
    f32, bf16 = _cfg2("f32"), _cfg2("bf16")
    assert bench.kept_flops(f32, t) == 2 * (64 * 28 * 28) * t * 8          # 7.40 GFLOP
    x = 64 * 28 * 28 * 128
    expect = lambda es: x * es + x * es + t * 8 * es + t * 4 + 17 * 4      # X + Y + D + I + P
    assert bench.alg_bytes(f32, t) == expect(4)                             # 51.7 MB
    assert bench.alg_bytes(bf16, t) == expect(2)                            # 25.9 MB
    assert abs(bench.alg_bytes(f32, t) / 1e6 - 51.7) < 0.05
    assert abs(bench.alg_bytes(bf16, t) / 1e6 - 25.9) < 0.05


def test_strided_1x1_counts_only_the_input_it_reads():
    layer = wl.ConvLayer("s2", 2, 14, 14, 64, 64, 1, 1, 2, 0, 1, N=4, rate=0.5)
    t = 0
    x_read = bench.alg_bytes(layer, t) - layer.pixels * 64 * 4 - (64 // 4 + 1) * 4
    assert x_read == 2 * 7 * 7 * 64 * 4          # a quarter of the input
    # padding that no output reaches past the edge is not counted either
    assert bench._touched(10, 10, 3, 1, 1, 1) == 10
    assert bench._touched(10, 5, 1, 2, 0, 1) == 5


PK = {"hbm_gbs": 8000.0, "bf16_tflops": 2000.0, "bf16_tflops_sustained": 1800.0,
      "fp32_ffma_tflops": 80.0, "sm_max_mhz": 2000.0, "source": "measured"}


def test_roofline_tensor_leg_fp32_counts_three_tf32_products():
    # (with these peaks the kept flops take longer than the algorithmic bytes)
    layer, t, ms = _cfg2("f32"), 9216, 0.0616
    r = bench.leg_roofline(layer, t, "tc", ms, PK)
    peak = 2000.0 * 1.1 / 2.25
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s"
    assert r["peak"] == pytest.approx(peak)
    achieved = bench.kept_flops(layer, t) / (ms * 1e-3) / 1e12
    assert r["achieved"] == pytest.approx(achieved)
    assert r["frac"] == pytest.approx(achieved / peak)
    dense = 2 * layer.pixels * layer.K * layer.C_out
    assert r["issued_tflops"] == pytest.approx(3 * dense / (ms * 1e-3) / 1e12)


def test_roofline_picks_hbm_when_bytes_dominate():
    layer = wl.ConvLayer("1x1", 128, 56, 56, 64, 64, 1, 1, 1, 0, 1, N=4, rate=0.9, dtype="bf16")
    t = int(0.1 * (64 // 4) * 64)
    r = bench.leg_roofline(layer, t, "tc", 0.05, PK)
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and r["peak"] == 8000.0
    assert r["achieved"] == pytest.approx(bench.alg_bytes(layer, t) / 0.05e-3 / 1e9)
    assert r["frac"] == pytest.approx(r["achieved"] / 8000.0)


def test_roofline_ffma_leg_is_alu_bound_against_the_derived_peak():
    layer = _cfg2("f32")
    r = bench.leg_roofline(layer, 9216, "fma", 0.2, PK)
    assert r["bound"] == "alu" and r["peak"] == 80.0
    assert "issued_tflops" not in r


def test_clock_summary_median_under_load_and_reasons(tmp_path):
    cs = bench.ClockSampler(0)
    cs.path = str(tmp_path / "clocks.csv")
    cs.proc = object()                                   # as if nvidia-smi had run
    lines = ["0, 2070, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active",
             "0, 2055, 2070, 1390.0, 0x4, Not Active, Not Active, Not Active, Active",
             "0, 2070, 2070, 1380.5, 0x4, Not Active, Not Active, Not Active, Active",
             "0, 345, 2070, 120.0, 0x0, Not Active, Not Active, Not Active, Not Active",
             "garbage line"]
    (tmp_path / "clocks.csv").write_text("\n".join(lines) + "\n")
    s = cs.summary()
    assert s == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 4}
    assert not os.path.exists(cs.path)                   # the sample file is removed


def test_clock_summary_reports_thermal_slowdown(tmp_path):
    cs = bench.ClockSampler(0)
    cs.path = str(tmp_path / "c.csv")
    cs.proc = object()
    (tmp_path / "c.csv").write_text("0, 1500, 2070, 1000, 0x40, Not Active, Active, Not Active, Not Active\n")
    assert cs.summary()["reasons"] == ["hw_thermal_slowdown"]


def test_traffic_only_while_the_source_is_unchanged(tmp_path, monkeypatch):
    src = tmp_path / "kernel.cu"
    src.write_bytes(b"__global__ void k() {}\n")
    sha = hashlib.sha256(src.read_bytes()).hexdigest()[:16]
    (tmp_path / "profiles").mkdir()
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(
        {"tc_layer": {"source": "kernel.cu", "source_sha": sha, "dram_bytes_per_launch": 12345}}))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_for("tc_layer") == 12345
    assert bench.traffic_for("other_layer") is None
    src.write_bytes(b"__global__ void k() { /* changed */ }\n")
    assert bench.traffic_for("tc_layer") is None


def test_committed_traffic_records_name_existing_sources_and_profiles():
    with open(os.path.join(bench.ROOT, "profiles", "traffic.json")) as fh:
        recs = json.load(fh)
    assert recs
    for key, rec in recs.items():
        assert os.path.exists(os.path.join(bench.ROOT, rec["source"])), key
        assert os.path.exists(os.path.join(bench.ROOT, rec["profile"])), key
        assert rec["dram_bytes_per_launch"] > 0
