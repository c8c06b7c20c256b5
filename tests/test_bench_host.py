"""Host logic of bench.py (no GPU): the roofline object and the per-kernel rates.

A timed region under a second takes the burst bf16 peak and a longer one the
sustained peak; every fraction is the algorithmic rate (flops or bytes over the
kernel's mean event time) over the named peak; the roofline reports the slowest GEMM
and never the quantize; a recorded DRAM traffic whose kernel sources changed since the
capture reads as unknown."""
import math

import bench

PK = {"hbm_gbs": 6778.3, "bf16_tflops": 1933.1, "bf16_tflops_sustained": 1702.0}
FLOPS = 2.0 * 16384 * 8512 * 2048
QBYTES = 79.6e6


def _per(fwd=0.371, dx=0.391, dw=0.340, q=0.0286):
    return {"quantize": q, "fwd": fwd, "dx": dx, "dw": dw}


def test_short_region_takes_the_burst_peak():
    kinfo, roof = bench.roofline(_per(), 22.7, 20, PK, "measured", FLOPS, QBYTES)
    assert roof["peak"] == PK["bf16_tflops"]
    assert "burst" in roof["peak_kind"] and "under 1 s" in roof["peak_kind"]
    assert roof["kernel"] == "dx" and roof["bound"] == "tensor"
    ach = FLOPS / (0.391e-3) / 1e12
    assert math.isclose(roof["achieved"], round(ach, 1))
    assert math.isclose(roof["frac"], round(ach / PK["bf16_tflops"], 4))
    assert math.isclose(roof["frac_of_sustained"], round(ach / PK["bf16_tflops_sustained"], 4))
    assert roof["timed_region_ms"] == 22.7 and roof["algorithmic_per_launch"] == FLOPS


def test_long_region_takes_the_sustained_peak():
    kinfo, roof = bench.roofline(_per(), 1150.0, 1000, PK, "measured", FLOPS, QBYTES)
    assert roof["peak"] == PK["bf16_tflops_sustained"]
    assert "sustained" in roof["peak_kind"] and "at least 1 s" in roof["peak_kind"]
    assert math.isclose(kinfo["fwd"]["frac"], round(FLOPS / 0.371e-3 / 1e12 / 1702.0, 4))


def test_quantize_is_scored_against_hbm_and_never_the_roofline_kernel():
    # even when the quantize is the slowest launch, the roofline is a GEMM
    kinfo, roof = bench.roofline(_per(q=5.0), 22.7, 20, PK, "measured", FLOPS, QBYTES)
    assert roof["kernel"] == "dx"
    assert kinfo["quantize"]["unit"] == "GB/s"
    assert math.isclose(kinfo["quantize"]["frac"], round(QBYTES / 5e-3 / 1e9 / PK["hbm_gbs"], 4))


def test_slowest_gemm_is_the_roofline_kernel():
    _, roof = bench.roofline(_per(fwd=0.5), 22.7, 20, PK, "measured", FLOPS, QBYTES)
    assert roof["kernel"] == "fwd"


def test_stale_traffic_reads_as_unknown(monkeypatch):
    files = dict((n, f) for n, f, _ in bench.KERNELS)["dx"]
    monkeypatch.setattr(bench, "kernel_hash", lambda f: "0" * 16)
    assert bench.recorded_traffic("dx", files) is None
    _, roof = bench.roofline(_per(), 22.7, 20, PK, "measured", FLOPS, QBYTES)
    assert roof["traffic"] is None


def test_current_traffic_is_read_when_the_sources_match(monkeypatch):
    import json
    import os
    with open(os.path.join(bench.ROOT, "profiles", "traffic.json")) as f:
        rec = json.load(f)["dx"]
    files = dict((n, f) for n, f, _ in bench.KERNELS)["dx"]
    monkeypatch.setattr(bench, "kernel_hash", lambda f: rec["source_sha"])
    assert bench.recorded_traffic("dx", files) == rec["dram_bytes_per_launch"]
