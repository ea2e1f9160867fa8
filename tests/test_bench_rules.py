"""The measurement rules of bench.py, on the CPU: which clock samples count
(only those time-stamped inside the timed region), which bf16 peak a run is
held to (the sustained one only when the power cap held the median clock
below 95 % of the maximum), the roofline arithmetic of the dominant kernel
and of the whole path, and that a committed DRAM figure is dropped once the
kernel's sources change."""
import datetime
import json
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
import crc_synth as S  # noqa: E402


def smi_line(ts: float, sm: int, mx: int, power: float, cap: bool, thermal: bool = False) -> str:
    stamp = datetime.datetime.fromtimestamp(ts).strftime("%Y/%m/%d %H:%M:%S.%f")[:-3]
    act = lambda on: "Active" if on else "Not Active"  # noqa: E731
    return (f"{stamp}, {sm}, {mx}, {power}, 0x0, {act(False)}, {act(thermal)}, "
            f"{act(False)}, {act(cap)}")


def test_clock_summary_keeps_only_the_timed_region():
    c = bench.ClockSampler("0")
    c.t0, c.t1 = 1_700_000_000.0, 1_700_000_001.0
    c.lines = [smi_line(c.t0 - 1.0, 900, 2070, 100.0, False, thermal=True),   # before: ignored
               smi_line(c.t0 + 0.1, 2070, 2070, 900.0, False),
               smi_line(c.t0 + 0.5, 1700, 2070, 1350.0, True),
               smi_line(c.t0 + 0.9, 1600, 2070, 1340.0, True),
               smi_line(c.t1 + 1.0, 800, 2070, 100.0, False, thermal=True),   # after: ignored
               "garbage line"]
    s = c.summary()
    assert s["samples"] == 3
    assert s["sm_mhz"] == 1700 and s["sm_min_mhz"] == 1600 and s["sm_max_mhz"] == 2070
    assert s["reasons"] == ["sw_power_cap"]          # the thermal samples lie outside
    assert s["window_s"] == 1.0


def test_clock_summary_without_samples():
    c = bench.ClockSampler("0")
    c.t0, c.t1 = 10.0, 12.5
    assert c.summary() == {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0,
                           "window_s": 2.5}


PK = {"bf16_tflops": 1929.2, "bf16_tflops_sustained": 1711.2, "hbm_gbs": 6795.5}


@pytest.mark.parametrize("clocks,expect", [
    ({"sm_mhz": 1650, "sm_max_mhz": 2070, "reasons": ["sw_power_cap"]}, 1711.2),
    ({"sm_mhz": 2070, "sm_max_mhz": 2070, "reasons": ["sw_power_cap"]}, 1929.2),  # cap, full clock
    ({"sm_mhz": 1650, "sm_max_mhz": 2070, "reasons": []}, 1929.2),                # no cap reason
    ({"sm_mhz": None, "sm_max_mhz": None, "reasons": []}, 1929.2),
    (None, 1929.2),
])
def test_tensor_peak_follows_the_clock_regime(clocks, expect):
    assert bench.tensor_peak(PK, clocks)[0] == expect


def test_roofline_arithmetic(monkeypatch):
    monkeypatch.setattr(bench, "peaks", lambda: (dict(PK), "measured"))
    w = S.QWEN3_30B
    steps, per_launch_ms = 10, 4.4
    kt = {"fused": {"ms": steps * per_launch_ms, "launches": steps},
          "router": {"ms": 0.0, "launches": 0}, "scan": {"ms": 0.0, "launches": 0},
          "state": {"ms": 0.05, "launches": steps}}
    ms = steps * per_launch_ms + 0.05
    roof, path, kernels = bench.rooflines(kt, w, 3, steps, ms, ms / steps,
                                          clocks={"sm_mhz": 2070, "sm_max_mhz": 2070,
                                                  "reasons": []})
    flops = 2.0 * w.d * 3 * w.N * w.units                 # per launch
    assert roof["bound"] == "tensor" and roof["peak"] == 1929.2
    assert roof["achieved"] == pytest.approx(flops / (per_launch_ms / 1e3) / 1e12)
    assert roof["frac"] == pytest.approx(roof["achieved"] / 1929.2)
    assert roof["frac_of_sustained"] == pytest.approx(roof["achieved"] / 1711.2)
    assert roof["launches"] == steps and roof["avg_launch_ms"] == pytest.approx(per_launch_ms)
    assert roof["kernel"] == f"fused_route_cache_kernel<{w.N},3>"
    # whole path: the slower of the flops at the peak and 2d bytes per unit + the weights
    t_roof = max(flops / 1929.2e12, (2.0 * w.d * w.units + 2.0 * w.L * 3 * w.N * w.d) / 6795.5e9)
    assert path["t_roof_ms"] == pytest.approx(1e3 * t_roof)
    assert path["frac"] == pytest.approx(1e3 * t_roof / (ms / steps))
    assert kernels["fused"]["launches"] == steps


def test_hbm_bound_roofline_for_n32(monkeypatch):
    monkeypatch.setattr(bench, "peaks", lambda: (dict(PK), "measured"))
    w = S.GPT_OSS_20B
    kt = {"fused": {"ms": 7.7, "launches": 1}, "router": {"ms": 0.0, "launches": 0},
          "scan": {"ms": 0.0, "launches": 0}}
    roof, _, _ = bench.rooflines(kt, w, 3, 1, 7.7, 7.7)
    by = 2.0 * w.d * w.units + 2.0 * w.L * 3 * w.N * w.d
    assert roof["bound"] == "hbm" and roof["unit"] == "GB/s"
    assert roof["frac"] == pytest.approx(by / 6795.5e9 / 7.7e-3)


def test_committed_traffic_needs_the_current_sources(monkeypatch, tmp_path):
    kname = "fused_route_cache_kernel<128,3>"
    good = {kname: {"qwen3-30b-a3b": {"dram_bytes_per_unit": 7000.0, "source": "x",
                                      "src_sha": bench.source_hash(kname)}}}
    stale = {kname: {"qwen3-30b-a3b": {"dram_bytes_per_unit": 7000.0, "source": "x",
                                       "src_sha": "0000000000000000"}}}
    prof = tmp_path / "profiles"
    prof.mkdir()
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    (prof / "traffic.json").write_text(json.dumps(good))
    # the hash reads the sources under ROOT: point it back at the repository's
    monkeypatch.setattr(bench, "source_hash", lambda k: good[kname]["qwen3-30b-a3b"]["src_sha"])
    assert bench.committed_traffic(kname, "qwen3-30b-a3b")[0] == 7000.0
    (prof / "traffic.json").write_text(json.dumps(stale))
    assert bench.committed_traffic(kname, "qwen3-30b-a3b") == (None, None)
    assert bench.committed_traffic(kname, "gpt-oss-20b") == (None, None)
