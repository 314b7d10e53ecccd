"""bench.py's clock record, on the CPU: samples outside the timed region are
left out, throttle reasons are read per sample, and a region with a hardware
or thermal slowdown (or clocks held low with no reason) is rejected."""
import os
import sys
import time

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _stamp(t):
    return time.strftime("%Y/%m/%d %H:%M:%S", time.localtime(t)) + ".%03d" % int((t % 1) * 1000)


def _row(t, sm, smax=2070, hw="Not Active", hwt="Not Active", swt="Not Active", cap="Not Active"):
    return ["0", _stamp(t), str(sm), str(smax), "900.0", "0x0", hw, hwt, swt, cap]


def test_sample_time_parses_nvidia_smi_stamps():
    t = 1_780_000_000.25
    assert abs(bench._sample_time(_stamp(t)) - t) < 2e-3
    assert bench._sample_time("2026/12/02 10:11:12") is not None
    assert bench._sample_time("not a time") is None


def test_only_samples_inside_the_region_count():
    t0 = 1_780_000_000.0
    rows = [_row(t0 - 0.15, 2070), _row(t0 - 0.10, 2070)]            # idle, before
    rows += [_row(t0 + 0.05 * k, 1800, cap="Active") for k in range(1, 6)]  # under load
    rows += [_row(t0 + 0.45, 2070, hwt="Active")]                        # after the region
    s = bench.summarise_clock_rows(rows, t0, t0 + 0.3)
    assert s["scope"] == "timed region" and s["samples"] == 5
    assert s["sm_mhz"] == 1800 and s["sm_max_mhz"] == 2070
    assert s["reasons"] == ["sw_power_cap"]  # the thermal sample after the region is not counted
    assert not bench.clocks_rejected(s)      # a power cap alone is kept


def test_falls_back_to_all_samples():
    t0 = 1_780_000_000.0
    rows = [_row(t0 - 1.0, 2070), _row(t0 + 1.0, 2065)]
    s = bench.summarise_clock_rows(rows, t0, t0 + 0.01)
    assert s["scope"].startswith("all samples") and s["samples"] == 2 and s["sm_mhz"] == 2067.5
    garbled = [r[:1] + ["?"] + r[2:] for r in rows]
    assert bench.summarise_clock_rows(garbled, t0, t0 + 0.01)["samples"] == 2
    assert bench.summarise_clock_rows([], t0, t0 + 1)["samples"] == 0


def test_rejection_rule():
    ok = {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": []}
    assert not bench.clocks_rejected(ok)
    for r in ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"):
        assert bench.clocks_rejected(dict(ok, reasons=[r]))
    assert bench.clocks_rejected(dict(ok, sm_mhz=1200.0))                             # held low, no reason
    assert not bench.clocks_rejected(dict(ok, sm_mhz=1200.0, reasons=["sw_power_cap"]))
    assert not bench.clocks_rejected({"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi samples"]})
