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


class FakeClock:
    """Stands in for the nvidia-smi sampler: hands out prepared summaries."""

    def __init__(self, records):
        self.records = records

    def __call__(self):
        return self

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        return False

    def start(self):
        pass

    def stop(self):
        pass

    def summary(self):
        return dict(self.records.pop(0))


GOOD = {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": []}
THERMAL = {"sm_mhz": 1500.0, "sm_max_mhz": 2070.0, "reasons": ["hw_thermal_slowdown"]}


def _region_counter():
    runs = []

    def region():
        runs.append(len(runs))
        return len(runs)
    return region, runs


def test_good_clock_record_is_measured_once():
    region, runs = _region_counter()
    res, clocks, again = bench.measure_with_clock_check(region, lambda: None, FakeClock([GOOD]))
    assert runs == [0] and res == 1 and not again and clocks["sm_mhz"] == 2070.0


def test_bad_clock_record_is_measured_once_more():
    region, runs = _region_counter()
    res, clocks, again = bench.measure_with_clock_check(region, lambda: None, FakeClock([THERMAL, GOOD]))
    assert runs == [0, 1] and res == 2 and again and clocks["reasons"] == []
    # a second bad record is kept (and reported): there is no third run
    region, runs = _region_counter()
    res, clocks, again = bench.measure_with_clock_check(region, lambda: None, FakeClock([THERMAL, THERMAL]))
    assert runs == [0, 1] and again and clocks["reasons"] == ["hw_thermal_slowdown"]
