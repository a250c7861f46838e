"""The clock record of bench.py's timed region, parsed from nvidia-smi's CSV
(here a file written by the test; no GPU and no nvidia-smi involved): the SM
clock is the median of the samples under load (idle samples below half the
highest are left out), the maximum is the largest reported maximum, and a
throttle reason is listed when any sample shows it Active."""
import os

import bench


def _sampler(lines):
    cs = bench.ClockSampler(0)
    cs.proc = True          # stands in for the nvidia-smi process
    cs.f.write("\n".join(lines) + "\n")
    return cs


def test_median_under_load_and_active_reasons():
    na = "Not Active"
    cs = _sampler([
        f"0, 345, 2070, 120.0, 0x0, {na}, {na}, {na}, {na}",          # idle before the steps start
        f"0, 2070, 2070, 1180.5, 0x4, {na}, {na}, {na}, Active",
        f"0, 2055, 2070, 1390.0, 0x4, {na}, {na}, {na}, Active",
        f"0, 2070, 2070, 1201.2, 0x0, {na}, {na}, {na}, {na}",
        "garbage line",
    ])
    s = cs.summary()
    assert s == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 4}


def test_thermal_slowdown_is_reported():
    cs = _sampler(["0, 1500, 2070, 1400.0, 0x40, Not Active, Active, Not Active, Not Active"])
    assert cs.summary()["reasons"] == ["hw_thermal_slowdown"]


def test_no_sampler_no_record():
    cs = bench.ClockSampler(0)
    assert cs.summary() is None
    cs.f.close()
    os.unlink(cs.f.name)
