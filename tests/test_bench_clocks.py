"""Clock summary of the benchmark (host logic, no GPU): only nvidia-smi samples taken inside
the timed region count; throttle reasons are read from the sample fields."""

import datetime

import bench


def _line(ts, sm, power, reasons=("Not Active",) * 4):
    stamp = datetime.datetime.fromtimestamp(ts).strftime("%Y/%m/%d %H:%M:%S.%f")[:-3]
    return ", ".join([stamp, "0", str(sm), "2070", str(power), "0x0000000000000000", *reasons])


def test_samples_outside_the_timed_region_are_ignored():
    t0 = 1_800_000_000.0
    lines = [_line(t0 - 0.5, 2070, 150.0), _line(t0 + 0.10, 1800, 900.0), _line(t0 + 0.20, 1900, 950.0),
             _line(t0 + 0.30, 2000, 920.0), _line(t0 + 1.5, 2070, 160.0)]
    s = bench.ClockSampler.summarize(bench.ClockSampler.parse(lines), t0, t0 + 0.35)
    assert s["samples"] == 3 and s["window"] == "timed region"
    assert s["sm_mhz"] == 1900 and s["power_w_max"] == 950.0 and s["reasons"] == []


def test_reasons_and_a_region_shorter_than_the_sampling_period():
    t0 = 1_800_000_000.0
    lines = [_line(t0 - 0.03, 1500, 1300.0, ("Not Active", "Not Active", "Not Active", "Active")),
             _line(t0 + 0.2, 2070, 200.0), "garbage line", ""]
    s = bench.ClockSampler.summarize(bench.ClockSampler.parse(lines), t0, t0 + 0.005)
    assert s["window"].startswith("nearest samples")
    assert "sw_power_cap" in s["reasons"]
    assert bench.ClockSampler.summarize([], t0, t0 + 1)["samples"] == 0


def test_launch_count_claim_matches_the_committed_launch_list():
    """gpu_launches (kernels per step x steps) against the ncu launch list of the stress step
    (two steps captured): the per-step count the benchmark claims is the one ncu saw."""
    import os
    import re

    path = os.path.join(os.path.dirname(bench.__file__), "profiles", "launches_route_commit_cfg5_n65536_fill95.md")
    text = open(path).read()
    global_index = "prefix index: global" in text
    totals = [int(m.group(1)) for m in re.finditer(r"\| \*\*total\*\* \| (\d+) \|", text)]
    assert totals and all(t == 2 * bench.kernels_per_step(global_index) for t in totals)
