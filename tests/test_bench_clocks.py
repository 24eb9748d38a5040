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


def test_profiled_figures_are_read_only_while_the_sources_match(tmp_path):
    """A committed ncu summary's machine-readable figures count only while the kernel's
    sources (comments and blank space aside) hash to the recorded value."""
    src = tmp_path / "k.cu"
    src.write_text("__global__ void k() { int x = 1; }  // first version\n")
    sha = bench.hash_sources_sha256((str(src),))
    summ = tmp_path / "k.md"
    summ.write_text("# ncu\n\n- `traffic_bytes_per_launch`: `123`\n- `batch_requests`: `65536`\n"
                    f"- `instances`: `128`\n- `sources_sha256`: `{sha}`\n")
    f = bench.profiled_fields(str(summ), (str(src),))
    assert f["traffic_bytes_per_launch"] == "123" and f["instances"] == "128"
    src.write_text("__global__ void k() { int x = 1; }  /* a comment edit */\n")
    assert bench.profiled_fields(str(summ), (str(src),))["traffic_bytes_per_launch"] == "123"
    src.write_text("__global__ void k() { int x = 2; }\n")
    assert bench.profiled_fields(str(summ), (str(src),)) == {}


def test_selection_traffic_is_reported_for_the_captured_workload_only():
    """The per-class selection's DRAM bytes were captured on the stress batch (65,536 requests,
    128 instances): another workload gets no figure."""
    import os

    f = bench.profiled_fields(bench.SELECT_PROFILE, bench.SELECT_SOURCES)
    if not f:  # the kernel changed since the capture: nothing is reported at all
        assert bench.profiled_select_traffic(65536, 128) is None
        return
    assert bench.profiled_select_traffic(65536, 128) == int(f["traffic_bytes_per_launch"])
    assert bench.profiled_select_traffic(4096, 128) is None
    assert bench.profiled_select_traffic(65536, 64) is None
    assert os.path.exists(bench.SELECT_PROFILE)
