"""Host-side pieces of the benchmark that decide what its JSON line claims, checked without a GPU:
the clock sampler's parsing (median clock, throttle reasons, the timed window), the DRAM-traffic
lookup in the committed ncu summaries (refused once the kernel's source has changed), and the L2
statement of the workload's config."""
import os
import shutil
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _line(sm, mx=2070, reasons=("Not Active",) * 4, active="0x0"):
    return ", ".join([str(sm), str(mx), "900.0", active, *reasons])


def test_clock_summary_median_window_and_reasons():
    c = bench.Clocks(0)
    c.marks = {"timed_start": 10.0, "timed_end": 12.0}
    c.lines = [
        (9.0, _line(1200)),  # warm-up: counted in the overall median only
        (10.5, _line(2070)),
        (11.0, _line(2055, reasons=("Not Active", "Not Active", "Not Active", "Active"))),
        (11.9, _line(2070)),
        (13.0, _line(1980)),
        (13.5, "garbage line"),
        (13.6, "[N/A], [N/A], 1, 2, 3, 4, 5, 6"),
    ]
    s = c.summary()
    assert s["samples"] == 5 and s["samples_timed"] == 3
    assert s["sm_mhz"] == 2055 and s["sm_mhz_timed"] == 2070
    assert s["sm_max_mhz"] == 2070
    assert s["reasons"] == ["sw_power_cap"]


def test_clock_summary_reports_each_slowdown_reason_by_name():
    c = bench.Clocks(0)
    c.lines = [(0.0, _line(1500, reasons=("Active", "Not Active", "Not Active", "Not Active"))),
               (0.1, _line(1400, reasons=("Not Active", "Active", "Active", "Not Active")))]
    s = c.summary()
    assert s["reasons"] == ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"]
    assert s["samples_timed"] == 0 and s["sm_mhz_timed"] is None


def test_clock_summary_without_samples():
    s = bench.Clocks(0).summary()
    assert s == {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}


@pytest.mark.parametrize("kernel", ["fwd", "bwd"])
def test_profiled_traffic_of_the_default_workload(kernel):
    t = bench._profiled_traffic(kernel, "packed64")
    assert isinstance(t, int) and t > 0
    assert bench._profiled_traffic(kernel, "no_such_workload") is None


def test_profiled_traffic_is_refused_after_a_source_change(tmp_path, monkeypatch):
    csrc = tmp_path / "paper_1906_11786_gb300" / "csrc"
    csrc.mkdir(parents=True)
    src = os.path.join(ROOT, "paper_1906_11786_gb300", "csrc")
    for f in ("band_tc.cu", "tc_util.cuh"):
        shutil.copy(os.path.join(src, f), csrc / f)
    shutil.copytree(os.path.join(ROOT, "profiles"), tmp_path / "profiles")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench._profiled_traffic("fwd", "packed64") == bench_traffic("fwd")
    with open(csrc / "band_tc.cu", "a") as fh:
        fh.write("\n// edited\n")
    assert bench._profiled_traffic("fwd", "packed64") is None


def bench_traffic(kernel):
    for line in open(os.path.join(ROOT, "profiles", f"k_band_tc_{kernel}_packed64.md")):
        if line.startswith("dram_bytes_per_launch:"):
            return int(line.split(":", 1)[1])
    return None


def test_l2_statement_follows_the_working_set():
    big = {"P": 20, "S": 128, "H": 64, "T": 8}
    cfg = bench.fixed_config("packed64", [0] * 64, big, 1, 64, 72000, 72064, 563)
    # bit tiles 2 * 563 * 3 * 20 * 128^2 / 8 = 138 MB alone
    assert "> 129 MB L2" in cfg["l2"] and cfg["parallelism"] == "dp1 (one supergraph per GPU)"
    small = {"P": 4, "S": 64, "H": 64, "T": 1}
    cfg = bench.fixed_config("single512", [0], small, 2, 1, 512, 512, 8)
    assert "fits the 129 MB L2" in cfg["l2"]
    assert cfg["parallelism"].startswith("dp2") and "all-reduce" in cfg["parallelism"]
    for k in ("workload", "graphs", "packed", "n_real", "n_pad", "K", "S", "P", "H", "T"):
        assert k in cfg
