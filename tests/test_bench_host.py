"""Host logic of bench.py that decides whether a measurement stands: the summary
of the nvidia-smi clock samples taken during the timed region (median SM clock
under load, the maximum clock, and every throttle reason seen).  CPU only: the
samples are written to the sampler's file by hand."""
import tempfile

import pytest

pytest.importorskip("torch")
import bench  # noqa: E402


def summarise(lines):
    cs = bench.ClockSampler(0)
    cs.proc = object()  # a sampler that ran; summary() reads only its file
    cs.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
    cs.f.write("".join(line + "\n" for line in lines))
    cs.f.flush()
    return cs.summary()


NA = "Not Active"


def row(sm, mx, *, hw=NA, hw_th=NA, sw_th=NA, cap=NA):
    # the sampler's query order: index, clocks.sm, clocks.max.sm, power.draw,
    # reasons bitmask, hw_slowdown, hw_thermal_slowdown, sw_thermal_slowdown, sw_power_cap
    return f"0, {sm}, {mx}, 812.5, 0x0000000000000000, {hw}, {hw_th}, {sw_th}, {cap}"


def test_clean_run_reports_the_median_clock_and_no_reason():
    s = summarise([row(2070, 2070), row(2055, 2070), row(2070, 2070)])
    assert s["sm_mhz"] == 2070 and s["sm_max_mhz"] == 2070
    assert s["reasons"] == [] and s["samples"] == 3


def test_every_throttle_reason_seen_is_reported():
    s = summarise([row(2070, 2070), row(1900, 2070, cap="Active"), row(1500, 2070, hw_th="Active"),
                   row(1600, 2070, sw_th="Active", hw="Active")])
    assert s["reasons"] == sorted(["sw_power_cap", "hw_thermal_slowdown", "sw_thermal_slowdown", "hw_slowdown"])
    assert s["sm_mhz"] == pytest.approx((1900 + 1600) / 2)


def test_unreadable_values_and_short_lines_are_skipped():
    s = summarise([row("[N/A]", 2070), "0, 2070", row(2070, 2070), ""])
    assert s["samples"] == 2 and s["sm_mhz"] == 2070


def test_no_samples_and_no_sampler_are_flagged():
    assert summarise([])["reasons"] == ["no samples"]
    assert bench.ClockSampler(0).summary()["reasons"] == ["nvidia-smi unavailable"]


def test_reference_arm_prints_one_contract_line():
    # the reference arm is the fp64 oracle on the host cores (no GPU needed)
    import json
    import os
    import subprocess
    import sys

    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--steps", "1", "--warmup", "1"],
                       cwd=root, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [x for x in r.stdout.splitlines() if x.strip().startswith("{")]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["metric"] == "rows/s" and line["unit"] == "rows/s"
    assert line["higher_is_better"] is True and line["value"] > 0 and line["warmup"] >= 3
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["value"] == line["value"]
    assert line["cpu_baseline"]["cores"] >= 1
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"], "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
