"""CPU checks of bench.py's host logic: the clock and throttle-reason sampler
(against a stand-in nvidia-smi on PATH) and the gate that reports the recorded
ncu traffic only for the kernel sources it was measured on."""
import os
import stat
import sys
import textwrap

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _fake_smi(tmp_path, rows):
    """An executable named nvidia-smi that prints `rows` as its query output and
    then waits to be terminated, as `nvidia-smi -lms` does."""
    script = tmp_path / "nvidia-smi"
    script.write_text(textwrap.dedent(f"""\
        #!{sys.executable}
        import sys, time
        for line in {rows!r}:
            print(line, flush=True)
        time.sleep(60)
        """))
    script.chmod(script.stat().st_mode | stat.S_IXUSR)
    return str(tmp_path)


def _row(sm, util, hw="Not Active", hwt="Not Active", swt="Not Active", swp="Not Active", smax=2070):
    # index, clocks.sm, clocks.max.sm, power.draw, utilization.gpu, reasons.active, then the four reasons
    return f"0, {sm}, {smax}, 900.0, {util}, 0x0, {hw}, {hwt}, {swt}, {swp}"


def _sample(monkeypatch, tmp_path, rows):
    monkeypatch.setenv("PATH", _fake_smi(tmp_path, rows) + os.pathsep + os.environ["PATH"])
    c = bench.ClockSampler(0)
    c.start()
    return c.stop()


def test_clock_sampler_reads_loaded_samples(monkeypatch, tmp_path):
    rows = [_row(345, 0), _row(2070, 100), _row(2055, 98), _row(2070, 100), _row(1980, 100, swp="Active"),
            _row(600, 10)]
    got = _sample(monkeypatch, tmp_path, rows)
    # idle samples (utilization below 50 %) are left out of the median and the reasons
    assert got["samples"] == 4
    assert got["sm_mhz"] == pytest.approx(2062.5)
    assert got["sm_max_mhz"] == 2070
    assert got["reasons"] == ["sw_power_cap"]


def test_clock_sampler_reports_slowdowns(monkeypatch, tmp_path):
    rows = [_row(1500, 100, hw="Active"), _row(1400, 100, hwt="Active", swt="Active"), "garbage line", ""]
    got = _sample(monkeypatch, tmp_path, rows)
    assert got["reasons"] == ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown"]
    assert got["samples"] == 2


def test_clock_sampler_without_nvidia_smi(monkeypatch, tmp_path):
    monkeypatch.setenv("PATH", str(tmp_path))  # nothing named nvidia-smi here
    c = bench.ClockSampler(0)
    c.start()
    assert c.stop() is None


def test_traffic_is_reported_only_for_the_measured_sources(monkeypatch):
    sha = bench.kernel_sources_sha256()
    monkeypatch.setattr(bench, "TRAFFIC", {"pixart": {"bytes_per_launch": 123, "sources_sha256": sha}})
    assert bench.measured_traffic("pixart") == 123
    assert bench.measured_traffic("sana") is None
    monkeypatch.setattr(bench, "TRAFFIC", {"pixart": {"bytes_per_launch": 123, "sources_sha256": "0" * 64}})
    assert bench.measured_traffic("pixart") is None
