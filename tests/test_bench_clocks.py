"""bench.py's clock record (no GPU): the median SM clock under load, the maximum, and the throttle
reasons seen, parsed from the CSV lines nvidia-smi prints during the timed region."""
import types

import bench


def _stopped(lines):
    s = bench.ClockSampler(0)
    s.proc = types.SimpleNamespace(terminate=lambda: None, wait=lambda timeout=None: 0, kill=lambda: None)
    s.t = types.SimpleNamespace(join=lambda timeout=None: None)
    s.lines = list(lines)
    return s.stop()


def line(sm, smax, hw="Not Active", hwt="Not Active", swt="Not Active", pcap="Not Active"):
    return f"0, {sm}, {smax}, 812.50, 0x0000000000000000, {hw}, {hwt}, {swt}, {pcap}"


def test_quiet_run():
    r = _stopped([line(2070, 2070)] * 5 + [line(1995, 2070)])
    assert r["sm_mhz"] == 2070.0 and r["sm_max_mhz"] == 2070.0 and r["reasons"] == [] and r["samples"] == 6


def test_throttle_reasons_are_reported():
    r = _stopped([line(2070, 2070), line(1800, 2070, hw="Active"), line(1900, 2070, pcap="Active"),
                  line(2000, 2070, swt="Active"), line(2010, 2070, hwt="Active")])
    assert r["reasons"] == ["hw_slowdown", "hw_thermal_slowdown", "sw_power_cap", "sw_thermal_slowdown"]
    assert r["sm_mhz"] == 2000.0


def test_malformed_lines_are_skipped():
    r = _stopped(["", "garbage", "0, [N/A], 2070, 1, 0x0, Not Active, Not Active, Not Active, Not Active",
                  line(2070, 2070)])
    assert r["samples"] == 1 and r["sm_mhz"] == 2070.0


def test_no_nvidia_smi():
    s = bench.ClockSampler(0)
    assert s.stop()["reasons"] == ["nvidia-smi unavailable"]
