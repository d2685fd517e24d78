"""The benchmark's clock record (bench.ClockSampler) from nvidia-smi output.

A bench line whose clock record shows a thermal or hardware slowdown, or SM
clocks far below their maximum, is not a valid measurement, so the record
must carry every throttle reason seen during the timed region and the
median SM clock under load (idle samples excluded). The nvidia-smi process
is replaced by a fake that returns fixed CSV lines.
"""
import bench


class _FakeProc:
    def __init__(self, out):
        self.out = out

    def terminate(self):
        pass

    def kill(self):
        pass

    def communicate(self, timeout=None):
        return self.out, ""


def _record(lines):
    s = bench.ClockSampler(0)
    s.proc = _FakeProc("\n".join(lines) + "\n")
    return s.stop()


def _line(sm, mx=2070, hw="Not Active", hwt="Not Active", swt="Not Active", cap="Not Active"):
    return f"0, {sm}, {mx}, 900.5, 0x0000000000000000, {hw}, {hwt}, {swt}, {cap}"


def test_median_under_load_and_no_reasons():
    rec = _record([_line(345), _line(2070), _line(2070), _line(1995), _line(360)])
    assert rec == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": [], "samples": 5}


def test_every_throttle_reason_is_reported():
    rec = _record([_line(2070, cap="Active"), _line(1800, hwt="Active"), _line(1900, swt="Active"),
                   _line(1700, hw="Active")])
    assert rec["reasons"] == ["hw_slowdown", "hw_thermal_slowdown", "sw_power_cap",
                              "sw_thermal_slowdown"]
    assert rec["sm_mhz"] == 1850.0


def test_malformed_lines_are_skipped_and_no_samples_gives_none():
    assert _record(["garbage", "0, [N/A], 2070, 1, 0, a, b, c, d"]) is None
    rec = _record(["short, line", _line(2070)])
    assert rec["samples"] == 1


def test_sampler_without_nvidia_smi_reports_nothing():
    s = bench.ClockSampler(0)
    assert s.stop() is None
