"""Host-side pieces of bench.py that need no GPU: the clock-sample summary."""
import datetime
import os
import tempfile

import bench


class _FakeProc:
    def terminate(self):
        pass

    def wait(self, timeout=None):
        return 0


def _sampler_with(lines):
    s = bench.ClockSampler(False)
    fd, s.path = tempfile.mkstemp(suffix=".csv")
    with os.fdopen(fd, "w") as fh:
        fh.write("\n".join(lines) + "\n")
    s.fh = open(os.devnull, "w")
    s.proc = _FakeProc()
    return s


def _row(t, mhz, watts, reasons=("Not Active",) * 4):
    stamp = datetime.datetime.fromtimestamp(t).strftime("%Y/%m/%d %H:%M:%S.%f")[:-3]
    return ", ".join([stamp, str(mhz), "2070", str(watts), *reasons])


def test_clock_summary_keeps_only_the_timed_region():
    t0 = 1_800_000_000.0
    lines = [_row(t0 - 1.0, 1200, 150)]                     # warm-up, idle clocks
    lines += [_row(t0 + 0.1 * i, 2070, 680) for i in range(5)]
    lines += [_row(t0 + 2.0, 900, 100, ("Active", "Not Active", "Not Active", "Not Active"))]
    out = _sampler_with(lines).stop((t0, t0 + 0.45))
    assert out["samples"] == 5 and out["samples_from"] == "timed region"
    assert out["sm_mhz"] == 2070.0 and out["reasons"] == []      # the late slowdown is outside
    assert out["power_w_max"] == 680.0


def test_clock_summary_reports_reasons_and_falls_back_without_a_window():
    t0 = 1_800_000_000.0
    lines = [_row(t0, 1900, 700, ("Not Active", "Not Active", "Not Active", "Active")),
             "garbage line", _row(t0 + 0.1, 2000, 650)]
    out = _sampler_with(lines).stop()
    assert out["samples"] == 2 and out["samples_from"] == "warm-up and timed region"
    assert out["reasons"] == ["sw_power_cap"]
