"""bench.py's clock sampler on CPU, driven by a stand-in for nvidia-smi that
prints CSV rows in its query format: the sampler must be live before the timed
region, keep only rows from inside it, and report throttle reasons."""
import os
import sys
import time

FAKE = r'''
import sys, time
period = float(sys.argv[sys.argv.index("-lms") + 1]) * 1e-3
print("0, 1000, 2070, 100.0, 0x0, Not Active, Not Active, Not Active, Not Active", flush=True)
i = 0
while True:
    time.sleep(period)
    cap = "Active" if i == 1 else "Not Active"
    print("0, 2070, 2070, 900.0, 0x4, Not Active, Not Active, Not Active, " + cap, flush=True)
    i += 1
'''


def _sampler(tmp_path, **kw):
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    fake = tmp_path / "fake_smi.py"
    fake.write_text(FAKE)
    return bench.ClockSampler(0, cmd=[sys.executable, str(fake)], **kw)


def test_samples_inside_the_region_only(tmp_path):
    with _sampler(tmp_path, period_ms=50) as clk:
        assert clk.stamped, "the sampler must be live before the region starts"
        time.sleep(0.5)
    s = clk.summary()
    # the first row (1000 MHz) arrived before the region and is dropped
    assert s["sm_mhz"] == 2070.0 and s["sm_max_mhz"] == 2070.0
    assert s["samples"] >= 5
    assert s["reasons"] == ["sw_power_cap"]
    assert clk.proc.poll() is not None


def test_missing_tool_reports_no_samples(tmp_path):
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    with bench.ClockSampler(0, cmd=[str(tmp_path / "no_such_tool")]) as clk:
        pass
    assert clk.summary() == {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
