"""Host-side pieces of bench.py that need no GPU: the clock record of the timed region,
the byte count of what the host call's kernels write into host memory, and the CPU
baseline's repetitions of its sample."""
import datetime
import os
import sys
import time

sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))


def _line(t, sm, reasons):
    ts = datetime.datetime.fromtimestamp(t).strftime("%Y/%m/%d %H:%M:%S.%f")[:-3]
    flags = ", ".join("Active" if r else "Not Active" for r in reasons)
    return f"{ts}, 0, {sm}, 2070, 1000.0, 0x0, {flags}"


def test_clock_samples_are_those_of_the_timed_region():
    import bench
    t = time.time()
    lines = [_line(t - 2.0, 1000, (1, 0, 0, 0)),   # warm-up, throttled: not in the region
             _line(t, 2070, (0, 0, 0, 1)),
             _line(t + 0.05, 2050, (0, 0, 0, 0)),
             _line(t + 2.0, 900, (0, 1, 0, 0))]    # after the region
    c = bench.ClockSampler.parse(lines, t - 0.01, t + 0.06, pad=0.1)
    assert c["samples"] == 2 and c["window"] == "timed region"
    assert c["sm_mhz"] == 2060.0 and c["sm_max_mhz"] == 2070.0
    assert c["reasons"] == ["sw_power_cap"]


def test_clock_record_falls_back_to_the_whole_run():
    import bench
    t = time.time()
    lines = [_line(t - 2.0, 1800, (0, 0, 0, 0)), "garbage", _line(t + 2.0, 2070, (0, 0, 0, 0))]
    c = bench.ClockSampler.parse(lines, t, t + 0.01, pad=0.1)
    assert c["samples"] == 2 and c["window"] == "whole run" and c["sm_mhz"] == 1935.0


def test_host_copy_bytes_count_what_the_kernels_write_to_host_memory():
    import bench
    # hour1: K = 64, n_prev = 1, one frame per unit: ids, expansion, frames, counts, status
    assert bench.host_copy_bytes(64, 128, 1) == 256 + 512 + 512 + 16 + 4
    assert bench.host_copy_bytes(1, 2, 2) == 4 + 8 + 16 + 16 + 4


def test_cpu_baseline_repeats_its_sample_for_the_set_cpu_time(monkeypatch):
    import bench
    from paper_2609_02780_gb300 import synth
    w = synth.PRESETS["tiny"].replace(n_frames=8, n_planted=1)
    data = synth.make_workload(w, device="cpu")
    monkeypatch.setattr(bench, "CPU_BASELINE_SECONDS", 0.2)
    b = bench.cpu_baseline(w, data["keys"], data["q"], frames=8)
    keys = w.n_slabs * 8 * w.tokens_per_frame
    assert b["repetitions"] >= 1 and b["seconds"] >= 0.2
    # `seconds` is rounded to the millisecond
    assert abs(b["value"] - keys * b["repetitions"] / b["seconds"]) <= 1e-2 * b["value"]
    assert f"{b['repetitions']} times" in b["sample"] and b["kind"] == "oracle"
