"""Host-side logic of bench.py on CPU: the clock sampler's parsing and its
bracketing of short timed regions (against a fake nvidia-smi), the traffic
record's source-hash check, and the algorithmic byte counts of verify."""
import json
import os
import sys
import threading
import time

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402

LINE = "{sm}, 2070, 900.5, {hw}, Not Active, Not Active, {cap}"


def _line(sm=2070, hw="Not Active", cap="Not Active"):
    return LINE.format(sm=sm, hw=hw, cap=cap)


def test_summary_parses_clocks_and_reasons():
    clk = bench.ClockSampler("GPU-x")
    clk.lines = [_line(1980), _line(2070, cap="Active"), _line(2070), "garbage", ""]
    s = clk.summary()
    assert s["samples"] == 3
    assert s["sm_mhz"] == 2070 and s["sm_max_mhz"] == 2070
    assert s["reasons"] == ["sw_power_cap"]
    clk.lines = [_line(hw="Active")]
    assert clk.summary()["reasons"] == ["hw_slowdown"]


def test_summary_without_samples_says_so():
    s = bench.ClockSampler("GPU-x").summary()
    assert s == {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}


def test_summary_starts_at_the_region():
    clk = bench.ClockSampler("GPU-x")
    clk.lines = [_line(600), _line(700), _line(2070), _line(2070)]
    clk.first = 2  # samples before the region (the idle clocks) are not counted
    assert clk.summary()["sm_mhz"] == 2070 and clk.summary()["samples"] == 2


class _FakeSmi:
    """Stands in for `nvidia-smi -lms 20`: a line every `period` seconds."""

    def __init__(self, period):
        self.period = period
        self.stop = threading.Event()
        self.stdout = self._lines()

    def _lines(self):
        while not self.stop.is_set():
            time.sleep(self.period)
            yield _line() + "\n"

    def terminate(self):
        self.stop.set()

    def wait(self, timeout=None):
        return 0

    def kill(self):
        self.stop.set()


def test_short_region_is_bracketed_by_samples(monkeypatch):
    monkeypatch.setattr(bench.subprocess, "Popen", lambda *a, **k: _FakeSmi(0.05))
    with bench.ClockSampler("GPU-x") as clk:
        clk.start_region()
        assert len(clk.lines) >= 1  # the sampler was running before the region began
        time.sleep(0.001)            # a region much shorter than the sampling period
        clk.end_region()
    s = clk.summary()
    assert s["samples"] >= 2 and s["reasons"] == []


def test_sampler_without_nvidia_smi_reports_unsampled(monkeypatch):
    def boom(*a, **k):
        raise FileNotFoundError("nvidia-smi")
    monkeypatch.setattr(bench.subprocess, "Popen", boom)
    t0 = time.perf_counter()
    with bench.ClockSampler("GPU-x") as clk:
        clk.start_region()
        clk.end_region()
    assert time.perf_counter() - t0 < 1.0  # no wait for lines that cannot come
    assert clk.summary()["reasons"] == ["unsampled"]


def test_traffic_follows_the_source_hash():
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        rec = json.load(f)
    for kernel, files in (("distill", bench.DISTILL_SOURCES), ("verify", bench.VERIFY_SOURCES)):
        want = rec[kernel]["dram_bytes_per_launch"] if rec[kernel]["source_sha"] == bench._source_hash(files) else None
        assert bench._traffic(kernel, files) == want
        assert rec[kernel]["alg_bytes_per_launch_full"] > 0
    assert bench._traffic("no-such-kernel", bench.DISTILL_SOURCES) is None


@pytest.mark.parametrize("B,k,V,s_in", [(32, 5, 32000, 2), (256, 8, 128256, 2), (4, 4, 32000, 4)])
def test_verify_bytes(B, k, V, s_in):
    # every draft row (B k) and target row (B (k+1)) read once; greedy reads only the target rows
    assert bench._bytes_verify(B, k, V, s_in, False) == (B * k + B * (k + 1)) * V * s_in
    assert bench._bytes_verify(B, k, V, s_in, True) == B * (k + 1) * V * s_in
    if (B, k, V, s_in) == (256, 8, 128256, 2):
        assert bench._bytes_verify(B, k, V, s_in, False) == 1116340224


def test_gpus_flag_starts_that_many_ranks():
    """`bench.py --gpus 2` outside torchrun starts two ranks itself; on the
    CPU-only launcher check (gloo, no GPU work) the line reports both ranks and
    the slower rank's time (rank r sleeps (r + 1) ms a step)."""
    import subprocess
    env = {k: v for k, v in os.environ.items() if k not in ("WORLD_SIZE", "RANK", "LOCAL_RANK")}
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--gpus", "2", "--launcher-check",
                        "--steps", "4", "--warmup", "0"], capture_output=True, text=True, timeout=300, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    line = json.loads([ln for ln in r.stdout.splitlines() if ln.startswith("{")][-1])
    assert line["check"] == "launcher" and line["n_gpus"] == 2
    assert line["ms_per_step"] >= 2.0
    assert line["value"] == pytest.approx(2 / (line["ms_per_step"] / 1e3), rel=1e-3)


def test_cpu_model_names_something():
    assert isinstance(bench.cpu_model(), str) and bench.cpu_model()
