"""bench.py end to end on the small workload: one JSON line carrying every key of the bench's
contract (throughput, timing, roofline, end-to-end copies, clocks, launch count)."""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_bench_prints_one_complete_line():
    cmd = [sys.executable, "bench.py", "--workload", "quadratic-n4-P1M", "--steps", "3", "--warmup", "3", "--no-cpu"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "e2e", "gpu_launches", "roofline", "clocks"):
        assert key in d, key
    assert d["n_gpus"] == 1 and d["steps"] == 3 and d["warmup"] == 3 and d["higher_is_better"] is True
    assert d["value"] > 0 and d["ms_per_step"] > 0 and d["config"]["workload"] == "quadratic-n4-P1M"
    w = d["config"]
    assert abs(d["value"] - w["n"] * w["P"] * w["K"] / (d["ms_per_step"] / 1e3)) <= 1e-6 * d["value"]
    rf = d["roofline"]
    assert rf["bound"] == "hbm" and rf["unit"] == "GB/s" and rf["peak"] > 0 and 0 < rf["frac"] < 2
    assert abs(rf["frac"] - rf["achieved"] / rf["peak"]) < 1e-9
    assert abs(rf["achieved"] - rf["bytes_per_launch"] / (rf["ms_per_launch"] / 1e3) / 1e9) < 1e-6 * rf["achieved"]
    e = d["e2e"]
    assert e["value"] > 0 and e["unit"] == d["unit"] and e["h2d_bytes_per_step"] == 12 * w["P"]
    assert e["d2h_bytes_per_step"] in (4 * w["P"], 4 * w["n"] * w["P"])
    assert d["gpu_launches"] > 0
    assert set(("sm_mhz", "sm_max_mhz", "reasons")) <= set(d["clocks"])
