"""bench.py's JSON line on a GPU: one short run checked against the fields its consumers read.

The run is the default int16 8192^3 workload with few steps and no per-workload table or CPU
baseline, so it takes seconds; the test checks the line's keys, units and internal consistency
(the roofline fraction is its achieved value over its peak, the end-to-end leg copies the bytes
of A, B and C in and C out, every timed launch is one of the library's kernels).
"""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_bench_line_has_the_contract_fields():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--steps", "3", "--warmup", "3",
                        "--no-extra", "--no-cpu-baseline"], capture_output=True, text=True, timeout=900, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1, r.stdout[-2000:]
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "roofline", "e2e", "gpu_launches", "clocks"):
        assert key in d, key
    assert d["n_gpus"] == 1 and d["steps"] == 3 and d["warmup"] == 3 and d["higher_is_better"] is True
    assert d["unit"] == "TOPS" and d["value"] > 0 and d["dtype"] == "int64"
    assert d["config"]["workload"] == "i16_8192"
    # value is 2mnk per step over the measured step time
    assert d["value"] == pytest.approx(2 * 8192 ** 3 / (d["ms_per_step"] * 1e-3) / 1e12, rel=1e-6)
    roof = d["roofline"]
    assert roof["bound"] == "tensor" and roof["unit"] == "TOPS"
    assert roof["frac"] == pytest.approx(roof["achieved"] / roof["peak"], rel=1e-9)
    assert 0.3 < roof["frac"] < 1.3, roof
    e2e = d["e2e"]
    assert e2e["value"] > 0 and e2e["unit"] == "TOPS"
    assert e2e["h2d_bytes_per_step"] == 8192 * 8192 * (2 + 2 + 8)
    assert e2e["d2h_bytes_per_step"] == 8192 * 8192 * 8
    # device-resident steps: one operand split and one pair GEMM each
    assert d["gpu_launches"] == 2 * 3
    assert {"sm_mhz", "sm_max_mhz", "reasons"} <= set(d["clocks"])
