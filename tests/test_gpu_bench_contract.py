"""bench.py's JSON line keeps the contract the driver reads: one line on
stdout with the metric, the whole-job value, the timing keys, the roofline,
the CPU baseline, the e2e leg, the launch count and the clocks. Run on the toy
workload, so it takes seconds."""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_bench_line_has_every_contract_key():
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--workload", "toy",
           "--steps", "2", "--warmup", "3"]
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
                "roofline", "cpu_baseline", "e2e", "gpu_launches", "clocks"):
        assert key in d, key
    assert d["n_gpus"] == 1 and d["steps"] == 2 and d["warmup"] == 3
    assert d["value"] > 0 and d["ms_per_step"] > 0 and d["higher_is_better"] is True
    assert d["config"]["workload"] == "toy"
    roof = d["roofline"]
    for key in ("bound", "achieved", "peak", "unit", "frac", "traffic"):
        assert key in roof, key
    assert roof["bound"] in ("hbm", "alu") and 0 < roof["frac"] < 2
    cpu = d["cpu_baseline"]
    assert cpu["kind"] == "oracle" and cpu["value"] > 0 and cpu["cores"] >= 1 and cpu["sample"]
    e2e = d["e2e"]
    nbytes = 2 ** 20 * 4
    assert e2e["value"] > 0 and e2e["h2d_bytes_per_step"] == nbytes
    assert e2e["d2h_bytes_per_step"] == nbytes
    # one launch per member and one fused update per generation
    assert d["gpu_launches"] == 2 * (8 + 1)
    assert {"sm_mhz", "sm_max_mhz", "reasons"} <= set(d["clocks"])
