"""bench.py's own arm on the GPU: one JSON line with every key the output
contract asks for, and values that are consistent with each other."""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_bench_json_line_on_the_gpu():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--workload", "single256", "--steps", "5",
                          "--warmup", "3"], capture_output=True, text=True, timeout=900, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, out.stdout
    d = json.loads(lines[0])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
              "vs_baseline", "dtype", "data", "config", "roofline", "cpu_baseline", "e2e", "gpu_launches", "clocks"):
        assert k in d, k
    assert d["n_gpus"] == 1 and d["steps"] == 5 and d["warmup"] >= 3 and d["higher_is_better"] is False
    assert d["value"] > 0 and d["value"] == d["ms_per_step"] and d["config"]["workload"] == "single256"
    r = d["roofline"]
    assert r["bound"] in ("tensor", "hbm") and r["peak"] > 0 and 0 < r["frac"] < 1.5
    assert abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-9
    assert d["gpu_launches"] == d["kernels_per_step"] * d["steps"] and d["gpu_launches"] > 0
    e = d["e2e"]
    assert e["value"] > 0 and e["h2d_bytes_per_step"] == 4 * 256 * 256 and e["d2h_bytes_per_step"] == 4 * 256 * 256
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] > 0 and cb["cores"] >= 1 and cb["sample"]
    c = d["clocks"]
    assert c["sm_max_mhz"] > 0 and "reasons" in c
