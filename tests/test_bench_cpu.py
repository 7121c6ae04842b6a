"""bench.py's output contract, checked through the reference arm (the fp64
oracle on the host cores), which needs no GPU."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(*args):
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], capture_output=True, text=True,
                         timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [l for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, out.stdout
    return json.loads(lines[0])


def test_reference_arm_json_line():
    d = _run("--impl", "reference", "--workload", "single256", "--steps", "2", "--warmup", "3")
    for k in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
              "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["impl"] == "reference" and d["higher_is_better"] is False and d["steps"] == 2 and d["timed_steps"] == 2
    assert d["value"] > 0 and d["unit"] == "ms/step" and d["config"]["workload"] == "single256"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    e = d["e2e"]
    assert e["value"] == d["value"] and e["h2d_bytes_per_step"] == 0 and e["d2h_bytes_per_step"] == 0


def test_reference_arm_follows_the_update_rule():
    d = _run("--impl", "reference", "--workload", "single256", "--steps", "1", "--warmup", "3", "--update-rule", "muon")
    assert d["config"]["update_rule"] == "Eq. (6)"


def test_oracle_sample_estimates_what_the_budget_leaves_out():
    """The bounded oracle sample always times the cheapest shape class and
    estimates a class it has no time for from the measured flop rate and the
    oracle's own flop count (Eq. (5) as written)."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2609_35701_gb300 import workloads as W

    wl = W.first_layers(W.get_workload("llama130m"), 1)
    assert wl.numel == 4 * 768 * 768 + 3 * 768 * 2048 and len(wl.shapes) == 7
    ms_all, timed, est = bench.oracle_sample(wl)
    assert est == [] and sorted(timed) == ["2048x768", "768x2048", "768x768"] and ms_all > 0
    ms, timed, est = bench.oracle_sample(wl, budget_s=1e-9)
    assert timed == ["768x768"] and sorted(est) == ["2048x768", "768x2048"] and ms > 0
    # the literal Eq. (5) costs the tall class (Gram side 2048) more than the wide one
    assert bench.oracle_flops(2048, 768, 0) > bench.oracle_flops(768, 2048, 0) > bench.oracle_flops(768, 768, 0)
