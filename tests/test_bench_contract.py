"""The reference arm of bench.py (the CPU oracle on a bounded sample) prints the
one JSON line the benchmark contract asks for; runs on the host only."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_the_contract_line():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "0",
                        "--steps", "2", "--warmup", "1"], capture_output=True, text=True, timeout=300, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
              "vs_baseline", "dtype", "data", "config", "impl", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["impl"] == "reference" and d["steps"] == 2 and d["warmup"] == 1 and d["value"] > 0
    assert d["higher_is_better"] is True and d["unit"] == "tokens/s"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    cfg = d["config"]
    assert cfg["workload"].startswith("tiny-f32") or "(workload 0)" in cfg["workload"]
    assert cfg["tokens_valid"] <= cfg["tokens_executed"] <= cfg["tokens_full"]


def test_reference_arm_suite_line_describes_the_headline_workload():
    # the default bench run leads with the video-shaped layer (workload 4): the
    # reference arm reports the same config, its oracle sample extrapolated from a
    # key/value pass and sampled query rows (the ~12k-row layer would take about a
    # minute of fp64 work)
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                        "--warmup", "0"], capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    cfg = d["config"]
    assert "(workload 4)" in cfg["workload"] and "suite" in cfg
    assert cfg["batch"] == 4 and cfg["window"] == 2048
    assert cfg["route"]["pad_rows"] >= 0 and cfg["tokens_valid"] <= cfg["tokens_executed"] <= cfg["tokens_full"]
    assert d["value"] > 0 and d["cpu_baseline"]["value"] == d["value"]
    assert "extrapolated" in d["cpu_baseline"]["sample"]
