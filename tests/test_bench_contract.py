"""bench.py's reference arm (the fp64 oracle timed on the host cores) prints the contract's JSON line.

Runs on the CPU: the reference arm needs no GPU.  The tiny workload keeps it to seconds.
"""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_one_contract_line():
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload", "tiny", "--steps", "3",
                        "--warmup", "1", "--reference-step-seconds", "0.05"],
                       cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip().startswith("{")]
    assert len(lines) == 1, r.stdout
    j = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
                "scaling", "vs_baseline", "dtype", "data", "config", "e2e", "cpu_baseline", "gpu_launches"):
        assert key in j, key
    assert j["impl"] == "reference"
    assert j["steps"] == 3 and j["warmup"] == 1 and j["n_gpus"] == 1
    assert j["value"] > 0 and j["ms_per_step"] > 0 and j["higher_is_better"] is True
    assert j["unit"] == "TFLOP/s" and j["dtype"] == "f64"
    assert j["config"]["workload"].startswith("tiny")
    # the same config dict as the GPU arm prints, so that the two lines compare
    sys.path.insert(0, ROOT)
    import bench
    from paper_2608_13499_gb300 import workloads as W
    assert j["config"] == json.loads(json.dumps(bench.bench_config(W.tiny(), 1)))
    assert j["e2e"] == {"value": j["value"], "unit": j["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    cb = j["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == j["value"] and cb["cores"] >= 1 and cb["sample"]
    assert j["gpu_launches"] == 0
