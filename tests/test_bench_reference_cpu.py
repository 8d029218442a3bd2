"""bench.py's reference arm (the oracle timed on the host cores) keeps the bench
line contract without a GPU: the main arm's metric, unit and workload keys, the
requested steps and warm-up, a cpu_baseline describing the run, and an e2e
object without host-device copies."""
import json
import os
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_line():
    sys.path.insert(0, ROOT)
    import bench

    t0 = time.perf_counter()
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--steps", "2", "--warmup", "3"],
                         cwd=ROOT, capture_output=True, text=True, timeout=900)
    wall = time.perf_counter() - t0
    assert out.returncode == 0, out.stderr[-2000:]
    line = json.loads(out.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference"
    assert line["metric"] == bench.METRIC
    assert line["unit"] == "tokens/s" and line["higher_is_better"] is True
    assert line["steps"] == 2 and line["warmup"] == 3
    for k, v in bench.workload_config(bench.K_DRAFT, 1).items():
        assert line["config"][k] == v
    assert line["value"] > 0 and line["ms_per_step"] > 0
    # the timed steps were executed: they fit inside the run's wall time
    assert line["ms_per_step"] * line["steps"] / 1000.0 <= wall
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == line["value"] and cb["cores"] >= 1
    assert "oracle" in cb["sample"] and cb["cpu_model"]
    assert cb["tokens_per_iteration"] >= 1.0 and cb["full_depth_iteration_s"] > 0
    assert line["e2e"] == {"value": line["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
