"""The benchmark's reference arm on the CPU: `bench.py --impl reference` times
the oracle on the host cores and prints one JSON line with the keys the
benchmark contract asks for.  Needs no GPU (the workload is generated on the
CPU and the oracle is plain C)."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_one_line():
    import oracle.oracle as O
    O.lib()  # builds the oracle library when it is missing
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--config", "1",
                        "--steps", "3", "--warmup", "4"],
                       cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip().startswith("{")]
    assert len(lines) == 1
    j = json.loads(lines[0])
    assert j["impl"] == "reference"
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "config", "cpu_baseline", "e2e"):
        assert k in j, k
    assert j["value"] > 0 and j["unit"] == "steps/s" and j["higher_is_better"] is True
    assert j["cpu_baseline"]["kind"] == "oracle" and j["cpu_baseline"]["cores"] == 1
    assert j["e2e"]["h2d_bytes_per_step"] == 0 and j["e2e"]["value"] == j["value"]
    assert j["config"]["workload"] == "c1-tiny"
    # the reference arm honours the requested steps and warm-up, and describes
    # the workload with the same dict as the GPU arm
    assert j["steps"] == 3 and j["warmup"] == 4
    import bench
    from paper_2205_11048_gb300 import workload as W
    assert j["config"] == bench.config_dict(W.config(1), 1)
