"""bench.py's command line on the CPU: the reference arm (the oracle timed on the host
cores) prints one JSON line with the keys the driver reads."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_prints_one_json_line():
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload", "softmax",
                        "--steps", "2", "--warmup", "1"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    line = json.loads(lines[0])
    for key in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
                "cpu_baseline", "e2e"):
        assert key in line, key
    assert line["impl"] == "reference"
    assert line["value"] > 0 and line["higher_is_better"] is True
    assert line["steps"] == 2 and line["warmup"] == 1
    assert line["config"]["workload"].startswith("softmax")
    # the same config dict as the GPU arm's line, so the two arms compare one workload
    sys.path.insert(0, ROOT)
    import bench
    from paper_1903_05133_gb300 import configs
    assert line["config"] == json.loads(json.dumps(bench.run_config(configs.SHORT["softmax"], 1)))
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == line["value"]
    assert cb["unit"] == line["unit"] and cb["sample"].startswith("extrapolated")
    e2e = line["e2e"]
    assert e2e["value"] == line["value"] and e2e["unit"] == line["unit"]
    assert e2e["h2d_bytes_per_step"] == 0 and e2e["d2h_bytes_per_step"] == 0


def test_dominant_kernel_sample_cycles_through_the_round():
    import math
    sys.path.insert(0, ROOT)
    import bench
    # 28 update+forward launches per round at 3072-2048-2048-10 (K1 = 8): every 7th
    # would always land on the first step of a block
    assert bench.dom_sample(28) == 9
    assert bench.dom_sample(24) == bench.DOM_SAMPLE
    for per_round in range(1, 200):
        n = bench.dom_sample(per_round)
        assert n >= bench.DOM_SAMPLE and math.gcd(n, per_round) == 1
        assert {(k * n) % per_round for k in range(per_round)} == set(range(per_round))
