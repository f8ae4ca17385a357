"""bench.py on the CPU: the reference arm (the oracle timed on the host cores) prints one
JSON line with the keys the driver reads; the sampling, extrapolation and roofline
arithmetic behind the GPU arm's line."""
import json
import os
import subprocess
import sys

import pytest

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


def test_round_extrapolation_of_the_oracle_sample():
    # A round of the 32-learner ImageNet-shaped workload: P * K1 * K2 = 1024 learner
    # steps, K2 * P / S = 32 cluster averages and a global average over P rows, which
    # the sample counts as (P - 1) / (S - 1) cluster averages (a tree over P values
    # takes P - 1 additions, one over S takes S - 1).
    sys.path.insert(0, ROOT)
    import bench
    from paper_1903_05133_gb300 import configs
    w = configs.MLP4096_P32
    smp = bench.OracleSample.__new__(bench.OracleSample)
    smp.w, smp.steps, smp.avg_split = w, 1, 8
    t_step, t_avg = 0.5, 0.01
    want = 1024 * t_step + (32 + 31 / 7) * t_avg * 8
    assert smp.round_seconds(t_step, t_avg) == pytest.approx(want)
    smp.steps = 4                                    # four steps timed: a quarter each
    assert smp.round_seconds(4 * t_step, t_avg) == pytest.approx(want)


def test_gemm_report_against_the_hbm_bound_ceiling():
    sys.path.insert(0, ROOT)
    import bench
    # 18 flop per byte against a 6790 GB/s copy rate and 1724 TFLOP/s: the HBM roofline
    # allows 18 * 6.79 = 122.2 TFLOP/s, 0.0709 of the tensor rate
    by, fl, ms = 1e12, 18e12, 10_000.0               # 1 TB and 18 PFLOP in 10 s
    r = bench.gemm_report(by, fl, ms, 6790.0, 1724.0)
    assert r["TFLOPs"] == pytest.approx(1.8, abs=1e-2)
    assert r["flop_per_byte"] == pytest.approx(18.0)
    assert r["hbm_bound_tensor_frac_ceiling"] == pytest.approx(18 * 6.79 / 1724, abs=1e-4)
    assert r["frac_of_hbm_bound_ceiling"] == pytest.approx(1.8 / (18 * 6.79), abs=1e-4)
    # a compute-bound intensity is capped by the tensor rate itself
    r = bench.gemm_report(1e9, 1e15, 1000.0, 6790.0, 1724.0)
    assert r["hbm_bound_tensor_frac_ceiling"] == pytest.approx(1.0)
