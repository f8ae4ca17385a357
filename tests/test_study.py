"""The synthetic convergence study: report formatting (CPU) and a short training run
whose global model's loss must fall (GPU)."""
import math

import pytest
import torch

from paper_1903_05133_gb300 import study


def test_interp_and_report():
    c = [(0, 2.0), (100, 1.0), (200, 0.5)]
    assert study._interp(c, 0) == 2.0
    assert math.isclose(study._interp(c, 50), 1.5)
    assert math.isclose(study._interp(c, 150), 0.75)
    text = study.report({"sec": {"run a": [c, [(0, 2.0), (100, 1.2), (200, 0.7)]]}}, [100, 200])
    assert "run a" in text and "1.1000 ± 0.1414" in text and "0.6000 ± 0.1414" in text


def test_paired_differences():
    a = [[(0, 2.0), (100, 1.0)], [(0, 2.0), (100, 1.2)], [(0, 2.0), (100, 0.9)]]
    b = [[(0, 2.0), (100, 1.1)], [(0, 2.0), (100, 1.25)], [(0, 2.0), (100, 1.0)]]
    text = study.paired({"sec": {"a": a, "b": b}}, [("sec", "a", "b")], [100])
    # differences -0.1, -0.05, -0.1: mean -0.08333, std 0.02887, t = -5.0, 3 of 3 below
    assert "-0.08333 ± 0.02887 (t = -5.0, 3/3 below)" in text


def test_pairs_name_existing_runs():
    runs = {section: {r.label for r in rs} for section, rs in study.STUDY}
    for section, a, b in study.PAIRS:
        assert a in runs[section] and b in runs[section]


def test_every_global_interval_divides_the_default_budget():
    for _section, runs in study.STUDY:
        for r in runs:
            assert 2752 % r.G == 0, r


@pytest.mark.gpu
def test_short_run_lowers_the_loss():
    w = study.base_workload(0).replace(N=512)
    X, y = study.learner_data(w, device="cuda")
    layers0 = study.initial_layers(w, device="cuda")
    curve = study.run_one(w, study.Run("x", 4, 4, 16), 64, X, y, layers0)
    assert len(curve) == 5 and all(math.isfinite(l) for _, l in curve)
    assert curve[-1][1] < 0.9 * curve[0][1]
    assert [s for s, _ in curve] == [0, 512, 1024, 1536, 2048]
