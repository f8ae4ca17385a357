"""Synthetic convergence study of Hier-AVG on one GPU.

Observes, on seeded Gaussian-mixture data (no CIFAR or ImageNet here), the training
behaviour the paper states:
  * Theorem 3.5 (Sec. 3.3): with the global interval fixed, the bounds increase with
    K1 and decrease with S, so lower training loss is expected for smaller K1 and
    larger S (the paper's figures: P = 16, 32 steps per global average, K1 = 4 vs 8,
    S = 2 vs 4);
  * Sec. 3.4 / 4.3: Hier-AVG with twice K-AVG's global interval and S = 4 converges
    at least as fast as K-AVG for the same data processed, with half the global
    averages (K-AVG is S = 1, K1 = K);
  * the non-integer beta of the ImageNet run (K1 = 20, 43 steps per global average).
Every run processes the same number of samples.  After each global average all
learners hold the global model, whose mean cross-entropy over every learner's whole
data set is recorded (evaluated in plain fp32 PyTorch, outside the learner step).

    python -m paper_1903_05133_gb300.study [--seeds 6] [--steps 2752] [--out study.md]

(2752 local steps = lcm of the global intervals 16, 32, 64 and 43: every run reads
exactly the same samples.)
"""
from __future__ import annotations

import argparse
import math
import time
from dataclasses import dataclass
from typing import Dict, List, Sequence, Tuple

import torch

from . import configs
from .hier_avg import HierAvg
from .inputs import initial_layers, learner_data


@dataclass(frozen=True)
class Run:
    label: str
    S: int
    K1: int
    G: int            # local steps per global average


def base_workload(seed: int) -> configs.Workload:
    """3072 -> 512 -> 10 on 16 learners, B = 32, harder classes than the bench's data."""
    return configs.MLP512_P16.replace(name="study_mlp512", sigma_mu=0.05, seed=seed)


@torch.no_grad()
def global_loss(ha: HierAvg, X: torch.Tensor, y: torch.Tensor, chunk: int = 8192) -> float:
    """Mean cross-entropy of learner 0's model over all learners' data (fp32)."""
    layers = [(W[0].float(), b[0].float()) for W, b in ha.unpack(ha.params)]
    Xf = X.reshape(-1, X.shape[-1])
    yf = y.reshape(-1).long()
    total = 0.0
    for i in range(0, Xf.shape[0], chunk):
        h = Xf[i:i + chunk].float()
        for l, (W, b) in enumerate(layers):
            h = h @ W.T + b
            if l + 1 < len(layers):
                h = torch.relu(h)
        total += float(torch.nn.functional.cross_entropy(h, yf[i:i + chunk], reduction="sum"))
    return total / Xf.shape[0]


def run_one(w: configs.Workload, r: Run, steps: int, X, y, layers0) -> List[Tuple[int, float]]:
    """Train for `steps` local steps; the global model's loss after every global average."""
    if steps % r.G:
        raise ValueError("steps must be a multiple of the global interval")
    ha = HierAvg(w.P, r.S, r.K1, 1, w.lr, w.B, w.dims, w.precision)
    params = ha.pack(layers0, device=X.device)
    ha.bind(params, X, y)
    ha.set_global_steps(r.G)
    curve = [(0, global_loss(ha, X, y))]
    for n in range(steps // r.G):
        ha.round()
        curve.append(((n + 1) * r.G * w.B, global_loss(ha, X, y)))
    ha.check()
    ha.destroy()
    return curve


# (section, runs): the paper's comparisons at P = 16
STUDY: Sequence[Tuple[str, Sequence[Run]]] = (
    ("Theorem 3.5, K1 (S = 4, 32 steps per global average)",
     [Run(f"K1 = {k}", 4, k, 32) for k in (2, 4, 8, 16)]),
    ("Theorem 3.5, S (K1 = 4, 32 steps per global average)",
     [Run(f"S = {s}", s, 4, 32) for s in (1, 2, 4, 8, 16)]),
    ("Sec. 4.3: K-AVG with K vs Hier-AVG with 2K steps per global average, S = 4",
     [Run("K-AVG, K = 16", 1, 16, 16), Run("Hier-AVG, 32 steps, K1 = 2", 4, 2, 32),
      Run("Hier-AVG, 32 steps, K1 = 4", 4, 4, 32), Run("K-AVG, K = 32", 1, 32, 32),
      Run("Hier-AVG, 64 steps, K1 = 4", 4, 4, 64)]),
    ("non-integer beta (K1 = 20, 43 steps per global average, S = 4) vs K-AVG, K = 43",
     [Run("K-AVG, K = 43", 1, 43, 43), Run("Hier-AVG, 43 steps, K1 = 20", 4, 20, 43)]),
)


def study(seeds: Sequence[int], steps: int, device="cuda") -> Dict[str, Dict[str, List[list]]]:
    out: Dict[str, Dict[str, List[list]]] = {}
    for seed in seeds:
        w = base_workload(seed)
        X, y = learner_data(w, device=device)
        layers0 = initial_layers(w, device=device)
        for section, runs in STUDY:
            for r in runs:
                curve = run_one(w, r, steps, X, y, layers0)
                out.setdefault(section, {}).setdefault(r.label, []).append(curve)
        del X, y
    return out


# Paired comparisons (a, b): per seed, loss(a) - loss(b) at the same samples; a
# negative mean says run a trains faster.  The runs of one seed share data and
# initialisation, so the per-seed difference removes what the seeds move together.
PAIRS: Sequence[Tuple[str, str, str]] = (
    ("Theorem 3.5, K1 (S = 4, 32 steps per global average)", "K1 = 2", "K1 = 16"),
    ("Theorem 3.5, K1 (S = 4, 32 steps per global average)", "K1 = 4", "K1 = 8"),
    ("Theorem 3.5, S (K1 = 4, 32 steps per global average)", "S = 16", "S = 1"),
    ("Theorem 3.5, S (K1 = 4, 32 steps per global average)", "S = 4", "S = 2"),
    ("Sec. 4.3: K-AVG with K vs Hier-AVG with 2K steps per global average, S = 4",
     "Hier-AVG, 32 steps, K1 = 4", "K-AVG, K = 16"),
    ("Sec. 4.3: K-AVG with K vs Hier-AVG with 2K steps per global average, S = 4",
     "Hier-AVG, 64 steps, K1 = 4", "K-AVG, K = 32"),
    ("non-integer beta (K1 = 20, 43 steps per global average, S = 4) vs K-AVG, K = 43",
     "Hier-AVG, 43 steps, K1 = 20", "K-AVG, K = 43"),
)


def paired(res: Dict[str, Dict[str, List[list]]], pairs: Sequence[Tuple[str, str, str]],
           marks: Sequence[int]) -> str:
    """Per-seed paired differences loss(a) - loss(b): mean ± std over seeds, the
    t statistic mean / (std / sqrt(n)), and how many seeds have a < b."""
    lines = ["| a − b | " + " | ".join(f"{m} samples" for m in marks) + " |",
             "|---|" + "---|" * len(marks)]
    for section, a, b in pairs:
        ca, cb = res[section][a], res[section][b]
        cells = []
        for m in marks:
            d = [_interp(x, m) - _interp(y, m) for x, y in zip(ca, cb)]
            n = len(d)
            mu = sum(d) / n
            sd = math.sqrt(sum((x - mu) ** 2 for x in d) / max(1, n - 1))
            t = mu / (sd / math.sqrt(n)) if sd > 0 else float("inf") * (1 if mu >= 0 else -1)
            wins = sum(1 for x in d if x < 0)
            cells.append(f"{mu:+.5f} ± {sd:.5f} (t = {t:+.1f}, {wins}/{n} below)")
        lines.append(f"| {a} − {b} | " + " | ".join(cells) + " |")
    return "\n".join(lines) + "\n"


def _interp(curve: List[Tuple[int, float]], samples: int) -> float:
    """The loss after `samples` samples per learner (linear between global averages)."""
    for (s0, l0), (s1, l1) in zip(curve, curve[1:]):
        if s0 <= samples <= s1:
            return l0 + (l1 - l0) * (samples - s0) / (s1 - s0)
    return curve[-1][1]


def report(res: Dict[str, Dict[str, List[list]]], marks: Sequence[int]) -> str:
    lines = []
    for section, runs in res.items():
        lines.append(f"**{section}** — global model's training loss after the given samples per "
                     f"learner (mean ± std over {len(next(iter(runs.values())))} seeds)\n")
        lines.append("| run | " + " | ".join(f"{m} samples" for m in marks) + " |")
        lines.append("|---|" + "---|" * len(marks))
        for label, curves in runs.items():
            cells = []
            for m in marks:
                v = [_interp(c, m) for c in curves]
                mu = sum(v) / len(v)
                sd = math.sqrt(sum((x - mu) ** 2 for x in v) / max(1, len(v) - 1))
                cells.append(f"{mu:.4f} ± {sd:.4f}")
            lines.append(f"| {label} | " + " | ".join(cells) + " |")
        lines.append("")
    return "\n".join(lines)


def main() -> None:
    ap = argparse.ArgumentParser()
    ap.add_argument("--seeds", type=int, default=6)
    ap.add_argument("--steps", type=int, default=2752,
                    help="local steps per run, a multiple of every global interval")
    ap.add_argument("--out", default=None)
    args = ap.parse_args()
    t0 = time.time()
    res = study(list(range(args.seeds)), args.steps)
    B = base_workload(0).B
    marks = [args.steps * B // 4, args.steps * B // 2, args.steps * B]
    text = report(res, marks)
    text += ("\n**Paired differences** (per seed, loss(a) − loss(b) at equal samples; "
             "negative: a trains faster)\n\n")
    text += paired(res, PAIRS, marks)
    text += f"\n({args.seeds} seeds, {args.steps} local steps per run, {time.time() - t0:.0f} s)\n"
    print(text)
    if args.out:
        with open(args.out, "w") as f:
            f.write(text)


if __name__ == "__main__":
    main()
