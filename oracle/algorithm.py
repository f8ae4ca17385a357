"""Algorithm 1 (Hier-AVG, Sec. 3.1) driven over P simulated learners.

State: a list of learner-indexed arrays (each with leading axis P).  One global
round is

    for b in 0 .. beta-1:            (beta = K2 here: local averages per round)
        for k in 1 .. K1:  every learner j takes one local SGD step
        local average within every cluster of S learners
    global average over all P learners (every learner is then synchronised)

The global step counter t counts local SGD steps from 0 and continues across
rounds.  Reading of "randomly sample a mini-batch": the per-learner data are i.i.d.
draws, so learner j at step t takes rows (t*B + s) mod N, s = 0..B-1, of its own
data set.

Sec. 3.1 takes the global interval K1 * beta with beta an integer for the analysis
and leaves it free in practice (the ImageNet run of Sec. 4 uses 43 local steps per
global average with K1 = 20).  Reading of a free global interval of G local steps:
within a round, every K1-th step is followed by a local average (counting from the
round's start, as Algorithm 1's loops do), and the round's G-th step by the global
average, preceded by a local average exactly when K1 divides G.  G = K1 * beta is
Algorithm 1 itself.  The step size gamma_n and batch size B_n of round n (Theorem
3.3's diminishing step sizes and growing batches) are ``lr`` and ``B`` at the time of
the round's steps.  With a batch size that changes, each learner reads its data
sequentially: the batch of a step starts where the previous one ended, at row
(sum of the earlier steps' batch sizes) mod N, which is t * B for a constant B.
"""
from __future__ import annotations

from typing import List

import numpy as np

from .averaging import global_average, local_average
from .learner import sgd_update


def batch_rows(t: int, B: int, N: int) -> np.ndarray:
    """Row indices of the mini-batch at local step t (constant batch size B)."""
    return batch_rows_from(t * B, B, N)


def batch_rows_from(start: int, B: int, N: int) -> np.ndarray:
    """Row indices of a mini-batch of B rows that starts at row `start` (mod N)."""
    return (start + np.arange(B)) % N


class HierAvgOracle:
    def __init__(self, P: int, S: int, K1: int, K2: int, lr: float, problem,
                 params: List[np.ndarray], mode: str = "fp32", global_steps: int = 0):
        if min(P, S, K1, K2) < 1 or P % S != 0:
            raise ValueError("need P, S, K1, K2 >= 1 and S | P")
        if global_steps < 0:
            raise ValueError("global_steps must be >= 0 (0: K1 * K2)")
        # local SGD steps per global round
        self.G = global_steps if global_steps > 0 else K1 * K2
        for p in params:
            if p.shape[0] != P:
                raise ValueError("every parameter array must have leading axis P")
        self.P, self.S, self.K1, self.K2, self.lr = P, S, K1, K2, lr
        self.problem, self.mode = problem, mode
        dt = np.float64 if mode == "f64" else np.float32
        self.params = [np.array(p, dtype=dt, copy=True) for p in params]
        self.t = 0
        self.B = getattr(problem, "B", 0)       # batch size of the following steps
        self.cursor = 0                         # rows read so far (per learner)

    def step(self) -> None:
        """One local SGD step on every learner (Algorithm 1, innermost loop)."""
        X = getattr(self.problem, "X", None)
        rows = None if X is None else batch_rows_from(self.cursor, self.B, X.shape[1])
        for j in range(self.P):
            pj = [p[j] for p in self.params]
            grads = self.problem.gradients(j, rows, pj)
            for p, g in zip(self.params, grads):
                p[j] = sgd_update(p[j], g, self.lr, self.mode)
        self.t += 1
        self.cursor += self.B

    def local_average(self) -> None:
        for p in self.params:
            local_average(p, self.S)

    def global_average(self) -> None:
        for p in self.params:
            global_average(p)

    def round(self) -> None:
        """One global round: G local steps, a local average after every K1-th of them,
        then the global average (Algorithm 1 when G = K1 * K2)."""
        for r in range(1, self.G + 1):
            self.step()
            if r % self.K1 == 0:
                self.local_average()
        self.global_average()
