"""Local and global averaging of Algorithm 1 (Sec. 3.1), written out plainly.

Paper: after K1 local steps every learner of a local cluster (|P_lc| = S, S | P,
Sec. 2) is replaced by (1/S) * sum over the cluster; after beta such blocks every
learner is replaced by (1/P) * sum over all P learners.

Reading adopted for floating point (the paper states the means in exact
arithmetic): the n values are summed by the canonical adjacent-pair tree

    for h = 1, 2, 4, ... while h < n:
        for i = 0, 2h, 4h, ...:
            if i + h < n:  v[i] = v[i] + v[i + h]     # unpaired v[i] is carried up

in the dtype of the input (fp32 for parity with the GPU, fp64 for exact-math
pins), and the mean is the correctly rounded quotient v[0] / n.  Clusters are the
contiguous learner blocks [g*S, (g+1)*S).
"""
from __future__ import annotations

import numpy as np


def tree_sum(rows: np.ndarray) -> np.ndarray:
    """Sum over axis 0 of ``rows`` [n, ...] in the canonical adjacent-pair order."""
    n = rows.shape[0]
    if n == 0:
        raise ValueError("empty reduction")
    v = [rows[i].copy() for i in range(n)]
    h = 1
    while h < n:
        for i in range(0, n, 2 * h):
            if i + h < n:
                v[i] = v[i] + v[i + h]
        h *= 2
    return v[0]


def group_mean(rows: np.ndarray) -> np.ndarray:
    """(1/n) * sum of the n rows: tree sum, then one division by n."""
    n = rows.shape[0]
    return tree_sum(rows) / rows.dtype.type(n)


def local_average(w: np.ndarray, S: int) -> None:
    """In place: every learner of cluster g gets the mean of rows [g*S, (g+1)*S).

    Algorithm 1, "locally average and synchronize" (Sec. 3.1)."""
    P = w.shape[0]
    if S < 1 or P % S != 0:
        raise ValueError(f"S={S} must divide P={P}")
    for g in range(P // S):
        m = group_mean(w[g * S:(g + 1) * S])
        w[g * S:(g + 1) * S] = m


def global_average(w: np.ndarray) -> None:
    """In place: every learner gets the mean over all P rows.

    Algorithm 1, "globally average and synchronize" plus the synchronisation of
    every learner to the new global parameter at the top of the next round."""
    m = group_mean(w)
    w[:] = m
