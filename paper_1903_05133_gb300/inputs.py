"""Seeded synthetic inputs shared by the CUDA path and the CPU oracle.

This module only draws random numbers; it holds none of Hier-AVG's arithmetic
(no sampling rule, no gradient, no averaging).  Both sides of every parity check
consume the very same bytes produced here.

Recipe (stand-in for CIFAR-10 / ImageNet-1K, which are not used):
  * class means   mu_c ~ N(0, sigma_mu^2 I) in R^{d_0}, shared by all learners
  * labels        y ~ Uniform{0 .. C-1}, drawn per learner
  * samples       x = mu_y + N(0, I), drawn per learner, stored bf16 (fp32 for
                  fp32 workloads)
  * initial model one w0 shared by every learner (Algorithm 1 initialises a single
                  global parameter): He-normal W_l ~ N(0, 2 / d_{l-1}) and zero
                  biases, or all zeros
Learner j draws from its own generator seeded with ``seed * 1000003 + j``.
"""
from __future__ import annotations

from typing import List, Sequence, Tuple

import torch

from .configs import Workload


def _gen(seed: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def class_means(w: Workload, device="cpu") -> torch.Tensor:
    """[C, d_0] fp32 class means ~ N(0, sigma_mu^2)."""
    g = _gen(w.seed * 7919 + 17, device)
    mu = torch.randn(w.classes, w.dims[0], generator=g, device=device, dtype=torch.float32)
    return mu * w.sigma_mu


def learner_data(w: Workload, device="cpu", N: int | None = None,
                 learners: Sequence[int] | None = None) -> Tuple[torch.Tensor, torch.Tensor]:
    """Per-learner datasets: X [P, N, d_0] (bf16, or fp32 for fp32 workloads), y [P, N] int32.
    With ``learners``, only those learners' data sets (the same bytes), stacked in
    that order."""
    N = w.N if N is None else N
    ids = list(range(w.P)) if learners is None else list(learners)
    dtype = torch.float32 if w.precision == "fp32" else torch.bfloat16
    mu = class_means(w, device)
    X = torch.empty(len(ids), N, w.dims[0], dtype=dtype, device=device)
    y = torch.empty(len(ids), N, dtype=torch.int32, device=device)
    for i, j in enumerate(ids):
        g = _gen(w.seed * 1000003 + j, device)
        yj = torch.randint(0, w.classes, (N,), generator=g, device=device, dtype=torch.int64)
        xj = torch.randn(N, w.dims[0], generator=g, device=device, dtype=torch.float32)
        xj += mu[yj]
        X[i].copy_(xj)
        y[i].copy_(yj.to(torch.int32))
    return X, y


def initial_layers(w: Workload, device="cpu") -> List[Tuple[torch.Tensor, torch.Tensor]]:
    """One shared w0 as [(W_l [d_l, d_{l-1}] fp32, b_l [d_l] fp32), ...]."""
    g = _gen(w.seed * 31337 + 5, device)
    layers = []
    for fan_in, fan_out in zip(w.dims[:-1], w.dims[1:]):
        if w.init == "zeros":
            Wl = torch.zeros(fan_out, fan_in, dtype=torch.float32, device=device)
        elif w.init == "he":
            Wl = torch.randn(fan_out, fan_in, generator=g, device=device, dtype=torch.float32)
            Wl *= (2.0 / fan_in) ** 0.5
        else:
            raise ValueError(f"unknown init {w.init!r}")
        layers.append((Wl, torch.zeros(fan_out, dtype=torch.float32, device=device)))
    return layers


def replica_matrix(P: int, D: int, seed: int = 0, device="cpu") -> torch.Tensor:
    """[P, D] fp32 ~ N(0, 1): the learner replicas of the averaging-only sweep."""
    g = _gen(seed * 104729 + P * 131 + 7, device)
    return torch.randn(P, D, generator=g, device=device, dtype=torch.float32)


def perturbed_layers(w: Workload, scale: float, seed: int, device="cpu"
                     ) -> List[List[Tuple[torch.Tensor, torch.Tensor]]]:
    """Per-learner parameter sets w0 + scale * N(0, 1): distinct learner states
    for one-step checks started from a state where the learners disagree."""
    base = initial_layers(w, device)
    out = []
    for j in range(w.P):
        g = _gen(seed * 1000033 + j, device)
        lj = []
        for Wl, bl in base:
            lj.append((Wl + scale * torch.randn(Wl.shape, generator=g, device=device),
                       bl + scale * torch.randn(bl.shape, generator=g, device=device)))
        out.append(lj)
    return out
