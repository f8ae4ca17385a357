"""The five Hier-AVG workloads this library is measured and checked on.

Notation follows Sec. 2 and Algorithm 1 (Sec. 3.1) of Zhou & Cong, "A Distributed
Hierarchical Averaging SGD Algorithm": P learners, local clusters of S learners,
K1 local SGD steps between local averages, mini-batch B, step size gamma (``lr``).

``K2`` here counts LOCAL AVERAGES per global average, i.e. the paper's beta
(Sec. 3.1 writes the global interval as K1 * beta local steps).  The paper's own
global averaging interval in local SGD steps is therefore ``K1 * K2``.

Every input is synthetic: Gaussian-mixture samples shaped like CIFAR-10
(32x32x3 -> 3072 features, 10 classes) or down-sampled ImageNet-1K
(64x64x3 -> 12288 features, 1000 classes); see ``inputs.py``.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Tuple


@dataclass(frozen=True)
class Workload:
    name: str
    P: int                    # learners (Sec. 2: "total number of learners")
    S: int                    # learners per local cluster, S | P (Sec. 2)
    K1: int                   # local SGD steps per local average (Sec. 2)
    K2: int                   # local averages per global average (= beta, Sec. 3.1)
    rounds: int               # global averaging rounds (outer loop of Algorithm 1)
    dims: Tuple[int, ...]     # layer widths d_0 .. d_L (d_0 = features, d_L = classes)
    precision: str            # "fp32" or "bf16" (bf16 GEMM operands, fp32 master)
    N: int                    # samples per learner
    B: int                    # mini-batch per learner step
    lr: float                 # constant step size gamma
    sigma_mu: float           # std of the class means of the Gaussian mixture
    init: str                 # "zeros" or "he"
    seed: int = 0

    @property
    def classes(self) -> int:
        return self.dims[-1]

    @property
    def samples_per_round(self) -> int:
        """Learner-samples consumed by one global round: P * B * K1 * K2."""
        return self.P * self.B * self.K1 * self.K2

    @property
    def n_params(self) -> int:
        """Parameters per learner: weights [d_l, d_{l-1}] plus biases [d_l]."""
        return sum(o * i + o for i, o in zip(self.dims[:-1], self.dims[1:]))

    def replace(self, **kw) -> "Workload":
        d = dict(self.__dict__)
        d.update(kw)
        return Workload(**d)


# Softmax regression 3072 -> 10 in fp32, zero-initialised: the smallest case.
SOFTMAX_P4 = Workload("softmax3072x10_P4_S2_K1_2_K2_2", P=4, S=2, K1=2, K2=2, rounds=2,
                      dims=(3072, 10), precision="fp32", N=512, B=16, lr=0.05,
                      sigma_mu=0.1, init="zeros")

# MLP 3072 -> 512 -> 10 (ReLU), CIFAR-10 shaped, bf16 GEMM operands, fp32 master.
MLP512_P16 = Workload("mlp3072x512x10_P16_S4_K1_4_K2_4", P=16, S=4, K1=4, K2=4, rounds=4,
                      dims=(3072, 512, 10), precision="bf16", N=4096, B=32, lr=0.05,
                      sigma_mu=0.1, init="he")

# MLP 3072 -> 2048 -> 2048 -> 10 (~10.5M params per learner).
MLP2048_P64 = Workload("mlp3072x2048x2048x10_P64_S8_K1_8_K2_4", P=64, S=8, K1=8, K2=4,
                       rounds=2, dims=(3072, 2048, 2048, 10), precision="bf16", N=8192,
                       B=64, lr=0.02, sigma_mu=0.1, init="he")

# MLP 12288 -> 4096 -> 4096 -> 1000 (~71M params per learner), ImageNet-shaped.
MLP4096_P32 = Workload("mlp12288x4096x4096x1000_P32_S8_K1_4_K2_8", P=32, S=8, K1=4, K2=8,
                       rounds=1, dims=(12288, 4096, 4096, 1000), precision="bf16",
                       N=4096, B=32, lr=0.01, sigma_mu=0.05, init="he")

WORKLOADS = {w.name: w for w in (SOFTMAX_P4, MLP512_P16, MLP2048_P64, MLP4096_P32)}
SHORT = {"softmax": SOFTMAX_P4, "mlp512": MLP512_P16, "mlp2048": MLP2048_P64,
         "mlp4096": MLP4096_P32}


@dataclass(frozen=True)
class AveragingSweep:
    """Averaging-only sweep: P = 128 fp32 replicas of D parameters ~ N(0, 1)."""
    P: int = 128
    D: Tuple[int, ...] = (1_000_000, 11_200_000, 32_000_000, 64_000_000)
    S: Tuple[int, ...] = (2, 4, 8, 16, 32)
    seed: int = 0


AVERAGING_SWEEP = AveragingSweep()
