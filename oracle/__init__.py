"""CPU oracle for Hier-AVG (Zhou & Cong, "A Distributed Hierarchical Averaging SGD
Algorithm: Trading Local Reductions for Global Reductions").

TEST INFRASTRUCTURE ONLY.  Nothing in the product path imports, calls or links
this package: only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline
leg of ``bench.py`` may use it.  It shares no code with the CUDA path; both sides
see the same seeded inputs and nothing else.

It is plain and slow on purpose: numpy arrays, explicit loops over learners,
groups and tree levels, numpy matrix products as the only library primitive.

Modules
  averaging  local and global averages of Algorithm 1 (Sec. 3.1), fixed-order tree
  learner    one learner's minibatch SGD step (Algorithm 1 inner loop) for a ReLU
             MLP with mean softmax cross-entropy, in three precision modes
  algorithm  the Algorithm 1 driver (rounds, local blocks, local steps)

Parity pins live in ``tests/test_oracle_*.py``.  The theorem bounds of Sec. 3.2-3.5
contain unknown constants (L, M, M_G) and are not computed here.
"""
from .averaging import tree_sum, group_mean, local_average, global_average
from .learner import (bf16_round, softmax_xent_grad, mlp_forward_backward, sgd_update,
                      MLPProblem, QuadraticProblem)
from .algorithm import HierAvgOracle, batch_rows, batch_rows_from

__all__ = [
    "tree_sum", "group_mean", "local_average", "global_average",
    "bf16_round", "softmax_xent_grad", "mlp_forward_backward", "sgd_update",
    "MLPProblem", "QuadraticProblem", "HierAvgOracle", "batch_rows", "batch_rows_from",
]
