"""Hier-AVG (Zhou & Cong, hierarchical averaging SGD) on one GB300: all P learners
as rows of a learner-indexed fp32 matrix, local SGD steps on tcgen05 tensor cores,
local and global averages as in-memory reductions over the learner axis.

The CUDA library is loaded lazily on first use and there is no CPU fallback.
"""
from .configs import WORKLOADS, SHORT, Workload, AVERAGING_SWEEP  # noqa: F401


def __getattr__(name):
    if name in ("HierAvg", "local_average_buffer", "global_average_buffer",
                "local_global_average_buffer"):
        from . import hier_avg
        return getattr(hier_avg, name)
    raise AttributeError(name)
