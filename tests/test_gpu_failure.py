"""Failure detection on the GPU without a fault: a bounded device wait that runs
out.  hier_avg_wait_selftest runs the library's two kinds of bounded wait (an
acquire spin on a global flag, an mbarrier phase wait) on conditions nothing
satisfies, with a short limit; the kernel records the timeout and returns, the
host reads HA_ETIMEOUT from hier_avg_check, and the same handle then steps
normally, bit for bit like a handle that never timed out."""
import time

import pytest
import torch

from paper_1903_05133_gb300 import configs
from paper_1903_05133_gb300._lib import HierAvgError
from paper_1903_05133_gb300.hier_avg import HierAvg
from paper_1903_05133_gb300.inputs import learner_data, perturbed_layers

pytestmark = pytest.mark.gpu

HA_ETIMEOUT = -5
W = configs.Workload("tiny_mlp_bf16", P=4, S=2, K1=2, K2=2, rounds=1, dims=(256, 192, 10),
                     precision="bf16", N=96, B=48, lr=0.05, sigma_mu=0.1, init="he")


def _handle():
    X, y = learner_data(W, device="cuda")
    ha = HierAvg(W.P, W.S, W.K1, W.K2, W.lr, W.B, W.dims, W.precision)
    ha.bind(ha.pack(perturbed_layers(W, 0.01, seed=5)), X, y)
    return ha


def test_bounded_wait_times_out_and_the_context_stays_usable(lib):
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    ha, ref = _handle(), _handle()
    ha.check()
    limit_ms = 50.0
    t0 = time.perf_counter()
    ha.wait_selftest(limit_ms)
    with pytest.raises(HierAvgError) as e:
        ha.check()                        # synchronises, then reads the error word
    elapsed = time.perf_counter() - t0
    assert e.value.status == HA_ETIMEOUT
    # two waits of limit_ms each at the peak clock (longer at a lower clock)
    assert 2 * limit_ms / 1e3 * 0.9 <= elapsed < 10.0
    # the word was cleared by the check; the handle and the context work as before
    ha.check()
    for h in (ha, ref):
        h.round()
        h.check()
    assert torch.equal(ha.params.view(torch.int32), ref.params.view(torch.int32))


def test_wait_selftest_rejects_bad_limits(lib):
    ha = _handle()
    for bad in (0.0, 2e4):                # 0 ms and 20 s
        with pytest.raises(HierAvgError) as e:
            ha.wait_selftest(bad)
        assert e.value.status == -1       # HA_EINVAL
    ha.check()
