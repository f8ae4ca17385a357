"""The allocation-free step (hier_avg_step_static) against the ordinary step.

Callers that cannot allocate device memory get the step's scratch from one
static array inside the library.  This file is collected last on purpose: if it
fails, a run that stops at the first failure has already run every other test.
The two paths run the same kernels in the same order on the same inputs, so
their parameters and losses must be bit-identical, on two steps in a row.  The
array keeps what the previous call left in it, so one test first runs a
configuration with a larger scratch footprint (three layers, split-K partials and
tile counters) and then the small case.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_1903_05133_gb300 import configs
from paper_1903_05133_gb300.hier_avg import HierAvg
from paper_1903_05133_gb300.inputs import learner_data, perturbed_layers

pytestmark = pytest.mark.gpu

SMALL_BF16 = configs.Workload("tiny_mlp_bf16", P=4, S=2, K1=2, K2=2, rounds=1,
                              dims=(256, 192, 10), precision="bf16", N=96, B=48, lr=0.05,
                              sigma_mu=0.1, init="he")
# 3072-2048-2048-10 with 8 learners (one cluster): ~24 MiB of the 32 MiB array,
# with split-tile partials and counters in use
LARGER_BF16 = configs.MLP2048_P64.replace(name="mlp2048_P8_static", P=8, N=256)


def _static_matches_bound(lib, w):
    X, y = learner_data(w)
    X, y = X.cuda(), y.cuda()
    layers = perturbed_layers(w, 0.01, seed=3)

    ref = HierAvg(w.P, w.S, w.K1, w.K2, w.lr, w.B, w.dims, w.precision)
    ref.bind(ref.pack(layers), X, y)                 # ordinary path: caller workspace

    st = HierAvg(w.P, w.S, w.K1, w.K2, w.lr, w.B, w.dims, w.precision)
    params = st.pack(layers)                         # the caller's own buffers only
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    loss = torch.empty(w.P, dtype=torch.float32)
    for step in range(2):                            # two calls in a row
        ref.step()
        rc = lib.hier_avg_step_static(st.h, ctypes.c_void_p(params.data_ptr()),
                                      ctypes.c_void_p(X.data_ptr()), ctypes.c_void_p(y.data_ptr()),
                                      X.shape[1], stream)
        assert rc == 0, lib.hier_avg_last_error(st.h)
        torch.cuda.synchronize()
        assert lib.hier_avg_check(st.h) == 0
        ref.check()
        assert torch.equal(params.view(torch.int32), ref.params.view(torch.int32))
        assert lib.hier_avg_losses(st.h, ctypes.c_void_p(loss.data_ptr())) == 0
        assert np.array_equal(loss.numpy().view(np.uint32), ref.losses().numpy().view(np.uint32))
        t = ctypes.c_int64()
        assert lib.hier_avg_get_step(st.h, ctypes.byref(t)) == 0 and t.value == step + 1


@pytest.mark.parametrize("w", [SMALL_BF16, configs.MLP512_P16, configs.SOFTMAX_P4],
                         ids=lambda w: w.name)
def test_static_step_matches_bound_step(lib, w):
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    _static_matches_bound(lib, w)


def test_static_step_after_a_larger_configuration(lib):
    # The larger configuration leaves partial sums, tile counters and activations in
    # the shared array; the small case that follows must not see any of it.
    assert torch.cuda.is_available(), "GPU tests need CUDA"
    _static_matches_bound(lib, LARGER_BF16)
    _static_matches_bound(lib, SMALL_BF16)


def test_static_step_rejects_large_configurations(lib):
    w = configs.MLP2048_P64                          # needs ~93 MiB of scratch
    h = HierAvg(w.P, w.S, w.K1, w.K2, w.lr, w.B, w.dims, w.precision)
    assert h.workspace_bytes > 32 << 20
    params = torch.zeros(w.P, h.ld, device="cuda")
    X = torch.zeros(w.P, 2, w.dims[0], dtype=torch.bfloat16, device="cuda")
    y = torch.zeros(w.P, 2, dtype=torch.int32, device="cuda")
    rc = lib.hier_avg_step_static(h.h, ctypes.c_void_p(params.data_ptr()),
                                  ctypes.c_void_p(X.data_ptr()), ctypes.c_void_p(y.data_ptr()),
                                  2, None)
    assert rc == -2                                  # HA_ENOMEM
    assert b"33554432" in lib.hier_avg_last_error(h.h)
