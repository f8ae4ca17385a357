"""GPU parity of the local / global averages (Algorithm 1, Sec. 3.1): the CUDA
kernels, called through the C ABI, must be bit-identical to the oracle's
fixed-order tree on the same inputs."""
import numpy as np
import pytest
import torch

import oracle
from paper_1903_05133_gb300 import hier_avg as ha
from paper_1903_05133_gb300.inputs import replica_matrix

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda(lib):
    assert torch.cuda.is_available(), "GPU tests need CUDA"


def _bits(a: np.ndarray) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)


def _gpu(w_host: np.ndarray, op, S=None, ld=None, offset=0):
    P, D = w_host.shape
    ld = D if ld is None else ld
    big = torch.full((P, ld + offset + 8), float("nan"), dtype=torch.float32, device="cuda")
    view = big[:, offset:offset + D]
    view.copy_(torch.from_numpy(w_host))
    if op == "local":
        ha.local_average_buffer(view, S)
    elif op == "global":
        ha.global_average_buffer(view)
    else:
        ha.local_global_average_buffer(view, S)
    torch.cuda.synchronize()
    out = big.cpu().numpy()
    # nothing outside the [P, D] window may change
    assert np.all(np.isnan(out[:, :offset])) and np.all(np.isnan(out[:, offset + D:]))
    return out[:, offset:offset + D]


def _oracle(w_host, op, S=None):
    w = w_host.copy()
    if op == "local":
        oracle.local_average(w, S)
    elif op == "global":
        oracle.global_average(w)
    else:
        oracle.local_average(w, S)
        oracle.global_average(w)
    return w


CASES = [(4, 2, 1000), (4, 2, 8), (8, 4, 4099), (6, 3, 1001), (16, 4, 4096), (128, 32, 10000),
         (128, 2, 33333), (16, 16, 777), (5, 5, 64), (7, 1, 100), (12, 4, 4099), (64, 8, 65536),
         (32, 8, 12345), (1, 1, 17), (3, 1, 5), (128, 128, 2048), (24, 6, 3000)]


@pytest.mark.parametrize("P,S,D", CASES)
@pytest.mark.parametrize("op", ["local", "global", "local_global"])
def test_bitexact(P, S, D, op):
    w = replica_matrix(P, D, seed=P * 1000 + S).numpy()
    got = _gpu(w, op, S)
    want = _oracle(w, op, S)
    assert np.array_equal(_bits(got), _bits(want))


@pytest.mark.parametrize("offset,ld_extra", [(1, 3), (0, 5), (2, 0), (4, 60)])
def test_strided_and_misaligned(offset, ld_extra):
    # unaligned base and odd leading dimensions take the scalar path for part or all
    P, S, D = 8, 4, 1037
    w = replica_matrix(P, D, seed=77).numpy()
    for op in ("local", "global", "local_global"):
        got = _gpu(w, op, S, ld=D + ld_extra, offset=offset)
        assert np.array_equal(_bits(got), _bits(_oracle(w, op, S)))


def test_edge_values():
    P, S, D = 8, 2, 64
    rng = np.random.default_rng(5)
    w = rng.standard_normal((P, D)).astype(np.float32)
    w[:, 0] = -0.0
    w[::2, 1] = 0.0
    w[:, 2] = np.float32(1e-45) * np.arange(1, P + 1)            # subnormals
    w[:, 3] = np.float32(1e-40)
    w[0, 4] = np.inf
    w[:, 5] = np.float32(3e38)                                     # sums overflow to inf
    w[:, 6] = np.float32([1, 2 ** 24, 1, -2 ** 24, 3, 5, 7, 11])   # order-sensitive
    w[:, 7] = np.float32(1.17549435e-38)                           # smallest normal
    for op in ("local", "global", "local_global"):
        got = _gpu(w, op, S)
        want = _oracle(w, op, S)
        assert np.array_equal(_bits(got), _bits(want)), op


def test_invariants_after_average():
    P, S, D = 16, 4, 5000
    w = replica_matrix(P, D, seed=3).numpy()
    got = _gpu(w, "local", S)
    for g in range(P // S):
        blk = _bits(got[g * S:(g + 1) * S])
        assert np.all(blk == blk[0])
    got = _gpu(w, "local_global", S)
    assert np.all(_bits(got) == _bits(got[0]))


@pytest.mark.parametrize("D", [1_000_000, 64_000_000])
def test_sweep_size_sampled(D):
    # The averaging sweep at its full size (P = 128): every column is independent,
    # so the oracle checks a random sample of columns one by one.
    P = 128
    torch.manual_seed(0)
    w = torch.randn(P, D, device="cuda", dtype=torch.float32)
    cols = torch.randint(0, D, (512,), device="cuda")
    cols = torch.cat([cols, torch.tensor([0, D - 1], device="cuda")])
    for op, S in (("local", 2), ("local", 32), ("local_global", 8), ("global", None)):
        src = w[:, cols].cpu().numpy()
        work = w.clone()
        if op == "local":
            ha.local_average_buffer(work, S)
        elif op == "global":
            ha.global_average_buffer(work)
        else:
            ha.local_global_average_buffer(work, S)
        torch.cuda.synchronize()
        got = work[:, cols].cpu().numpy()
        del work
        assert np.array_equal(_bits(got), _bits(_oracle(src, op, S))), (op, S)
