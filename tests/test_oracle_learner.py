"""Pins of the oracle's local SGD step (Algorithm 1 inner loop): the bf16 operand
rounding against torch's converter, the softmax cross-entropy gradient against
torch, and the MLP backward pass against finite differences and torch autograd."""
import numpy as np
import pytest
import torch

from oracle import learner as ln


def _torch_bf16(x: np.ndarray) -> np.ndarray:
    return torch.from_numpy(x).to(torch.bfloat16).to(torch.float32).numpy()


def test_bf16_round_random():
    rng = np.random.default_rng(0)
    x = (rng.standard_normal(1_000_000) * 10.0 ** rng.integers(-40, 38, 1_000_000)).astype(np.float32)
    got, want = ln.bf16_round(x), _torch_bf16(x)
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


def test_bf16_round_edges():
    f = np.float32
    one = f(1.0)
    x = np.array([
        0.0, -0.0, np.inf, -np.inf,
        np.finfo(np.float32).max, -np.finfo(np.float32).max,
        1e-45, -1e-45, 1.1754942e-38, 1.17549435e-38,
        one + f(2.0 ** -8),            # tie between 1 and 1+2^-7 -> even (1)
        one + f(3 * 2.0 ** -8),        # tie between 1+2^-7 and 1+2^-6 -> even (1+2^-6)
        one + f(2.0 ** -8) + f(2.0 ** -20),   # just above the tie -> up
        f(3.3895314e38),               # rounds up to Inf
    ], dtype=np.float32)
    got, want = ln.bf16_round(x), _torch_bf16(x)
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))
    assert got[10] == 1.0 and got[11] == np.float32(1 + 2.0 ** -6)
    nan = np.array([np.nan, -np.nan], dtype=np.float32)
    r = ln.bf16_round(nan)
    assert np.all(np.isnan(r))
    assert np.array_equal(np.signbit(r), np.signbit(nan))


def test_softmax_xent_against_torch():
    rng = np.random.default_rng(1)
    for B, C in ((4, 3), (16, 10), (32, 1000)):
        Z = rng.standard_normal((B, C)) * 5
        y = rng.integers(0, C, B)
        loss, dZ = ln.softmax_xent_grad(Z, y, B)
        zt = torch.tensor(Z, dtype=torch.float64, requires_grad=True)
        lt = torch.nn.functional.cross_entropy(zt, torch.tensor(y), reduction="mean")
        lt.backward()
        assert abs(loss - lt.item()) < 1e-12 * max(1, abs(lt.item()))
        assert np.allclose(dZ, zt.grad.numpy(), rtol=1e-12, atol=1e-15)


def _tiny_net(dims, B, seed):
    rng = np.random.default_rng(seed)
    Ws = [rng.standard_normal((o, i)) * np.sqrt(2.0 / i) for i, o in zip(dims[:-1], dims[1:])]
    bs = [rng.standard_normal(o) * 0.1 for o in dims[1:]]
    X = rng.standard_normal((B, dims[0]))
    y = rng.integers(0, dims[-1], B)
    return Ws, bs, X, y


def test_mlp_gradient_finite_differences():
    Ws, bs, X, y = _tiny_net((7, 5, 3), 4, 11)
    loss, gW, gb = ln.mlp_forward_backward(Ws, bs, X, y, "f64")
    h = 1e-6

    def L(Ws_, bs_):
        return ln.mlp_forward_backward(Ws_, bs_, X, y, "f64")[0]

    for l in range(2):
        for idx in np.ndindex(Ws[l].shape):
            Wp = [w.copy() for w in Ws]
            Wm = [w.copy() for w in Ws]
            Wp[l][idx] += h
            Wm[l][idx] -= h
            fd = (L(Wp, bs) - L(Wm, bs)) / (2 * h)
            assert abs(fd - gW[l][idx]) < 1e-7, (l, idx)
        for k in range(bs[l].shape[0]):
            bp = [b.copy() for b in bs]
            bm = [b.copy() for b in bs]
            bp[l][k] += h
            bm[l][k] -= h
            fd = (L(Ws, bp) - L(Ws, bm)) / (2 * h)
            assert abs(fd - gb[l][k]) < 1e-7


def test_mlp_gradient_against_autograd():
    dims = (12, 9, 7, 4)
    Ws, bs, X, y = _tiny_net(dims, 6, 12)
    loss, gW, gb = ln.mlp_forward_backward(Ws, bs, X, y, "f64")
    tW = [torch.tensor(w, requires_grad=True) for w in Ws]
    tb = [torch.tensor(b, requires_grad=True) for b in bs]
    h = torch.tensor(X)
    for l in range(3):
        h = h @ tW[l].T + tb[l]
        if l < 2:
            h = torch.relu(h)
    lt = torch.nn.functional.cross_entropy(h, torch.tensor(y))
    lt.backward()
    assert abs(loss - lt.item()) < 1e-12
    for l in range(3):
        assert np.allclose(gW[l], tW[l].grad.numpy(), rtol=1e-12, atol=1e-14)
        assert np.allclose(gb[l], tb[l].grad.numpy(), rtol=1e-12, atol=1e-14)


@pytest.mark.parametrize("mode,tol", [("fp32", 1e-5), ("bf16", 3e-2), ("bf16_acc32", 3e-2)])
def test_reduced_precision_modes_track_f64(mode, tol):
    Ws, bs, X, y = _tiny_net((64, 48, 10), 16, 13)
    X = ln.bf16_round(X.astype(np.float32)).astype(np.float64)
    Ws32 = [w.astype(np.float32) for w in Ws]
    bs32 = [b.astype(np.float32) for b in bs]
    _, gW, gb = ln.mlp_forward_backward([w.astype(np.float64) for w in Ws32],
                                        [b.astype(np.float64) for b in bs32], X, y, "f64")
    _, gW2, gb2 = ln.mlp_forward_backward(Ws32, bs32, X, y, mode)
    for a, b in zip(gW + gb, gW2 + gb2):
        assert np.max(np.abs(a - b)) <= tol * np.max(np.abs(a))
        assert b.dtype == np.float64


def test_bf16_mode_rounds_operands():
    # With W exactly bf16-representable and a single layer, the bf16 and fp32
    # modes see identical operands in the forward pass, so their losses agree.
    Ws, bs, X, y = _tiny_net((32, 10), 8, 14)
    Ws = [ln.bf16_round(w.astype(np.float32)).astype(np.float64) for w in Ws]
    X = ln.bf16_round(X.astype(np.float32)).astype(np.float64)
    l1 = ln.mlp_forward_backward(Ws, bs, X, y, "bf16")[0]
    l2 = ln.mlp_forward_backward(Ws, bs, X, y, "fp32")[0]
    assert l1 == l2
    # ... while a W that is not bf16-exact changes the bf16 loss.
    Ws2 = [w + 1e-3 * np.float64(2.0 ** -9) for w in Ws]
    assert ln.mlp_forward_backward(Ws2, bs, X, y, "bf16")[0] != ln.mlp_forward_backward(Ws2, bs, X, y, "fp32")[0]


def test_sgd_update_fp32_is_separate_multiply_subtract():
    rng = np.random.default_rng(15)
    p = rng.standard_normal(1000).astype(np.float32)
    g = rng.standard_normal(1000).astype(np.float32)
    got = ln.sgd_update(p, g, 0.05, "fp32")
    lr = np.float32(0.05)
    # reference through float64: each fp32 op is the exact result rounded once
    step = (np.float64(lr) * g.astype(np.float64)).astype(np.float32)
    want = (p.astype(np.float64) - step.astype(np.float64)).astype(np.float32)
    assert np.array_equal(got, want)
    assert got.dtype == np.float32


def _bf16_step_in_torch(Ws, bs, X, y):
    """One bf16-mode step written independently of the oracle, in torch float64:
    every GEMM operand is cast explicitly with .to(bfloat16).to(float64), every
    stored value with .to(float32).to(float64).  Operands: X, W_l and H_{l-1} in
    the forward; dZ_l and H_{l-1} in dW_l; dZ_l and W_l (before its update) in the
    dX product.  Bias add, ReLU, softmax cross-entropy and the bias gradient stay
    in fp32 storage."""
    f64, f32, b16 = torch.float64, torch.float32, torch.bfloat16

    def bf(t):
        return t.to(f32).to(b16).to(f64)

    def st(t):
        return t.to(f32).to(f64)

    Wt = [torch.tensor(w, dtype=f64) for w in Ws]
    bt = [torch.tensor(b, dtype=f64) for b in bs]
    yt = torch.tensor(y)
    B = X.shape[0]
    Hs = [bf(torch.tensor(X, dtype=f64))]
    Zs = []
    for l in range(len(Wt)):
        z = st(st(Hs[l] @ bf(Wt[l]).T) + bt[l])
        Zs.append(z)
        if l < len(Wt) - 1:
            Hs.append(bf(st(torch.relu(z))))
    z = Zs[-1].clone().requires_grad_(True)
    loss = torch.nn.functional.cross_entropy(z, yt, reduction="mean")
    loss.backward()
    dz = st(z.grad)
    gW, gb = [None] * len(Wt), [None] * len(Wt)
    for l in reversed(range(len(Wt))):
        gW[l] = st(bf(dz).T @ Hs[l])
        gb[l] = st(dz.sum(dim=0))
        if l > 0:
            dh = st(bf(dz) @ bf(Wt[l]))
            dz = st(dh * (Hs[l] > 0).to(f64))
    return loss.item(), [g.numpy() for g in gW], [g.numpy() for g in gb]


@pytest.mark.parametrize("dims,B", [((40, 24, 16, 10), 12), ((96, 72, 56, 13), 20)])
def test_bf16_mode_operand_placement_against_torch(dims, B):
    # Pins WHICH operands the bf16 mode rounds: a dropped or extra bf16 rounding of
    # any one GEMM operand moves a gradient by ~2^-9 relative, far above 1e-12.
    # X is drawn off the bf16 grid so that its rounding is checked too.
    Ws, bs, X, y = _tiny_net(dims, B, 21)
    Ws = [w.astype(np.float32).astype(np.float64) for w in Ws]
    bs = [b.astype(np.float32).astype(np.float64) for b in bs]
    X = X.astype(np.float32).astype(np.float64)
    loss, gW, gb = ln.mlp_forward_backward(Ws, bs, X, y, "bf16")
    loss_t, gW_t, gb_t = _bf16_step_in_torch(Ws, bs, X, y)
    assert abs(loss - loss_t) <= 1e-12 * max(1.0, abs(loss_t))
    for l in range(len(Ws)):
        for a, b in ((gW[l], gW_t[l]), (gb[l], gb_t[l])):
            assert np.max(np.abs(a - b)) <= 1e-12 * np.max(np.abs(b)), l
    # the placement matters at this size: the fp32 mode differs from it
    _, gW32, _ = ln.mlp_forward_backward(Ws, bs, X, y, "fp32")
    assert all(np.max(np.abs(a - b)) > 1e-6 * np.max(np.abs(b)) for a, b in zip(gW32, gW_t))
