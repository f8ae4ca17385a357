"""Pins of the oracle's Algorithm 1 driver against what the paper fixes:
special cases that reduce to synchronous SGD and K-AVG (Sec. 3.1), the
synchronisation invariants, and the closed-form trajectory of a noise-free
least-squares problem."""
import numpy as np
import pytest
import torch

from oracle import HierAvgOracle, MLPProblem, QuadraticProblem, batch_rows, batch_rows_from
from oracle import learner as ln


def _mlp_setup(P, dims, N, B, seed=0):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((P, N, dims[0]))
    y = rng.integers(0, dims[-1], (P, N))
    params = []
    for i, o in zip(dims[:-1], dims[1:]):
        W = rng.standard_normal((o, i)) * np.sqrt(2.0 / i)
        b = rng.standard_normal(o) * 0.1
        params += [np.broadcast_to(W, (P, o, i)).copy(), np.broadcast_to(b, (P, o)).copy()]
    return X, y, params


def _torch_big_batch_step(params0, X, y, rows_per_learner, lr, dims):
    """One SGD step on the union of all learners' mini-batches (batch P*B), with
    torch autograd in float64: an implementation independent of the oracle."""
    P = X.shape[0]
    Xb = np.concatenate([X[j, rows_per_learner] for j in range(P)])
    yb = np.concatenate([y[j, rows_per_learner] for j in range(P)])
    t = [torch.tensor(p[0], requires_grad=True) for p in params0]
    h = torch.tensor(Xb)
    L = len(dims) - 1
    for l in range(L):
        h = h @ t[2 * l].T + t[2 * l + 1]
        if l < L - 1:
            h = torch.relu(h)
    torch.nn.functional.cross_entropy(h, torch.tensor(yb)).backward()
    return [(p - lr * p.grad).detach().numpy() for p in t]


@pytest.mark.parametrize("P,S", [(4, 2), (4, 1), (6, 3), (4, 4)])
def test_sync_sgd_special_case(P, S):
    # K1 = 1 and one local average per round: a round is one step of minibatch
    # SGD with batch P*B (Sec. 3.1: K2 = K1 = 1 gives synchronous parallel SGD).
    dims, N, B, lr = (6, 5, 3), 40, 4, 0.1
    X, y, params = _mlp_setup(P, dims, N, B, seed=P + S)
    o = HierAvgOracle(P, S, 1, 1, lr, MLPProblem(X, y, B, 2, "f64"), params, "f64")
    o.round()
    want = _torch_big_batch_step(params, X, y, batch_rows(0, B, N), lr, dims)
    for got, w in zip(o.params, want):
        for j in range(P):
            assert np.allclose(got[j], w, rtol=1e-12, atol=1e-13)


def test_sync_sgd_with_growing_batch():
    # Theorem 3.3's growing batch: round n uses B_n rows per learner, read where the
    # previous step's batch ended.  With K1 = 1, S = P the round is one step of
    # minibatch SGD on the P * B_n rows (torch autograd, independent of the oracle),
    # including the wrap past the end of the data.
    P, dims, N, lr = 4, (6, 5, 3), 20, 0.1
    X, y, params = _mlp_setup(P, dims, N, 4, seed=11)
    o = HierAvgOracle(P, P, 1, 1, lr, MLPProblem(X, y, 4, 2, "f64"), params, "f64")
    start, cur = 0, [p.copy() for p in params]
    for Bn in (2, 3, 5, 8, 7):
        o.B = Bn
        o.round()
        want = _torch_big_batch_step(cur, X, y, batch_rows_from(start, Bn, N), lr, dims)
        start += Bn
        for got, w in zip(o.params, want):
            for j in range(P):
                assert np.allclose(got[j], w, rtol=1e-12, atol=1e-13)
        cur = [p.copy() for p in o.params]
    assert o.cursor == 25 and o.t == 5


def test_batch_rows_from_continues_a_cursor():
    assert list(batch_rows_from(18, 4, 20)) == [18, 19, 0, 1]
    assert list(batch_rows_from(8, 4, 10)) == list(batch_rows(2, 4, 10))


def _kavg(params, problem, P, K, lr, rounds):
    """K-AVG written independently: K local steps per learner, then the mean over
    learners (numpy mean, not the oracle's tree)."""
    ps = [p.copy() for p in params]
    t = 0
    for _ in range(rounds):
        for _k in range(K):
            for j in range(P):
                g = problem.gradients(j, batch_rows(t, problem.B, problem.X.shape[1]),
                                      [p[j] for p in ps])
                for p, gg in zip(ps, g):
                    p[j] = p[j] - lr * gg
            t += 1
        for p in ps:
            p[:] = p.mean(axis=0)
    return ps


@pytest.mark.parametrize("K1,K2", [(2, 3), (3, 1), (1, 4)])
def test_s1_is_kavg(K1, K2):
    # S = 1: the local average is the identity, so Hier-AVG is K-AVG with
    # K = K1 * K2 local steps per global average (Sec. 3.1).
    P, dims, N, B, lr = 4, (6, 5, 3), 64, 4, 0.1
    X, y, params = _mlp_setup(P, dims, N, B, seed=K1 * 10 + K2)
    o = HierAvgOracle(P, 1, K1, K2, lr, MLPProblem(X, y, B, 2, "f64"), params, "f64")
    o.round()
    o.round()
    want = _kavg(params, MLPProblem(X, y, B, 2, "f64"), P, K1 * K2, lr, 2)
    for a, b in zip(o.params, want):
        assert np.allclose(a, b, rtol=1e-12, atol=1e-13)


@pytest.mark.parametrize("P,S,K1", [(4, 2, 3), (6, 3, 2), (8, 4, 1)])
def test_one_local_block_is_kavg(P, S, K1):
    # beta = 1 (the paper's K2 = K1): the global mean of equal-size cluster means
    # is the global mean, so a round equals K-AVG with K = K1.
    dims, N, B, lr = (6, 5, 3), 64, 4, 0.1
    X, y, params = _mlp_setup(P, dims, N, B, seed=P * S + K1)
    o = HierAvgOracle(P, S, K1, 1, lr, MLPProblem(X, y, B, 2, "f64"), params, "f64")
    o.round()
    want = _kavg(params, MLPProblem(X, y, B, 2, "f64"), P, K1, lr, 1)
    for a, b in zip(o.params, want):
        assert np.allclose(a, b, rtol=1e-12, atol=1e-13)


def test_synchronisation_invariants_fp32():
    P, S, dims, N, B = 8, 4, (16, 12, 5), 64, 8
    X, y, params = _mlp_setup(P, dims, N, B, seed=3)
    X = ln.bf16_round(X.astype(np.float32)).astype(np.float64)
    o = HierAvgOracle(P, S, 2, 2, 0.05, MLPProblem(X, y, B, 2, "bf16"), params, "bf16")
    o.step()
    o.step()
    assert not np.array_equal(o.params[0][0], o.params[0][1])     # learners diverged
    o.local_average()
    for p in o.params:
        for g in range(P // S):
            blk = p[g * S:(g + 1) * S].view(np.uint32)
            assert np.all(blk == blk[0])
    assert not np.array_equal(o.params[0][0], o.params[0][S])     # clusters differ
    o.global_average()
    for p in o.params:
        assert np.all(p.view(np.uint32) == p[0].view(np.uint32))
        assert p.dtype == np.float32


@pytest.mark.parametrize("P,S,K1,K2", [(4, 2, 3, 2), (6, 3, 2, 4), (8, 8, 1, 3), (8, 1, 5, 2),
                                       (12, 4, 4, 1)])
def test_quadratic_closed_form(P, S, K1, K2):
    # f_j(w) = 0.5 ||w - c_j||^2: each step maps w - c_j to (1 - g)(w - c_j).  From
    # Algorithm 1, after b local blocks a cluster G holds
    #     cbar_G + (1 - g)^(b K1) (w~ - cbar_G),
    # and after a round w~' - cbar = (1 - g)^(K1 K2) (w~ - cbar) for every S and K1.
    D, gamma = 5, 0.3
    rng = np.random.default_rng(P + S + K1 + K2)
    c = rng.standard_normal((P, D))
    w0 = rng.standard_normal(D)
    o = HierAvgOracle(P, S, K1, K2, gamma, QuadraticProblem(c),
                      [np.broadcast_to(w0, (P, D)).copy()], "f64")
    r = 1.0 - gamma
    wt = w0.copy()
    cbar = c.mean(axis=0)
    for _round in range(3):
        for b in range(1, K2 + 1):
            for _ in range(K1):
                o.step()
            o.local_average()
            for g in range(P // S):
                cg = c[g * S:(g + 1) * S].mean(axis=0)
                want = cg + r ** (b * K1) * (wt - cg)
                assert np.allclose(o.params[0][g * S:(g + 1) * S], want, rtol=0, atol=1e-12)
        o.global_average()
        wt = cbar + r ** (K1 * K2) * (wt - cbar)
        assert np.allclose(o.params[0], wt, rtol=0, atol=1e-12)


@pytest.mark.parametrize("P,S,K1,G", [(8, 4, 20, 43), (8, 2, 3, 7), (4, 2, 5, 5), (6, 3, 4, 2),
                                      (8, 1, 3, 8), (12, 4, 2, 9)])
def test_quadratic_free_global_interval(P, S, K1, G):
    # Free global interval of G local steps (Sec. 3.1; Sec. 4's ImageNet run: K1 = 20,
    # G = 43) and a diminishing step size gamma_n = gamma_0 / (n + 1) (Theorem 3.3).
    # With f_j(w) = 0.5 ||w - c_j||^2 and q = G // K1 local averages inside the round
    # (r = 1 - gamma_n): after the b-th, cluster C holds cbar_C + r^(b K1) (w~ - cbar_C);
    # before the global average learner j holds c_j + r^(G - q K1) (w_C - c_j), where
    # w_C is its cluster's value after the q-th average (w~ if q = 0); and the round
    # maps w~ - cbar to r^G (w~ - cbar).
    D, gamma0 = 4, 0.25
    rng = np.random.default_rng(P + S + K1 + G)
    c = rng.standard_normal((P, D))
    w0 = rng.standard_normal(D)
    o = HierAvgOracle(P, S, K1, 1, gamma0, QuadraticProblem(c),
                      [np.broadcast_to(w0, (P, D)).copy()], "f64", global_steps=G)
    assert o.G == G
    q, rem = divmod(G, K1)
    wt = w0.copy()
    cbar = c.mean(axis=0)
    cl = np.repeat(c.reshape(P // S, S, D).mean(axis=1), S, axis=0)   # cbar of j's cluster
    for n in range(3):
        o.lr = gamma0 / (n + 1)
        r = 1.0 - o.lr
        for step in range(1, G + 1):
            o.step()
            if step % K1 == 0:
                o.local_average()
                b = step // K1
                assert np.allclose(o.params[0], cl + r ** (b * K1) * (wt - cl), rtol=0, atol=1e-12)
        wc = cl + r ** (q * K1) * (wt - cl) if q > 0 else np.broadcast_to(wt, (P, D))
        assert np.allclose(o.params[0], c + r ** rem * (wc - c), rtol=0, atol=1e-12)
        o.global_average()
        wt = cbar + r ** G * (wt - cbar)
        assert np.allclose(o.params[0], wt, rtol=0, atol=1e-12)


@pytest.mark.parametrize("K1,G", [(20, 43), (3, 7), (4, 2)])
def test_round_with_free_interval_follows_its_definition(K1, G):
    # round() = G steps with a local average after every K1-th and the global average
    # at the end; checked against the same sequence of calls on a second oracle (MLP).
    P, S, dims, N, B = 4, 2, (12, 8, 5), 40, 4
    X, y, params = _mlp_setup(P, dims, N, B, seed=5)
    o1 = HierAvgOracle(P, S, K1, 1, 0.05, MLPProblem(X, y, B, 2, "fp32"), params, "fp32",
                       global_steps=G)
    o2 = HierAvgOracle(P, S, K1, 1, 0.05, MLPProblem(X, y, B, 2, "fp32"), params, "fp32")
    o1.round()
    for step in range(1, G + 1):
        o2.step()
        if step % K1 == 0:
            o2.local_average()
    o2.global_average()
    assert o1.t == o2.t == G
    for a, b in zip(o1.params, o2.params):
        assert np.array_equal(a, b)


def test_default_global_interval_is_k1_times_k2():
    o = HierAvgOracle(4, 2, 3, 5, 0.1, None, [np.zeros((4, 2))])
    assert o.G == 15


def test_batch_rows_cycle():
    # mini-batch of step t: rows (t*B + s) mod N
    assert list(batch_rows(0, 4, 10)) == [0, 1, 2, 3]
    assert list(batch_rows(2, 4, 10)) == [8, 9, 0, 1]


def test_rejects_bad_config():
    with pytest.raises(ValueError):
        HierAvgOracle(4, 2, 1, 1, 0.1, None, [np.zeros((4, 2))], global_steps=-1)
    with pytest.raises(ValueError):
        HierAvgOracle(6, 4, 1, 1, 0.1, None, [np.zeros((6, 2))])
    with pytest.raises(ValueError):
        HierAvgOracle(4, 2, 0, 1, 0.1, None, [np.zeros((4, 2))])
