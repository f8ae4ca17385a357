"""Pins of the oracle's local and global averages (Algorithm 1, Sec. 3.1) against
hand-derived cases, exact arithmetic, error bounds and the invariants the
algorithm fixes."""
import math
import os
from fractions import Fraction

import numpy as np
import pytest

from oracle import averaging as av

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "averaging_tree_order.txt")


def _golden_cases():
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip():
            continue
        n, vals, exp = line.split(";")
        yield int(n), [float(x) for x in vals.split()], float(exp)


@pytest.mark.parametrize("case", list(_golden_cases()), ids=lambda c: f"n{c[0]}")
def test_tree_order_golden(case):
    n, vals, expected = case
    v = np.array(vals, dtype=np.float32).reshape(n, 1)
    got = av.group_mean(v)
    assert got.dtype == np.float32
    assert got[0] == np.float32(expected)


def test_integer_values_are_exact():
    # Small integers: every partial sum is exact in fp32, so the tree sum equals
    # the exact integer sum and a power-of-two mean is exact.
    rng = np.random.default_rng(1)
    for n in (1, 2, 3, 4, 5, 7, 8, 16, 33, 128):
        ints = rng.integers(-1000, 1000, size=(n, 257))
        s = av.tree_sum(ints.astype(np.float32))
        assert np.array_equal(s.astype(np.int64), ints.sum(axis=0))
        if n & (n - 1) == 0:
            m = av.group_mean(ints.astype(np.float32))
            assert np.array_equal(m.astype(np.float64), ints.sum(axis=0) / n)


def _fp32_round(q: Fraction) -> float:
    """Round an exact rational to the nearest fp32 (ties to even), independently of
    numpy: scale to a 24-bit significand and round the integer."""
    if q == 0:
        return 0.0
    sign = -1 if q < 0 else 1
    a = abs(q)
    e = math.floor(math.log2(a.numerator) - math.log2(a.denominator))
    while Fraction(2) ** e > a:
        e -= 1
    while Fraction(2) ** (e + 1) <= a:
        e += 1
    e = max(e, -126)                      # subnormal range keeps the fixed quantum
    quantum = Fraction(2) ** (e - 23)
    k = a / quantum
    fl = math.floor(k)
    rem = k - fl
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and fl % 2 == 1):
        fl += 1
    return sign * float(fl * quantum)


def test_division_is_correctly_rounded():
    # The mean is one correctly rounded fp32 division of the tree sum by n.
    rng = np.random.default_rng(2)
    for n in (3, 5, 6, 7, 12, 24):
        v = rng.standard_normal((n, 64)).astype(np.float32)
        s = av.tree_sum(v)
        m = av.group_mean(v)
        for k in range(64):
            assert m[k] == np.float32(_fp32_round(Fraction(float(s[k])) / n))


def test_fp32_additions_match_exact_model():
    # Each fp32 add of the tree is the exact sum rounded to nearest even: checked
    # for n = 2 (one add) against an exact rational model.
    rng = np.random.default_rng(3)
    v = (rng.standard_normal((2, 2000)) * 10.0 ** rng.integers(-30, 30, (2, 2000))).astype(np.float32)
    s = av.tree_sum(v)
    for k in range(v.shape[1]):
        exact = Fraction(float(v[0, k])) + Fraction(float(v[1, k]))
        assert s[k] == np.float32(_fp32_round(exact))


def test_error_bound_pairwise():
    # Pairwise summation: |tree - exact| <= ceil(log2 n) * u * sum|v| (u = 2^-24).
    rng = np.random.default_rng(4)
    for n in (2, 3, 8, 17, 64, 128):
        v = rng.standard_normal((n, 500)).astype(np.float32)
        s = av.tree_sum(v).astype(np.float64)
        exact = np.array([math.fsum(v[:, k].astype(np.float64)) for k in range(500)])
        bound = math.ceil(math.log2(n)) * 2.0 ** -24 * np.abs(v.astype(np.float64)).sum(axis=0)
        assert np.all(np.abs(s - exact) <= bound * 1.0000001)


def test_f64_mode_matches_fsum():
    rng = np.random.default_rng(5)
    v = rng.standard_normal((37, 100))
    s = av.tree_sum(v)
    exact = np.array([math.fsum(v[:, k]) for k in range(100)])
    assert np.allclose(s, exact, rtol=1e-14, atol=1e-14)


def test_brute_force_tiny():
    # P=4, S=2, D=8: each local mean is (a+b)/2, the only order there is.
    rng = np.random.default_rng(6)
    w = rng.standard_normal((4, 8)).astype(np.float32)
    want = np.empty_like(w)
    for g in range(2):
        for d in range(8):
            pair = Fraction(float(w[2 * g, d])) + Fraction(float(w[2 * g + 1, d]))
            want[2 * g:2 * g + 2, d] = _fp32_round(Fraction(_fp32_round(pair)) / 2)
    got = w.copy()
    av.local_average(got, 2)
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


@pytest.mark.parametrize("P,S", [(4, 2), (8, 4), (6, 3), (12, 4), (128, 32), (5, 5), (7, 1)])
def test_invariants(P, S):
    rng = np.random.default_rng(P * 100 + S)
    w = rng.standard_normal((P, 301)).astype(np.float32)
    orig = w.copy()
    av.local_average(w, S)
    for g in range(P // S):
        blk = w[g * S:(g + 1) * S].view(np.uint32)
        assert np.all(blk == blk[0])                     # members bitwise identical
    if S == 1:
        assert np.array_equal(w.view(np.uint32), orig.view(np.uint32))   # identity
    w2 = orig.copy()
    av.global_average(w2)
    assert np.all(w2.view(np.uint32) == w2[0].view(np.uint32))
    w3 = orig.copy()
    av.local_average(w3, P)                               # S = P is the global average
    assert np.array_equal(w3.view(np.uint32), w2.view(np.uint32))


def test_signed_zero_and_subnormals():
    tiny = np.float32(1e-45)   # smallest fp32 subnormal
    w = np.array([[-0.0, tiny, 3 * tiny, -0.0],
                  [-0.0, tiny, -tiny, 0.0]], dtype=np.float32)
    av.local_average(w, 2)
    # -0 + -0 = -0 and -0/2 = -0; tiny + tiny = 2 tiny, /2 = tiny (exact, no flush);
    # 3 tiny - tiny = 2 tiny -> tiny; -0 + 0 = +0.
    assert np.signbit(w[0, 0]) and w[0, 0] == 0
    assert w[0, 1] == tiny and w[0, 2] == tiny
    assert w[0, 3] == 0 and not np.signbit(w[0, 3])


def test_rejects_bad_groups():
    with pytest.raises(ValueError):
        av.local_average(np.zeros((6, 3), np.float32), 4)
    with pytest.raises(ValueError):
        av.tree_sum(np.zeros((0, 3), np.float32))
