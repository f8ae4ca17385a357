"""One learner's local SGD step (Algorithm 1 inner loop, Sec. 3.1), plainly.

Paper: w <- w - (gamma / B) * sum_{s=1..B} grad f(w; xi_s) on the learner's own
mini-batch.  The objective here is the mean softmax cross-entropy of a ReLU MLP
(weights W_l [d_l, d_{l-1}], biases b_l [d_l]); the 1/B of the update is the mean
over the batch.

Precision modes (the paper computes in exact arithmetic; the method as built fixes
fp32 master weights and, optionally, bf16 GEMM operands with fp32 accumulation):
  "f64"   every value float64 (used for exact-math pins)
  "fp32"  stored values (products' accumulators, bias sums, activations, gradients,
          weights) are rounded to fp32; products are accumulated in float64 first
  "bf16"  as "fp32", and every operand of a matrix product is first rounded to
          bf16 (round-to-nearest-even): the input X, W_l, H_{l-1} and dZ_l
  "bf16_acc32"  as "bf16" but each product is accumulated in fp32 (numpy's
          float32 matrix product, in its own summation order): a second valid
          order of the same computation, used to measure how far two correct
          implementations drift apart through rounding-boundary decisions
Readings: ReLU'(z) is taken as [h > 0] on the stored (operand) activation h;
the update is w - fl(lr * g), a rounded product followed by a rounded subtraction.
"""
from __future__ import annotations

from typing import List, Sequence, Tuple

import numpy as np

MODES = ("f64", "fp32", "bf16", "bf16_acc32")


def bf16_round(x) -> np.ndarray:
    """fp32 -> nearest bf16 (ties to even), returned as fp32 values.

    Written from the format: bf16 keeps the top 16 bits of an fp32 word.  Adding
    0x7FFF plus the lowest kept bit and truncating rounds to nearest, ties to the
    even kept pattern; the carry handles mantissa overflow (including to Inf).
    NaN is returned as a quiet NaN of the same sign."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    u = x.view(np.uint32).astype(np.uint64)
    lsb = (u >> np.uint64(16)) & np.uint64(1)
    r = ((u + np.uint64(0x7FFF) + lsb) >> np.uint64(16)) << np.uint64(16)
    out = (r & np.uint64(0xFFFFFFFF)).astype(np.uint32)
    nan = np.isnan(x)
    if nan.any():
        q = ((x.view(np.uint32)[nan] >> np.uint32(16)) << np.uint32(16)) | np.uint32(0x00400000)
        out[nan] = q
    return out.view(np.float32).reshape(x.shape)


def _mm64(a, b):
    return a @ b


def _mm32(a, b):
    return (np.asarray(a, np.float32) @ np.asarray(b, np.float32)).astype(np.float64)


def _modes(mode: str):
    if mode == "f64":
        def operand(a):
            return np.asarray(a, dtype=np.float64)
        store = operand
    elif mode == "fp32":
        def operand(a):
            return np.asarray(a, dtype=np.float32).astype(np.float64)
        store = operand
    elif mode in ("bf16", "bf16_acc32"):
        def operand(a):
            return bf16_round(np.asarray(a, dtype=np.float32)).astype(np.float64)

        def store(a):
            return np.asarray(a, dtype=np.float32).astype(np.float64)
    else:
        raise ValueError(f"mode must be one of {MODES}")
    return operand, store, (_mm32 if mode == "bf16_acc32" else _mm64)


def softmax_xent_grad(Z: np.ndarray, y: np.ndarray, B: int) -> Tuple[float, np.ndarray]:
    """Mean softmax cross-entropy over the rows of Z [B, C] and its gradient.

    loss = (1/B) sum_b [log sum_c exp(z_bc) - z_{b,y_b}];
    dL/dz_bc = (softmax(z_b)_c - [c == y_b]) / B.   (float64)"""
    Z = np.asarray(Z, dtype=np.float64)
    m = Z.max(axis=1, keepdims=True)
    e = np.exp(Z - m)
    s = e.sum(axis=1, keepdims=True)
    p = e / s
    rows = np.arange(Z.shape[0])
    loss = float(np.mean(np.log(s[:, 0]) + m[:, 0] - Z[rows, y]))
    onehot = np.zeros_like(p)
    onehot[rows, y] = 1.0
    return loss, (p - onehot) / B


def mlp_forward_backward(Ws: Sequence[np.ndarray], bs: Sequence[np.ndarray],
                         X: np.ndarray, y: np.ndarray, mode: str, preacts: list | None = None
                         ) -> Tuple[float, List[np.ndarray], List[np.ndarray]]:
    """Loss and gradients (dW_l, db_l) of the mean softmax cross-entropy of a
    ReLU MLP on one mini-batch X [B, d_0], y [B].  If ``preacts`` is a list, the
    pre-activations Z_l of every layer are appended to it (for inspection only)."""
    operand, store, mm = _modes(mode)
    L = len(Ws)
    B = X.shape[0]
    H = [operand(X)]                     # operand form of every layer input
    Zs = []
    for l in range(L):
        z = store(mm(H[l], operand(Ws[l]).T))
        z = store(z + np.asarray(bs[l], dtype=np.float64))
        Zs.append(z)
        if preacts is not None:
            preacts.append(z)
        if l < L - 1:
            H.append(operand(store(np.maximum(z, 0.0))))
    loss, dz = softmax_xent_grad(Zs[-1], y, B)
    dz = store(dz)
    gW: List[np.ndarray] = [None] * L  # type: ignore[list-item]
    gb: List[np.ndarray] = [None] * L  # type: ignore[list-item]
    for l in reversed(range(L)):
        gW[l] = store(mm(operand(dz).T, H[l]))
        gb[l] = store(dz.sum(axis=0))
        if l > 0:
            dh = store(mm(operand(dz), operand(Ws[l])))  # uses W_l before its update
            dz = store(dh * (H[l] > 0))
    return loss, gW, gb


def sgd_update(p: np.ndarray, g: np.ndarray, lr: float, mode: str) -> np.ndarray:
    """w - lr * g: float64 in mode "f64", else fp32 multiply then fp32 subtract."""
    if mode == "f64":
        return np.asarray(p, np.float64) - lr * np.asarray(g, np.float64)
    lr32 = np.float32(lr)
    step = (lr32 * np.asarray(g, dtype=np.float32)).astype(np.float32)
    return (np.asarray(p, dtype=np.float32) - step).astype(np.float32)


class MLPProblem:
    """Learner j's mini-batch gradient of the MLP objective on its own data.

    X [P, N, d_0] (float values; bf16 data passed as its exact fp32 values),
    y [P, N] integer labels; B is the default batch size.  A step's rows are chosen by
    the caller (``batch_rows_from``)."""

    def __init__(self, X: np.ndarray, y: np.ndarray, B: int, n_layers: int, mode: str):
        self.X, self.y, self.B, self.L, self.mode = X, y, B, n_layers, mode
        self.last_loss = np.zeros(X.shape[0])
        self.last_preacts: dict = {}

    def gradients(self, j: int, rows: np.ndarray, params_j: List[np.ndarray]) -> List[np.ndarray]:
        Ws, bs = params_j[0::2], params_j[1::2]
        pre: list = []
        loss, gW, gb = mlp_forward_backward(Ws, bs, self.X[j, rows], self.y[j, rows], self.mode,
                                            preacts=pre)
        self.last_loss[j] = loss
        self.last_preacts[j] = pre
        out = []
        for a, b in zip(gW, gb):
            out += [a, b]
        return out


class QuadraticProblem:
    """Noise-free least squares with identity design: f_j(w) = 0.5 * ||w - c_j||^2,
    whose exact gradient is w - c_j (float64)."""

    def __init__(self, c: np.ndarray):
        self.c = np.asarray(c, dtype=np.float64)
        self.mode = "f64"

    def gradients(self, j: int, rows, params_j: List[np.ndarray]) -> List[np.ndarray]:
        return [params_j[0] - self.c[j]]
