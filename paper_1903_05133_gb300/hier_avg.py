"""Python binding of the Hier-AVG C ABI: argument marshalling only.

PyTorch provides the device memory (parameters, workspace, data) and the CUDA
stream; every step of the computation runs in the library's CUDA kernels.  The
function and method names are those of include/hier_avg.h without the
``hier_avg_`` prefix.
"""
from __future__ import annotations

import ctypes
from typing import List, NamedTuple, Optional, Sequence, Tuple

import torch

from . import _lib
from ._lib import c_double, c_int, c_int64, c_void_p, check

PREC = {"fp32": 0, "bf16": 1}
KERNEL_KINDS = {"gather": 0, "forward": 1, "xent": 2, "backward": 3, "local_avg": 4,
                "global_avg": 5, "head": 6, "update_forward": 7}


class ProfileTotals(NamedTuple):
    total_ms: float
    launches: int
    bytes: float
    flops: float


def _stream(stream) -> c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return c_void_p(stream.cuda_stream)


def _rows(w: torch.Tensor) -> Tuple[int, int, int]:
    if w.dtype != torch.float32 or not w.is_cuda or w.dim() != 2 or w.stride(1) != 1:
        raise ValueError("w must be a CUDA fp32 matrix [P, D] with unit column stride")
    return w.shape[0], w.shape[1], w.stride(0)


def local_average_buffer(w: torch.Tensor, S: int, stream=None) -> None:
    """Local average (Algorithm 1, Sec. 3.1) of the rows of w in place."""
    P, D, ld = _rows(w)
    check(_lib.load().hier_avg_local_average_buffer(c_void_p(w.data_ptr()), P, S, D, ld,
                                                    _stream(stream)), "local_average_buffer")


def global_average_buffer(w: torch.Tensor, stream=None) -> None:
    """Global average (Algorithm 1, Sec. 3.1) of the rows of w in place."""
    P, D, ld = _rows(w)
    check(_lib.load().hier_avg_global_average_buffer(c_void_p(w.data_ptr()), P, D, ld,
                                                     _stream(stream)), "global_average_buffer")


def local_global_average_buffer(w: torch.Tensor, S: int, stream=None) -> None:
    """Last local average of a round fused with the global average, in place."""
    P, D, ld = _rows(w)
    check(_lib.load().hier_avg_local_global_average_buffer(c_void_p(w.data_ptr()), P, S, D, ld,
                                                           _stream(stream)),
          "local_global_average_buffer")


class HierAvg:
    """P learners of a ReLU MLP ``dims`` trained by Hier-AVG on one GPU."""

    def __init__(self, P: int, S: int, K1: int, K2: int, lr: float, B: int,
                 dims: Sequence[int], precision: str = "bf16"):
        lib = _lib.load()
        self._lib = lib
        self.h = c_void_p()
        arr = (c_int * len(dims))(*dims)
        check(lib.hier_avg_create(P, S, K1, K2, float(lr), B, arr, len(dims), PREC[precision],
                                  ctypes.byref(self.h)), "create")
        self.P, self.S, self.K1, self.K2, self.lr, self.B = P, S, K1, K2, lr, B
        self.dims, self.precision = tuple(dims), precision
        self.L = len(dims) - 1
        D, ld = c_int64(), c_int64()
        offs = (c_int64 * (2 * self.L))()
        check(lib.hier_avg_param_layout(self.h, ctypes.byref(D), ctypes.byref(ld), offs),
              "param_layout", self.h)
        self.D, self.ld = D.value, ld.value
        self.offsets = [(offs[2 * l], offs[2 * l + 1]) for l in range(self.L)]
        wb = c_int64()
        check(lib.hier_avg_workspace_bytes(self.h, ctypes.byref(wb)), "workspace_bytes", self.h)
        self.workspace_bytes = wb.value
        self.params: Optional[torch.Tensor] = None
        self.workspace: Optional[torch.Tensor] = None

    @classmethod
    def create(cls, P, S, K1, K2, lr, B, dims, precision="bf16") -> "HierAvg":
        return cls(P, S, K1, K2, lr, B, dims, precision)

    # ------------------------------------------------------------ parameters
    def new_params(self, device="cuda") -> torch.Tensor:
        return torch.zeros(self.P, self.ld, dtype=torch.float32, device=device)

    def pack(self, layers, device="cuda") -> torch.Tensor:
        """[P, ld] parameter matrix from one shared [(W, b), ...] (every learner
        gets the same w0) or from a per-learner list of such lists."""
        out = self.new_params(device)
        per_learner = isinstance(layers[0], (list, tuple)) and isinstance(layers[0][0], (list, tuple))
        for j in range(self.P):
            lj = layers[j] if per_learner else layers
            for l, (W, b) in enumerate(lj):
                wo, bo = self.offsets[l]
                out[j, wo:wo + W.numel()] = W.reshape(-1).to(out.device, torch.float32)
                out[j, bo:bo + b.numel()] = b.reshape(-1).to(out.device, torch.float32)
        return out

    def unpack(self, params: torch.Tensor) -> List[Tuple[torch.Tensor, torch.Tensor]]:
        """Per-layer views [(W [P, out, in], b [P, out]), ...] of a [P, ld] matrix."""
        res = []
        for l in range(self.L):
            i, o = self.dims[l], self.dims[l + 1]
            wo, bo = self.offsets[l]
            res.append((params[:, wo:wo + o * i].reshape(self.P, o, i), params[:, bo:bo + o]))
        return res

    # ------------------------------------------------------------ binding
    def bind(self, params: torch.Tensor, X: torch.Tensor, y: torch.Tensor, stream=None) -> None:
        want_dtype = torch.bfloat16 if self.precision == "bf16" else torch.float32
        if params.shape != (self.P, self.ld) or params.dtype != torch.float32 or not params.is_contiguous():
            raise ValueError(f"params must be a contiguous fp32 [{self.P}, {self.ld}] CUDA tensor")
        if X.dtype != want_dtype or X.dim() != 3 or X.shape[0] != self.P or X.shape[2] != self.dims[0]:
            raise ValueError(f"X must be {want_dtype} [P, N, {self.dims[0]}]")
        if y.dtype != torch.int32 or tuple(y.shape) != tuple(X.shape[:2]):
            raise ValueError("y must be int32 [P, N]")
        if not (X.is_contiguous() and y.is_contiguous()):
            raise ValueError("X and y must be contiguous")
        self.workspace = torch.empty(self.workspace_bytes, dtype=torch.uint8, device=params.device)
        self.params, self.X, self.y = params, X, y
        self._stream_obj = stream
        check(self._lib.hier_avg_bind(self.h, c_void_p(params.data_ptr()),
                                      c_void_p(self.workspace.data_ptr()), self.workspace_bytes,
                                      c_void_p(X.data_ptr()), c_void_p(y.data_ptr()), X.shape[1],
                                      _stream(stream)), "bind", self.h)

    # ------------------------------------------------------------ Algorithm 1
    def step(self) -> None:
        check(self._lib.hier_avg_step(self.h), "step", self.h)

    def local_average(self) -> None:
        check(self._lib.hier_avg_local_average(self.h), "local_average", self.h)

    def global_average(self) -> None:
        check(self._lib.hier_avg_global_average(self.h), "global_average", self.h)

    def round(self) -> None:
        check(self._lib.hier_avg_round(self.h), "round", self.h)

    def round_host(self, X_host: torch.Tensor, y_host: torch.Tensor,
                   loss_host: Optional[torch.Tensor] = None) -> torch.Tensor:
        """One round with the data read from host memory (pinned recommended)."""
        if loss_host is None:
            loss_host = torch.empty(self.P, dtype=torch.float32, pin_memory=True)
        if X_host.shape != self.X.shape or X_host.dtype != self.X.dtype or y_host.shape != self.y.shape:
            raise ValueError("host data must match the bound device data set")
        check(self._lib.hier_avg_round_host(self.h, c_void_p(X_host.data_ptr()),
                                            c_void_p(y_host.data_ptr()),
                                            c_void_p(loss_host.data_ptr())), "round_host", self.h)
        return loss_host

    # ------------------------------------------------------------ state and checks
    def get_step(self) -> int:
        t = c_int64()
        check(self._lib.hier_avg_get_step(self.h, ctypes.byref(t)), "get_step", self.h)
        return t.value

    def set_step(self, t: int) -> None:
        check(self._lib.hier_avg_set_step(self.h, t), "set_step", self.h)

    def losses(self) -> torch.Tensor:
        out = torch.empty(self.P, dtype=torch.float32)
        check(self._lib.hier_avg_losses(self.h, c_void_p(out.data_ptr())), "losses", self.h)
        return out

    def check(self) -> None:
        check(self._lib.hier_avg_check(self.h), "check", self.h)

    def wait_selftest(self, limit_ms: float) -> None:
        """Run the library's bounded device waits on conditions nothing satisfies, each
        limited to limit_ms; the next check() raises HA_ETIMEOUT (see the header)."""
        check(self._lib.hier_avg_wait_selftest(self.h, int(round(limit_ms * 1000))),
              "wait_selftest", self.h)

    def profile(self, enable) -> None:
        """Start (and clear) kernel timing: True for every kind, an iterable of kind
        names for a subset; False stops it."""
        if isinstance(enable, bool) or enable is None:
            check(self._lib.hier_avg_profile(self.h, 1 if enable else 0), "profile", self.h)
            return
        mask = 0
        for k in enable:
            mask |= 1 << KERNEL_KINDS[k]
        check(self._lib.hier_avg_profile_kinds(self.h, mask), "profile", self.h)

    def set_global_steps(self, steps: int) -> None:
        """Local steps per global average (0: K1 * K2); see hier_avg_set_global_steps."""
        check(self._lib.hier_avg_set_global_steps(self.h, int(steps)), "set_global_steps", self.h)

    def set_lr(self, lr: float) -> None:
        """Step size of the following local steps (per-round schedules)."""
        check(self._lib.hier_avg_set_lr(self.h, float(lr)), "set_lr", self.h)
        self.lr = float(lr)

    def set_batch(self, B: int) -> None:
        """Mini-batch size of the following local steps (<= the B given at creation)."""
        check(self._lib.hier_avg_set_batch(self.h, int(B)), "set_batch", self.h)

    def launches(self) -> int:
        """Kernels this handle has launched since it was created."""
        n = c_int64()
        check(self._lib.hier_avg_launches(self.h, ctypes.byref(n)), "launches", self.h)
        return n.value

    def profile_every(self, every: int) -> None:
        """Time only every n-th launch of each enabled kind."""
        check(self._lib.hier_avg_profile_every(self.h, int(every)), "profile_every", self.h)

    def profile_read(self, kind: str) -> "ProfileTotals":
        """(total_ms, launches, bytes, flops) of the timed launches of one kernel kind."""
        ms, n, by, fl = c_double(), c_int64(), c_double(), c_double()
        check(self._lib.hier_avg_profile_read(self.h, KERNEL_KINDS[kind], ctypes.byref(ms),
                                              ctypes.byref(n), ctypes.byref(by), ctypes.byref(fl)),
              "profile_read", self.h)
        return ProfileTotals(ms.value, n.value, by.value, fl.value)

    def destroy(self) -> None:
        if self.h:
            self._lib.hier_avg_destroy(self.h)
            self.h = c_void_p()

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass
