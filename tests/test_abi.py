"""Host-side checks of the C ABI: the library loads, exports every function the
public header declares, and rejects bad arguments before touching the GPU."""
import ctypes
import os
import re

import pytest

from paper_1903_05133_gb300 import _lib as L
from paper_1903_05133_gb300.configs import MLP512_P16, MLP2048_P64, MLP4096_P32, SOFTMAX_P4

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include",
                      "hier_avg.h")


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(hier_avg_\w+)\s*\(", text)))


def test_header_declares_the_abi():
    names = declared_functions()
    for must in ("hier_avg_create", "hier_avg_step", "hier_avg_local_average",
                 "hier_avg_global_average", "hier_avg_round"):
        assert must in names
    assert set(names) == set(L.SIGNATURES), "binding and header disagree"


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def _create(lib, P=4, S=2, K1=1, K2=1, lr=0.1, B=16, dims=(64, 10), prec=1):
    h = ctypes.c_void_p()
    arr = (ctypes.c_int * len(dims))(*dims)
    rc = lib.hier_avg_create(P, S, K1, K2, lr, B, arr, len(dims), prec, ctypes.byref(h))
    return rc, h


@pytest.mark.parametrize("kw,status", [
    (dict(S=3), -1), (dict(P=0), -1), (dict(K1=0), -1), (dict(K2=0), -1), (dict(B=0), -1),
    (dict(lr=float("nan")), -1), (dict(lr=float("inf")), -1), (dict(dims=(64,)), -1),
    (dict(dims=(64, 0)), -1), (dict(prec=7), -1),
    (dict(B=65), -6), (dict(dims=(60, 10)), -6),
])
def test_create_rejects(lib, kw, status):
    rc, h = _create(lib, **kw)
    assert rc == status
    assert not h.value


def test_layout_and_workspace(lib):
    for w in (SOFTMAX_P4, MLP512_P16, MLP2048_P64, MLP4096_P32):
        rc, h = _create(lib, P=w.P, S=w.S, K1=w.K1, K2=w.K2, lr=w.lr, B=w.B, dims=w.dims,
                        prec=0 if w.precision == "fp32" else 1)
        assert rc == 0
        D, ld = ctypes.c_int64(), ctypes.c_int64()
        L_ = len(w.dims) - 1
        offs = (ctypes.c_int64 * (2 * L_))()
        assert lib.hier_avg_param_layout(h, ctypes.byref(D), ctypes.byref(ld), offs) == 0
        assert D.value == w.n_params
        assert ld.value % 64 == 0 and ld.value >= D.value
        prev_end = 0
        for l in range(L_):
            i, o = w.dims[l], w.dims[l + 1]
            assert offs[2 * l] % 64 == 0 and offs[2 * l] >= prev_end
            assert offs[2 * l + 1] % 64 == 0 and offs[2 * l + 1] >= offs[2 * l] + i * o
            prev_end = offs[2 * l + 1] + o
        assert prev_end <= ld.value
        wb = ctypes.c_int64()
        assert lib.hier_avg_workspace_bytes(h, ctypes.byref(wb)) == 0 and wb.value > 0
        lib.hier_avg_destroy(h)


def test_calls_before_bind_fail_cleanly(lib):
    rc, h = _create(lib)
    assert rc == 0
    assert lib.hier_avg_step(h) == -4
    assert lib.hier_avg_round(h) == -4
    assert lib.hier_avg_local_average(h) == -4
    assert lib.hier_avg_wait_selftest(h, 1000) == -4
    assert b"bind" in lib.hier_avg_last_error(h)
    assert lib.hier_avg_bind(h, None, None, 0, None, None, 1, None) == -1
    assert lib.hier_avg_set_step(h, 5) == 0
    t = ctypes.c_int64()
    assert lib.hier_avg_get_step(h, ctypes.byref(t)) == 0 and t.value == 5
    assert lib.hier_avg_profile(h, 1) == 0
    assert lib.hier_avg_profile_every(h, 0) == -1
    assert lib.hier_avg_profile_every(h, 7) == 0
    assert lib.hier_avg_profile_kinds(h, 1 << 8) == -1          # no such kernel kind
    assert lib.hier_avg_profile_kinds(h, 1 << 7) == 0
    assert lib.hier_avg_profile_kinds(h, (1 << 1) | (1 << 3)) == 0
    assert lib.hier_avg_profile_read(h, 99, None, None, None, None) == -1
    assert lib.hier_avg_set_global_steps(h, -1) == -1
    assert lib.hier_avg_set_global_steps(h, 43) == 0 and lib.hier_avg_set_global_steps(h, 0) == 0
    assert lib.hier_avg_set_global_steps(None, 5) == -1
    assert lib.hier_avg_set_lr(h, float("nan")) == -1 and lib.hier_avg_set_lr(h, float("inf")) == -1
    assert lib.hier_avg_set_lr(h, 0.01) == 0
    assert lib.hier_avg_set_batch(h, 0) == -1 and lib.hier_avg_set_batch(h, 10 ** 6) == -1
    assert lib.hier_avg_set_batch(None, 1) == -1
    assert lib.hier_avg_set_batch(h, 1) == 0
    n = ctypes.c_int64(-1)
    assert lib.hier_avg_launches(h, ctypes.byref(n)) == 0 and n.value == 0   # nothing ran
    assert lib.hier_avg_launches(h, None) == -1
    assert lib.hier_avg_launches(None, ctypes.byref(n)) == -1
    lib.hier_avg_destroy(h)
    lib.hier_avg_destroy(None)


def test_stateless_averages_validate(lib):
    assert lib.hier_avg_local_average_buffer(None, 6, 4, 10, 10, None) == -1     # S does not divide P
    assert lib.hier_avg_local_average_buffer(None, 4, 2, 10, 5, None) == -1      # ld < D
    assert lib.hier_avg_global_average_buffer(None, 0, 10, 10, None) == -1
    assert lib.hier_avg_local_global_average_buffer(None, 4, 2, 10, 10, None) == -1   # NULL
    assert lib.hier_avg_local_average_buffer(None, 4, 2, 0, 0, None) == 0        # empty: no-op
    # more than 65535 clusters in one launch is rejected before any launch
    assert lib.hier_avg_local_average_buffer(None, 2 * 65536, 2, 0, 0, None) == -6
    assert lib.hier_avg_global_average_buffer(None, 2 * 65536, 0, 0, None) == 0
    assert lib.hier_avg_local_global_average_buffer(None, 2 * 65536, 2, 0, 0, None) == 0


def test_status_strings(lib):
    for s in (0, -1, -2, -3, -4, -5, -6):
        assert lib.hier_avg_strerror(s)
    assert lib.hier_avg_strerror(-99) == b"unknown status"
