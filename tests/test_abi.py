"""The C ABI library loads, exports every function include/mcpu.h declares,
and rejects bad arguments on the host before touching a GPU."""
import ctypes
import os
import re

import pytest
import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2608_22167_gb300 import build

    path = build.build()
    return ctypes.CDLL(path)


def _declared_functions():
    src = open(os.path.join(ROOT, "include", "mcpu.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(mcpu_[a-z_]+)\s*\(", src)))


def test_header_declares_the_two_hot_path_calls():
    names = _declared_functions()
    assert "mcpu_kv_append" in names and "mcpu_paged_attention_forward" in names


def test_every_declared_symbol_is_exported(lib):
    for name in _declared_functions():
        assert hasattr(lib, name), name


def test_binding_uses_the_same_names():
    from paper_2608_22167_gb300 import mcpu

    for name in _declared_functions():
        assert hasattr(mcpu, name), name


class Dims(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("num_seqs", "total_q", "max_pages_per_seq", "num_pages",
                                              "num_q_heads", "num_kv_heads", "head_dim", "page_size")]


def _fn(lib, name):
    f = getattr(lib, name)
    f.restype = ctypes.c_int
    return f


def test_workspace_size(lib):
    lib.mcpu_workspace_size.restype = ctypes.c_size_t
    ok = Dims(4, 4, 19, 34, 8, 2, 64, 16)
    n = lib.mcpu_workspace_size(ctypes.byref(ok))
    assert n > 0 and n % 256 == 0
    bigger = Dims(400, 40000, 19, 34, 8, 2, 64, 16)
    assert lib.mcpu_workspace_size(ctypes.byref(bigger)) > n
    for bad in (Dims(4, 4, 19, 34, 8, 3, 64, 16),     # H_q not a multiple of H_kv
                Dims(4, 4, 19, 34, 8, 2, 128, 16),    # head_dim unsupported
                Dims(4, 4, 19, 34, 8, 2, 64, 32),     # page size unsupported
                Dims(4, 4, 19, 34, 48, 2, 64, 16),    # group 24 unsupported
                Dims(5000, 4, 19, 34, 8, 2, 64, 16),  # too many rows
                Dims(-1, 4, 19, 34, 8, 2, 64, 16)):
        assert lib.mcpu_workspace_size(ctypes.byref(bad)) == 0
    assert lib.mcpu_workspace_size(None) == 0


def test_host_validation_errors(lib):
    fwd = _fn(lib, "mcpu_paged_attention_forward")
    fwd.argtypes = [ctypes.c_void_p] * 6 + [ctypes.c_int32, ctypes.c_float, ctypes.POINTER(Dims)] + \
        [ctypes.c_void_p] * 3 + [ctypes.c_size_t, ctypes.c_void_p, ctypes.c_void_p]
    d = Dims(4, 4, 19, 34, 8, 2, 64, 16)
    P = 1 << 20  # a 256-byte-aligned fake address: never dereferenced by these calls
    lib.mcpu_workspace_size.restype = ctypes.c_size_t
    need = lib.mcpu_workspace_size(ctypes.byref(d))
    args = [P] * 6 + [0, 0.125, ctypes.byref(d), P, P, P, need, None, None]
    # dims NULL
    a = list(args); a[8] = None
    assert fwd(*a) == 1
    # workspace too small
    a = list(args); a[12] = need - 1
    assert fwd(*a) == 3
    # misaligned workspace
    a = list(args); a[11] = P + 8
    assert fwd(*a) == 1
    # NaN scale
    a = list(args); a[7] = float("nan")
    assert fwd(*a) == 1
    # unsupported head dim
    d2 = Dims(4, 4, 19, 34, 8, 2, 128, 16)
    a = list(args); a[8] = ctypes.byref(d2)
    assert fwd(*a) == 2
    # misaligned q (needs 16 bytes)
    a = list(args); a[0] = P + 2
    assert fwd(*a) == 1
    # null output
    a = list(args); a[9] = None
    assert fwd(*a) == 1
    # empty batch: nothing to do, no launch, OK
    d3 = Dims(0, 0, 19, 34, 8, 2, 64, 16)
    a = list(args); a[8] = ctypes.byref(d3); a[12] = lib.mcpu_workspace_size(ctypes.byref(d3))
    assert fwd(*a) == 0


def test_kv_append_host_validation(lib):
    app = _fn(lib, "mcpu_kv_append")
    app.argtypes = [ctypes.c_void_p] * 7 + [ctypes.POINTER(Dims), ctypes.c_void_p, ctypes.c_void_p]
    d = Dims(4, 4, 19, 34, 2, 2, 64, 16)
    P = 1 << 20
    assert app(P, P, P, P, P, P, P, ctypes.byref(d), None, None) == 1      # no status word
    assert app(P + 4, P, P, P, P, P, P, ctypes.byref(d), P, None) == 1     # misaligned k_new
    d0 = Dims(0, 0, 19, 34, 2, 2, 64, 16)
    assert app(P, P, P, P, P, P, P, ctypes.byref(d0), P, None) == 0        # empty: no-op


def test_fp8_host_validation(lib):
    fwd = _fn(lib, "mcpu_paged_attention_forward_fp8")
    fwd.argtypes = [ctypes.c_void_p] * 5 + [ctypes.c_int32, ctypes.c_float, ctypes.POINTER(Dims)] + \
        [ctypes.c_void_p] * 3 + [ctypes.c_size_t, ctypes.c_void_p, ctypes.c_void_p]
    d = Dims(4, 4, 19, 34, 8, 2, 64, 16)
    P = 1 << 20
    lib.mcpu_workspace_size.restype = ctypes.c_size_t
    need = lib.mcpu_workspace_size(ctypes.byref(d))
    args = [P] * 5 + [0, 0.125, ctypes.byref(d), P, P, P, need, None, None]
    a = list(args); a[1] = None           # no pool
    assert fwd(*a) == 1
    a = list(args); a[1] = P + 8          # misaligned pool
    assert fwd(*a) == 1
    d_app = Dims(4, 9, 19, 34, 8, 2, 64, 16)  # 9 query tokens over 4 rows: some row appends
    a = list(args); a[7] = ctypes.byref(d_app); a[11] = lib.mcpu_workspace_size(ctypes.byref(d_app))
    assert fwd(*a) == 2
    d0 = Dims(0, 0, 19, 34, 8, 2, 64, 16)
    a = list(args); a[7] = ctypes.byref(d0); a[11] = lib.mcpu_workspace_size(ctypes.byref(d0))
    assert fwd(*a) == 0
    app = _fn(lib, "mcpu_kv_append_fp8")
    app.argtypes = [ctypes.c_void_p] * 6 + [ctypes.POINTER(Dims), ctypes.c_void_p, ctypes.c_void_p]
    assert app(P, P, None, P, P, P, ctypes.byref(d), P, None) == 1   # no pool
    assert app(P, P, P + 4, P, P, P, ctypes.byref(d), P, None) == 1  # misaligned pool
    assert app(P, P, P, P, P, P, ctypes.byref(d), None, None) == 1   # no status word


def test_status_strings(lib):
    lib.mcpu_status_string.restype = ctypes.c_char_p
    seen = set()
    for code in range(11):
        s = lib.mcpu_status_string(code)
        assert s and s not in seen
        seen.add(s)


def test_timeout_selftest_host_checks(lib):
    f = _fn(lib, "mcpu_selftest_wait_timeout")
    f.argtypes = [ctypes.c_void_p] * 3
    P = 1 << 20
    assert f(None, P, None) == 1
    assert f(P, None, None) == 1
    assert f(P + 2, P, None) == 1  # status word not 4-byte aligned
    assert f(P, P + 4, None) == 1  # report not 8-byte aligned


def test_append_abort_selftest_host_checks(lib):
    f = _fn(lib, "mcpu_selftest_append_abort")
    f.argtypes = [ctypes.c_void_p] * 6 + [ctypes.c_float, ctypes.POINTER(Dims)] + [ctypes.c_void_p] * 3 + \
        [ctypes.c_size_t, ctypes.c_int32, ctypes.c_void_p, ctypes.c_void_p]
    d = Dims(2, 40, 19, 34, 16, 2, 64, 16)
    lib.mcpu_workspace_size.restype = ctypes.c_size_t
    need = lib.mcpu_workspace_size(ctypes.byref(d))
    P = 1 << 20
    args = lambda role, rep, ws=P, nbytes=need: (P, P, P, P, P, P, 0.125, ctypes.byref(d), P, P, ws,  # noqa: E731
                                                 nbytes, role, rep, None)
    assert f(*args(3, P)) == 1  # no such role
    assert f(*args(-1, P)) == 1
    assert f(*args(0, None)) == 1  # no report
    assert f(*args(0, P + 4)) == 1  # report not 8-byte aligned
    assert f(*args(0, P, ws=P + 16)) == 1  # workspace not 256-byte aligned
    assert f(*args(0, P, nbytes=need - 1)) == 3  # workspace too small
    bad = Dims(2, 40, 19, 34, 16, 2, 128, 16)
    assert f(P, P, P, P, P, P, 0.125, ctypes.byref(bad), P, P, P, need, 0, P, None) == 2  # head_dim 128


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the no-GPU error path")
def test_no_gpu_is_a_clean_error(lib):
    fwd = _fn(lib, "mcpu_paged_attention_forward")
    fwd.argtypes = [ctypes.c_void_p] * 6 + [ctypes.c_int32, ctypes.c_float, ctypes.POINTER(Dims)] + \
        [ctypes.c_void_p] * 3 + [ctypes.c_size_t, ctypes.c_void_p, ctypes.c_void_p]
    d = Dims(4, 4, 19, 34, 8, 2, 64, 16)
    lib.mcpu_workspace_size.restype = ctypes.c_size_t
    need = lib.mcpu_workspace_size(ctypes.byref(d))
    P = 1 << 20
    assert fwd(P, P, P, P, P, P, 0, 0.125, ctypes.byref(d), P, P, P, need, None, None) == 4


def test_host_slice_rows(lib):
    # row ranges of the host-buffer call: 0 .. B, strictly increasing, every
    # slice with tokens, each boundary the row start nearest its target
    import numpy as np

    f = lib.mcpu_host_slice_rows
    f.restype = ctypes.c_int32
    rng = np.random.default_rng(11)
    for trial in range(300):
        B = int(rng.integers(1, 40))
        L = rng.integers(0, 50, size=B)
        L[rng.random(B) < 0.2] = int(rng.integers(100, 2000))
        qsl = np.concatenate([[0], np.cumsum(L)]).astype(np.int32)
        T = int(qsl[-1])
        for slices in range(1, 9):
            rb = (ctypes.c_int32 * 9)()
            n = f(qsl.ctypes.data_as(ctypes.c_void_p), B, slices, ctypes.cast(rb, ctypes.c_void_p))
            got = [rb[i] for i in range(n + 1)]
            if T == 0:
                assert n == 1 and got == [0, B]
                continue
            assert 1 <= n <= slices and got[0] == 0 and got[-1] == B
            assert all(a < b for a, b in zip(got, got[1:]))
            for a, b in zip(got[:-2], got[1:-1]):  # interior slices carry tokens
                assert qsl[b] > qsl[a]
            # brute force: boundary k is the row start nearest round(T k / slices) after the last one
            exp = [0]
            for k in range(1, slices):
                target = (T * k + slices // 2) // slices
                cands = range(exp[-1] + 1, B)
                if not cands:
                    continue
                lo = next((r for r in cands if qsl[r] >= target), B)
                if lo - 1 > exp[-1] and target - qsl[lo - 1] < qsl[lo] - target:
                    lo -= 1
                if lo < B and qsl[lo] > qsl[exp[-1]]:
                    exp.append(lo)
            exp.append(B)
            assert got == exp, (qsl.tolist(), slices, got, exp)
    rb = (ctypes.c_int32 * 9)()
    qsl = np.zeros(1, np.int32)
    assert f(qsl.ctypes.data_as(ctypes.c_void_p), 0, 4, ctypes.cast(rb, ctypes.c_void_p)) == 0
    assert f(qsl.ctypes.data_as(ctypes.c_void_p), 0, 9, ctypes.cast(rb, ctypes.c_void_p)) == 0
    assert f(None, 3, 2, ctypes.cast(rb, ctypes.c_void_p)) == 0


def test_host_stage_host_checks(lib):
    # checks that return before any CUDA call: no stage, bad sizes
    null = ctypes.c_void_p()
    assert _fn(lib, "mcpu_host_stage_wait")(null, null) == 1
    assert _fn(lib, "mcpu_host_stage_sync")(null) == 1
    assert _fn(lib, "mcpu_host_stage_destroy")(null) == 0
    h = ctypes.c_void_p()
    create = _fn(lib, "mcpu_host_stage_create")
    assert create(0, 4, 8, 2, 2, ctypes.byref(h)) == 1
    assert create(16, 4, 8, 3, 2, ctypes.byref(h)) == 1  # H_q not a multiple of H_kv
    assert create(16, 4, 8, 2, 1, ctypes.byref(h)) == 1  # fewer than two slots
    assert create(16, 4, 8, 2, 5, ctypes.byref(h)) == 1  # more than MCPU_MAX_HOST_SLOTS
    assert create(16, 4, 8, 2, 2, None) == 1
    d = Dims(4, 4, 19, 34, 8, 2, 64, 16)
    call = _fn(lib, "mcpu_paged_attention_host")
    call.argtypes = [ctypes.c_void_p] * 9 + [ctypes.c_int32, ctypes.c_float, ctypes.c_void_p, ctypes.c_void_p,
                                             ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p,
                                             ctypes.c_int32, ctypes.c_void_p]
    assert call(None, None, None, None, None, None, None, None, None, 0, 0.125, ctypes.byref(d), None, None, None,
                0, None, 0, None) == 1
