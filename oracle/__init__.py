"""CPU oracle for the paged-attention hot path (test infrastructure only).

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package. The product path (the CUDA library and
its binding) never does, and this package imports nothing from it.

``mcpu_oracle.c`` is the plain definition (fp64 accumulation, bf16 rounding
at the end); ``brute.py`` is a second, independent numpy formulation used to
pin it on tiny inputs. Inputs are numpy arrays; bf16 travels as uint16 bits.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "mcpu_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "liboracle.so")
_lock = threading.Lock()
_lib = None

ERRORS = {1: "shape", 2: "length", 3: "page", 4: "nomem"}


class OracleError(RuntimeError):
    pass


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (-O2, OpenMP) into oracle/_build/."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", _SRC, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i32, i64, f64 = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
            lib.oracle_kv_append.argtypes = [P, P, P, P, P, P, P, i32, i32, i64, i32, i32, i32]
            lib.oracle_kv_append.restype = ctypes.c_int
            lib.oracle_paged_attention.argtypes = [
                P, P, P, P, P, P, i32, i32, i64, i32, i32, i32, i32, i32, f64, P, P, i32, P
            ]
            lib.oracle_paged_attention.restype = ctypes.c_int
            lib.oracle_paged_attention_sampled.argtypes = [
                P, P, P, P, P, P, i32, i32, i64, i32, i32, i32, i32, i32, f64, P, P, i64, P, P, i32, P
            ]
            lib.oracle_paged_attention_sampled.restype = ctypes.c_int
            lib.oracle_paged_attention_fp8.argtypes = [
                P, P, P, P, P, P, P, P, i32, i32, i64, i32, i32, i32, i32, i32, f64, P, P, i32, P
            ]
            lib.oracle_paged_attention_fp8.restype = ctypes.c_int
            lib.oracle_paged_attention_sampled_fp8.argtypes = [
                P, P, P, P, P, P, P, P, i32, i32, i64, i32, i32, i32, i32, i32, f64, P, P, i64, P, P, i32, P
            ]
            lib.oracle_paged_attention_sampled_fp8.restype = ctypes.c_int
            lib.oracle_kv_append_fp8.argtypes = [P, P, P, P, P, P, P, P, P, i32, i32, i64, i32, i32, i32]
            lib.oracle_kv_append_fp8.restype = ctypes.c_int
            lib.oracle_e4m3_to_double.argtypes = [ctypes.c_uint8]
            lib.oracle_e4m3_to_double.restype = f64
            lib.oracle_float_to_e4m3.argtypes = [ctypes.c_float]
            lib.oracle_float_to_e4m3.restype = ctypes.c_uint8
            lib.oracle_rope.argtypes = [P, i64, i32, i32, P, P, i64]
            lib.oracle_rope.restype = ctypes.c_int
            lib.oracle_double_to_bf16.argtypes = [f64]
            lib.oracle_double_to_bf16.restype = ctypes.c_uint16
            lib.oracle_max_threads.restype = ctypes.c_int
            _lib = lib
    return _lib


def _c(a, dtype):
    a = np.ascontiguousarray(a, dtype=dtype)
    return a, a.ctypes.data_as(ctypes.c_void_p)


def _check(rc):
    if rc != 0:
        raise OracleError(f"oracle rejected its inputs: {ERRORS.get(rc, rc)}")


def max_threads() -> int:
    return int(_load().oracle_max_threads())


def double_to_bf16(x: float) -> int:
    return int(_load().oracle_double_to_bf16(float(x)))


def kv_append(k_new, v_new, k_cache, v_cache, block_table, seq_lens, query_start_loc, page_size=16):
    """Return copies of (k_cache, v_cache) with the new rows written in."""
    lib = _load()
    k_cache = np.array(k_cache, dtype=np.uint16, copy=True, order="C")
    v_cache = np.array(v_cache, dtype=np.uint16, copy=True, order="C")
    kn, kn_p = _c(k_new, np.uint16)
    vn, vn_p = _c(v_new, np.uint16)
    bt, bt_p = _c(block_table, np.int32)
    sl, sl_p = _c(seq_lens, np.int32)
    qs, qs_p = _c(query_start_loc, np.int32)
    num_pages, hkv, page, d = k_cache.shape
    assert page == page_size
    rc = lib.oracle_kv_append(
        kn_p, vn_p, k_cache.ctypes.data_as(ctypes.c_void_p), v_cache.ctypes.data_as(ctypes.c_void_p),
        bt_p, sl_p, qs_p, sl.shape[0], bt.shape[1] if bt.ndim == 2 else 0, num_pages, hkv, d, page,
    )
    _check(rc)
    return k_cache, v_cache


def _sinks(sinks, hq):
    if sinks is None:
        return None, None
    a, p = _c(sinks, np.float32)
    assert a.shape == (hq,)
    return a, p


def paged_attention(q, k_cache, v_cache, block_table, seq_lens, query_start_loc, sliding_window,
                    softmax_scale, num_threads=0, sinks=None):
    """Return (out [T, Hq, D] uint16 bf16 bits, lse [T, Hq] float32).
    sinks: optional per-q-head sink logits [Hq] (natural-log units)."""
    lib = _load()
    q, q_p = _c(q, np.uint16)
    kc, kc_p = _c(k_cache, np.uint16)
    vc, vc_p = _c(v_cache, np.uint16)
    bt, bt_p = _c(block_table, np.int32)
    sl, sl_p = _c(seq_lens, np.int32)
    qs, qs_p = _c(query_start_loc, np.int32)
    T, hq, d = q.shape
    num_pages, hkv, page, d2 = kc.shape
    assert d == d2
    sk, sk_p = _sinks(sinks, hq)
    out = np.zeros((T, hq, d), np.uint16)
    lse = np.zeros((T, hq), np.float32)
    rc = lib.oracle_paged_attention(
        q_p, kc_p, vc_p, bt_p, sl_p, qs_p, sl.shape[0], bt.shape[1], num_pages, hq, hkv, d, page,
        int(sliding_window), float(softmax_scale), out.ctypes.data_as(ctypes.c_void_p),
        lse.ctypes.data_as(ctypes.c_void_p), int(num_threads), sk_p,
    )
    _check(rc)
    return out, lse


def paged_attention_sampled(q, k_cache, v_cache, block_table, seq_lens, query_start_loc,
                            sliding_window, softmax_scale, tokens, heads, num_threads=0, sinks=None):
    """The oracle at listed (token, q head) pairs: (out [n, D] bits, lse [n])."""
    lib = _load()
    q, q_p = _c(q, np.uint16)
    kc, kc_p = _c(k_cache, np.uint16)
    vc, vc_p = _c(v_cache, np.uint16)
    bt, bt_p = _c(block_table, np.int32)
    sl, sl_p = _c(seq_lens, np.int32)
    qs, qs_p = _c(query_start_loc, np.int32)
    tk, tk_p = _c(tokens, np.int64)
    hd, hd_p = _c(heads, np.int32)
    T, hq, d = q.shape
    num_pages, hkv, page, _ = kc.shape
    n = tk.shape[0]
    sk, sk_p = _sinks(sinks, hq)
    out = np.zeros((n, d), np.uint16)
    lse = np.zeros((n,), np.float32)
    rc = lib.oracle_paged_attention_sampled(
        q_p, kc_p, vc_p, bt_p, sl_p, qs_p, sl.shape[0], bt.shape[1], num_pages, hq, hkv, d, page,
        int(sliding_window), float(softmax_scale), tk_p, hd_p, n, out.ctypes.data_as(ctypes.c_void_p),
        lse.ctypes.data_as(ctypes.c_void_p), int(num_threads), sk_p,
    )
    _check(rc)
    return out, lse


def bf16_bits_to_float(a) -> np.ndarray:
    """uint16 bf16 bit patterns -> float32 values (exact)."""
    a = np.asarray(a, dtype=np.uint16)
    return (a.astype(np.uint32) << 16).view(np.float32)


def token_positions(seq_lens, query_start_loc) -> np.ndarray:
    """Position of every query token: S_r - L_r + i for token i of row r."""
    sl = np.asarray(seq_lens, np.int64)
    qsl = np.asarray(query_start_loc, np.int64)
    pos = np.zeros(int(qsl[-1]), np.int64)
    for r in range(len(sl)):
        L = qsl[r + 1] - qsl[r]
        pos[qsl[r]:qsl[r + 1]] = sl[r] - L + np.arange(L)
    return pos


def rope(x, positions, cos_sin):
    """Rotary embedding (step 4) of x [n, heads, D] bf16 bits at the given
    positions with the table cos_sin [max_position, D]; returns a copy."""
    lib = _load()
    x = np.array(x, dtype=np.uint16, copy=True, order="C")
    pos, pos_p = _c(positions, np.int64)
    cs, cs_p = _c(cos_sin, np.float32)
    n, heads, d = x.shape
    assert cs.shape[1] == d and pos.shape == (n,)
    rc = lib.oracle_rope(x.ctypes.data_as(ctypes.c_void_p), n, heads, d, pos_p, cs_p, cs.shape[0])
    _check(rc)
    return x


# ------------------------------------------------------------ fp8 pages (step 5)


def e4m3_to_float(code: int) -> float:
    return float(_load().oracle_e4m3_to_double(int(code)))


def float_to_e4m3(x: float) -> int:
    return int(_load().oracle_float_to_e4m3(float(x)))


def kv_append_fp8(k_new, v_new, k8, v8, k_scale, v_scale, block_table, seq_lens, query_start_loc, page_size=16):
    """Copies of the fp8 pools (codes uint8 [P, Hkv, page, D]) and scales
    (float32 [P, Hkv, page]) with the new rows quantized and written in."""
    lib = _load()
    k8 = np.array(k8, dtype=np.uint8, copy=True, order="C")
    v8 = np.array(v8, dtype=np.uint8, copy=True, order="C")
    ks = np.array(k_scale, dtype=np.float32, copy=True, order="C")
    vs = np.array(v_scale, dtype=np.float32, copy=True, order="C")
    kn, kn_p = _c(k_new, np.uint16)
    vn, vn_p = _c(v_new, np.uint16)
    bt, bt_p = _c(block_table, np.int32)
    sl, sl_p = _c(seq_lens, np.int32)
    qs, qs_p = _c(query_start_loc, np.int32)
    num_pages, hkv, page, d = k8.shape
    assert page == page_size
    P = ctypes.c_void_p
    rc = lib.oracle_kv_append_fp8(kn_p, vn_p, k8.ctypes.data_as(P), v8.ctypes.data_as(P), ks.ctypes.data_as(P),
                                  vs.ctypes.data_as(P), bt_p, sl_p, qs_p, sl.shape[0], bt.shape[1], num_pages, hkv,
                                  d, page)
    _check(rc)
    return k8, v8, ks, vs


def paged_attention_fp8(q, k8, v8, k_scale, v_scale, block_table, seq_lens, query_start_loc, sliding_window,
                        softmax_scale, num_threads=0, sinks=None):
    """Attention over fp8 pools: (out bf16 bits, lse)."""
    lib = _load()
    q, q_p = _c(q, np.uint16)
    k8, k8_p = _c(k8, np.uint8)
    v8, v8_p = _c(v8, np.uint8)
    ks, ks_p = _c(k_scale, np.float32)
    vs, vs_p = _c(v_scale, np.float32)
    bt, bt_p = _c(block_table, np.int32)
    sl, sl_p = _c(seq_lens, np.int32)
    qs, qs_p = _c(query_start_loc, np.int32)
    T, hq, d = q.shape
    num_pages, hkv, page, _ = k8.shape
    sk, sk_p = _sinks(sinks, hq)
    out = np.zeros((T, hq, d), np.uint16)
    lse = np.zeros((T, hq), np.float32)
    rc = lib.oracle_paged_attention_fp8(q_p, k8_p, v8_p, ks_p, vs_p, bt_p, sl_p, qs_p, sl.shape[0], bt.shape[1],
                                        num_pages, hq, hkv, d, page, int(sliding_window), float(softmax_scale),
                                        out.ctypes.data_as(ctypes.c_void_p), lse.ctypes.data_as(ctypes.c_void_p),
                                        int(num_threads), sk_p)
    _check(rc)
    return out, lse


def paged_attention_sampled_fp8(q, k8, v8, k_scale, v_scale, block_table, seq_lens, query_start_loc,
                                sliding_window, softmax_scale, tokens, heads, num_threads=0, sinks=None):
    lib = _load()
    q, q_p = _c(q, np.uint16)
    k8, k8_p = _c(k8, np.uint8)
    v8, v8_p = _c(v8, np.uint8)
    ks, ks_p = _c(k_scale, np.float32)
    vs, vs_p = _c(v_scale, np.float32)
    bt, bt_p = _c(block_table, np.int32)
    sl, sl_p = _c(seq_lens, np.int32)
    qs, qs_p = _c(query_start_loc, np.int32)
    tk, tk_p = _c(tokens, np.int64)
    hd, hd_p = _c(heads, np.int32)
    T, hq, d = q.shape
    num_pages, hkv, page, _ = k8.shape
    n = tk.shape[0]
    sk, sk_p = _sinks(sinks, hq)
    out = np.zeros((n, d), np.uint16)
    lse = np.zeros((n,), np.float32)
    rc = lib.oracle_paged_attention_sampled_fp8(q_p, k8_p, v8_p, ks_p, vs_p, bt_p, sl_p, qs_p, sl.shape[0],
                                                bt.shape[1], num_pages, hq, hkv, d, page, int(sliding_window),
                                                float(softmax_scale), tk_p, hd_p, n,
                                                out.ctypes.data_as(ctypes.c_void_p),
                                                lse.ctypes.data_as(ctypes.c_void_p), int(num_threads), sk_p)
    _check(rc)
    return out, lse
