"""Python face of the C decode-attention oracle (oracle/attention.c).

TEST INFRASTRUCTURE ONLY: see oracle/__init__.py for who may use it.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading
from typing import Optional, Sequence, Tuple

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "attention.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (plain C, OpenMP)."""
    if not force and os.path.exists(_LIB_PATH) and \
            os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC):
        return _LIB_PATH
    os.makedirs(_OUT_DIR, exist_ok=True)
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC",
                           "-shared", "-o", tmp, _SRC, "-lm"])
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def lib():
    global _lib
    with _lock:
        if _lib is None:
            path = build()
            L = ctypes.CDLL(path)
            u16p = ctypes.POINTER(ctypes.c_uint16)
            f64p = ctypes.POINTER(ctypes.c_double)
            L.oracle_decode_f64.argtypes = [
                ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                u16p, u16p, u16p, ctypes.c_double,
                ctypes.POINTER(ctypes.c_uint8), f64p, f64p, f64p]
            L.oracle_decode_f64.restype = ctypes.c_int
            L.oracle_decode_dev_f64.argtypes = [
                ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                u16p, u16p, u16p, ctypes.c_double,
                ctypes.POINTER(ctypes.c_uint8), f64p, f64p, f64p]
            L.oracle_decode_dev_f64.restype = ctypes.c_int
            L.oracle_decode_batch_f64.argtypes = [
                ctypes.c_int, ctypes.POINTER(ctypes.c_int), ctypes.c_int,
                ctypes.c_int, ctypes.c_int, u16p,
                ctypes.POINTER(u16p), ctypes.POINTER(u16p), ctypes.c_double, f64p]
            L.oracle_decode_batch_f64.restype = ctypes.c_int
            L.oracle_prefill_f64.argtypes = [
                ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int,
                u16p, u16p, u16p, ctypes.c_double,
                ctypes.POINTER(ctypes.c_uint8), f64p, f64p]
            L.oracle_prefill_f64.restype = ctypes.c_int
            L.oracle_num_threads.argtypes = []
            L.oracle_num_threads.restype = ctypes.c_int
            L.oracle_set_threads.argtypes = [ctypes.c_int]
            L.oracle_set_threads.restype = None
            _lib = L
    return _lib


def _u16(a: np.ndarray):
    assert a.dtype == np.uint16 and a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.POINTER(ctypes.c_uint16))


def num_threads() -> int:
    return int(lib().oracle_num_threads())


def set_threads(n: int) -> None:
    lib().oracle_set_threads(int(n))


def decode(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float,
           mask: Optional[np.ndarray] = None, want_weights: bool = False,
           want_lse: bool = False):
    """Decode attention of one sequence.

    q: uint16 bf16 bits [Hq, d]; k, v: uint16 bf16 bits [n, Hkv, d] in logical
    order; mask: optional bool/uint8 [n] (True = token removed).
    Returns out float64 [Hq, d] (and weights [Hq, n], lse [Hq] if asked).
    """
    q = np.ascontiguousarray(q, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    Hq, d = q.shape
    n, Hkv, d2 = k.shape
    assert d2 == d and v.shape == k.shape
    out = np.zeros((Hq, d), dtype=np.float64)
    w = np.zeros((Hq, n), dtype=np.float64) if want_weights else None
    lse = np.zeros((Hq,), dtype=np.float64) if want_lse else None
    m = None
    if mask is not None:
        m = np.ascontiguousarray(mask, dtype=np.uint8)
        assert m.shape == (n,)
    f64p = ctypes.POINTER(ctypes.c_double)
    rc = lib().oracle_decode_f64(
        n, Hq, Hkv, d, _u16(q), _u16(k), _u16(v), float(scale),
        m.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8)) if m is not None else None,
        out.ctypes.data_as(f64p),
        w.ctypes.data_as(f64p) if w is not None else None,
        lse.ctypes.data_as(f64p) if lse is not None else None)
    if rc != 0:
        raise ValueError(f"oracle_decode_f64 rejected the input (rc={rc})")
    res = [out]
    if want_weights:
        res.append(w)
    if want_lse:
        res.append(lse)
    return res[0] if len(res) == 1 else tuple(res)


def decode_dev(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float,
               mask: Optional[np.ndarray] = None):
    """Decode attention of one sequence plus two weighted spreads of V used
    by error analyses (not part of the method): returns (out, dev, absv),
    each float64 [Hq, d], with dev[h, e] = sum_t w_t |V[t, g, e] - out[h, e]|
    and absv[h, e] = sum_t w_t |V[t, g, e]| for the exact softmax weights w.
    Arguments as for decode()."""
    q = np.ascontiguousarray(q, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    Hq, d = q.shape
    n, Hkv, d2 = k.shape
    assert d2 == d and v.shape == k.shape
    out = np.zeros((Hq, d), dtype=np.float64)
    dev = np.zeros((Hq, d), dtype=np.float64)
    absv = np.zeros((Hq, d), dtype=np.float64)
    m = None
    if mask is not None:
        m = np.ascontiguousarray(mask, dtype=np.uint8)
        assert m.shape == (n,)
    f64p = ctypes.POINTER(ctypes.c_double)
    rc = lib().oracle_decode_dev_f64(
        n, Hq, Hkv, d, _u16(q), _u16(k), _u16(v), float(scale),
        m.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8)) if m is not None else None,
        out.ctypes.data_as(f64p), dev.ctypes.data_as(f64p), absv.ctypes.data_as(f64p))
    if rc != 0:
        raise ValueError(f"oracle_decode_dev_f64 rejected the input (rc={rc})")
    return out, dev, absv


def decode_batch(q: np.ndarray, ks: Sequence[np.ndarray], vs: Sequence[np.ndarray],
                 scale: float) -> np.ndarray:
    """One decode step of a batch: q uint16 [S, Hq, d]; ks[i], vs[i] uint16
    [n_i, Hkv, d].  Returns float64 [S, Hq, d]."""
    q = np.ascontiguousarray(q, dtype=np.uint16)
    S, Hq, d = q.shape
    assert len(ks) == S and len(vs) == S
    ks = [np.ascontiguousarray(k, dtype=np.uint16) for k in ks]
    vs = [np.ascontiguousarray(v, dtype=np.uint16) for v in vs]
    Hkv = ks[0].shape[1]
    ns = (ctypes.c_int * S)(*[int(k.shape[0]) for k in ks])
    u16p = ctypes.POINTER(ctypes.c_uint16)
    kp = (u16p * S)(*[_u16(k) for k in ks])
    vp = (u16p * S)(*[_u16(v) for v in vs])
    out = np.zeros((S, Hq, d), dtype=np.float64)
    rc = lib().oracle_decode_batch_f64(S, ns, Hq, Hkv, d, _u16(q), kp, vp,
                                       float(scale),
                                       out.ctypes.data_as(ctypes.POINTER(ctypes.c_double)))
    if rc != 0:
        raise ValueError(f"oracle_decode_batch_f64 rejected the input (rc={rc})")
    return out


def removed_mask(n: int, spans: Sequence[Tuple[int, int]]) -> np.ndarray:
    """uint8 [n]: 1 for tokens inside any half-open span (start, end)."""
    m = np.zeros(n, dtype=np.uint8)
    for a, b in spans:
        m[int(a):int(b)] = 1
    return m


def prefill(q: np.ndarray, k: np.ndarray, v: np.ndarray, scale: float,
            spans: Sequence[Tuple[int, int]] = (), want_lse: bool = False):
    """Masked prefill attention (Algorithm 2's BuildMask): the last n_q tokens
    of the sequence query it causally with the spans' tokens removed.

    q: uint16 bf16 bits [n_q, Hq, d]; k, v: uint16 [n, Hkv, d] in logical
    order; spans: half-open (start, end) token ranges to remove.
    Returns out float64 [n_q, Hq, d] (and lse [n_q, Hq], natural log, -inf
    for a query that sees no token)."""
    q = np.ascontiguousarray(q, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    n_q, Hq, d = q.shape
    n, Hkv, d2 = k.shape
    assert d2 == d and v.shape == k.shape
    m = removed_mask(n, spans)
    out = np.zeros((n_q, Hq, d), dtype=np.float64)
    lse = np.zeros((n_q, Hq), dtype=np.float64)
    f64p = ctypes.POINTER(ctypes.c_double)
    rc = lib().oracle_prefill_f64(n, n_q, Hq, Hkv, d, _u16(q), _u16(k), _u16(v),
                                  float(scale),
                                  m.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8)),
                                  out.ctypes.data_as(f64p), lse.ctypes.data_as(f64p))
    if rc != 0:
        raise ValueError(f"oracle_prefill_f64 rejected the input (rc={rc})")
    return (out, lse) if want_lse else out
