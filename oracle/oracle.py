"""ctypes wrapper around oracle/twinkv_oracle.c.

TEST INFRASTRUCTURE ONLY (see the package docstring).  Every function here is
argument marshalling; the arithmetic is in the C file, which cites the paper passage
each step follows.  ``build()`` compiles the C file with gcc into ``oracle/_build``.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "twinkv_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libtwinkv_oracle.so")
_lock = threading.Lock()
_lib = None

_P = ctypes.c_void_p


def build(force: bool = False) -> str:
    """Compile the oracle into a shared library (OpenMP when gcc supports it)."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    os.makedirs(_BUILD, exist_ok=True)
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    base = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True,
                       capture_output=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            lib.twk_oracle_round_bf16.argtypes = [_P, _P, ctypes.c_long]
            lib.twk_oracle_sim.argtypes = [_P, _P, ctypes.c_int]
            lib.twk_oracle_sim.restype = ctypes.c_double
            lib.twk_oracle_audit.argtypes = [
                _P, ctypes.c_int, ctypes.c_int, ctypes.c_int, _P, ctypes.c_int, _P,
                ctypes.c_int, _P, _P, _P, _P, _P, _P]
            lib.twk_oracle_count.argtypes = [
                _P, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_int, ctypes.c_float,
                ctypes.c_double, _P, ctypes.c_int, _P, _P, _P]
            lib.twk_oracle_policy_select.argtypes = [
                ctypes.c_int, ctypes.c_int, _P, ctypes.c_int, ctypes.c_int, _P, _P, _P]
            lib.twk_oracle_repair_dedup.argtypes = [
                ctypes.c_int, ctypes.c_int, _P, _P, _P, _P, ctypes.c_float, ctypes.c_int,
                ctypes.c_int, _P, _P, _P, _P]
            for name in ("twk_oracle_repair", "twk_oracle_repair_f32"):
                getattr(lib, name).argtypes = [
                    ctypes.c_int, ctypes.c_int, _P, _P, _P, ctypes.c_float, ctypes.c_int,
                    ctypes.c_int, _P, _P, _P, _P, _P, _P]
            _lib = lib
    return _lib


def _ptr(a):
    return None if a is None else a.ctypes.data


def round_bf16(x) -> np.ndarray:
    """float32 array -> bf16 bit patterns (uint16), round to nearest even."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    _load().twk_oracle_round_bf16(_ptr(x), _ptr(out), x.size)
    return out


def _keys3(keys) -> np.ndarray:
    keys = np.ascontiguousarray(keys)
    if keys.dtype == np.float32:
        keys = round_bf16(keys)
    if keys.dtype != np.uint16:
        raise TypeError("keys must be bf16 bit patterns (uint16) or float32")
    if keys.ndim == 2:
        keys = keys[None]
    if keys.ndim == 4:
        keys = keys.reshape(-1, keys.shape[-2], keys.shape[-1])
    return np.ascontiguousarray(keys)


def sim(keys, u: int, i: int, j: int) -> float:
    """Eq. 1 similarity of keys i and j of unit u (keys [U,N,d] or [N,d])."""
    k = _keys3(keys)
    return float(_load().twk_oracle_sim(_ptr(k[u, i]), _ptr(k[u, j]), k.shape[2]))


def audit(keys, mask=None, window: int = 32, rows=None) -> dict:
    """Best twin over all keys and over the retained keys (Eq. 4), per unit and row.

    keys: uint16 bf16 bits (or float32, rounded to bf16 first), shape [U,N,d],
    [L,H,N,d] or [N,d].  mask: [U,N] uint8 (or matching leading dims) or None.
    rows: optional 1-D list of row positions evaluated in every unit.
    Returns arrays of shape [U, nrows]: b_all, t_all, b_all2 and, with a mask,
    b_ret, t_ret, b_ret2 (b*2 = second-largest value of that scan).
    """
    k = _keys3(keys)
    U, N, d = k.shape
    m = None
    if mask is not None:
        m = np.ascontiguousarray(np.asarray(mask, dtype=np.uint8).reshape(U, N))
    r = None
    nrows = N
    if rows is not None:
        r = np.ascontiguousarray(np.asarray(rows, dtype=np.int32).ravel())
        nrows = r.size
    out = {
        "b_all": np.empty((U, nrows), np.float64),
        "t_all": np.empty((U, nrows), np.int32),
        "b_all2": np.empty((U, nrows), np.float64),
    }
    if m is not None:
        out["b_ret"] = np.empty((U, nrows), np.float64)
        out["t_ret"] = np.empty((U, nrows), np.int32)
        out["b_ret2"] = np.empty((U, nrows), np.float64)
    _load().twk_oracle_audit(
        _ptr(k), U, N, d, _ptr(m), int(window), _ptr(r), nrows, _ptr(out["b_all"]),
        _ptr(out["t_all"]), _ptr(out["b_all2"]), _ptr(out.get("b_ret")),
        _ptr(out.get("t_ret")), _ptr(out.get("b_ret2")))
    return out


def _repair(fn, b, mask, threshold, n_sink, n_recent, budget, dtype):
    b = np.ascontiguousarray(np.asarray(b, dtype=dtype))
    U = b.shape[0] if b.ndim == 2 else 1
    b = b.reshape(U, -1)
    N = b.shape[1]
    m = np.ascontiguousarray(np.asarray(mask, dtype=np.uint8).reshape(U, N))
    bud = None
    if budget is not None:
        bud = np.ascontiguousarray(np.asarray(budget, dtype=np.int32).reshape(U))
    out = {
        "mask": np.empty((U, N), np.uint8),
        "swaps": np.full((U, N // 2, 2), -1, np.int32),
        "nswaps": np.empty(U, np.int32),
        "status": np.empty(U, np.int32),
        "orphan": np.empty((U, N), np.uint8),
        "donor": np.empty((U, N), np.uint8),
    }
    fn(U, N, _ptr(b), _ptr(m), _ptr(bud), ctypes.c_float(threshold), int(n_sink),
       int(n_recent), _ptr(out["mask"]), _ptr(out["swaps"]), _ptr(out["nswaps"]),
       _ptr(out["status"]), _ptr(out["orphan"]), _ptr(out["donor"]))
    return out


def repair(b_ret, mask, threshold: float, n_sink: int = 4, n_recent: int = 64,
           budget=None) -> dict:
    """Sec. 3.4 repair on fp64 b values [U,N]; threshold is rounded to float first."""
    return _repair(_load().twk_oracle_repair, b_ret, mask, threshold, n_sink, n_recent,
                   budget, np.float64)


def repair_f32(b_ret, mask, threshold: float, n_sink: int = 4, n_recent: int = 64,
               budget=None) -> dict:
    """Selection-only entry: the same repair on float32 b values (e.g. a GPU's own)."""
    return _repair(_load().twk_oracle_repair_f32, b_ret, mask, threshold, n_sink,
                   n_recent, budget, np.float32)


def count(keys, threshold: float, window: int = 32, band: float = 0.0, rows=None) -> dict:
    """Redundancy counts of Eq. 2 per unit and row: r (sim > tau, tau rounded to float),
    r_lo (sim > tau + band) and r_hi (sim > tau - band), each [U, nrows] int32."""
    k = _keys3(keys)
    U, N, d = k.shape
    r = None
    nrows = N
    if rows is not None:
        r = np.ascontiguousarray(np.asarray(rows, dtype=np.int32).ravel())
        nrows = r.size
    out = {n: np.empty((U, nrows), np.int32) for n in ("r", "r_lo", "r_hi")}
    _load().twk_oracle_count(_ptr(k), U, N, d, int(window), ctypes.c_float(threshold),
                             float(band), _ptr(r), nrows, _ptr(out["r"]), _ptr(out["r_lo"]),
                             _ptr(out["r_hi"]))
    return out


def policy_select(r, budget, n_sink: int = 4, n_recent: int = 64) -> dict:
    """The standalone policy of Sec. 3.2 (Eq. 3) on counts r [U,N]: keep budget[u]
    positions ordered by (protected, s = -r/N descending, position).  Returns mask
    [U,N] uint8 and status [U]."""
    r = np.ascontiguousarray(np.asarray(r, dtype=np.int32))
    U = r.shape[0] if r.ndim == 2 else 1
    r = r.reshape(U, -1)
    N = r.shape[1]
    bud = np.ascontiguousarray(np.broadcast_to(np.asarray(budget, dtype=np.int32), (U,)))
    out = {"mask": np.empty((U, N), np.uint8), "status": np.empty(U, np.int32)}
    _load().twk_oracle_policy_select(U, N, _ptr(r), int(n_sink), int(n_recent), _ptr(bud),
                                     _ptr(out["mask"]), _ptr(out["status"]))
    return out


def policy(keys, threshold: float, budget, window: int = 32, n_sink: int = 4,
           n_recent: int = 64) -> dict:
    """Counts (Eq. 2) and the policy's retained set (Eq. 3) for keys [U,N,d]."""
    c = count(keys, threshold, window)
    p = policy_select(c["r"], budget, n_sink, n_recent)
    return {"r": c["r"], **p}


def repair_dedup(b_ret, t_ret, mask, threshold: float, n_sink: int = 4, n_recent: int = 64,
                 budget=None) -> dict:
    """Sec. 3.4 repair that never evicts both members of a twin pair: donors walked in
    severity order, a donor skipped when its twin (t_ret) is already being evicted or
    when it is the twin of an evicted donor.
    b_ret fp64 [U,N], t_ret int32 [U,N]."""
    b = np.ascontiguousarray(np.asarray(b_ret, dtype=np.float64))
    U = b.shape[0] if b.ndim == 2 else 1
    b = b.reshape(U, -1)
    N = b.shape[1]
    t = np.ascontiguousarray(np.asarray(t_ret, dtype=np.int32).reshape(U, N))
    m = np.ascontiguousarray(np.asarray(mask, dtype=np.uint8).reshape(U, N))
    bud = None
    if budget is not None:
        bud = np.ascontiguousarray(np.asarray(budget, dtype=np.int32).reshape(U))
    out = {
        "mask": np.empty((U, N), np.uint8),
        "swaps": np.full((U, N // 2, 2), -1, np.int32),
        "nswaps": np.empty(U, np.int32),
        "status": np.empty(U, np.int32),
    }
    _load().twk_oracle_repair_dedup(U, N, _ptr(b), _ptr(t), _ptr(m), _ptr(bud),
                                    ctypes.c_float(threshold), int(n_sink), int(n_recent),
                                    _ptr(out["mask"]), _ptr(out["swaps"]), _ptr(out["nswaps"]),
                                    _ptr(out["status"]))
    return out
