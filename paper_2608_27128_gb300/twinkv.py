"""Python binding of libtwinkv (include/twinkv.h): argument marshalling only.

Each function has the name of the C entry point it calls.  Tensors are torch CUDA
tensors (torch supplies device memory and streams); every computation runs in the
library's CUDA kernels.  There is no CPU fallback: if the library is missing or the
device is not an sm_103 GPU, calls raise.

Paper: TwinKV (arXiv 2608.27128) Sec. 3.2 (Eq. 1, twin window, protected regions) and
Sec. 3.4 (Eq. 4, orphans, donors, the budget-exact swap).
"""
from __future__ import annotations

import ctypes
import math
import os
import threading

import torch

from . import build as _build

(OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_BUDGET, ERR_CUDA, ERR_TIMEOUT, ERR_WORKSPACE,
 ERR_TOO_LARGE) = range(8)
NOALLOC_MAX_POSITIONS = 262144
BF16, F32 = 0, 1
(OP_REDUNDANCY, OP_REPAIR, OP_REPAIR_SELECT, OP_POLICY, OP_REPAIR_SELECT_DEDUP,
 OP_REDUNDANCY_SYMMETRIC) = range(6)
KERNEL_PREP, KERNEL_AUDIT, KERNEL_REPAIR, KERNEL_REFINE = 0, 1, 2, 3
KERNEL_NAMES = ("prep", "audit", "repair", "refine")

EXPORTED = (
    "twinkv_abi_version", "twinkv_default_params", "twinkv_swaps_capacity",
    "twinkv_workspace_size", "twinkv_redundancy", "twinkv_repair", "twinkv_repair_select",
    "twinkv_status_string", "twinkv_get_last_error", "twinkv_set_wait_timeout_ns",
    "twinkv_wait_probe", "twinkv_profile_begin", "twinkv_profile_end",
    "twinkv_repair_select_noalloc", "twinkv_host_arena_size", "twinkv_host_default_chunk",
    "twinkv_repair_host",
    "twinkv_policy", "twinkv_repair_dedup", "twinkv_repair_select_dedup",
    "twinkv_redundancy_symmetric",
)


class Shape(ctypes.Structure):
    _fields_ = [("L", ctypes.c_int32), ("H", ctypes.c_int32), ("N", ctypes.c_int32),
                ("d", ctypes.c_int32), ("dtype", ctypes.c_int32)]


class Params(ctypes.Structure):
    _fields_ = [("threshold", ctypes.c_float), ("window", ctypes.c_int32),
                ("n_sink", ctypes.c_int32), ("n_recent", ctypes.c_int32)]


class TwinKVError(RuntimeError):
    def __init__(self, status: int, what: str = ""):
        self.status = status
        super().__init__(f"{what}: {status_string(status)} (status {status})")


_P = ctypes.c_void_p
_lock = threading.Lock()
_lib = None


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True):
    """Load libtwinkv.so (building it with nvcc first when it is missing or stale)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = _build.LIB
        if build_if_missing:
            path = _build.build()
        if not os.path.exists(path):
            raise RuntimeError(f"libtwinkv.so not found at {path}; run "
                               "`python -m paper_2608_27128_gb300.build`")
        lib = ctypes.CDLL(path)
        lib.twinkv_abi_version.restype = ctypes.c_int32
        lib.twinkv_default_params.restype = Params
        lib.twinkv_swaps_capacity.argtypes = [Shape]
        lib.twinkv_swaps_capacity.restype = ctypes.c_size_t
        lib.twinkv_workspace_size.argtypes = [Shape, ctypes.c_int32]
        lib.twinkv_workspace_size.restype = ctypes.c_size_t
        lib.twinkv_redundancy.argtypes = [_P, Shape, ctypes.c_int32, _P, _P, _P,
                                          ctypes.c_size_t, _P]
        lib.twinkv_redundancy_symmetric.argtypes = lib.twinkv_redundancy.argtypes
        lib.twinkv_repair.argtypes = [_P, Shape, _P, _P, ctypes.c_float,
                                      ctypes.POINTER(Params), _P, _P, _P, _P, _P, _P, _P, _P,
                                      _P, ctypes.c_size_t, _P]
        lib.twinkv_repair_select.argtypes = [_P, Shape, _P, _P, ctypes.c_float,
                                             ctypes.POINTER(Params), _P, _P, _P, _P, _P,
                                             ctypes.c_size_t, _P]
        lib.twinkv_repair_select_noalloc.argtypes = [_P, Shape, _P, _P, ctypes.c_float,
                                                     ctypes.POINTER(Params), _P, _P, _P, _P,
                                                     _P]
        lib.twinkv_host_arena_size.argtypes = [Shape, ctypes.c_int32]
        lib.twinkv_host_arena_size.restype = ctypes.c_size_t
        lib.twinkv_host_default_chunk.argtypes = [Shape]
        lib.twinkv_host_default_chunk.restype = ctypes.c_int32
        lib.twinkv_repair_host.argtypes = [_P, Shape, _P, _P, ctypes.c_float,
                                           ctypes.POINTER(Params), _P, _P, _P, _P, _P, _P, _P,
                                           _P, ctypes.c_int32, _P, ctypes.c_size_t, _P]
        lib.twinkv_repair_dedup.argtypes = lib.twinkv_repair.argtypes
        lib.twinkv_repair_select_dedup.argtypes = [_P, _P, Shape, _P, _P, ctypes.c_float,
                                                   ctypes.POINTER(Params), _P, _P, _P, _P, _P,
                                                   ctypes.c_size_t, _P]
        lib.twinkv_policy.argtypes = [_P, Shape, _P, ctypes.c_float, ctypes.POINTER(Params),
                                      _P, _P, _P, _P, ctypes.c_size_t, _P]
        lib.twinkv_status_string.argtypes = [ctypes.c_int]
        lib.twinkv_status_string.restype = ctypes.c_char_p
        lib.twinkv_set_wait_timeout_ns.argtypes = [ctypes.c_uint64]
        lib.twinkv_wait_probe.argtypes = [ctypes.c_uint64, ctypes.POINTER(ctypes.c_int32), _P]
        lib.twinkv_profile_end.argtypes = [ctypes.POINTER(ctypes.c_int32),
                                           ctypes.POINTER(ctypes.c_double)]
        for name in ("twinkv_redundancy", "twinkv_redundancy_symmetric", "twinkv_repair",
                     "twinkv_repair_select",
                     "twinkv_repair_select_noalloc", "twinkv_repair_host", "twinkv_policy",
                     "twinkv_repair_dedup", "twinkv_repair_select_dedup",
                     "twinkv_get_last_error", "twinkv_set_wait_timeout_ns",
                     "twinkv_wait_probe", "twinkv_profile_begin", "twinkv_profile_end"):
            getattr(lib, name).restype = ctypes.c_int
        _lib = lib
        return lib


def status_string(status: int) -> str:
    try:
        return load().twinkv_status_string(int(status)).decode()
    except Exception:  # the library itself failed to load
        return f"status {status}"


def _check(status: int, what: str):
    if status != OK:
        raise TwinKVError(status, what)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _need(t, name, dtype, shape, device):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch tensor")
    if t.device != device or not t.is_cuda:
        raise ValueError(f"{name} must live on {device}")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t


def _out(t, name, dtype, shape, device):
    if t is None:
        return torch.empty(shape, dtype=dtype, device=device)
    return _need(t, name, dtype, shape, device)


def shape_of(keys) -> Shape:
    if keys.dim() != 4:
        raise ValueError("keys must be [L, H, N, d]")
    if keys.dtype == torch.bfloat16:
        dt = BF16
    elif keys.dtype == torch.float32:
        dt = F32
    else:
        raise ValueError("keys must be bfloat16 or float32")
    L, H, N, d = (int(x) for x in keys.shape)
    return Shape(L, H, N, d, dt)


def twinkv_default_params() -> Params:
    return load().twinkv_default_params()


def twinkv_swaps_capacity(shape: Shape) -> int:
    return int(load().twinkv_swaps_capacity(shape))


def twinkv_workspace_size(shape: Shape, op: int) -> int:
    return int(load().twinkv_workspace_size(shape, int(op)))


def workspace(shape: Shape, op: int, device) -> torch.Tensor:
    """A device workspace of the size `op` needs (torch's allocator: 512-byte aligned)."""
    n = twinkv_workspace_size(shape, op)
    return torch.empty(max(n, 1), dtype=torch.uint8, device=device)


def _ws(ws, shape, op, device):
    need = twinkv_workspace_size(shape, op)
    if ws is None:
        ws = workspace(shape, op, device)
    if ws.numel() < need:
        raise ValueError(f"workspace needs {need} bytes, got {ws.numel()}")
    return ws


def twinkv_redundancy(keys, window: int = 32, out_score=None, out_twin=None, ws=None,
                      stream=None):
    """Best twin of every key over all other keys outside the +-window band.

    keys: [L,H,N,d] bf16/float32 CUDA tensor.  Returns (score float64 [L,H,N],
    twin int32 [L,H,N]); score = -1 and twin = -1 where no position lies beyond w.
    """
    s = shape_of(keys)
    dev = keys.device
    _need(keys, "keys", keys.dtype, keys.shape, dev)
    out_score = _out(out_score, "out_score", torch.float64, keys.shape[:3], dev)
    out_twin = _out(out_twin, "out_twin", torch.int32, keys.shape[:3], dev)
    ws = _ws(ws, s, OP_REDUNDANCY, dev)
    st = load().twinkv_redundancy(_ptr(keys), s, int(window), _ptr(out_score), _ptr(out_twin),
                                  _ptr(ws), ws.numel(), _stream(stream))
    _check(st, "twinkv_redundancy")
    return out_score, out_twin


def twinkv_redundancy_symmetric(keys, window: int = 32, out_score=None, out_twin=None,
                                ws=None, stream=None):
    """twinkv_redundancy from the upper-triangle similarity tiles only (each tile serves
    its rows and its columns); same arguments and results."""
    s = shape_of(keys)
    dev = keys.device
    _need(keys, "keys", keys.dtype, keys.shape, dev)
    out_score = _out(out_score, "out_score", torch.float64, keys.shape[:3], dev)
    out_twin = _out(out_twin, "out_twin", torch.int32, keys.shape[:3], dev)
    ws = _ws(ws, s, OP_REDUNDANCY_SYMMETRIC, dev)
    st = load().twinkv_redundancy_symmetric(_ptr(keys), s, int(window), _ptr(out_score),
                                            _ptr(out_twin), _ptr(ws), ws.numel(),
                                            _stream(stream))
    _check(st, "twinkv_redundancy_symmetric")
    return out_score, out_twin


def _params(params, threshold, window, n_sink, n_recent):
    p = twinkv_default_params() if params is None else params
    p = Params(p.threshold, p.window, p.n_sink, p.n_recent)
    if threshold is not None:
        p.threshold = float(threshold)
    if window is not None:
        p.window = int(window)
    if n_sink is not None:
        p.n_sink = int(n_sink)
    if n_recent is not None:
        p.n_recent = int(n_recent)
    return p


def twinkv_repair_dedup(keys, retained_mask, budget=None, threshold=None, params=None,
                        **kw) -> dict:
    """twinkv_repair, but a donor is never evicted together with its twin (see the C
    header); same arguments and outputs."""
    return twinkv_repair(keys, retained_mask, budget, threshold, params, _fn="twinkv_repair_dedup",
                         **kw)


def twinkv_repair(keys, retained_mask, budget=None, threshold=None, params=None, *,
                  window=None, n_sink=None, n_recent=None, want_ret=True, want_all=False,
                  out=None, ws=None, stream=None, _fn="twinkv_repair") -> dict:
    """Audit of the retained set S0 and the budget-exact orphan/donor swap.

    keys [L,H,N,d] bf16/float32; retained_mask [L,H,N] uint8; budget [L*H] int32 or None.
    Returns a dict of CUDA tensors: mask (S1), swaps [L*H, N//2, 2], nswaps, status,
    and score_ret/twin_ret (b_i(S0)) if want_ret, score_all/twin_all if want_all.
    ``out`` may hold preallocated tensors under the same keys.
    """
    s = shape_of(keys)
    dev = keys.device
    _need(keys, "keys", keys.dtype, keys.shape, dev)
    L, H, N = s.L, s.H, s.N
    _need(retained_mask, "retained_mask", torch.uint8, (L, H, N), dev)
    if budget is not None:
        _need(budget, "budget", torch.int32, (L * H,), dev)
    p = _params(params, threshold, window, n_sink, n_recent)
    out = dict(out or {})
    o = {
        "mask": _out(out.get("mask"), "mask", torch.uint8, (L, H, N), dev),
        "swaps": _out(out.get("swaps"), "swaps", torch.int32, (L * H, N // 2, 2), dev),
        "nswaps": _out(out.get("nswaps"), "nswaps", torch.int32, (L * H,), dev),
        "status": _out(out.get("status"), "status", torch.int32, (L * H,), dev),
    }
    if want_ret:
        o["score_ret"] = _out(out.get("score_ret"), "score_ret", torch.float64, (L, H, N), dev)
        o["twin_ret"] = _out(out.get("twin_ret"), "twin_ret", torch.int32, (L, H, N), dev)
    if want_all:
        o["score_all"] = _out(out.get("score_all"), "score_all", torch.float64, (L, H, N), dev)
        o["twin_all"] = _out(out.get("twin_all"), "twin_all", torch.int32, (L, H, N), dev)
    ws = _ws(ws, s, OP_REPAIR, dev)
    st = getattr(load(), _fn)(
        _ptr(keys), s, _ptr(retained_mask), _ptr(budget), ctypes.c_float(p.threshold),
        ctypes.byref(p), _ptr(o["mask"]), _ptr(o["swaps"]), _ptr(o["nswaps"]),
        _ptr(o.get("score_ret")), _ptr(o.get("twin_ret")), _ptr(o.get("score_all")),
        _ptr(o.get("twin_all")), _ptr(o["status"]), _ptr(ws), ws.numel(), _stream(stream))
    _check(st, _fn)
    return o


def twinkv_repair_select_dedup(score_ret, twin_ret, retained_mask, budget=None, threshold=None,
                               params=None, *, n_sink=None, n_recent=None, out=None, ws=None,
                               stream=None) -> dict:
    """The dedup selection alone, on given float64 b_i(S0) and int32 twins [L,H,N]."""
    if score_ret.dim() != 3:
        raise ValueError("score_ret must be [L, H, N]")
    L, H, N = (int(x) for x in score_ret.shape)
    dev = score_ret.device
    _need(score_ret, "score_ret", torch.float64, (L, H, N), dev)
    _need(twin_ret, "twin_ret", torch.int32, (L, H, N), dev)
    _need(retained_mask, "retained_mask", torch.uint8, (L, H, N), dev)
    if budget is not None:
        _need(budget, "budget", torch.int32, (L * H,), dev)
    s = Shape(L, H, N, 64, BF16)
    p = _params(params, threshold, None, n_sink, n_recent)
    out = dict(out or {})
    o = {
        "mask": _out(out.get("mask"), "mask", torch.uint8, (L, H, N), dev),
        "swaps": _out(out.get("swaps"), "swaps", torch.int32, (L * H, N // 2, 2), dev),
        "nswaps": _out(out.get("nswaps"), "nswaps", torch.int32, (L * H,), dev),
        "status": _out(out.get("status"), "status", torch.int32, (L * H,), dev),
    }
    ws = _ws(ws, s, OP_REPAIR_SELECT_DEDUP, dev)
    st = load().twinkv_repair_select_dedup(
        _ptr(score_ret), _ptr(twin_ret), s, _ptr(retained_mask), _ptr(budget),
        ctypes.c_float(p.threshold), ctypes.byref(p), _ptr(o["mask"]), _ptr(o["swaps"]),
        _ptr(o["nswaps"]), _ptr(o["status"]), _ptr(ws), ws.numel(), _stream(stream))
    _check(st, "twinkv_repair_select_dedup")
    return o


def twinkv_repair_select(score_ret, retained_mask, budget=None, threshold=None, params=None,
                         *, n_sink=None, n_recent=None, out=None, ws=None,
                         stream=None) -> dict:
    """The classification, ranking and swap alone, on given float64 b_i(S0) [L,H,N]."""
    if score_ret.dim() != 3:
        raise ValueError("score_ret must be [L, H, N]")
    L, H, N = (int(x) for x in score_ret.shape)
    dev = score_ret.device
    _need(score_ret, "score_ret", torch.float64, (L, H, N), dev)
    _need(retained_mask, "retained_mask", torch.uint8, (L, H, N), dev)
    if budget is not None:
        _need(budget, "budget", torch.int32, (L * H,), dev)
    s = Shape(L, H, N, 64, BF16)
    p = _params(params, threshold, None, n_sink, n_recent)
    out = dict(out or {})
    o = {
        "mask": _out(out.get("mask"), "mask", torch.uint8, (L, H, N), dev),
        "swaps": _out(out.get("swaps"), "swaps", torch.int32, (L * H, N // 2, 2), dev),
        "nswaps": _out(out.get("nswaps"), "nswaps", torch.int32, (L * H,), dev),
        "status": _out(out.get("status"), "status", torch.int32, (L * H,), dev),
    }
    ws = _ws(ws, s, OP_REPAIR_SELECT, dev)
    st = load().twinkv_repair_select(
        _ptr(score_ret), s, _ptr(retained_mask), _ptr(budget), ctypes.c_float(p.threshold),
        ctypes.byref(p), _ptr(o["mask"]), _ptr(o["swaps"]), _ptr(o["nswaps"]),
        _ptr(o["status"]), _ptr(ws), ws.numel(), _stream(stream))
    _check(st, "twinkv_repair_select")
    return o


def twinkv_repair_select_noalloc(score_ret, retained_mask, budget=None, threshold=None,
                                 params=None, *, n_sink=None, n_recent=None, out=None,
                                 stream=None) -> dict:
    """twinkv_repair_select without a workspace, for callers that may not allocate
    device memory: the library's own fixed scratch array holds the sort buffers, so at
    most NOALLOC_MAX_POSITIONS positions (L*H*N) per call, and calls that may run
    concurrently on the GPU must be ordered on one stream.  Output tensors are created
    here when ``out`` does not supply them; pass them in ``out`` to allocate nothing."""
    if score_ret.dim() != 3:
        raise ValueError("score_ret must be [L, H, N]")
    L, H, N = (int(x) for x in score_ret.shape)
    dev = score_ret.device
    _need(score_ret, "score_ret", torch.float64, (L, H, N), dev)
    _need(retained_mask, "retained_mask", torch.uint8, (L, H, N), dev)
    if budget is not None:
        _need(budget, "budget", torch.int32, (L * H,), dev)
    s = Shape(L, H, N, 64, BF16)
    p = _params(params, threshold, None, n_sink, n_recent)
    out = dict(out or {})
    o = {
        "mask": _out(out.get("mask"), "mask", torch.uint8, (L, H, N), dev),
        "swaps": _out(out.get("swaps"), "swaps", torch.int32, (L * H, N // 2, 2), dev),
        "nswaps": _out(out.get("nswaps"), "nswaps", torch.int32, (L * H,), dev),
        "status": _out(out.get("status"), "status", torch.int32, (L * H,), dev),
    }
    st = load().twinkv_repair_select_noalloc(
        _ptr(score_ret), s, _ptr(retained_mask), _ptr(budget), ctypes.c_float(p.threshold),
        ctypes.byref(p), _ptr(o["mask"]), _ptr(o["swaps"]), _ptr(o["nswaps"]),
        _ptr(o["status"]), _stream(stream))
    _check(st, "twinkv_repair_select_noalloc")
    return o


def budget_for_ratio(N: int, ratio: float) -> int:
    """Retained count of Sec. 3.1: |S| = ceil((1 - rho) n)."""
    return int(math.ceil((1.0 - float(ratio)) * N - 1e-9))


def twinkv_policy(keys, budget, threshold=None, params=None, *, window=None, n_sink=None,
                  n_recent=None, want_count=True, out=None, ws=None, stream=None) -> dict:
    """The standalone TwinKV policy (Sec. 3.2, Eq. 2-3) on keys [L,H,N,d].

    budget: int32 CUDA tensor [L*H], or an int used for every unit.  Returns a dict of
    CUDA tensors: mask [L,H,N] uint8 (kept positions), status [L*H] int32 and, with
    want_count, count [L,H,N] int32 (r_i of Eq. 2).
    """
    s = shape_of(keys)
    dev = keys.device
    _need(keys, "keys", keys.dtype, keys.shape, dev)
    L, H, N = s.L, s.H, s.N
    if not isinstance(budget, torch.Tensor):
        budget = torch.full((L * H,), int(budget), dtype=torch.int32, device=dev)
    _need(budget, "budget", torch.int32, (L * H,), dev)
    p = _params(params, threshold, window, n_sink, n_recent)
    out = dict(out or {})
    o = {
        "mask": _out(out.get("mask"), "mask", torch.uint8, (L, H, N), dev),
        "status": _out(out.get("status"), "status", torch.int32, (L * H,), dev),
    }
    if want_count:
        o["count"] = _out(out.get("count"), "count", torch.int32, (L, H, N), dev)
    ws = _ws(ws, s, OP_POLICY, dev)
    st = load().twinkv_policy(
        _ptr(keys), s, _ptr(budget), ctypes.c_float(p.threshold), ctypes.byref(p),
        _ptr(o["mask"]), _ptr(o.get("count")), _ptr(o["status"]), _ptr(ws), ws.numel(),
        _stream(stream))
    _check(st, "twinkv_policy")
    return o


def _need_host(t, name, dtype, shape):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch tensor")
    if t.device.type != "cpu":
        raise ValueError(f"{name} must be a host tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t


def _out_host(t, name, dtype, shape, pin):
    if t is None:
        return torch.empty(shape, dtype=dtype, pin_memory=pin)
    return _need_host(t, name, dtype, shape)


def twinkv_host_default_chunk(shape: Shape) -> int:
    """Units per chunk twinkv_repair_host uses when chunk_units is 0."""
    return int(load().twinkv_host_default_chunk(shape))


def twinkv_host_arena_size(shape: Shape, chunk_units: int = 0) -> int:
    return int(load().twinkv_host_arena_size(shape, int(chunk_units)))


def host_arena(shape: Shape, chunk_units: int = 0, device=None) -> torch.Tensor:
    """A device arena for twinkv_repair_host (torch's allocator: 512-byte aligned)."""
    n = twinkv_host_arena_size(shape, chunk_units)
    if n == 0:
        raise ValueError("invalid shape or chunk size")
    return torch.empty(n, dtype=torch.uint8, device=device or torch.cuda.current_device())


_arenas = {}


def _cached_arena(shape: Shape, chunk_units: int) -> torch.Tensor:
    """The binding's own arena for the current device, grown on demand.  It stays alive
    between calls because the library's copy streams may still be using it when a call
    returns; the library orders successive calls' use of it."""
    dev = torch.cuda.current_device()
    n = twinkv_host_arena_size(shape, chunk_units)
    if n == 0:
        raise ValueError("invalid shape or chunk size")
    a = _arenas.get(dev)
    if a is None or a.numel() < n:
        if a is not None:
            torch.cuda.synchronize(dev)   # the old arena may still be in use
        a = _arenas[dev] = torch.empty(n, dtype=torch.uint8, device=dev)
    return a


def twinkv_repair_host(keys, retained_mask, budget=None, threshold=None, params=None, *,
                       window=None, n_sink=None, n_recent=None, want_ret=True, want_all=False,
                       chunk_units=0, out=None, arena=None, stream=None) -> dict:
    """twinkv_repair on HOST tensors (a cache held in host memory): the units go to the
    device in chunks whose copies overlap the computation of other chunks.  Inputs and
    the returned outputs are CPU tensors (pinned ones copy asynchronously); the outputs
    are valid once ``stream`` (default: the current stream) has completed.  ``arena`` is
    a device uint8 tensor of twinkv_host_arena_size bytes that the caller keeps alive
    until the stream has completed (a cached one of the binding's when not given)."""
    s = shape_of(keys)
    _need_host(keys, "keys", keys.dtype, keys.shape)
    L, H, N = s.L, s.H, s.N
    _need_host(retained_mask, "retained_mask", torch.uint8, (L, H, N))
    if budget is not None:
        _need_host(budget, "budget", torch.int32, (L * H,))
    p = _params(params, threshold, window, n_sink, n_recent)
    pin = keys.is_pinned()
    out = dict(out or {})
    o = {
        "mask": _out_host(out.get("mask"), "mask", torch.uint8, (L, H, N), pin),
        "swaps": _out_host(out.get("swaps"), "swaps", torch.int32, (L * H, N // 2, 2), pin),
        "nswaps": _out_host(out.get("nswaps"), "nswaps", torch.int32, (L * H,), pin),
        "status": _out_host(out.get("status"), "status", torch.int32, (L * H,), pin),
    }
    if want_ret:
        o["score_ret"] = _out_host(out.get("score_ret"), "score_ret", torch.float64,
                                   (L, H, N), pin)
        o["twin_ret"] = _out_host(out.get("twin_ret"), "twin_ret", torch.int32, (L, H, N), pin)
    if want_all:
        o["score_all"] = _out_host(out.get("score_all"), "score_all", torch.float64,
                                   (L, H, N), pin)
        o["twin_all"] = _out_host(out.get("twin_all"), "twin_all", torch.int32, (L, H, N), pin)
    if arena is None:
        arena = _cached_arena(s, chunk_units)
    if not arena.is_cuda or arena.dtype != torch.uint8:
        raise ValueError("arena must be a CUDA uint8 tensor")
    st = load().twinkv_repair_host(
        _ptr(keys), s, _ptr(retained_mask), _ptr(budget), ctypes.c_float(p.threshold),
        ctypes.byref(p), _ptr(o["mask"]), _ptr(o["swaps"]), _ptr(o["nswaps"]),
        _ptr(o.get("score_ret")), _ptr(o.get("twin_ret")), _ptr(o.get("score_all")),
        _ptr(o.get("twin_all")), _ptr(o["status"]), int(chunk_units), _ptr(arena),
        arena.numel(), _stream(stream))
    _check(st, "twinkv_repair_host")
    return o


def twinkv_get_last_error() -> int:
    return int(load().twinkv_get_last_error())


def twinkv_set_wait_timeout_ns(ns: int):
    _check(load().twinkv_set_wait_timeout_ns(int(ns)), "twinkv_set_wait_timeout_ns")


def twinkv_wait_probe(timeout_ns: int, stream=None) -> int:
    out = ctypes.c_int32(-1)
    _check(load().twinkv_wait_probe(int(timeout_ns), ctypes.byref(out), _stream(stream)),
           "twinkv_wait_probe")
    return int(out.value)


def twinkv_profile_begin():
    _check(load().twinkv_profile_begin(), "twinkv_profile_begin")


def twinkv_profile_end() -> dict:
    k = len(KERNEL_NAMES)
    n = (ctypes.c_int32 * k)()
    ms = (ctypes.c_double * k)()
    _check(load().twinkv_profile_end(n, ms), "twinkv_profile_end")
    return {KERNEL_NAMES[i]: (int(n[i]), float(ms[i])) for i in range(k)}
