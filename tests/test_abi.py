"""The C ABI without a GPU: the library loads, exports every entry point the header
declares, and rejects host-visible argument errors before touching any device."""
import ctypes
import os
import re

import pytest

from paper_2608_27128_gb300 import twinkv as tk

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include",
                      "twinkv.h")
FAKE = ctypes.c_void_p(1 << 20)     # never dereferenced: validation fails first


@pytest.fixture(scope="module")
def lib():
    return tk.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(twinkv_[a-z_0-9]+)\s*\(", text)))


def test_header_and_binding_agree():
    assert declared_functions() == sorted(tk.EXPORTED)


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_defaults_and_sizes(lib):
    p = tk.twinkv_default_params()
    assert (round(p.threshold, 6), p.window, p.n_sink, p.n_recent) == (0.85, 32, 4, 64)
    assert lib.twinkv_abi_version() == 1
    s = tk.Shape(36, 8, 16384, 128, tk.BF16)
    assert tk.twinkv_swaps_capacity(s) == 36 * 8 * 8192 * 2
    assert tk.twinkv_swaps_capacity(tk.Shape(1, 1, 7, 64, tk.BF16)) == 6
    r = tk.twinkv_workspace_size(s, tk.OP_REDUNDANCY)
    f = tk.twinkv_workspace_size(s, tk.OP_REPAIR)
    sel = tk.twinkv_workspace_size(s, tk.OP_REPAIR_SELECT)
    assert 0 < r < f and 0 < sel < f
    # the repair workspace holds a retained-first copy of every unit's keys
    assert f > 36 * 8 * 16384 * 128 * 2
    assert tk.twinkv_workspace_size(tk.Shape(36, 8, 16384, 128, tk.F32), tk.OP_REPAIR) > f
    for bad in (tk.Shape(0, 1, 10, 64, 0), tk.Shape(1, 1, 10, 96, 0),
                tk.Shape(1, 1, 10, 64, 7), tk.Shape(1, 1, (1 << 20) + 1, 64, 0)):
        assert tk.twinkv_workspace_size(bad, tk.OP_REPAIR) == 0
    assert tk.twinkv_workspace_size(s, 9) == 0


def test_status_strings(lib):
    for st in range(8):
        assert tk.status_string(st)
    assert "unknown" in tk.status_string(99)


def _redundancy(lib, keys=FAKE, shape=None, window=32, score=FAKE, twin=FAKE, ws=FAKE,
                wsb=1 << 40):
    shape = shape or tk.Shape(1, 2, 300, 64, tk.BF16)
    return lib.twinkv_redundancy(keys, shape, window, score, twin, ws, wsb, None)


def test_redundancy_argument_errors(lib):
    assert _redundancy(lib, keys=None) == tk.ERR_INVALID_ARG
    assert _redundancy(lib, score=None) == tk.ERR_INVALID_ARG
    assert _redundancy(lib, twin=None) == tk.ERR_INVALID_ARG
    assert _redundancy(lib, window=-1) == tk.ERR_INVALID_ARG
    assert _redundancy(lib, shape=tk.Shape(1, 1, 300, 80, tk.BF16)) == tk.ERR_INVALID_ARG
    assert _redundancy(lib, shape=tk.Shape(1, 1, 0, 64, tk.BF16)) == tk.ERR_INVALID_ARG
    assert _redundancy(lib, ws=None) == tk.ERR_WORKSPACE
    assert _redundancy(lib, ws=ctypes.c_void_p((1 << 20) + 8)) == tk.ERR_WORKSPACE
    assert _redundancy(lib, wsb=16) == tk.ERR_WORKSPACE


def _repair(lib, threshold=0.85, params=None, mask=FAKE, out_mask=FAKE, ws=FAKE, wsb=1 << 40):
    shape = tk.Shape(2, 2, 500, 128, tk.BF16)
    pp = ctypes.byref(params) if params is not None else None
    return lib.twinkv_repair(FAKE, shape, mask, None, ctypes.c_float(threshold), pp, out_mask,
                             FAKE, FAKE, None, None, None, None, None, ws, wsb, None)


def test_repair_argument_errors(lib):
    assert _repair(lib, threshold=float("nan")) == tk.ERR_INVALID_ARG
    assert _repair(lib, threshold=float("inf")) == tk.ERR_INVALID_ARG
    assert _repair(lib, mask=None) == tk.ERR_INVALID_ARG
    assert _repair(lib, out_mask=None) == tk.ERR_INVALID_ARG
    assert _repair(lib, params=tk.Params(0.85, -1, 4, 64)) == tk.ERR_INVALID_ARG
    assert _repair(lib, params=tk.Params(0.85, 32, -4, 64)) == tk.ERR_INVALID_ARG
    assert _repair(lib, wsb=1024) == tk.ERR_WORKSPACE


def test_select_argument_errors(lib):
    shape = tk.Shape(1, 1, 100, 0, 0)     # d and dtype are not used here
    r = lib.twinkv_repair_select(None, shape, FAKE, None, ctypes.c_float(0.5), None, FAKE,
                                 FAKE, FAKE, None, FAKE, 1 << 30, None)
    assert r == tk.ERR_INVALID_ARG
    r = lib.twinkv_repair_select(FAKE, shape, FAKE, None, ctypes.c_float(0.5), None, FAKE,
                                 FAKE, FAKE, None, FAKE, 8, None)
    assert r == tk.ERR_WORKSPACE


def test_timeout_setting(lib):
    """Limits below 10 ms are refused on the host: with a tiny limit a CTA could give up
    while its own copies or MMAs are still in flight."""
    for ns in (0, 1, 1000, 9_999_999):
        assert lib.twinkv_set_wait_timeout_ns(ns) == tk.ERR_INVALID_ARG
    assert lib.twinkv_set_wait_timeout_ns(10_000_000) == tk.OK
    assert lib.twinkv_set_wait_timeout_ns(2_000_000_000) == tk.OK


def test_binding_rejects_bad_tensors():
    import torch
    with pytest.raises((ValueError, TypeError)):
        tk.twinkv_redundancy(torch.zeros(2, 3, 4), 32)           # not 4-D
    with pytest.raises((ValueError, TypeError)):
        tk.twinkv_redundancy(torch.zeros(1, 1, 4, 64, dtype=torch.float16), 32)
