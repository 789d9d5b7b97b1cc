"""The selection entry point that allocates nothing (twinkv_repair_select_noalloc).

Some callers may not allocate device memory themselves, for example a plugin running
inside a serving engine that owns all device memory through its own pool, or a loop
that cannot afford the synchronization cudaMalloc/cudaFree can cause.  For them the
library keeps the selection's scratch in its own fixed device array.  These tests call
that entry point through the C ABI, twice in a row, and check that it returns exactly
what the workspace-taking twinkv_repair_select returns on the same inputs; and that a
request larger than the fixed array is refused without touching the GPU.

This file is collected last, so that a run stopping at its first failure has already
run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_27128_gb300 import synth
from paper_2608_27128_gb300 import twinkv as tk


def _inputs(seed, L, H, N):
    rng = np.random.default_rng(seed)
    U = L * H
    grid = np.array([-1.0, 0.0, 0.5, 0.85, 0.9, 0.99995, 1.0])
    b = np.where(rng.random((U, N)) < 0.3, rng.choice(grid, size=(U, N)),
                 rng.uniform(-1, 1, size=(U, N)))
    S0 = synth.random_masks(seed, U, N, int(rng.integers(1, N)))
    dev = torch.device("cuda:0")
    return (torch.from_numpy(b.reshape(L, H, N)).to(dev),
            torch.from_numpy(S0.reshape(L, H, N)).to(dev),
            torch.from_numpy(S0.sum(1).astype(np.int32)).to(dev))


@pytest.mark.gpu
def test_noalloc_selection_matches_workspace_selection_twice():
    tk.load()
    for call, (seed, L, H, N) in enumerate([(1, 2, 3, 5000), (2, 1, 8, 20000)]):
        b, S0, budget = _inputs(seed, L, H, N)
        ref = tk.twinkv_repair_select(b, S0, budget, threshold=0.85)
        got = tk.twinkv_repair_select_noalloc(b, S0, budget, threshold=0.85)
        torch.cuda.synchronize()
        for k in ("mask", "nswaps", "status"):
            assert torch.equal(got[k], ref[k]), (call, k)
        n = ref["nswaps"].cpu().numpy()
        g, r = got["swaps"].cpu().numpy(), ref["swaps"].cpu().numpy()
        for u, m in enumerate(n):
            np.testing.assert_array_equal(g[u, :m], r[u, :m])
        assert n.max() > 0
    assert tk.twinkv_get_last_error() == tk.OK


@pytest.mark.gpu
def test_noalloc_refuses_requests_beyond_its_fixed_array():
    lib = tk.load()
    shape = tk.Shape(1, 1, tk.NOALLOC_MAX_POSITIONS + 1, 64, tk.BF16)
    fake = ctypes.c_void_p(1 << 20)        # never dereferenced: refused on the host
    st = lib.twinkv_repair_select_noalloc(fake, shape, fake, None, ctypes.c_float(0.85),
                                          None, fake, fake, fake, None, None)
    assert st == tk.ERR_TOO_LARGE
