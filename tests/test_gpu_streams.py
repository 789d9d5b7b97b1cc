"""Calls on different streams, each with its own workspace and outputs, may run at the
same time on the GPU (GPU): the library keeps no per-call state outside the caller's
buffers (the no-allocation selection, which shares a fixed array, is the documented
exception).  Two repairs of different shapes and head dimensions, issued back to back on
two streams several times, must give what serial calls give, bit for bit."""
import numpy as np
import pytest
import torch

from gpu_harness import device, keys_tensor
from paper_2608_27128_gb300 import synth
from paper_2608_27128_gb300 import twinkv as tk

pytestmark = pytest.mark.gpu


def _inputs(seed, L, H, N, d, keep):
    keys = synth.random_keys(seed, L * H, N, d)
    rng = np.random.default_rng(seed)
    for u in range(L * H):
        for _ in range(N // 16):
            i, j = rng.choice(N, 2, replace=False)
            keys[u, j] = keys[u, i]
    mask = synth.random_masks(seed + 1, L * H, N, keep).reshape(L, H, N)
    return keys_tensor(keys, L, H), torch.from_numpy(mask).to(device())


def _same(got, want):
    for name in want:
        if name != "swaps":
            assert torch.equal(got[name], want[name]), name
    for u, m in enumerate(want["nswaps"].tolist()):
        assert torch.equal(got["swaps"][u, :max(m, 0)], want["swaps"][u, :max(m, 0)]), u


def test_repairs_on_two_streams_at_once():
    ka, ma = _inputs(21, 2, 4, 6000, 128, 3000)
    kb, mb = _inputs(23, 2, 3, 4100, 64, 1500)
    want_a = tk.twinkv_repair(ka, ma, None, threshold=0.85, want_all=True)
    want_b = tk.twinkv_repair(kb, mb, None, threshold=0.90, want_all=True)
    torch.cuda.synchronize()
    sa, sb = torch.cuda.Stream(), torch.cuda.Stream()
    wsa = tk.workspace(tk.shape_of(ka), tk.OP_REPAIR, device())
    wsb = tk.workspace(tk.shape_of(kb), tk.OP_REPAIR, device())
    out_a = {k: torch.empty_like(v) for k, v in want_a.items()}
    out_b = {k: torch.empty_like(v) for k, v in want_b.items()}
    for _ in range(3):
        for v in list(out_a.values()) + list(out_b.values()):
            v.fill_(7 if v.dtype == torch.uint8 else -7)
        sa.wait_stream(torch.cuda.current_stream())
        sb.wait_stream(torch.cuda.current_stream())
        for _ in range(2):   # several calls in flight on each stream
            tk.twinkv_repair(ka, ma, None, threshold=0.85, want_all=True, out=out_a, ws=wsa,
                             stream=sa)
            tk.twinkv_repair(kb, mb, None, threshold=0.90, want_all=True, out=out_b, ws=wsb,
                             stream=sb)
        torch.cuda.synchronize()
        _same(out_a, want_a)
        _same(out_b, want_b)
    assert tk.twinkv_get_last_error() == tk.OK
