"""The calls replay in a CUDA graph (GPU): a serving loop captures its work once and
replays it on new contents of the same buffers.  Every call only enqueues work on the
caller's stream, and everything that depends on the data (retained counts, the split of
the work items, the cut of the selection) is computed on the device, so a replay on new
keys and masks must give what an eager call on them gives, bit for bit."""
import numpy as np
import pytest
import torch

from gpu_harness import device, keys_tensor
from paper_2608_27128_gb300 import synth
from paper_2608_27128_gb300 import twinkv as tk

pytestmark = pytest.mark.gpu


def _inputs(seed, L, H, N, d, keep):
    keys = synth.random_keys(seed, L * H, N, d)
    # planted duplicates and near-duplicates, so that twins, orphans and donors occur
    rng = np.random.default_rng(seed)
    for u in range(L * H):
        for _ in range(N // 16):
            i, j = rng.choice(N, 2, replace=False)
            keys[u, j] = keys[u, i]
    mask = synth.random_masks(seed + 1, L * H, N, keep).reshape(L, H, N)
    return keys_tensor(keys, L, H), torch.from_numpy(mask).to(device())


def _capture(fn):
    """fn() once on a side stream (the calls' first-use setup), then captured."""
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        fn()
    torch.cuda.current_stream().wait_stream(s)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    return g


@pytest.mark.parametrize("L,H,N,d", [(2, 4, 3000, 128), (1, 3, 2100, 64)])
def test_repair_replays_on_new_inputs(L, H, N, d):
    keys, mask = _inputs(5, L, H, N, d, N // 2)
    s = tk.shape_of(keys)
    ws = tk.workspace(s, tk.OP_REPAIR, device())
    ref = tk.twinkv_repair(keys, mask, None, threshold=0.85, want_all=True)
    out = {k: torch.empty_like(v) for k, v in ref.items()}

    def step():
        tk.twinkv_repair(keys, mask, None, threshold=0.85, want_all=True, out=out, ws=ws)

    g = _capture(step)
    for seed, keep in ((5, N // 2), (7, N // 3), (9, (2 * N) // 3)):
        k2, m2 = _inputs(seed, L, H, N, d, keep)
        keys.copy_(k2)
        mask.copy_(m2)
        for v in out.values():
            v.fill_(-7 if v.dtype != torch.uint8 else 7)
        g.replay()
        want = tk.twinkv_repair(k2, m2, None, threshold=0.85, want_all=True)
        torch.cuda.synchronize()
        for name in want:
            if name != "swaps":
                assert torch.equal(out[name], want[name]), (seed, name)
        # only the first nswaps[u] pairs of a unit's swap list are written
        for u, m in enumerate(want["nswaps"].tolist()):
            assert torch.equal(out["swaps"][u, :max(m, 0)], want["swaps"][u, :max(m, 0)]), (seed, u)
        assert int(want["nswaps"].max()) > 0   # the swap path ran


def test_redundancy_and_policy_replay_on_new_inputs():
    L, H, N, d = 1, 4, 2500, 128
    keys, mask = _inputs(11, L, H, N, d, N // 2)
    ref_s, ref_t = tk.twinkv_redundancy(keys, 32)
    sc, tw = torch.empty_like(ref_s), torch.empty_like(ref_t)
    budget = torch.full((L * H,), N // 2, dtype=torch.int32, device=device())
    pol = tk.twinkv_policy(keys, budget, threshold=0.85)
    pout = {k: torch.empty_like(v) for k, v in pol.items()}

    def step():
        tk.twinkv_redundancy(keys, 32, out_score=sc, out_twin=tw)
        tk.twinkv_policy(keys, budget, threshold=0.85, out=pout)

    g = _capture(step)
    k2, _ = _inputs(13, L, H, N, d, N // 2)
    keys.copy_(k2)
    sc.fill_(-7)
    tw.fill_(-7)
    for v in pout.values():
        v.fill_(7 if v.dtype == torch.uint8 else -7)
    g.replay()
    want_s, want_t = tk.twinkv_redundancy(k2, 32)
    want_p = tk.twinkv_policy(k2, budget, threshold=0.85)
    torch.cuda.synchronize()
    assert torch.equal(sc, want_s) and torch.equal(tw, want_t)
    for name in want_p:
        assert torch.equal(pout[name], want_p[name]), name
