"""The dedup repair variant on the GPU (a donor is never evicted together with its
twin), through the C ABI.  The audit part is the one of twinkv_repair, so b_i(S0)
and the twins must equal that call's bit for bit; the selection must equal the
oracle's dedup walk fed the GPU's own b and twins, bit for bit (split check).
Covered: the hand-derived golden cases, the workload recipes at reduced size, the
selection-only entry on random twin graphs with ties and data errors, the size limit,
and the Qwen3-4B shape in one launch."""
import numpy as np
import pytest
import torch

import oracle
from golden_io import read_worked_example
from gpu_harness import device, keys_tensor
from paper_2608_27128_gb300 import synth
from paper_2608_27128_gb300 import twinkv as tk

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _setup():
    oracle.build()
    tk.load()
    torch.cuda.init()


def split_check_dedup(h, S0, tau, n_sink, n_recent, budget=None):
    U, N = S0.shape
    rf = oracle.repair_dedup(h["score_ret"].reshape(U, N), h["twin_ret"].reshape(U, N), S0,
                             tau, n_sink=n_sink, n_recent=n_recent, budget=budget)
    np.testing.assert_array_equal(h["status"], rf["status"])
    np.testing.assert_array_equal(h["nswaps"], rf["nswaps"])
    np.testing.assert_array_equal(h["mask"].reshape(U, N), rf["mask"])
    for u in range(U):
        m = int(rf["nswaps"][u])
        if m > 0:
            np.testing.assert_array_equal(h["swaps"][u, :m], rf["swaps"][u, :m])
    return rf


def run_both(keys, S0, L, H, tau, n_sink=synth.N_SINK, n_recent=synth.N_RECENT):
    U, N, _ = keys.shape
    kt = keys_tensor(keys, L, H)
    mt = torch.from_numpy(S0.reshape(L, H, N).copy()).to(device())
    bt = torch.from_numpy(S0.sum(1).astype(np.int32)).to(device())
    kw = dict(threshold=tau, window=synth.WINDOW, n_sink=n_sink, n_recent=n_recent)
    lit = tk.twinkv_repair(kt, mt, bt, **kw)
    dd = tk.twinkv_repair_dedup(kt, mt, bt, **kw)
    torch.cuda.synchronize()
    assert tk.twinkv_get_last_error() == tk.OK
    hl = {k: v.cpu().numpy() for k, v in lit.items()}
    hd = {k: v.cpu().numpy() for k, v in dd.items()}
    # the audit is shared: identical b_i(S0) and twins
    np.testing.assert_array_equal(hd["score_ret"], hl["score_ret"])
    np.testing.assert_array_equal(hd["twin_ret"], hl["twin_ret"])
    rf = split_check_dedup(hd, S0, tau, n_sink, n_recent)
    assert np.all(hd["nswaps"] <= hl["nswaps"])
    return hl, hd, rf


def test_golden_cases():
    head, cases = read_worked_example()
    keys = np.zeros((1, head["N"], 64), np.float32)
    keys[0, :, :head["d"]] = head["keys"]
    for c in cases:
        S0 = c["S0"].astype(np.uint8)[None]
        kt = keys_tensor(keys, 1, 1)
        out = tk.twinkv_repair_dedup(kt, torch.from_numpy(S0.reshape(1, 1, -1)).to(device()),
                                     None, threshold=c["tau"], window=head["window"],
                                     n_sink=head["n_sink"], n_recent=head["n_recent"])
        torch.cuda.synchronize()
        m = int(out["nswaps"][0])
        np.testing.assert_array_equal(out["swaps"][0, :m].cpu().numpy().ravel(),
                                      c["dedup_swaps"])
        np.testing.assert_array_equal(out["mask"].cpu().numpy().ravel(), c["dedup_S1"])


@pytest.mark.parametrize("name,over,ratio", [
    ("tiny", {}, 0.5),
    ("llama", {"L": 1, "H": 2, "N": 2048}, 0.3),
    ("qwen", {"L": 1, "H": 2, "N": 2048}, 0.5),
    ("retrieval", {"L": 1, "H": 2, "N": 4096}, 0.3),
    ("long", {"L": 1, "H": 1, "N": 4096}, 0.5),
])
def test_workload_recipes(name, over, ratio):
    w = synth.get(name, **over)
    keys, _ = synth.keys(w)
    S0 = synth.masks(w, ratio)
    hl, hd, _ = run_both(keys, S0, w.L, w.H, w.tau)
    if name == "llama":
        # twin pairs both retained and donors scarcer than orphans: dedup bites
        assert np.any(hd["nswaps"] < hl["nswaps"])
    # no evicted donor's twin is evicted
    U = S0.shape[0]
    for u in range(U):
        m = int(hd["nswaps"][u])
        ev = set(hd["swaps"][u, :m, 0].tolist())
        tw = hd["twin_ret"].reshape(U, -1)[u]
        assert not any(int(tw[d]) in ev for d in ev)


def test_pyramid_budgets():
    w = synth.get("llama", L=4, H=2, N=1500)
    keys, _ = synth.keys(w)
    S0 = synth.masks(w, 0.5, schedule="pyramid")
    hl, hd, _ = run_both(keys, S0, w.L, w.H, w.tau)
    np.testing.assert_array_equal(hd["mask"].reshape(w.units, -1).sum(1), S0.sum(1))


@pytest.mark.parametrize("seed", range(5))
def test_select_dedup_on_random_twin_graphs(seed):
    rng = np.random.default_rng(100 + seed)
    L, H, N = 1, 3, int(rng.integers(2, 6000))
    U = L * H
    S0 = synth.random_masks(seed, U, N, max(1, N // 2))
    b = rng.choice([0.2, 0.5, 0.85, 0.9, 1.0], size=(U, N)) + \
        np.where(rng.random((U, N)) < 0.5, rng.uniform(-1e-3, 1e-3, (U, N)), 0.0)
    t = np.empty((U, N), np.int32)
    for u in range(U):
        ret = np.flatnonzero(S0[u])
        t[u] = rng.choice(ret, size=N)
        same = t[u] == np.arange(N)
        t[u][same] = -1                       # no self twins (the window excludes them)
    budget = S0.sum(1).astype(np.int32)
    if seed == 3:
        budget[1] += 1                        # a budget mismatch
    out = tk.twinkv_repair_select_dedup(
        torch.from_numpy(b.reshape(L, H, N)).to(device()),
        torch.from_numpy(t.reshape(L, H, N)).to(device()),
        torch.from_numpy(S0.reshape(L, H, N)).to(device()),
        torch.from_numpy(budget).to(device()), threshold=0.85, n_sink=3, n_recent=7)
    torch.cuda.synchronize()
    h = {k: v.cpu().numpy() for k, v in out.items()}
    h["score_ret"], h["twin_ret"] = b, t
    split_check_dedup(h, S0, 0.85, 3, 7, budget=budget)


def test_select_dedup_with_more_than_4096_donors():
    """All donors are sorted before the walk: more than 4096 of them takes the radix
    passes instead of the shared-memory sort."""
    rng = np.random.default_rng(21)
    L, H, N = 1, 2, 20000
    U = L * H
    S0 = synth.random_masks(21, U, N, N // 2)
    b = np.round(rng.uniform(0.0, 1.0, size=(U, N)), 3)
    t = np.empty((U, N), np.int32)
    for u in range(U):
        ret = np.flatnonzero(S0[u])
        t[u] = rng.choice(ret, size=N)
        t[u][t[u] == np.arange(N)] = -1
    out = tk.twinkv_repair_select_dedup(
        torch.from_numpy(b.reshape(L, H, N)).to(device()),
        torch.from_numpy(t.reshape(L, H, N)).to(device()),
        torch.from_numpy(S0.reshape(L, H, N)).to(device()),
        torch.from_numpy(S0.sum(1).astype(np.int32)).to(device()), threshold=0.3)
    torch.cuda.synchronize()
    h = {k: v.cpu().numpy() for k, v in out.items()}
    h["score_ret"], h["twin_ret"] = b, t
    nd = ((S0 == 1) & (b >= np.float32(0.3)))[:, 4:N - 64].sum(1)
    assert np.all(nd > 4096), nd
    split_check_dedup(h, S0, 0.3, synth.N_SINK, synth.N_RECENT)


def test_size_limit_is_reported():
    N = (1 << 19) + 1
    z = torch.zeros((1, 1, N), dtype=torch.float64, device=device())
    with pytest.raises(tk.TwinKVError) as e:
        tk.twinkv_repair_select_dedup(z, torch.zeros((1, 1, N), dtype=torch.int32,
                                                     device=device()),
                                      torch.zeros((1, 1, N), dtype=torch.uint8,
                                                  device=device()), threshold=0.5)
    assert e.value.status == tk.ERR_UNSUPPORTED


def test_full_qwen_shape():
    """36x8x16384x128 in one call: the split check on every unit."""
    w = synth.get("qwen")
    keys, _ = synth.keys(w)
    S0 = synth.masks(w, 0.5)
    run_both(keys, S0, w.L, w.H, w.tau)
