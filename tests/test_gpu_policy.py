"""Parity of the standalone policy (Sec. 3.2, Eq. 2-3) on the GPU, through the C ABI,
with the fp64 oracle.

- Counts: each row's r_i must lie in [r(tau + BAND), r(tau - BAND)] of the oracle, so
  it equals the oracle's count wherever no pair's similarity lies within BAND of tau.
  BAND = 1e-4 is far below the score tie band of 4e-3 and far above the fp32
  error of the kernel's decision (about 1e-6).
- Selection: the oracle's selection fed the GPU's own counts reproduces the mask and
  statuses bit for bit (split check).
Covered: the hand-derived worked example, ragged shapes (several 128-row blocks and
256-column tiles with tails), windows wider than N, negative and zero thresholds,
zero keys, fp32 keys, budget edges, and the five workload recipes at reduced size."""
import numpy as np
import pytest
import torch

import oracle
from golden_io import read_worked_example
from gpu_harness import device, keys_tensor
from paper_2608_27128_gb300 import synth
from paper_2608_27128_gb300 import twinkv as tk

pytestmark = pytest.mark.gpu

BAND = 1e-4


@pytest.fixture(scope="module", autouse=True)
def _setup():
    oracle.build()
    tk.load()
    torch.cuda.init()


def run_policy(keys, L, H, tau, budget, window=32, n_sink=4, n_recent=64, rows=None):
    """GPU policy vs the oracle; returns the GPU counts and mask [U,N]."""
    U, N, d = keys.shape
    bud = np.broadcast_to(np.asarray(budget, np.int32), (U,)).copy()
    out = tk.twinkv_policy(keys_tensor(keys, L, H), torch.from_numpy(bud).to(device()),
                           threshold=tau, window=window, n_sink=n_sink, n_recent=n_recent)
    torch.cuda.synchronize()
    assert tk.twinkv_get_last_error() == tk.OK
    cnt = out["count"].reshape(U, N).cpu().numpy()
    mask = out["mask"].reshape(U, N).cpu().numpy()
    status = out["status"].cpu().numpy()
    ref = oracle.count(keys, tau, window, band=BAND, rows=rows)
    sel = np.arange(N) if rows is None else np.asarray(rows)
    lo_ok = cnt[:, sel] >= ref["r_lo"]
    hi_ok = cnt[:, sel] <= ref["r_hi"]
    bad = np.argwhere(~(lo_ok & hi_ok))
    assert bad.size == 0, [(int(u), int(sel[i]), int(cnt[u, sel[i]]), int(ref["r"][u, i]))
                           for u, i in bad[:10]]
    # split check: the oracle's selection on the GPU's counts, bit for bit
    sp = oracle.policy_select(cnt, bud, n_sink, n_recent)
    np.testing.assert_array_equal(mask, sp["mask"])
    np.testing.assert_array_equal(status, sp["status"])
    return cnt, mask, ref


def test_worked_example():
    head, cases = read_worked_example("worked_policy.txt")
    keys = np.zeros((1, head["N"], 64), np.float32)
    keys[0, :, :head["d"]] = head["keys"]
    kb = synth.f32_to_bf16_bits(keys)
    for c in cases:
        for kk, ss in (("K", "S"), ("K2", "S2")):
            if kk not in c:
                continue
            cnt, mask, _ = run_policy(kb, 1, 1, c["tau"], int(c[kk][0]), head["window"],
                                      head["n_sink"], head["n_recent"])
            np.testing.assert_array_equal(cnt[0], c["r"])
            np.testing.assert_array_equal(mask[0], c[ss])


@pytest.mark.parametrize("L,H,N,d,w,tau", [
    (1, 1, 1, 64, 32, 0.5), (1, 2, 5, 128, 1, 0.0), (1, 1, 33, 64, 40, 0.2),
    (2, 1, 129, 128, 0, 0.1), (1, 3, 257, 64, 7, 0.1), (1, 1, 300, 128, 32, -0.05),
    (2, 2, 700, 64, 32, 0.15), (1, 1, 1025, 128, 5, 0.12), (1, 1, 2053, 64, 32, 0.2),
])
def test_counts_and_selection_match_oracle(L, H, N, d, w, tau):
    keys = synth.random_keys(30 + N, L * H, N, d)
    U = L * H
    budgets = np.linspace(0, N, U + 2).astype(np.int32)[1:-1] if U > 1 else [N // 2]
    run_policy(keys, L, H, tau, budgets, window=w)


def test_budget_edges_and_status():
    N = 300
    keys = synth.random_keys(5, 6, N, 64)
    bud = np.array([0, N, 10, N + 1, -1, 68], np.int32)   # 10 < 68 protected positions
    cnt, mask, _ = run_policy(keys, 2, 3, 0.1, bud)
    assert mask[0].sum() == 0 and mask[1].sum() == N
    np.testing.assert_array_equal(np.flatnonzero(mask[2]), np.r_[0:4, 236:242])
    assert mask[3].sum() == 0 and mask[4].sum() == 0


def test_zero_keys_and_fp32_keys():
    rng = np.random.default_rng(8)
    x = rng.standard_normal((2, 400, 64)).astype(np.float32)
    x[0, 100] = 0.0
    x[1, ::50] = 0.0
    x[0, 300] = x[0, 20]                  # a twin far apart
    for tau in (0.5, -0.05):
        run_policy(x, 1, 2, tau, 200)
    kb = synth.f32_to_bf16_bits(x)
    cnt_b, _, _ = run_policy(kb, 1, 2, 0.5, 200)
    cnt_f, _, _ = run_policy(x, 1, 2, 0.5, 200)
    np.testing.assert_array_equal(cnt_b, cnt_f)   # fp32 keys are rounded to bf16 first
    assert cnt_b[0, 20] >= 1 and cnt_b[0, 300] >= 1


@pytest.mark.parametrize("name,over,ratio", [
    ("tiny", {}, 0.5),
    ("llama", {"L": 1, "H": 2, "N": 2048}, 0.5),
    ("qwen", {"L": 1, "H": 2, "N": 2048}, 0.3),
    ("retrieval", {"L": 1, "H": 1, "N": 4096}, 0.7),
    ("long", {"L": 1, "H": 1, "N": 4096}, 0.5),
])
def test_workload_recipes(name, over, ratio):
    w = synth.get(name, **over)
    keys, truths = synth.keys(w)
    K = tk.budget_for_ratio(w.N, ratio)
    n_sink, n_recent = (0, 0) if name == "tiny" else (synth.N_SINK, synth.N_RECENT)
    cnt, mask, ref = run_policy(keys, w.L, w.H, w.tau, K, synth.WINDOW, n_sink, n_recent)
    if name == "tiny":
        # planted margin: no pair near tau, so the counts are exact
        np.testing.assert_array_equal(cnt, ref["r"])
    for u, t in enumerate(truths):
        for s_, c in np.concatenate([t.pairs, t.exact_pairs]).reshape(-1, 2):
            if c - s_ > synth.WINDOW:
                assert cnt[u, s_] >= 1 and cnt[u, c] >= 1
        if name == "retrieval":
            # needles have no twin: r = 0, the highest score, all kept
            assert np.all(cnt[u, t.needles] == 0)
            assert np.all(mask[u, t.needles] == 1)


def test_full_qwen_shape_sampled_rows():
    """The Qwen3-4B cache shape (36x8x16384x128) in one launch; the oracle checks 2
    units on 256 sampled rows each against all columns, and the selection of every
    unit on the GPU's counts."""
    w = synth.get("qwen")
    units = [(0, 0), (35, 7)]
    L, H, N = w.L, w.H, w.N
    keys_all = synth.random_keys(77, L * H, N, w.d)
    sub, _ = synth.keys(w, units=units)
    for k, (l, h) in enumerate(units):
        keys_all[l * H + h] = sub[k]
    K = tk.budget_for_ratio(N, 0.5)
    out = tk.twinkv_policy(keys_tensor(keys_all, L, H),
                           torch.full((L * H,), K, dtype=torch.int32, device=device()),
                           threshold=w.tau)
    torch.cuda.synchronize()
    assert tk.twinkv_get_last_error() == tk.OK
    cnt = out["count"].reshape(L * H, N).cpu().numpy()
    mask = out["mask"].reshape(L * H, N).cpu().numpy()
    rows = np.random.default_rng(4).choice(N, 256, replace=False)
    for k, (l, h) in enumerate(units):
        ref = oracle.count(sub[k:k + 1], w.tau, synth.WINDOW, band=BAND, rows=rows)
        c = cnt[l * H + h, rows]
        assert np.all(c >= ref["r_lo"][0]) and np.all(c <= ref["r_hi"][0])
    sp = oracle.policy_select(cnt, np.full(L * H, K, np.int32))
    np.testing.assert_array_equal(mask, sp["mask"])
    assert np.all(mask.sum(1) == K)
