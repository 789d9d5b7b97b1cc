"""The large workloads at full size, in the launch configuration bench.py times (one
twinkv_repair call over every layer and head, with b_i(all)), and twinkv_redundancy at
full N over enough units that every CTA of the persistent audit takes many work items.

Checked per workload and retention ratio:
  * every unit: the bit-exact split check (oracle repair on the GPU's own b_i(S0)), the
    budget and swap invariants of Sec. 3.4, and the planted ground truth (twins of
    planted pairs farther apart than w; evicted needles admitted as orphans), all exact
    with nothing excused;
  * every unit: a random sample of rows (different in each unit) against the fp64
    oracle, b_i(S0), b_i(all) and both twins;
  * a few whole units: full comparison with the oracle (scores, twins, S1, swaps).
Each configuration's failures and excused items are recorded (gpu_harness.record).
"""
import numpy as np
import pytest
import torch

import oracle
from comparator import Report, compare_best, compare_repair
from gpu_harness import device, keys_tensor, record, sampled_rows, split_check
from paper_2608_27128_gb300 import synth
from paper_2608_27128_gb300 import twinkv as tk

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


def run_full(w, ratio, schedule="uniform"):
    keys, truths = synth.keys(w)
    S0 = synth.masks(w, ratio, schedule=schedule)
    U, N = S0.shape
    kt = keys_tensor(keys, w.L, w.H)
    mt = torch.from_numpy(S0.reshape(w.L, w.H, N)).to(device())
    bud = torch.from_numpy(S0.sum(1).astype(np.int32)).to(device())
    out = tk.twinkv_repair(kt, mt, bud, threshold=w.tau, want_all=True)
    torch.cuda.synchronize()
    assert tk.twinkv_get_last_error() == tk.OK
    h = {k: v.cpu().numpy() for k, v in out.items()}
    for k in ("mask", "score_ret", "twin_ret", "score_all", "twin_all"):
        h[k] = h[k].reshape(U, N)
    del kt, mt, out
    torch.cuda.empty_cache()
    return keys, truths, S0, h


def invariants(S0, h, tau):
    U, N = S0.shape
    assert np.all(h["status"] == 0)
    np.testing.assert_array_equal(h["mask"].sum(1), S0.sum(1))            # |S1| = |S0|
    prot = np.zeros(N, bool)
    prot[:synth.N_SINK] = True
    prot[N - synth.N_RECENT:] = True
    tau_d = float(np.float32(tau))
    for u in range(U):
        m = int(h["nswaps"][u])
        out_, in_ = h["swaps"][u, :m, 0], h["swaps"][u, :m, 1]
        assert np.all(S0[u, out_] == 1) and np.all(S0[u, in_] == 0)
        assert np.all(h["score_ret"][u, out_] >= tau_d) and not np.any(prot[out_])
        assert np.all(h["score_ret"][u, in_] < tau_d)
        changed = np.flatnonzero(h["mask"][u] != S0[u])
        assert changed.size == 2 * m
        assert np.all(h["score_ret"][u] <= h["score_all"][u])
        t = h["twin_ret"][u]
        ok = t >= 0
        assert np.all(S0[u, t[ok]] == 1)
        assert np.all(np.abs(t[ok] - np.flatnonzero(ok)) > synth.WINDOW)


def planted(truths, h, S0, check_needles=False):
    """Asserts the planted ground truth exactly; returns the number of planted items
    checked (twin pairs, and evicted needles)."""
    n = 0
    for u, t in enumerate(truths):
        for s, c in t.pairs:
            if c - s > synth.WINDOW:
                assert h["twin_all"][u, s] == c and h["twin_all"][u, c] == s
                n += 1
        if check_needles:
            ev = t.needles[S0[u, t.needles] == 0]
            assert ev.size > 0
            assert np.all(h["score_ret"][u, ev] < 0.85)
            assert np.all(h["mask"][u, ev] == 1)
            n += ev.size
    return n


def full_units(keys, S0, h, units, tau):
    rep = Report()
    for u in units:
        a = oracle.audit(keys[u:u + 1], S0[u:u + 1], window=synth.WINDOW)
        sim = (lambda uu: (lambda i, j: oracle.sim(keys, uu, i, j)))(u)
        rep.add(compare_best(h["score_ret"][u], h["twin_ret"][u], a["b_ret"][0],
                             a["t_ret"][0], a["b_ret2"][0], sim, synth.WINDOW, S0=S0[u]))
        rep.add(compare_best(h["score_all"][u], h["twin_all"][u], a["b_all"][0],
                             a["t_all"][0], a["b_all2"][0], sim, synth.WINDOW))
        r = oracle.repair(a["b_ret"], S0[u:u + 1], tau, budget=S0[u:u + 1].sum(1))
        rep.add(compare_repair(S0[u], h["mask"][u], h["swaps"][u], int(h["nswaps"][u]),
                               {k: r[k][0] for k in r}, a["b_ret"][0], tau, synth.N_SINK,
                               synth.N_RECENT))
    return rep


# rows sampled per unit (the long workload samples 4096 rows of each of its 8 units)
ROWS = {"llama": 256, "qwen": 128, "retrieval": 96, "long": 4096, "largest": 256}


def check_config(name, w, ratio, keys, truths, S0, h, full, schedule="uniform",
                 needles=False, seed=0):
    split_check(h, S0, w.tau, synth.N_SINK, synth.N_RECENT)
    invariants(S0, h, w.tau)
    n_planted = planted(truths, h, S0, check_needles=needles)
    rep_ret, rep_all, n_rows = sampled_rows(keys, S0, h, ROWS[name], seed, synth.WINDOW)
    rep_full = full_units(keys, S0, h, full, w.tau)
    record(workload=name, ratio=ratio, schedule=schedule, units=w.units, N=w.N, d=w.d,
           rows_sampled=n_rows, full_units=len(full),
           n_fail=rep_ret.n_fail + rep_all.n_fail + rep_full.n_fail,
           excused_twin_ret=rep_ret.n_excused, excused_twin_all=rep_all.n_excused,
           excused_full_units=rep_full.n_excused, planted_checked=n_planted,
           planted_excused=0,
           max_dev_same_twin=max(rep_ret.max_dev_same_twin, rep_all.max_dev_same_twin,
                                 rep_full.max_dev_same_twin))
    for rep in (rep_ret, rep_all, rep_full):
        assert rep.n_fail == 0, rep.notes
        assert rep.max_dev_same_twin < 1e-9


@pytest.mark.parametrize("ratio", [0.3, 0.5, 0.7])
def test_llama_full(ratio):
    w = synth.get("llama")
    keys, truths, S0, h = run_full(w, ratio)
    check_config("llama", w, ratio, keys, truths, S0, h, [0, 77], seed=int(ratio * 10))


@pytest.mark.parametrize("ratio", [0.3, 0.5, 0.7])
def test_qwen_full(ratio):
    w = synth.get("qwen")
    keys, truths, S0, h = run_full(w, ratio)
    check_config("qwen", w, ratio, keys, truths, S0, h, [5], seed=int(ratio * 10))


def test_qwen_full_pyramid_budgets():
    """Per-layer budgets at full size: layer 0 keeps all 16384 keys (no evicted
    segment), the last layer keeps 6554; one launch covers them all."""
    w = synth.get("qwen")
    keys, truths, S0, h = run_full(w, 0.3, schedule="pyramid")
    k = np.repeat(synth.pyramid_budgets(w, 0.3), w.H)
    np.testing.assert_array_equal(S0.sum(1), k)
    for u in range(w.H):   # layer 0: nothing evicted
        np.testing.assert_array_equal(h["score_ret"][u], h["score_all"][u])
        assert h["nswaps"][u] == 0
    check_config("qwen", w, 0.3, keys, truths, S0, h, [1, w.units - 1], schedule="pyramid",
                 seed=9)


def test_retrieval_full():
    w = synth.get("retrieval")
    keys, truths, S0, h = run_full(w, 0.3)
    check_config("retrieval", w, 0.3, keys, truths, S0, h, [3], needles=True, seed=4)


def test_long_full_sampled_rows():
    w = synth.get("long")
    keys, truths, S0, h = run_full(w, 0.5)
    check_config("long", w, 0.5, keys, truths, S0, h, [], seed=5)


def test_repair_at_the_largest_n():
    """N = 2^20, the largest the ABI accepts, on the long-stress recipe (2 heads,
    d = 128; the selection runs each unit on a cluster of 16 CTAs): the split check and
    the invariants on every position, every planted twin exact, and 256 random rows of
    each unit against the oracle over all 2^20 columns."""
    w = synth.get("long", H=2, N=1 << 20)
    keys, truths, S0, h = run_full(w, 0.5)
    assert int(h["nswaps"].min()) > 0
    check_config("largest", w, 0.5, keys, truths, S0, h, [], seed=6)


@pytest.mark.parametrize("name", ["qwen", "llama"])
def test_redundancy_full_size_many_items_per_cta(name):
    """twinkv_redundancy (columns in position order) at full N over 2 layers x 8 heads:
    2048 (Qwen3-4B shape, d = 128) or 1024 (Llama-3.2-1B shape, d = 64) 128-row work
    items on the persistent grid, so every CTA runs many items and both A buffers,
    both accumulators and the metadata ring wrap around many times.  4096 random rows
    of every unit against the oracle; planted twins exact."""
    w = synth.get(name, L=2)
    keys, truths = synth.keys(w)
    U, N = w.units, w.N
    kt = keys_tensor(keys, w.L, w.H)
    score, twin = tk.twinkv_redundancy(kt, synth.WINDOW)
    torch.cuda.synchronize()
    assert tk.twinkv_get_last_error() == tk.OK
    s = score.reshape(U, N).cpu().numpy()
    t = twin.reshape(U, N).cpu().numpy()
    del kt, score, twin
    torch.cuda.empty_cache()
    rng = np.random.default_rng(17)
    rep = Report()
    n_rows = 0
    for u in range(U):
        rows = np.sort(rng.choice(N, size=4096, replace=False))
        a = oracle.audit(keys[u:u + 1], window=synth.WINDOW, rows=rows)
        sim = (lambda uu: (lambda i, j: oracle.sim(keys, uu, i, j)))(u)
        rep.add(compare_best(s[u, rows], t[u, rows], a["b_all"][0], a["t_all"][0],
                             a["b_all2"][0], sim, synth.WINDOW, rows=rows, what=f"u{u}"))
        n_rows += rows.size
    n_planted = planted(truths, {"twin_all": t}, None)
    record(workload=name, call="twinkv_redundancy", units=U, N=N, d=w.d, rows_sampled=n_rows,
           n_fail=rep.n_fail, excused_twin_all=rep.n_excused, planted_checked=n_planted,
           planted_excused=0, max_dev_same_twin=rep.max_dev_same_twin)
    assert rep.n_fail == 0, rep.notes
    assert rep.max_dev_same_twin < 1e-9


def test_symmetric_redundancy_full_qwen_shape():
    """twinkv_redundancy_symmetric at the full Qwen3-4B shape (36 x 8 x 16384 x 128):
    128 random rows of every unit against the oracle, every planted twin exact, and the
    twins equal to the full-tile audit's wherever that one is not a near tie."""
    w = synth.get("qwen")
    keys, truths = synth.keys(w)
    U, N = w.units, w.N
    kt = keys_tensor(keys, w.L, w.H)
    score, twin = tk.twinkv_redundancy_symmetric(kt, synth.WINDOW)
    torch.cuda.synchronize()
    assert tk.twinkv_get_last_error() == tk.OK
    s = score.reshape(U, N).cpu().numpy()
    t = twin.reshape(U, N).cpu().numpy()
    del kt, score, twin
    torch.cuda.empty_cache()
    rng = np.random.default_rng(23)
    rep = Report()
    n_rows = 0
    for u in range(U):
        rows = np.sort(rng.choice(N, size=128, replace=False))
        a = oracle.audit(keys[u:u + 1], window=synth.WINDOW, rows=rows)
        sim = (lambda uu: (lambda i, j: oracle.sim(keys, uu, i, j)))(u)
        rep.add(compare_best(s[u, rows], t[u, rows], a["b_all"][0], a["t_all"][0],
                             a["b_all2"][0], sim, synth.WINDOW, rows=rows, what=f"u{u}"))
        n_rows += rows.size
    n_planted = planted(truths, {"twin_all": t}, None)
    record(workload="qwen", call="twinkv_redundancy_symmetric", units=U, N=N, d=w.d,
           rows_sampled=n_rows, n_fail=rep.n_fail, excused_twin_all=rep.n_excused,
           planted_checked=n_planted, planted_excused=0,
           max_dev_same_twin=rep.max_dev_same_twin)
    assert rep.n_fail == 0, rep.notes
    assert rep.max_dev_same_twin < 1e-9
