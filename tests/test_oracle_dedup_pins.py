"""Pins for the oracle's dedup repair variant (Sec. 3.4 read so that a twin pair never
loses both members: evicting a donor keeps its twin): the hand-derived cases of
tests/golden/worked_repair.txt, and invariants that characterise the rule on planted
and random inputs.  None needs a GPU."""
import numpy as np
import pytest

from golden_io import read_worked_example
from paper_2608_27128_gb300 import synth


def bf16(x):
    return synth.f32_to_bf16_bits(np.asarray(x, np.float32))


def test_worked_example(oracle_mod):
    head, cases = read_worked_example()
    keys = bf16(head["keys"])[None]
    for case in cases:
        S0 = case["S0"].astype(np.uint8)[None]
        a = oracle_mod.audit(keys, S0, window=head["window"])
        r = oracle_mod.repair_dedup(a["b_ret"], a["t_ret"], S0, case["tau"],
                                    n_sink=head["n_sink"], n_recent=head["n_recent"],
                                    budget=[int(S0.sum())])
        m = r["nswaps"][0]
        np.testing.assert_array_equal(r["swaps"][0, :m].ravel(), case["dedup_swaps"])
        np.testing.assert_array_equal(r["mask"][0], case["dedup_S1"])


def check_invariants(oracle_mod, b, t, S0, tau, n_sink, n_recent):
    """The dedup result, checked against the literal repair and the rule itself."""
    U, N = b.shape
    lit = oracle_mod.repair(b, S0, tau, n_sink=n_sink, n_recent=n_recent)
    dd = oracle_mod.repair_dedup(b, t, S0, tau, n_sink=n_sink, n_recent=n_recent)
    tau_f = float(np.float32(tau))
    i = np.arange(N)
    prot = (i < n_sink) | (i >= N - n_recent)
    for u in range(U):
        m = int(dd["nswaps"][u])
        ev = dd["swaps"][u, :m, 0]
        ad = dd["swaps"][u, :m, 1]
        donors = np.flatnonzero(lit["donor"][u])
        orphans = np.flatnonzero(lit["orphan"][u])
        # |S1| = |S0|; evicted are donors, admitted are orphans; at most the literal m
        assert dd["mask"][u].sum() == S0[u].sum()
        assert set(ev) <= set(donors) and set(ad) <= set(orphans)
        assert m <= lit["nswaps"][u]
        # the admitted orphans are the literal ranking's first m
        np.testing.assert_array_equal(ad, lit["swaps"][u, :m, 1])
        # no evicted donor's twin is evicted too
        evs = set(ev.tolist())
        assert not any(int(t[u, d]) in evs for d in ev)
        # the walk: donors by (b desc, position asc); a donor is passed over exactly
        # when its twin was evicted before it, or it is the twin of a donor evicted
        # before it; acceptance stops at |O|
        order = donors[np.lexsort((donors, -b[u, donors]))]
        rank = {int(d): k for k, d in enumerate(order)}
        ev_rank = [rank[int(d)] for d in ev]
        assert ev_rank == sorted(ev_rank)
        last = ev_rank[-1] if m else -1
        for k, d in enumerate(order[:last + 1]):
            d = int(d)
            earlier = set(int(x) for x in ev if rank[int(x)] < k)
            blocked = int(t[u, d]) in earlier or any(int(t[u, e]) == d for e in earlier)
            assert (d in evs) == (not blocked), (u, d)
        if m < len(orphans):   # ran out of donors: every later donor is blocked
            for d in order[last + 1:]:
                d = int(d)
                assert int(t[u, d]) in evs or any(int(t[u, e]) == d for e in ev), (u, d)
        assert all(b[u, d] >= tau_f and not prot[d] for d in ev)
    return lit, dd


@pytest.mark.parametrize("name,over,ratio", [
    ("tiny", {}, 0.5),
    ("llama", {"L": 1, "H": 2, "N": 1024}, 0.3),
    ("retrieval", {"L": 1, "H": 1, "N": 2048}, 0.3),
])
def test_invariants_on_planted_workloads(oracle_mod, name, over, ratio):
    w = synth.get(name, **over)
    keys, _ = synth.keys(w)
    S0 = synth.masks(w, ratio)
    a = oracle_mod.audit(keys, S0, window=synth.WINDOW)
    lit, dd = check_invariants(oracle_mod, a["b_ret"], a["t_ret"], S0, w.tau, synth.N_SINK,
                               synth.N_RECENT)
    if name == "retrieval":
        # 256 filler templates: many retained twin pairs, so dedup must bite
        assert np.any(dd["nswaps"] < lit["nswaps"]) or np.all(lit["nswaps"] == 0)


@pytest.mark.parametrize("seed", range(6))
def test_invariants_on_random_twin_graphs(oracle_mod, seed):
    """Random b and twin arrays (each twin a retained position other than itself, as
    the window guarantees), many ties."""
    rng = np.random.default_rng(seed)
    U, N = 3, int(rng.integers(20, 400))
    S0 = synth.random_masks(seed, U, N, N // 2)
    b = rng.choice([0.2, 0.5, 0.9, 0.95, 1.0], size=(U, N)).astype(np.float64)
    t = np.empty((U, N), np.int32)
    for u in range(U):
        ret = np.flatnonzero(S0[u])
        for i in range(N):
            t[u, i] = rng.choice(ret[ret != i])
    check_invariants(oracle_mod, b, t, S0, 0.85, 2, 5)


def test_no_donor_chains_gives_the_literal_repair(oracle_mod):
    """When every donor's twin is protected, nothing is skipped: dedup = literal."""
    rng = np.random.default_rng(3)
    U, N = 2, 300
    S0 = synth.random_masks(9, U, N, 150)
    S0[:, :4] = 1
    b = rng.uniform(0.0, 1.0, size=(U, N))
    t = rng.integers(0, 4, size=(U, N)).astype(np.int32)   # twins among the 4 sinks
    lit = oracle_mod.repair(b, S0, 0.6, n_sink=4, n_recent=0)
    dd = oracle_mod.repair_dedup(b, t, S0, 0.6, n_sink=4, n_recent=0)
    for k in ("mask", "nswaps", "status"):
        np.testing.assert_array_equal(dd[k], lit[k])
    for u in range(U):
        m = lit["nswaps"][u]
        np.testing.assert_array_equal(dd["swaps"][u, :m], lit["swaps"][u, :m])


def test_status_codes(oracle_mod):
    N = 50
    S0 = np.zeros((2, N), np.uint8)
    S0[:, :20] = 1
    S0[1, 30] = 2
    b = np.full((2, N), 0.5)
    t = np.zeros((2, N), np.int32)
    dd = oracle_mod.repair_dedup(b, t, S0, 0.6, budget=[19, 21])
    np.testing.assert_array_equal(dd["status"], [3, 1])
    np.testing.assert_array_equal(dd["nswaps"], [-1, -1])
    np.testing.assert_array_equal(dd["mask"], S0)
