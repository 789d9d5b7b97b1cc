"""The comparator itself, on the CPU: what it excuses and what it fails.

The GPU parity tests rest on tests/comparator.py, so it is pinned here on planted
differences built with the oracle's own repair (Sec. 3.4): an identical result passes
with nothing excused; a flag flip whose b lies within BAND of tau, and the swaps that
follow from it, are excused; a change to a protected position, a twin that is not a
near tie, a score off by more than TOL, or a swap count that no flip explains fail."""
import numpy as np

import oracle
from comparator import BAND, TOL, compare_best, compare_repair

N, TAU = 400, 0.5


def unit(seed=0, K=200):
    rng = np.random.default_rng(seed)
    b = rng.uniform(-0.2, 1.0, N)
    S0 = np.zeros(N, np.uint8)
    S0[rng.permutation(N)[:K]] = 1
    return b, S0


def run(b, S0):
    r = oracle.repair(b[None], S0[None], TAU)
    return {k: v[0] for k, v in r.items()}


def test_identical_result_passes_clean():
    b, S0 = unit()
    o = run(b, S0)
    rep = compare_repair(S0, o["mask"], o["swaps"], int(o["nswaps"]), o, b, TAU)
    assert rep.n_fail == 0 and rep.n_excused == 0
    assert int(o["nswaps"]) > 0


def test_flag_flip_near_tau_and_its_extra_swap_are_excused():
    b, S0 = unit(1)
    o = run(b, S0)
    n_o, n_d = int(o["orphan"].sum()), int(o["donor"].sum())
    assert n_o != n_d
    # flip one candidate of the shorter side across tau, as a GPU whose b is off by
    # less than BAND would: m grows by one
    if n_o < n_d:
        i = int(np.flatnonzero((S0 == 0) & (b >= TAU))[0])
        b_gpu = b.copy()
        b[i] = TAU + 0.5 * BAND
        b_gpu[i] = TAU - 0.5 * BAND
    else:
        pos = np.arange(N)
        i = int(np.flatnonzero((S0 == 1) & (b < TAU) & (pos >= 4) & (pos < N - 64))[0])
        b_gpu = b.copy()
        b[i] = TAU - 0.5 * BAND
        b_gpu[i] = TAU + 0.5 * BAND
    o = run(b, S0)
    g = run(b_gpu, S0)
    assert int(g["nswaps"]) == int(o["nswaps"]) + 1
    rep = compare_repair(S0, g["mask"], g["swaps"], int(g["nswaps"]), o, b, TAU)
    assert rep.n_fail == 0, rep.notes
    assert rep.n_excused >= 1


def test_protected_position_change_fails_even_near_tau():
    b, S0 = unit(2)
    S0[0] = 1
    b[0] = TAU + 0.1 * BAND          # near tau, but position 0 is a sink: never a donor
    o = run(b, S0)
    assert o["mask"][0] == 1
    S1 = o["mask"].copy()
    S1[0] = 0
    rep = compare_repair(S0, S1, o["swaps"], int(o["nswaps"]), o, b, TAU)
    assert rep.n_fail >= 1


def test_unexplained_swap_count_fails():
    b, S0 = unit(3)
    o = run(b, S0)
    m = int(o["nswaps"])
    rep = compare_repair(S0, o["mask"], o["swaps"], m + 1, o, np.where(
        np.abs(b - TAU) <= BAND, TAU + 3 * BAND, b), TAU)
    assert rep.n_fail >= 1


def test_swapped_order_beyond_band_fails():
    b, S0 = unit(4)
    o = run(b, S0)
    m = int(o["nswaps"])
    assert m >= 2
    sw = o["swaps"].copy()
    d0, d1 = sw[0, 0], sw[m - 1, 0]
    assert abs(b[d0] - b[d1]) > BAND
    sw[0, 0], sw[m - 1, 0] = d1, d0
    rep = compare_repair(S0, o["mask"], sw, m, o, b, TAU)
    assert rep.n_fail >= 1


def test_compare_best_rules():
    b_orc = np.array([0.9, 0.5, -1.0, 0.7])
    t_orc = np.array([10, 20, -1, 30])
    b2 = np.array([0.9 - 0.5 * BAND, 0.3, -1.0, 0.7 - 0.5 * BAND])
    sims = {(0, 11): 0.9 - 0.5 * BAND, (3, 31): 0.7 - 2 * BAND}
    sim = lambda i, j: sims[(i, j)]   # noqa: E731
    # identical
    rep = compare_best(b_orc, t_orc, b_orc, t_orc, b2, sim, window=0)
    assert rep.n_fail == 0 and rep.n_excused == 0
    # a near tie at row 0 (gap <= BAND, the GPU's twin scores within BAND): excused
    rep = compare_best(b_orc, np.array([11, 20, -1, 30]), b_orc, t_orc, b2, sim, window=0)
    assert rep.n_fail == 0 and rep.n_excused == 1
    # row 3's other twin scores more than BAND below the best: a failure
    rep = compare_best(b_orc, np.array([10, 20, -1, 31]), b_orc, t_orc, b2, sim, window=0)
    assert rep.n_fail == 1
    # a twin inside the window is never excused
    rep = compare_best(b_orc, np.array([11, 20, -1, 30]), b_orc, t_orc, b2, sim, window=11)
    assert rep.n_fail == 1
    # a score off by more than TOL, and a candidate where the oracle has none
    rep = compare_best(b_orc + np.array([0, 2 * TOL, 0, 0]), t_orc, b_orc, t_orc, b2, sim,
                       window=0)
    assert rep.n_fail == 1
    rep = compare_best(b_orc, np.array([10, 20, 5, 30]), b_orc, t_orc, b2, sim, window=0)
    assert rep.n_fail == 1
