"""Pins for the reference oracle, checked against things other than itself.

Each test fixes the oracle to a closed form, a hand-derived worked example, a float64
numpy computation it does not use, a brute-force ranking, or an invariant the paper
states (Sec. 3.2 Eq. 1 and the twin relation; Sec. 3.4 Eq. 4, the orphan/donor rule
and the budget-preserving swap; Sec. 4.1 no-op check).  None needs a GPU.
"""
import numpy as np
import pytest

from golden_io import read_worked_example
from paper_2608_27128_gb300 import synth


def bf16(x):
    return synth.f32_to_bf16_bits(np.asarray(x, np.float32))


def hadamard(n):
    h = np.array([[1.0]])
    while h.shape[0] < n:
        h = np.block([[h, h], [h, -h]])
    return h


# ---------------------------------------------------------------- worked example

def test_worked_example_audit_and_repair(oracle_mod):
    head, cases = read_worked_example()
    keys = bf16(head["keys"])[None]
    w = head["window"]
    for case in cases:
        S0 = case["S0"].astype(np.uint8)
        a = oracle_mod.audit(keys, S0[None], window=w)
        np.testing.assert_allclose(a["b_all"][0], head["b_all"], atol=1e-12)
        np.testing.assert_array_equal(a["t_all"][0], head["t_all"])
        np.testing.assert_allclose(a["b_ret"][0], case["b_ret"], atol=1e-12)
        np.testing.assert_array_equal(a["t_ret"][0], case["t_ret"])
        r = oracle_mod.repair(a["b_ret"], S0[None], case["tau"], n_sink=head["n_sink"],
                              n_recent=head["n_recent"], budget=[int(S0.sum())])
        assert r["status"][0] == 0
        np.testing.assert_array_equal(np.flatnonzero(r["orphan"][0]), case["orphans"])
        np.testing.assert_array_equal(np.flatnonzero(r["donor"][0]), case["donors"])
        m = r["nswaps"][0]
        np.testing.assert_array_equal(r["swaps"][0, :m].ravel(), case["swaps"])
        np.testing.assert_array_equal(r["mask"][0], case["S1"])


def test_worked_example_zero_padding_keeps_results(oracle_mod):
    """Zero channels change neither dots nor norms (Eq. 1): d=4 embeds in d=64."""
    head, cases = read_worked_example()
    k4 = bf16(head["keys"])[None]
    k64 = np.zeros((1, head["N"], 64), np.uint16)
    k64[0, :, :4] = k4[0]
    S0 = cases[0]["S0"].astype(np.uint8)[None]
    a4 = oracle_mod.audit(k4, S0, window=1)
    a64 = oracle_mod.audit(k64, S0, window=1)
    for k in ("b_all", "t_all", "b_ret", "t_ret"):
        np.testing.assert_array_equal(a4[k], a64[k])


# ---------------------------------------------------------------- Eq. 1 closed forms

def test_sim_closed_forms(oracle_mod):
    k = bf16([[3, 4, 0, 0], [0, 1, 0, 0], [1, 1, 1, 1], [-3, -4, 0, 0], [0, 0, 0, 0],
              [6, 8, 0, 0]])[None]
    assert oracle_mod.sim(k, 0, 0, 1) == pytest.approx(0.8, abs=1e-15)
    assert oracle_mod.sim(k, 0, 2, 0) == pytest.approx(0.7, abs=1e-15)
    assert oracle_mod.sim(k, 0, 0, 3) == pytest.approx(-1.0, abs=1e-15)
    assert oracle_mod.sim(k, 0, 0, 5) == pytest.approx(1.0, abs=1e-15)   # scale invariance
    assert oracle_mod.sim(k, 0, 4, 0) == 0.0                             # zero key
    assert oracle_mod.sim(k, 0, 1, 2) == pytest.approx(0.5, abs=1e-15)


def test_hadamard_rows_are_orthogonal_and_ties_go_to_lowest_position(oracle_mod):
    """Scaled Hadamard rows: every off-diagonal sim is exactly 0, so each row's best
    twin is the lowest position outside its window, and the second best is also 0."""
    rng = np.random.default_rng(11)
    H = hadamard(64) * (2.0 ** rng.integers(-3, 4, size=64))[:, None]
    keys = bf16(H)[None]
    for w in (0, 5, 31):
        a = oracle_mod.audit(keys, window=w)
        i = np.arange(64)
        expect_t = np.where(i > w, 0, i + w + 1)
        assert np.all(a["b_all"][0] == 0.0)
        np.testing.assert_array_equal(a["t_all"][0], expect_t)
        n_elig = np.maximum(i - w, 0) + np.maximum(64 - (i + w + 1), 0)
        expect2 = np.where(n_elig >= 2, 0.0, -np.inf)
        np.testing.assert_array_equal(a["b_all2"][0], expect2)


def test_scaled_and_negated_copies(oracle_mod):
    """A positively scaled copy gives sim exactly 1 (normalisation, Eq. 1); a negated
    copy gives -1 and never beats an orthogonal key."""
    H = hadamard(64)
    keys = bf16(H.copy())
    keys[40] = bf16(4.0 * H[3])
    keys[50] = bf16(-0.5 * H[7])
    a = oracle_mod.audit(keys[None], window=2)
    assert a["b_all"][0, 3] == 1.0 and a["t_all"][0, 3] == 40
    assert a["b_all"][0, 40] == 1.0 and a["t_all"][0, 40] == 3
    assert a["b_all"][0, 7] == 0.0 and a["t_all"][0, 7] == 0
    assert a["b_all"][0, 50] == 0.0
    # only negated partners eligible: the best is -1, a real twin (not the empty -1)
    k3 = bf16([[1, 2, 0, 0], [-1, -2, 0, 0], [-2, -4, 0, 0]])[None]
    b = oracle_mod.audit(k3, window=0)
    assert b["b_all"][0, 0] == pytest.approx(-1.0, abs=1e-15)
    assert b["t_all"][0, 0] == 1


def test_window_boundary(oracle_mod):
    """|i-j| = w is excluded and |i-j| = w+1 included (Sec. 3.2 twin relation)."""
    rng = np.random.default_rng(5)
    w = 5
    x = rng.standard_normal((100, 64)).astype(np.float32)
    x[10 + w] = x[10]          # distance w: not a twin
    x[10 + w + 1] = x[10]      # distance w+1: a twin
    keys = bf16(x)[None]
    a = oracle_mod.audit(keys, window=w)
    assert a["t_all"][0, 10] == 16 and a["b_all"][0, 10] == pytest.approx(1.0, abs=1e-14)
    assert a["t_all"][0, 16] == 10
    assert a["b_all"][0, 15] < 0.9          # its copies at distance w and 1 are excluded
    assert a["t_all"][0, 15] not in (10, 16)


# ---------------------------------------------------------------- dense library check

@pytest.mark.parametrize("U,N,d,w", [(2, 300, 64, 7), (1, 129, 128, 32), (1, 70, 64, 0)])
def test_against_float64_numpy_dense_matrix(oracle_mod, U, N, d, w):
    """Eq. 1 as a float64 numpy matmul on normalised keys, the window and retained
    masks applied to the dense matrix, then numpy max/argmax (first maximum)."""
    keys = synth.random_keys(1, U, N, d)
    S0 = synth.random_masks(2, U, N, N // 3)
    a = oracle_mod.audit(keys, S0, window=w)
    kf = synth.bf16_bits_to_f32(keys).astype(np.float64)
    for u in range(U):
        kh = kf[u] / np.linalg.norm(kf[u], axis=1, keepdims=True)
        S = kh @ kh.T
        i, j = np.meshgrid(np.arange(N), np.arange(N), indexing="ij")
        S_all = np.where(np.abs(i - j) > w, S, -np.inf)
        S_ret = np.where(S0[u][None, :] != 0, S_all, -np.inf)
        np.testing.assert_allclose(a["b_all"][u], S_all.max(1), atol=1e-12)
        np.testing.assert_array_equal(a["t_all"][u], S_all.argmax(1))
        has = np.isfinite(S_ret.max(1))
        np.testing.assert_allclose(a["b_ret"][u][has], S_ret.max(1)[has], atol=1e-12)
        np.testing.assert_array_equal(a["t_ret"][u][has], S_ret.argmax(1)[has])
        assert np.all(a["b_ret"][u][~has] == -1) and np.all(a["t_ret"][u][~has] == -1)
        srt = np.sort(S_all, axis=1)
        np.testing.assert_allclose(a["b_all2"][u], srt[:, -2], atol=1e-12)


def test_row_subset_matches_full(oracle_mod):
    keys = synth.random_keys(3, 2, 200, 64)
    S0 = synth.random_masks(4, 2, 200, 90)
    full = oracle_mod.audit(keys, S0, window=32)
    rows = np.array([0, 7, 199, 100, 33])
    sub = oracle_mod.audit(keys, S0, window=32, rows=rows)
    for k in full:
        np.testing.assert_array_equal(sub[k], full[k][:, rows])


# ---------------------------------------------------------------- Eq. 4 invariants

def test_empty_candidate_sets_give_minus_one(oracle_mod):
    keys = synth.random_keys(6, 1, 40, 64)
    a = oracle_mod.audit(keys, np.ones((1, 40), np.uint8), window=39)
    assert np.all(a["b_all"] == -1) and np.all(a["t_all"] == -1)
    a = oracle_mod.audit(keys, np.zeros((1, 40), np.uint8), window=3)
    assert np.all(a["b_ret"] == -1) and np.all(a["t_ret"] == -1)
    assert np.all(a["t_all"] >= 0)
    # the middle row of N = 2w+1 has no position farther than w
    a = oracle_mod.audit(synth.random_keys(6, 1, 11, 64), window=5)
    assert a["b_all"][0, 5] == -1 and a["t_all"][0, 5] == -1
    assert np.all(a["t_all"][0, np.arange(11) != 5] >= 0)


def test_retained_everything_equals_all(oracle_mod):
    keys = synth.random_keys(7, 2, 150, 64)
    a = oracle_mod.audit(keys, np.ones((2, 150), np.uint8), window=4)
    np.testing.assert_array_equal(a["b_ret"], a["b_all"])
    np.testing.assert_array_equal(a["t_ret"], a["t_all"])


def test_retained_max_invariants(oracle_mod):
    keys = synth.random_keys(8, 3, 257, 64)
    S0 = synth.random_masks(9, 3, 257, 100)
    w = 6
    a = oracle_mod.audit(keys, S0, window=w)
    assert np.all(a["b_ret"] <= a["b_all"])
    for u in range(3):
        t = a["t_ret"][u]
        assert np.all(S0[u][t] == 1)
        assert np.all(np.abs(t - np.arange(257)) > w)
        in_s0 = S0[u][a["t_all"][u]] == 1
        np.testing.assert_array_equal(a["b_ret"][u][in_s0], a["b_all"][u][in_s0])
        np.testing.assert_array_equal(a["t_ret"][u][in_s0], a["t_all"][u][in_s0])


def test_reversal_equivariance(oracle_mod):
    """Reversing positions reverses every output and maps twin j to N-1-j."""
    N = 180
    keys = synth.random_keys(10, 1, N, 64)
    S0 = synth.random_masks(11, 1, N, 70)
    a = oracle_mod.audit(keys, S0, window=9)
    r = oracle_mod.audit(keys[:, ::-1].copy(), S0[:, ::-1].copy(), window=9)
    np.testing.assert_allclose(r["b_all"][0][::-1], a["b_all"][0], atol=1e-14)
    np.testing.assert_array_equal(N - 1 - r["t_all"][0][::-1], a["t_all"][0])
    np.testing.assert_array_equal(N - 1 - r["t_ret"][0][::-1], a["t_ret"][0])


def test_planted_tiny_workload(oracle_mod):
    """Tiny workload: every planted pair (copy + N(0, 0.01^2)) and exact duplicate is
    found as twin in both directions; cos >= 1/sqrt(1 + 4 sigma^2 d / |k|^2)."""
    w = synth.get("tiny")
    keys, truth = synth.keys(w)
    a = oracle_mod.audit(keys, window=synth.WINDOW)
    for s, c in truth[0].pairs:
        assert a["t_all"][0, s] == c and a["t_all"][0, c] == s
        assert a["b_all"][0, s] > 0.999
    for s, c in truth[0].exact_pairs:
        assert a["t_all"][0, c] == s
        assert a["b_all"][0, c] == pytest.approx(1.0, abs=1e-14)


# ---------------------------------------------------------------- bf16 decoding

def test_round_bf16_bit_patterns(oracle_mod):
    x = np.array([1.0, 1.0 + 2**-8, 1.0 + 3 * 2**-8, 1.0 + 2**-8 + 2**-20, -2.5,
                  0.0, 3.0e38, 1.0 - 2**-9], np.float32)
    expect = np.array([0x3F80, 0x3F80, 0x3F82, 0x3F81, 0xC020, 0x0000, 0x7F62, 0x3F80],
                      np.uint16)
    np.testing.assert_array_equal(oracle_mod.round_bf16(x), expect)


def test_fp32_keys_are_rounded_to_bf16(oracle_mod):
    x = np.random.default_rng(12).standard_normal((1, 90, 64)).astype(np.float32)
    a = oracle_mod.audit(x, window=3)
    b = oracle_mod.audit(oracle_mod.round_bf16(x), window=3)
    np.testing.assert_array_equal(a["b_all"], b["b_all"])


# ---------------------------------------------------------------- Sec. 3.4 repair

def _brute_force_repair(b, S0, tau, n_sink, n_recent):
    """Classification by definition, ranking by counting (O(n^2)): an orphan's rank
    is the number of orphans strictly more severe; likewise for donors."""
    N = b.size
    tau = float(np.float32(tau))
    prot = (np.arange(N) < n_sink) | (np.arange(N) >= N - n_recent)
    O = [i for i in range(N) if S0[i] == 0 and b[i] < tau]
    D = [i for i in range(N) if S0[i] == 1 and not prot[i] and b[i] >= tau]
    m = min(len(O), len(D))
    rank_o = {i: sum((b[j], j) < (b[i], i) for j in O) for i in O}
    rank_d = {i: sum((-b[j], j) < (-b[i], i) for j in D) for i in D}
    so = sorted((rank_o[i], i) for i in O if rank_o[i] < m)
    sd = sorted((rank_d[i], i) for i in D if rank_d[i] < m)
    S1 = S0.copy()
    for (_, i), (_, j) in zip(so, sd):
        S1[i], S1[j] = 1, 0
    return O, D, [(j, i) for (_, i), (_, j) in zip(so, sd)], S1


@pytest.mark.parametrize("seed", range(12))
def test_repair_matches_brute_force_ranking(oracle_mod, seed):
    rng = np.random.default_rng(seed)
    N = int(rng.integers(6, 40))
    tau = float(rng.choice([0.5, 0.75, 0.85]))
    # coarse grid values create exact ties in b and values exactly at tau
    b = rng.choice([-1.0, 0.0, 0.25, 0.5, 0.75, 0.85, 0.9, 1.0], size=N)
    K = int(rng.integers(0, N + 1))
    S0 = np.zeros(N, np.uint8)
    S0[rng.permutation(N)[:K]] = 1
    n_sink, n_recent = int(rng.integers(0, 3)), int(rng.integers(0, 4))
    r = oracle_mod.repair(b[None], S0[None], tau, n_sink=n_sink, n_recent=n_recent)
    O, D, swaps, S1 = _brute_force_repair(b, S0, tau, n_sink, n_recent)
    np.testing.assert_array_equal(np.flatnonzero(r["orphan"][0]), O)
    np.testing.assert_array_equal(np.flatnonzero(r["donor"][0]), D)
    m = r["nswaps"][0]
    assert m == len(swaps)
    assert [tuple(p) for p in r["swaps"][0, :m].tolist()] == swaps
    np.testing.assert_array_equal(r["mask"][0], S1)


def test_repair_invariants_on_the_tiny_workload(oracle_mod):
    w = synth.get("tiny")
    keys, _ = synth.keys(w)
    S0 = synth.masks(w, 0.5)
    a = oracle_mod.audit(keys, S0, window=synth.WINDOW)
    r = oracle_mod.repair(a["b_ret"], S0, w.tau, budget=S0.sum(1))
    S1 = r["mask"][0]
    m = r["nswaps"][0]
    assert S1.sum() == S0.sum()                                   # |S1| = |S0|
    out_, in_ = r["swaps"][0, :m, 0], r["swaps"][0, :m, 1]
    assert np.all(r["donor"][0][out_] == 1) and np.all(r["orphan"][0][in_] == 1)
    assert m == min(r["orphan"].sum(), r["donor"].sum())
    changed = np.flatnonzero(S1 != S0[0])
    np.testing.assert_array_equal(np.sort(changed), np.sort(np.concatenate([out_, in_])))
    prot = np.r_[0:4, 512 - 64:512]
    assert np.all(S1[prot] >= S0[0][prot])      # protected positions never leave
    assert m > 0


def test_no_op_when_selection_is_redundancy_consistent(oracle_mod):
    """Sec. 4.1 no-op check: retained keys are mutually orthogonal (no donors) and every
    evicted key is a copy of a retained one far enough away (no orphans): S1 = S0."""
    H = hadamard(64)
    N = 128
    keys = np.zeros((N, 64), np.float32)
    keys[:64] = H                      # retained, pairwise sim 0
    keys[64:] = H[np.arange(64)]       # evicted copies, distance 64 > w
    S0 = np.zeros(N, np.uint8)
    S0[:64] = 1
    a = oracle_mod.audit(bf16(keys)[None], S0[None], window=32)
    r = oracle_mod.repair(a["b_ret"], S0[None], 0.85, n_sink=0, n_recent=0)
    assert r["orphan"].sum() == 0 and r["donor"].sum() == 0
    assert r["nswaps"][0] == 0
    np.testing.assert_array_equal(r["mask"][0], S0)


def test_repair_status_codes(oracle_mod):
    b = np.zeros((2, 10))
    S0 = np.zeros((2, 10), np.uint8)
    S0[:, :4] = 1
    S0[1, 7] = 2
    r = oracle_mod.repair(b, S0, 0.5, budget=[3, 5])
    assert list(r["status"]) == [3, 1]
    assert list(r["nswaps"]) == [-1, -1]
    np.testing.assert_array_equal(r["mask"], S0)


def test_f32_entry_equals_f64_entry_on_float_values(oracle_mod):
    rng = np.random.default_rng(3)
    b = rng.uniform(-1, 1, size=(3, 500)).astype(np.float32)
    b[:, ::7] = np.float32(0.85)
    S0 = synth.random_masks(5, 3, 500, 240)
    r32 = oracle_mod.repair_f32(b, S0, 0.85)
    r64 = oracle_mod.repair(b.astype(np.float64), S0, 0.85)
    for k in r32:
        np.testing.assert_array_equal(r32[k], r64[k])


def test_similarity_is_symmetric_and_exact_for_duplicates(oracle_mod):
    """Eq. 1 is symmetric in (i, j): mutual twins carry bitwise-equal b; duplicates
    (also positively scaled by a power of two) score exactly 1."""
    keys = synth.random_keys(13, 1, 400, 128)
    keys[0, 300] = keys[0, 10]
    x = synth.bf16_bits_to_f32(keys[0, 20]) * 4.0
    keys[0, 350] = synth.f32_to_bf16_bits(x)
    a = oracle_mod.audit(keys, window=32)
    t, b = a["t_all"][0], a["b_all"][0]
    mutual = [i for i in range(400) if t[t[i]] == i]
    assert len(mutual) > 10
    for i in mutual:
        assert b[i] == b[t[i]]
    assert b[10] == 1.0 and t[10] == 300 and b[20] == 1.0 and t[20] == 350
    for i, j in [(3, 77), (200, 5), (10, 300)]:
        assert oracle_mod.sim(keys, 0, i, j) == oracle_mod.sim(keys, 0, j, i)
