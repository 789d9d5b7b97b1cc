"""Parity of the CUDA path (through the C ABI) with the fp64 oracle on seeded inputs:
shapes spanning several 128-row blocks and 256-column tiles with ragged tails, edge
cases (N = 1, empty and full retained sets, window wider than N, zero keys, exact
ties), the hand-derived worked example and the planted-twin workloads at reduced
sizes.  Scores within 2e-3; integer results exact outside the 4e-3 tie bands; the
repair kernel bit-exact on the GPU's own b values (split check)."""
import numpy as np
import pytest
import torch

import oracle
from golden_io import read_worked_example
from gpu_harness import (device, keys_tensor, redundancy_vs_oracle, repair_vs_oracle,
                         split_check)
from paper_2608_27128_gb300 import synth
from paper_2608_27128_gb300 import twinkv as tk

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _setup():
    oracle.build()
    tk.load()
    torch.cuda.init()


def hadamard(n):
    h = np.array([[1.0]])
    while h.shape[0] < n:
        h = np.block([[h, h], [h, -h]])
    return h


# ---------------------------------------------------------------- worked example

def test_worked_example():
    head, cases = read_worked_example()
    N = head["N"]
    k = np.zeros((1, N, 64), np.float32)
    k[0, :, :4] = head["keys"]
    keys = synth.f32_to_bf16_bits(k)
    score, twin = tk.twinkv_redundancy(keys_tensor(keys, 1, 1), head["window"])
    np.testing.assert_allclose(score.cpu().numpy().ravel(), head["b_all"], atol=2e-5)
    np.testing.assert_array_equal(twin.cpu().numpy().ravel(), head["t_all"])
    for case in cases:
        S0 = case["S0"].astype(np.uint8)
        out = tk.twinkv_repair(keys_tensor(keys, 1, 1),
                               torch.from_numpy(S0.reshape(1, 1, N)).to(device()),
                               torch.tensor([int(S0.sum())], dtype=torch.int32, device=device()),
                               threshold=case["tau"], window=head["window"],
                               n_sink=head["n_sink"], n_recent=head["n_recent"], want_all=True)
        h = {kk: v.cpu().numpy() for kk, v in out.items()}
        np.testing.assert_allclose(h["score_ret"].ravel(), case["b_ret"], atol=2e-5)
        np.testing.assert_array_equal(h["twin_ret"].ravel(), case["t_ret"])
        np.testing.assert_allclose(h["score_all"].ravel(), head["b_all"], atol=2e-5)
        np.testing.assert_array_equal(h["twin_all"].ravel(), head["t_all"])
        m = int(h["nswaps"][0])
        np.testing.assert_array_equal(h["swaps"][0, :m].ravel(), case["swaps"])
        np.testing.assert_array_equal(h["mask"].ravel(), case["S1"])
        assert h["status"][0] == 0


def test_exact_ties_go_to_lowest_position():
    """Scaled Hadamard rows: all off-diagonal sims are exactly 0 on both sides."""
    rng = np.random.default_rng(11)
    H = hadamard(128)[:, :128] * (2.0 ** rng.integers(-3, 4, size=128))[:, None]
    keys = synth.f32_to_bf16_bits(H.astype(np.float32))[None]
    for w in (0, 5, 31):
        score, twin = tk.twinkv_redundancy(keys_tensor(keys, 1, 1), w)
        i = np.arange(128)
        np.testing.assert_array_equal(twin.cpu().numpy().ravel(), np.where(i > w, 0, i + w + 1))
        assert np.all(score.cpu().numpy() == 0.0)


def simplex(n):
    """n keys whose pairwise similarities are all exactly -1/(n-1): the rows of a
    Hadamard matrix of order n with the all-ones first column zeroed (each row keeps
    n-1 entries of +-1, and two different rows have dot product 0 - 1 = -1)."""
    h = hadamard(n)
    h[:, 0] = 0.0
    return h


@pytest.mark.parametrize("n", [64, 128])
def test_exact_negative_ties_go_to_lowest_position(n):
    """Every candidate of every row ties at the same negative similarity: the twin is
    the lowest position beyond the window, in both the position-order audit and the
    retained-first audit of the repair (b_i(S0) and b_i(all)), with nothing excused."""
    d = n
    keys = synth.f32_to_bf16_bits(simplex(n).astype(np.float32))[None]
    i = np.arange(n)
    for w in (0, 5, 31):
        score, twin = tk.twinkv_redundancy(keys_tensor(keys, 1, 1), w)
        np.testing.assert_array_equal(twin.cpu().numpy().ravel(), np.where(i > w, 0, i + w + 1))
        np.testing.assert_allclose(score.cpu().numpy().ravel(), -1.0 / (n - 1), rtol=0,
                                   atol=1e-12)
        rep, s, t = redundancy_vs_oracle(keys, 1, 1, w)
        assert rep.n_fail == 0 and rep.n_excused == 0, rep.notes
    S0 = synth.random_masks(n, 1, n, n // 3)
    for w in (0, 7):
        rep, h, a, r = repair_vs_oracle(keys, S0, 1, 1, w, 0.85, n_sink=4, n_recent=8)
        assert rep.n_fail == 0 and rep.n_excused == 0, rep.notes
        ret = np.flatnonzero(S0[0])
        for row in range(n):
            cand = ret[np.abs(ret - row) > w]
            assert h["twin_ret"][0, row] == (cand[0] if cand.size else -1)
            assert h["twin_all"][0, row] == (0 if row > w else row + w + 1)


# ---------------------------------------------------------------- shape sweep

REDUNDANCY_CASES = [
    (1, 1, 1, 64, 0), (1, 1, 2, 64, 0), (1, 2, 33, 64, 32), (2, 1, 127, 128, 1),
    (1, 1, 129, 64, 5), (1, 1, 257, 128, 32), (1, 3, 300, 64, 32), (2, 2, 513, 128, 32),
    (1, 1, 1000, 64, 100), (1, 1, 2053, 128, 32), (1, 1, 600, 64, 700), (1, 1, 384, 128, 0),
]


@pytest.mark.parametrize("L,H,N,d,w", REDUNDANCY_CASES)
def test_redundancy_matches_oracle(L, H, N, d, w):
    keys = synth.random_keys(20 + N, L * H, N, d)
    rep, s, t = redundancy_vs_oracle(keys, L, H, w)
    assert rep.n_fail == 0, rep.notes
    assert rep.n_excused <= max(1, N // 100)
    assert rep.max_dev_same_twin < 1e-9


@pytest.mark.parametrize("L,H,N,d,w", REDUNDANCY_CASES + [(1, 2, 1500, 128, 3), (1, 1, 3000, 64, 32)])
def test_symmetric_redundancy_matches_oracle(L, H, N, d, w):
    """The upper-triangle audit: rows meet their earlier candidates through the column
    maxima of earlier row blocks, in the same packed (value, position) slot."""
    keys = synth.random_keys(20 + N, L * H, N, d)
    rep, s, t = redundancy_vs_oracle(keys, L, H, w, symmetric=True)
    assert rep.n_fail == 0, rep.notes
    assert rep.n_excused <= max(1, N // 100)
    assert rep.max_dev_same_twin < 1e-9


@pytest.mark.parametrize("n", [64, 128])
def test_symmetric_exact_ties_go_to_lowest_position(n):
    """Exact ties through both directions: simplex keys (every similarity -1/(n-1)) and
    Hadamard rows (every similarity 0), nothing excused."""
    keys = synth.f32_to_bf16_bits(simplex(n).astype(np.float32))[None]
    had = synth.f32_to_bf16_bits(hadamard(n).astype(np.float32))[None]
    i = np.arange(n)
    for w in (0, 5, 31):
        for k in (keys, had):
            score, twin = tk.twinkv_redundancy_symmetric(keys_tensor(k, 1, 1), w)
            np.testing.assert_array_equal(twin.cpu().numpy().ravel(), np.where(i > w, 0, i + w + 1))
            rep, s, t = redundancy_vs_oracle(k, 1, 1, w, symmetric=True)
            assert rep.n_fail == 0 and rep.n_excused == 0, rep.notes


def test_symmetric_planted_twins_across_row_blocks():
    """Planted copies whose source lies in an earlier row block (found only through the
    column direction) and in a later one (row direction), at several distances."""
    rng = np.random.default_rng(77)
    N, d = 2000, 128
    x = rng.standard_normal((1, N, d)).astype(np.float32)
    pairs = [(5, 1900), (130, 131 + 200), (700, 260), (1999, 3), (1024, 1500)]
    for src, dst in pairs:
        x[0, dst] = x[0, src] + 0.01 * rng.standard_normal(d).astype(np.float32)
    keys = synth.f32_to_bf16_bits(x)
    score, twin = tk.twinkv_redundancy_symmetric(keys_tensor(keys, 1, 1), 32)
    t = twin.cpu().numpy().ravel()
    for src, dst in pairs:
        assert t[dst] == src and t[src] == dst
    rep, s, tt = redundancy_vs_oracle(keys, 1, 1, 32, symmetric=True)
    assert rep.n_fail == 0, rep.notes


REPAIR_CASES = [
    # L, H, N, d, w, K, tau, n_sink, n_recent
    (1, 1, 1, 64, 0, 1, 0.85, 4, 64),
    (1, 1, 5, 64, 1, 2, 0.0, 0, 0),
    (1, 2, 65, 64, 2, 30, 0.2, 1, 3),
    (1, 1, 129, 128, 32, 0, 0.85, 4, 64),
    (1, 1, 129, 128, 32, 129, 0.85, 4, 64),
    (2, 1, 300, 64, 3, 150, 0.25, 4, 64),
    (1, 2, 511, 128, 32, 256, 0.3, 4, 64),
    (1, 1, 1025, 64, 7, 513, 0.3, 4, 64),
    (1, 1, 2053, 128, 32, 600, 0.28, 4, 64),
    (1, 1, 700, 64, 800, 350, 0.2, 4, 64),
    (1, 1, 258, 128, 0, 257, 0.3, 4, 64),
]


@pytest.mark.parametrize("L,H,N,d,w,K,tau,ns,nr", REPAIR_CASES)
def test_repair_matches_oracle(L, H, N, d, w, K, tau, ns, nr):
    keys = synth.random_keys(40 + N, L * H, N, d)
    S0 = synth.random_masks(41 + N, L * H, N, K)
    rep, h, a, r = repair_vs_oracle(keys, S0, L, H, w, tau, ns, nr)
    assert rep.n_fail == 0, rep.notes
    assert rep.max_dev_same_twin < 1e-9


def test_repair_without_b_all_skips_nothing_it_reports():
    keys = synth.random_keys(5, 2, 777, 128)
    S0 = synth.random_masks(6, 2, 777, 300)
    rep, h, a, r = repair_vs_oracle(keys, S0, 1, 2, 32, 0.3, want_all=False)
    assert rep.n_fail == 0, rep.notes
    assert "score_all" not in h


def test_zero_keys_have_similarity_zero():
    keys = synth.random_keys(8, 1, 300, 64)
    keys[0, [3, 100, 250]] = 0
    rep, s, t = redundancy_vs_oracle(keys, 1, 1, 4)
    assert rep.n_fail == 0, rep.notes
    assert s[0, 100] == 0.0


def test_fp32_keys_are_rounded_like_the_oracle():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((2, 400, 64)).astype(np.float32)
    rep, s, t = redundancy_vs_oracle(x, 1, 2, 32)
    assert rep.n_fail == 0 and rep.n_excused == 0, rep.notes


def test_non_default_stream():
    keys = synth.random_keys(9, 1, 500, 128)
    S0 = synth.random_masks(10, 1, 500, 200)
    st = torch.cuda.Stream()
    with torch.cuda.stream(st):
        rep, h, a, r = repair_vs_oracle(keys, S0, 1, 1, 32, 0.3, stream=st)
    assert rep.n_fail == 0, rep.notes


# ---------------------------------------------------------------- workloads (reduced)

@pytest.mark.parametrize("name,over,ratio", [
    ("tiny", {}, 0.5),
    ("llama", {"L": 1, "H": 2, "N": 2048}, 0.5),
    ("qwen", {"L": 1, "H": 2, "N": 2048}, 0.3),
    ("retrieval", {"L": 1, "H": 2, "N": 4096}, 0.3),
    ("long", {"L": 1, "H": 1, "N": 4096}, 0.5),
])
def test_workload_recipes(name, over, ratio):
    w = synth.get(name, **over)
    keys, truths = synth.keys(w)
    S0 = synth.masks(w, ratio)
    rep, h, a, r = repair_vs_oracle(keys, S0, w.L, w.H, synth.WINDOW, w.tau)
    assert rep.n_fail == 0, rep.notes
    assert rep.max_dev_same_twin < 1e-9
    if name == "tiny":
        assert rep.n_excused == 0, rep.notes
    # planted twins are found exactly, with no tie excuse
    for u, t in enumerate(truths):
        for s_, c in np.concatenate([t.pairs, t.exact_pairs]).reshape(-1, 2):
            if c - s_ > synth.WINDOW:
                assert h["twin_all"][u, s_] == a["t_all"][u, s_] == c
                assert h["twin_all"][u, c] == a["t_all"][u, c]
    if name == "retrieval":
        # evicted needles have no surviving twin: orphans, and all admitted
        for u, t in enumerate(truths):
            ev = t.needles[S0[u, t.needles] == 0]
            assert np.all(r["orphan"][u, ev] == 1)
            assert np.all(h["mask"][u, ev] == 1)


@pytest.mark.parametrize("name,over,ratio", [
    ("qwen", {"L": 4, "H": 2, "N": 2048}, 0.3),     # layer 0 keeps every key
    ("llama", {"L": 6, "H": 2, "N": 1500}, 0.5),
    ("qwen", {"L": 3, "H": 1, "N": 2053}, 0.7),     # ragged N
])
def test_pyramid_budgets(name, over, ratio):
    """Per-layer budgets in one call: every unit has its own |S0|, so the retained-first
    column layout, the tile counts of both segments and the selection sizes differ
    from unit to unit within the launch."""
    w = synth.get(name, **over)
    keys, _ = synth.keys(w)
    S0 = synth.masks(w, ratio, schedule="pyramid")
    k = np.repeat(synth.pyramid_budgets(w, ratio), w.H)
    assert len(set(k.tolist())) == w.L
    rep, h, a, r = repair_vs_oracle(keys, S0, w.L, w.H, synth.WINDOW, w.tau)
    assert rep.n_fail == 0, rep.notes
    assert rep.max_dev_same_twin < 1e-9
    np.testing.assert_array_equal(h["mask"].sum(1), k)
    full = np.flatnonzero(k == w.N)
    for u in full:
        # nothing evicted: b_i(S0) = b_i(all) for every row, and no swap
        np.testing.assert_array_equal(h["score_ret"][u], h["score_all"][u])
        np.testing.assert_array_equal(h["twin_ret"][u], h["twin_all"][u])
        assert h["nswaps"][u] == 0


# ---------------------------------------------------------------- selection alone

@pytest.mark.parametrize("seed", range(4))
def test_repair_select_is_bit_exact(seed):
    rng = np.random.default_rng(seed)
    L, H, N = 2, 3, int(rng.integers(50, 5000))
    U = L * H
    grid = np.array([-1.0, -0.0, 0.0, 0.25, 0.5, 0.75, 0.85, 0.9, 1.0,
                     float(np.float32(0.5)) + 1e-12])
    b = np.where(rng.random((U, N)) < 0.5, rng.choice(grid, size=(U, N)),
                 rng.uniform(-1, 1, size=(U, N)))
    S0 = synth.random_masks(seed, U, N, N // 2)
    tau = 0.5
    budget = S0.sum(1).astype(np.int32)
    budget[1] += 1                     # a budget mismatch
    S0[2, 7] = 3                       # a mask byte outside {0,1}
    out = tk.twinkv_repair_select(
        torch.from_numpy(b.reshape(L, H, N)).to(device()),
        torch.from_numpy(S0.reshape(L, H, N)).to(device()),
        torch.from_numpy(budget).to(device()), threshold=tau)
    h = {k: v.cpu().numpy() for k, v in out.items()}
    h["score_ret"] = b
    assert list(h["status"][:3]) == [0, 3, 1]
    split_check(h, S0, tau, 4, 64, budget=budget)


@pytest.mark.parametrize("N,frac", [(30000, 0.5), (24001, 0.35)])
def test_repair_select_lists_on_both_sides_of_the_shared_memory_sort(N, frac):
    """Units whose swap lists run from a few dozen items to well above 4096, at the
    cluster size the library picks for them, with many equal b values and ties at tau,
    bit-exact against the oracle's selection."""
    rng = np.random.default_rng(N)
    L, H = 1, 4
    U = L * H
    b = np.round(rng.uniform(-1.0, 1.0, size=(U, N)), 3)   # many exact ties
    b[:, ::97] = 0.0                                          # ties at tau
    K = np.array([N // 2, int(N * frac), N // 8, N - 64], np.int64)
    S0 = np.zeros((U, N), np.uint8)
    for u in range(U):
        S0[u, rng.permutation(N)[:K[u]]] = 1
    tau = 0.0
    out = tk.twinkv_repair_select(
        torch.from_numpy(b.reshape(L, H, N)).to(device()),
        torch.from_numpy(S0.reshape(L, H, N)).to(device()),
        torch.from_numpy(S0.sum(1).astype(np.int32)).to(device()), threshold=tau)
    h = {k: v.cpu().numpy() for k, v in out.items()}
    h["score_ret"] = b
    m = h["nswaps"]
    assert m.max() > 4096 and m.min() < 4096, m
    split_check(h, S0, tau, 4, 64)


@pytest.mark.parametrize("cluster", [1, 2, 4, 8, 16])
@pytest.mark.parametrize("N,K,tau", [(30000, 15000, 0.0), (24001, 8400, 0.25), (611, 300, 0.0),
                                     (50, 25, 0.0)])
def test_repair_select_every_cluster_size(cluster, N, K, tau, monkeypatch):
    """The literal selection on clusters of 1 to 16 CTAs per unit (forced; the library
    picks the size from the unit count): lists cut on either side; per-CTA shares of the
    swap list up to 2048 items (both sides sorted at once), from 2049 to 4096 (one side
    after the other) and above (radix passes over the workspace); slices that are empty,
    many equal b values and ties at tau, bit-exact against the oracle."""
    monkeypatch.setenv("TWINKV_SELECT_CLUSTER", str(cluster))
    rng = np.random.default_rng([N, K, cluster])
    L, H = 1, 3
    U = L * H
    b = np.round(rng.uniform(-1.0, 1.0, size=(U, N)), 3)   # many exact ties
    b[:, ::89] = tau                                          # ties at tau
    S0 = np.zeros((U, N), np.uint8)
    for u, k in enumerate((K, N - K, N // 7)):
        S0[u, rng.permutation(N)[:k]] = 1
    budget = S0.sum(1).astype(np.int32)
    out = tk.twinkv_repair_select(
        torch.from_numpy(b.reshape(L, H, N)).to(device()),
        torch.from_numpy(S0.reshape(L, H, N)).to(device()),
        torch.from_numpy(budget).to(device()), threshold=tau)
    h = {k: v.cpu().numpy() for k, v in out.items()}
    h["score_ret"] = b
    assert np.all(h["status"] == 0)
    split_check(h, S0, tau, 4, 64)


@pytest.mark.parametrize("d", [128, 64])
def test_keys_far_below_their_units_largest_norm(d):
    """The audit's packed resolution is relative to the unit's largest key norm: a key
    of norm ratio r to it has a near-tie band of about 2^-17 / r in similarity.  Down to
    r = 1/100 that band stays inside the 2e-3 tolerance: every key of these units is
    about 100 times shorter than one outlier key, with planted near-duplicates, and all
    compare with the oracle."""
    U, N = 2, 1500
    rng = np.random.default_rng(d)
    x = rng.standard_normal((U, N, d), dtype=np.float32)
    for u in range(U):
        src = rng.choice(N, 60, replace=False)
        dst = (src + rng.integers(40, 400, 60)) % N
        x[u, dst] = x[u, src] + np.float32(0.02) * rng.standard_normal((60, d), dtype=np.float32)
        x[u, 700] *= np.float32(100.0)          # the outlier sets the unit's scale
    rep, s, t = redundancy_vs_oracle(x, 1, U, 32)
    assert rep.n_fail == 0, rep.notes
    assert rep.max_dev_same_twin < 1e-9


def test_wait_probe_times_out_cleanly():
    assert tk.twinkv_wait_probe(2_000_000) == tk.ERR_TIMEOUT
    # the context stays usable and the sticky error word is untouched
    keys = synth.random_keys(1, 1, 200, 64)
    rep, s, t = redundancy_vs_oracle(keys, 1, 1, 32)
    assert rep.n_fail == 0
    assert tk.twinkv_get_last_error() == tk.OK
