"""Pins for the oracle's standalone policy (Sec. 3.2, Eq. 2-3), checked against things
other than itself: the hand-derived worked example in tests/golden/worked_policy.txt,
closed forms on orthogonal (Hadamard) keys and planted duplicates, a float64 numpy
dense matrix, Python's own sort as a brute-force ranking, and the rule's invariants.
None needs a GPU."""
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


def protected(N, n_sink, n_recent):
    i = np.arange(N)
    return (i < n_sink) | (i >= N - n_recent)


# ---------------------------------------------------------------- worked example

def test_worked_example_counts_and_policy(oracle_mod):
    head, cases = read_worked_example("worked_policy.txt")
    keys = bf16(head["keys"])[None]
    for c in cases:
        cnt = oracle_mod.count(keys, c["tau"], head["window"])
        np.testing.assert_array_equal(cnt["r"][0], c["r"], err_msg=c["name"])
        for kk, ss in (("K", "S"), ("K2", "S2")):
            if kk not in c:
                continue
            p = oracle_mod.policy_select(cnt["r"], int(c[kk][0]), head["n_sink"],
                                         head["n_recent"])
            np.testing.assert_array_equal(p["mask"][0], c[ss], err_msg=c["name"] + kk)
            assert p["status"][0] == 0


# ---------------------------------------------------------------- counts (Eq. 2)

def test_orthogonal_keys_closed_form(oracle_mod):
    """Scaled Hadamard rows: every off-diagonal sim is exactly 0.  Eq. 2 is strict, so
    tau = 0 counts nothing; tau < 0 counts every j outside the window."""
    rng = np.random.default_rng(3)
    N = 64
    H = hadamard(N) * (2.0 ** rng.integers(-3, 4, size=N))[:, None]
    keys = bf16(H)[None]
    i = np.arange(N)
    for w in (0, 4, 40):
        n_elig = np.maximum(i - w, 0) + np.maximum(N - (i + w + 1), 0)
        assert np.all(oracle_mod.count(keys, 0.5, w)["r"][0] == 0)
        assert np.all(oracle_mod.count(keys, 0.0, w)["r"][0] == 0)
        np.testing.assert_array_equal(oracle_mod.count(keys, -0.25, w)["r"][0], n_elig)


def test_planted_copies_and_window_boundary(oracle_mod):
    """A direction copied c times (positively scaled) on orthogonal background: each
    copy's r is the number of other copies outside its window; a copy at distance
    exactly w does not count, one at w + 1 does."""
    H = hadamard(128)
    x = H.copy()
    w = 6
    src = 10
    copies = [10, 10 + w, 10 + w + 1, 60, 100]        # 16 is at distance w from 10
    for p in copies:
        x[p] = H[src] * (2.0 ** (p % 3))
    keys = bf16(x)[None]
    r = oracle_mod.count(keys, 0.9, w)["r"][0]
    for p in copies:
        expect = sum(1 for q in copies if q != p and abs(q - p) > w)
        assert r[p] == expect, p
    others = np.setdiff1d(np.arange(128), copies)
    assert np.all(r[others] == 0)


def test_zero_key_counts_only_below_zero_threshold(oracle_mod):
    """A zero key has similarity 0 with everything (the design's reading)."""
    x = np.zeros((40, 8), np.float32)
    x[:, 0] = 1.0
    x[20] = 0.0
    keys = bf16(x)[None]
    r_pos = oracle_mod.count(keys, 0.5, 2)["r"][0]
    r_neg = oracle_mod.count(keys, -0.5, 2)["r"][0]
    assert r_pos[20] == 0 and r_neg[20] == 40 - 5
    assert r_pos[0] == 40 - 3 - 1          # j = 3..39 except the zero key at 20


@pytest.mark.parametrize("U,N,d,w,tau", [(2, 257, 64, 7, 0.1), (1, 200, 128, 32, 0.05),
                                         (1, 90, 64, 0, -0.05)])
def test_counts_against_float64_numpy_dense_matrix(oracle_mod, U, N, d, w, tau):
    """Eq. 2 from a float64 numpy matmul of normalised keys, windowed; pairs within
    1e-9 of tau would make the comparison fragile and are asserted absent."""
    keys = synth.random_keys(7, U, N, d)
    c = oracle_mod.count(keys, tau, w, band=0.01)
    t = float(np.float32(tau))
    kf = synth.bf16_bits_to_f32(keys).astype(np.float64)
    i, j = np.meshgrid(np.arange(N), np.arange(N), indexing="ij")
    far = np.abs(i - j) > w
    for u in range(U):
        kh = kf[u] / np.linalg.norm(kf[u], axis=1, keepdims=True)
        S = kh @ kh.T
        assert not np.any(far & (np.abs(S - t) < 1e-9))
        np.testing.assert_array_equal(c["r"][u], (far & (S > t)).sum(1))
        np.testing.assert_array_equal(c["r_lo"][u], (far & (S > t + 0.01)).sum(1))
        np.testing.assert_array_equal(c["r_hi"][u], (far & (S > t - 0.01)).sum(1))
    assert np.all(c["r_lo"] <= c["r"]) and np.all(c["r"] <= c["r_hi"])


def test_count_row_subset_matches_full(oracle_mod):
    keys = synth.random_keys(8, 2, 150, 64)
    full = oracle_mod.count(keys, 0.1, 5, band=0.02)
    rows = np.array([149, 0, 77, 3])
    sub = oracle_mod.count(keys, 0.1, 5, band=0.02, rows=rows)
    for k in full:
        np.testing.assert_array_equal(sub[k], full[k][:, rows])


# ---------------------------------------------------------------- selection (Eq. 3)

@pytest.mark.parametrize("seed", range(12))
def test_policy_matches_python_sort(oracle_mod, seed):
    """Brute force from the scores themselves: s_i = -r_i / N (Eq. 3), +inf on the
    protected regions (their maximum score, Sec. 3.2); Python's sorted() on
    (-s, position) and the first K kept."""
    rng = np.random.default_rng(seed)
    U = 3
    N = int(rng.integers(1, 300))
    n_sink, n_recent = int(rng.integers(0, 6)), int(rng.integers(0, 20))
    if seed % 4 == 3:
        n_recent = N + 3                                    # every position protected
    r = rng.integers(0, 6, size=(U, N)).astype(np.int32)   # many ties
    K = rng.integers(0, N + 1, size=U).astype(np.int32)
    p = oracle_mod.policy_select(r, K, n_sink, n_recent)
    prot = protected(N, n_sink, n_recent)
    for u in range(U):
        score = [float("inf") if prot[i] else -int(r[u, i]) / N for i in range(N)]
        order = sorted(range(N), key=lambda i: (-score[i], i))
        expect = np.zeros(N, np.uint8)
        expect[order[:K[u]]] = 1
        np.testing.assert_array_equal(p["mask"][u], expect)
        assert p["status"][u] == 0


def test_policy_invariants(oracle_mod):
    """|S| = K; protected positions kept when K covers them; every kept unprotected
    position has r no larger than any evicted one (Eq. 3: higher s kept)."""
    rng = np.random.default_rng(21)
    U, N, n_sink, n_recent = 4, 1000, 4, 64
    r = rng.integers(0, 40, size=(U, N)).astype(np.int32)
    K = np.array([68, 300, 700, 1000], np.int32)
    p = oracle_mod.policy_select(r, K, n_sink, n_recent)
    prot = protected(N, n_sink, n_recent)
    for u in range(U):
        S = p["mask"][u].astype(bool)
        assert S.sum() == K[u]
        assert np.all(S[prot])
        kept, ev = r[u][S & ~prot], r[u][~S & ~prot]
        if kept.size and ev.size:
            assert kept.max() <= ev.min()


def test_policy_budget_edges(oracle_mod):
    N = 100
    r = (N - np.arange(N, dtype=np.int32))[None].repeat(5, 0)   # fewer twins later
    K = np.array([0, N, 10, N + 1, -1], np.int32)
    p = oracle_mod.policy_select(r, K, 4, 64)
    assert p["mask"][0].sum() == 0 and p["status"][0] == 0
    assert p["mask"][1].sum() == N and p["status"][1] == 0
    # budget below the 68 protected positions: the lowest protected positions
    np.testing.assert_array_equal(np.flatnonzero(p["mask"][2]),
                                  np.r_[0:4, 36:42])
    for u in (3, 4):
        assert p["status"][u] == 1 and p["mask"][u].sum() == 0


def test_policy_of_planted_tiny_workload(oracle_mod):
    """On the tiny workload (tau 0.85, fp32 N(0,1) keys), only planted pairs exceed
    tau, so every planted key has r >= 1, every other key r = 0, and the policy
    evicts planted keys first."""
    w = synth.get("tiny")
    keys, truths = synth.keys(w)
    pol = oracle_mod.policy(keys, w.tau, budget=w.N - 40, window=synth.WINDOW,
                            n_sink=0, n_recent=0)
    t = truths[0]
    planted = np.unique(np.concatenate([t.pairs, t.exact_pairs]).ravel())
    r = pol["r"][0]
    assert np.all(r[np.setdiff1d(np.arange(w.N), planted)] == 0)
    assert np.all(r[planted] >= 1)
    assert np.all(pol["mask"][0][r == 0] == 1)
