"""Per-layer budgets (a pyramid schedule: more retained keys in lower layers, fewer in
higher ones, the total fixed) as inputs to the repair of Sec. 3.4.  The schedule is
input generation only; these tests pin its definition and check that the oracle's
repair keeps each unit's own budget.  None needs a GPU."""
import numpy as np
import pytest

from paper_2608_27128_gb300 import synth


@pytest.mark.parametrize("name", ["qwen", "llama"])
@pytest.mark.parametrize("ratio", [0.1, 0.3, 0.5, 0.7, 0.99])
def test_schedule_definition(name, ratio):
    w = synth.get(name)
    k = synth.pyramid_budgets(w, ratio)
    mean = synth.budget(w, ratio)
    lo = synth.N_SINK + synth.N_RECENT
    assert k.shape == (w.L,) and k.dtype == np.int64
    assert int(k.sum()) == w.L * mean                  # total budget unchanged
    assert np.all(k[:-1] >= k[1:])                     # shrinks with depth
    assert np.all((k >= min(lo, mean)) & (k <= w.N))
    # linear in the layer index up to rounding: second differences are within 1 + 1
    assert np.all(np.abs(np.diff(k, 2)) <= 2)
    # symmetric about the mean: first + last = 2 * mean up to rounding
    assert abs(int(k[0] + k[-1]) - 2 * mean) <= 2


def test_schedule_spread_and_caps():
    w = synth.get("qwen")
    k = synth.pyramid_budgets(w, 0.5)          # mean 8192, spread 0.5 fits
    assert k[0] == 12288 and k[-1] == 4096
    k = synth.pyramid_budgets(w, 0.3)          # mean 11469: the top end caps at N
    assert k[0] == w.N
    k = synth.pyramid_budgets(w, 0.5, spread=0.0)
    assert np.all(k == 8192)
    assert np.array_equal(synth.pyramid_budgets(synth.get("long"), 0.5), [65536])


@pytest.mark.parametrize("name,over,ratio", [
    ("qwen", {"L": 4, "H": 2, "N": 1024}, 0.3),
    ("llama", {"L": 6, "H": 2, "N": 700}, 0.5),
])
def test_masks_follow_schedule(name, over, ratio):
    w = synth.get(name, **over)
    k = synth.pyramid_budgets(w, ratio)
    S0 = synth.masks(w, ratio, schedule="pyramid")
    np.testing.assert_array_equal(S0.sum(1), np.repeat(k, w.H))
    # the protected regions the stand-in policies force stay retained
    assert np.all(S0[:, :synth.N_SINK] == 1) and np.all(S0[:, -synth.N_RECENT:] == 1)
    # a unit's mask depends only on its own (layer, head) and count
    sub = synth.masks(w, ratio, units=[(w.L - 1, 1)], schedule="pyramid")
    np.testing.assert_array_equal(sub[0], S0[(w.L - 1) * w.H + 1])
    with pytest.raises(ValueError):
        synth.masks(w, ratio, schedule="bogus")


def test_oracle_repair_keeps_each_units_budget(oracle_mod):
    w = synth.get("qwen", L=4, H=1, N=600)
    keys, _ = synth.keys(w)
    S0 = synth.masks(w, 0.3, schedule="pyramid")
    k = synth.pyramid_budgets(w, 0.3)
    assert k[0] == w.N                          # layer 0 keeps every key
    a = oracle_mod.audit(keys, S0, window=synth.WINDOW)
    r = oracle_mod.repair(a["b_ret"], S0, w.tau, budget=k.astype(np.int32))
    np.testing.assert_array_equal(r["status"], 0)
    np.testing.assert_array_equal(r["mask"].sum(1), k)
    # nothing evicted: no orphan, so no swap
    assert r["nswaps"][0] == 0 and not r["orphan"][0].any()
    # a budget that is not the unit's popcount is a data error for that unit only
    bad = k.astype(np.int32).copy()
    bad[2] += 1
    r2 = oracle_mod.repair(a["b_ret"], S0, w.tau, budget=bad)
    assert r2["status"][2] == 3 and r2["nswaps"][2] == -1
    np.testing.assert_array_equal(r2["status"][[0, 1, 3]], 0)
