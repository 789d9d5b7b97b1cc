"""Runs the CUDA path through the C ABI and scores it against the oracle."""
import json
import os

import numpy as np
import torch

import oracle
from comparator import Report, compare_best, compare_repair
from paper_2608_27128_gb300 import twinkv as tk


def device():
    return torch.device("cuda:0")


def keys_tensor(keys: np.ndarray, L: int, H: int) -> torch.Tensor:
    """bf16 bit patterns (uint16) or float32 [U,N,d] -> CUDA tensor [L,H,N,d]."""
    U, N, d = keys.shape
    if keys.dtype == np.float32:
        t = torch.from_numpy(keys.reshape(L, H, N, d).copy())
    else:
        t = torch.from_numpy(keys.view(np.int16).reshape(L, H, N, d).copy()).view(torch.bfloat16)
    return t.to(device())


def redundancy_vs_oracle(keys, L, H, window, rows=None, symmetric=False) -> Report:
    U, N, d = keys.shape
    call = tk.twinkv_redundancy_symmetric if symmetric else tk.twinkv_redundancy
    score, twin = call(keys_tensor(keys, L, H), window)
    torch.cuda.synchronize()
    s = score.reshape(U, N).cpu().numpy()
    t = twin.reshape(U, N).cpu().numpy()
    a = oracle.audit(keys, window=window, rows=rows)
    rep = Report()
    sel = np.arange(N) if rows is None else np.asarray(rows)
    for u in range(U):
        rep.add(compare_best(s[u, sel], t[u, sel], a["b_all"][u], a["t_all"][u], a["b_all2"][u],
                             lambda i, j: oracle.sim(keys, u, i, j), window, rows=sel,
                             what=f"u{u} all"))
    return rep, s, t


def repair_vs_oracle(keys, S0, L, H, window, tau, n_sink=4, n_recent=64, want_all=True,
                     stream=None):
    """Full repair call; returns (report, host outputs).  Also runs the bit-exact split
    check: the oracle's selection on the GPU's own b_ret must give identical S1,
    swap lists and counts."""
    U, N, d = keys.shape
    mask_t = torch.from_numpy(S0.reshape(L, H, N).copy()).to(device())
    budget = torch.from_numpy(S0.sum(1).astype(np.int32)).to(device())
    out = tk.twinkv_repair(keys_tensor(keys, L, H), mask_t, budget, threshold=tau,
                           window=window, n_sink=n_sink, n_recent=n_recent, want_all=want_all,
                           stream=stream)
    torch.cuda.synchronize()
    h = {k: v.cpu().numpy() for k, v in out.items()}
    for k in ("mask", "score_ret", "twin_ret", "score_all", "twin_all"):
        if k in h:
            h[k] = h[k].reshape(U, N)
    a = oracle.audit(keys, S0, window=window)
    rep = Report()
    for u in range(U):
        sim = (lambda uu: (lambda i, j: oracle.sim(keys, uu, i, j)))(u)
        rep.add(compare_best(h["score_ret"][u], h["twin_ret"][u], a["b_ret"][u], a["t_ret"][u],
                             a["b_ret2"][u], sim, window, S0=S0[u], what=f"u{u} ret"))
        if want_all:
            rep.add(compare_best(h["score_all"][u], h["twin_all"][u], a["b_all"][u],
                                 a["t_all"][u], a["b_all2"][u], sim, window, what=f"u{u} all"))
    r = oracle.repair(a["b_ret"], S0, tau, n_sink=n_sink, n_recent=n_recent,
                      budget=S0.sum(1))
    for u in range(U):
        ou = {k: r[k][u] for k in r}
        rep.add(compare_repair(S0[u], h["mask"][u], h["swaps"][u], int(h["nswaps"][u]), ou,
                               a["b_ret"][u], tau, n_sink, n_recent))
    split_check(h, S0, tau, n_sink, n_recent)
    assert np.all(h["status"] == 0)
    return rep, h, a, r


def split_check(h, S0, tau, n_sink, n_recent, budget=None):
    """The oracle's repair fed the GPU's own fp64 b_ret must reproduce S1, the swap
    lists and their lengths bit for bit."""
    U, N = S0.shape
    rf = oracle.repair(h["score_ret"].reshape(U, N), S0, tau, n_sink=n_sink,
                           n_recent=n_recent,
                           budget=S0.sum(1) if budget is None else budget)
    np.testing.assert_array_equal(h["nswaps"], rf["nswaps"])
    np.testing.assert_array_equal(h["mask"].reshape(U, N), rf["mask"])
    for u in range(U):
        m = int(rf["nswaps"][u])
        if m > 0:
            np.testing.assert_array_equal(h["swaps"][u, :m], rf["swaps"][u, :m])


def record(**fields):
    """One parity record per checked configuration (failures, excused items by kind,
    rows checked), printed and, when TWINKV_PARITY_LOG names a file, appended to it as
    a JSON line."""
    line = json.dumps(fields, sort_keys=True, default=float)
    print("parity", line)
    path = os.environ.get("TWINKV_PARITY_LOG")
    if path:
        with open(path, "a") as f:
            f.write(line + "\n")


def sampled_rows(keys, S0, h, rows_per_unit, seed, window, units=None):
    """b_i(S0), b_i(all) and their twins of `rows_per_unit` random rows of every unit
    (different rows in each unit) against the oracle.  Returns one Report per quantity
    and the number of rows checked."""
    U, N, _ = keys.shape
    rng = np.random.default_rng(seed)
    rep_ret, rep_all = Report(), Report()
    n_rows = 0
    for u in (range(U) if units is None else units):
        rows = np.sort(rng.choice(N, size=min(rows_per_unit, N), replace=False))
        a = oracle.audit(keys[u:u + 1], S0[u:u + 1], window=window, rows=rows)
        sim = (lambda uu: (lambda i, j: oracle.sim(keys, uu, i, j)))(u)
        rep_ret.add(compare_best(h["score_ret"][u, rows], h["twin_ret"][u, rows],
                                 a["b_ret"][0], a["t_ret"][0], a["b_ret2"][0], sim, window,
                                 rows=rows, S0=S0[u], what=f"u{u} ret"))
        rep_all.add(compare_best(h["score_all"][u, rows], h["twin_all"][u, rows],
                                 a["b_all"][0], a["t_all"][0], a["b_all2"][0], sim, window,
                                 rows=rows, what=f"u{u} all"))
        n_rows += rows.size
    return rep_ret, rep_all, n_rows
