"""Comparison of the CUDA path against the oracle, with the tie bands of the audit.

Similarities computed in fp32 from bf16 keys can differ from the fp64 oracle by a few
1e-6; scores must agree within TOL = 2e-3 absolute.  An integer result that a
similarity decides (a twin index, an orphan/donor flag, membership of the m swapped
items) must agree exactly unless the deciding similarity lies within BAND = 2*TOL of a
tie or of the threshold; those items are counted as excused, not as failures.
"""
from dataclasses import dataclass, field

import numpy as np

TOL = 2e-3
BAND = 2 * TOL


@dataclass
class Report:
    n_fail: int = 0
    n_excused: int = 0
    notes: list = field(default_factory=list)
    # largest |b_gpu - b_oracle| over rows whose twin agrees (the refined value)
    max_dev_same_twin: float = 0.0

    def fail(self, msg):
        self.n_fail += 1
        if len(self.notes) < 20:
            self.notes.append(msg)

    def add(self, other):
        self.n_fail += other.n_fail
        self.n_excused += other.n_excused
        self.max_dev_same_twin = max(self.max_dev_same_twin, other.max_dev_same_twin)
        self.notes += other.notes[: max(0, 20 - len(self.notes))]
        return self


def compare_best(b_gpu, t_gpu, b_orc, t_orc, b_orc2, sim, window, rows=None, S0=None,
                 what="b"):
    """One unit's (score, twin) against the oracle.

    b_gpu, t_gpu: GPU results for the rows in `rows` (all rows if None).
    b_orc, t_orc, b_orc2: oracle best, argmax and second best for the same rows.
    sim(i, j): oracle similarity, used to score a differing GPU twin.
    """
    rep = Report()
    rows = np.arange(len(b_orc)) if rows is None else np.asarray(rows)
    for k, i in enumerate(rows):
        bg, tg, bo, to, b2 = float(b_gpu[k]), int(t_gpu[k]), float(b_orc[k]), int(t_orc[k]), \
            float(b_orc2[k])
        if to < 0:
            if not (tg == -1 and bg == -1.0):
                rep.fail(f"{what} row {i}: oracle has no candidate, gpu ({bg}, {tg})")
            continue
        if abs(bg - bo) > TOL:
            rep.fail(f"{what} row {i}: score {bg} vs {bo}")
        if tg == to:
            rep.max_dev_same_twin = max(rep.max_dev_same_twin, abs(bg - bo))
            continue
        ok = (0 <= tg and abs(tg - i) > window and (S0 is None or S0[tg])
              and bo - b2 <= BAND and sim(i, tg) >= bo - BAND)
        if ok:
            rep.n_excused += 1
        else:
            rep.fail(f"{what} row {i}: twin {tg} vs {to} (best {bo}, second {b2})")
    return rep


def compare_repair(S0, S1_gpu, swaps_gpu, m_gpu, orc, b_orc, tau, n_sink=4, n_recent=64):
    """One unit's repair (S1, swap list) against the oracle run on fp64 b values.

    orc: oracle repair output for this unit (mask, swaps, nswaps, orphan, donor).
    Only positions the rule can move are ever excused: evicted positions (orphan
    candidates) and retained positions outside the protected sink and recent regions
    (donor candidates, Sec. 3.4).  A protected retained position that changes is a
    failure whatever its b.
    """
    rep = Report()
    N = len(S0)
    tau_f = float(np.float32(tau))
    m_orc = int(orc["nswaps"])
    pos = np.arange(N)
    prot = (pos < n_sink) | (pos >= N - n_recent)
    cand_o = S0 == 0
    cand_d = (S0 != 0) & ~prot
    # an orphan or donor flag that b within BAND of tau may flip
    near_tau = (cand_o | cand_d) & (np.abs(b_orc - tau_f) <= BAND)
    excusable = near_tau.copy()
    if m_orc > 0:
        so = orc["swaps"][:m_orc, 1]
        sd = orc["swaps"][:m_orc, 0]
        cut_o, cut_d = b_orc[so[-1]], b_orc[sd[-1]]
        excusable |= cand_o & (np.abs(b_orc - cut_o) <= BAND)
        excusable |= cand_d & (np.abs(b_orc - cut_d) <= BAND)
    if m_gpu != m_orc:
        flips = int(near_tau.sum())
        if abs(m_gpu - m_orc) > flips:
            rep.fail(f"m {m_gpu} vs {m_orc}")
        else:
            rep.n_excused += 1
            # the swaps past the shorter list follow from the flipped flags: the next
            # donors and orphans in severity order on the side that has more
            longer = swaps_gpu[m_orc:m_gpu] if m_gpu > m_orc else orc["swaps"][m_gpu:m_orc]
            for d_, o_ in np.asarray(longer).reshape(-1, 2):
                excusable[d_] |= bool(cand_d[d_])
                excusable[o_] |= bool(cand_o[o_])
    diff = np.flatnonzero(S1_gpu != orc["mask"])
    for i in diff:
        if excusable[i]:
            rep.n_excused += 1
        else:
            rep.fail(f"S1[{i}] {S1_gpu[i]} vs {orc['mask'][i]} (b {b_orc[i]})")
    m = min(m_gpu, m_orc)
    for k in range(m):
        for side in (0, 1):
            g, o = int(swaps_gpu[k, side]), int(orc["swaps"][k, side])
            if g == o:
                continue
            if (excusable[g] and excusable[o]) or abs(b_orc[g] - b_orc[o]) <= BAND:
                rep.n_excused += 1
            else:
                rep.fail(f"swap {k} side {side}: {g} vs {o}")
    return rep
