"""Seeded synthetic KV-cache workloads for the TwinKV audit and repair pass.

This module only draws inputs: keys (as bf16 bit patterns, or float32 for the tiny
case), retained masks from stand-in eviction policies, and the ground truth planted
into them.  It holds none of the method's arithmetic (no similarity, no maxima, no
orphan/donor rule), so the CUDA path and the reference oracle can both be fed from
it without sharing any of the computation they are compared on.

Every unit (one layer and KV head) is drawn from its own generator,
``numpy.random.default_rng([seed, layer, head, stream])``, so a unit can be
regenerated alone and sub-sampled workloads keep the values of the full ones.

The five workloads stand in for the paper's KV caches (Sec. 3.1 problem setup; Sec. 4
models Qwen3-4B and Llama-3.2-1B, thresholds 0.85 and 0.90; wrapped policies
StreamingLLM / SnapKV-like / heavy-tailed scores; sink 4 and recent 64 protected
regions of Sec. 3.2).  No model, dataset or checkpoint is used.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

WINDOW = 32      # local window w (Sec. 3.2 default)
N_SINK = 4       # protected leading sink tokens (Sec. 3.2)
N_RECENT = 64    # protected trailing recent window (Sec. 3.2)


@dataclass(frozen=True)
class Workload:
    name: str
    seed: int
    L: int
    H: int
    N: int
    d: int
    tau: float
    ratios: tuple
    fp32_keys: bool = False
    description: str = ""

    @property
    def units(self) -> int:
        return self.L * self.H


WORKLOADS = {
    "tiny": Workload(
        "tiny", 0, 1, 1, 512, 64, 0.85, (0.5,), fp32_keys=True,
        description="1x1x512x64 fp32 N(0,1); 64 near-duplicate pairs (sigma 0.01) and 8 "
                    "exact duplicates, distance > w; uniform-random policy scores"),
    "llama": Workload(
        "llama", 2, 16, 8, 8192, 64, 0.90, (0.3, 0.5, 0.7),
        description="Llama-3.2-1B cache shape 16x8x8192x64 bf16 N(0,1), 4 outlier "
                    "channels x8 per head; 10% copies (sigma 0.02) at distance > w; "
                    "Pareto(1.5) policy scores + sinks + recent"),
    "qwen": Workload(
        "qwen", 3, 36, 8, 16384, 128, 0.85, (0.3, 0.5, 0.7),
        description="Qwen3-4B cache shape 36x8x16384x128 bf16 N(0,1), RoPE-like rotation "
                    "per position (theta 1e6); 15% copies (sigma 0.02) of the rotated "
                    "key, distance uniform in 1..N-1; SnapKV-like policy scores"),
    "retrieval": Workload(
        "retrieval", 4, 36, 8, 32768, 128, 0.85, (0.3,),
        description="36x8x32768x128 bf16: 90% filler from 256 templates + N(0,0.01^2), 32 "
                    "unique needles, rest unique; 4 sinks + last positions retained"),
    "long": Workload(
        "long", 5, 1, 8, 131072, 128, 0.85, (0.5,),
        description="1x8x131072x128 bf16 N(0,1), 5% copies (sigma 0.02) at distance > w; "
                    "uniform-random policy scores + sinks + recent"),
}


def get(name: str, **overrides) -> Workload:
    """A workload by name, optionally with a smaller L, H or N (same recipe)."""
    w = WORKLOADS[name]
    if overrides:
        w = Workload(**{**w.__dict__, **overrides})
    return w


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (nearest, ties to even) and return the 16-bit patterns."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = b + np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1))
    return (rounded >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(h: np.ndarray) -> np.ndarray:
    return (np.asarray(h, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _rng(w: Workload, layer: int, head: int, stream: int) -> np.random.Generator:
    return np.random.default_rng([w.seed, layer, head, stream])


def plant_pairs(rng, N: int, n_pairs: int, dmin: int, dmax: int,
                forbidden=None) -> np.ndarray:
    """Disjoint (source, copy) position pairs with copy = source + delta.

    delta is drawn uniformly from [dmin, dmax], then the source uniformly from the
    positions that keep the copy inside [0, N).  Every position is used at most once
    (no chains), and positions in ``forbidden`` are never used.
    """
    used = np.zeros(N, dtype=bool)
    if forbidden is not None:
        used[np.asarray(forbidden, dtype=np.int64)] = True
    dmax = min(dmax, N - 1)
    pairs = []
    tries = 0
    while len(pairs) < n_pairs:
        batch = max(64, 2 * (n_pairs - len(pairs)))
        deltas = rng.integers(dmin, dmax + 1, size=batch)
        u = rng.random(batch)
        for delta, r in zip(deltas.tolist(), u.tolist()):
            s = int(r * (N - delta))
            c = s + delta
            if not used[s] and not used[c]:
                used[s] = used[c] = True
                pairs.append((s, c))
                if len(pairs) == n_pairs:
                    break
        tries += batch
        if tries > 200 * n_pairs + 10000:
            raise RuntimeError("could not place the planted pairs")
    return np.asarray(pairs, dtype=np.int64).reshape(-1, 2)


def _rope(x: np.ndarray, base: float = 1.0e6) -> np.ndarray:
    """Rotate dimension pairs (t, t + d/2) of row p by angle p * base**(-2t/d)."""
    N, d = x.shape
    half = d // 2
    theta = base ** (-2.0 * np.arange(half, dtype=np.float64) / d)
    ang = np.arange(N, dtype=np.float64)[:, None] * theta[None, :]
    c = np.cos(ang).astype(np.float32)
    s = np.sin(ang).astype(np.float32)
    a, b = x[:, :half], x[:, half:]
    return np.concatenate([a * c - b * s, a * s + b * c], axis=1)


@dataclass
class UnitTruth:
    """What was planted into one unit, for the tests."""
    pairs: np.ndarray = field(default_factory=lambda: np.zeros((0, 2), np.int64))
    exact_pairs: np.ndarray = field(default_factory=lambda: np.zeros((0, 2), np.int64))
    needles: np.ndarray = field(default_factory=lambda: np.zeros(0, np.int64))


def unit_keys(w: Workload, layer: int, head: int):
    """Keys of one unit as float32 [N, d] (exact bf16 values unless w.fp32_keys)."""
    rng = _rng(w, layer, head, 0)
    N, d = w.N, w.d
    truth = UnitTruth()
    if w.name == "tiny":
        x = rng.standard_normal((N, d), dtype=np.float32)
        pairs = plant_pairs(rng, N, 72, WINDOW + 1, N - 1)
        near, exact = pairs[:64], pairs[64:]
        x[near[:, 1]] = x[near[:, 0]] + 0.01 * rng.standard_normal((64, d), dtype=np.float32)
        x[exact[:, 1]] = x[exact[:, 0]]
        truth.pairs, truth.exact_pairs = near, exact
        return x, truth
    if w.name == "llama":
        x = rng.standard_normal((N, d), dtype=np.float32)
        ch = rng.choice(d, size=4, replace=False)
        x[:, ch] *= 8.0
        n = int(round(0.10 * N))
        pairs = plant_pairs(rng, N, n, WINDOW + 1, N - 1)
        x[pairs[:, 1]] = x[pairs[:, 0]] + 0.02 * rng.standard_normal((n, d), dtype=np.float32)
        truth.pairs = pairs
    elif w.name == "qwen":
        x = _rope(rng.standard_normal((N, d), dtype=np.float32))
        n = int(round(0.15 * N))
        pairs = plant_pairs(rng, N, n, 1, N - 1)
        x[pairs[:, 1]] = x[pairs[:, 0]] + 0.02 * rng.standard_normal((n, d), dtype=np.float32)
        truth.pairs = pairs
    elif w.name == "retrieval":
        templates = rng.standard_normal((256, d), dtype=np.float32)
        needles = np.sort(rng.choice(N, size=32, replace=False))
        rest = np.setdiff1d(np.arange(N), needles)
        filler = rng.choice(rest, size=int(round(0.90 * N)), replace=False)
        x = rng.standard_normal((N, d), dtype=np.float32)   # needles and unique keys
        tid = rng.integers(0, 256, size=filler.size)
        x[filler] = templates[tid] + 0.01 * rng.standard_normal((filler.size, d),
                                                                 dtype=np.float32)
        truth.needles = needles
    elif w.name == "long":
        x = rng.standard_normal((N, d), dtype=np.float32)
        n = int(round(0.05 * N))
        pairs = plant_pairs(rng, N, n, WINDOW + 1, N - 1)
        x[pairs[:, 1]] = x[pairs[:, 0]] + 0.02 * rng.standard_normal((n, d), dtype=np.float32)
        truth.pairs = pairs
    else:
        raise KeyError(w.name)
    return bf16_bits_to_f32(f32_to_bf16_bits(x)), truth


def keys(w: Workload, units=None):
    """Keys for all units (or the listed (layer, head) units).

    Returns (keys, truths): float32 [U, N, d] for the fp32 workload, otherwise uint16
    bf16 bit patterns [U, N, d]; truths is a list of UnitTruth.
    """
    if units is None:
        units = [(l, h) for l in range(w.L) for h in range(w.H)]
    dtype = np.float32 if w.fp32_keys else np.uint16
    out = np.empty((len(units), w.N, w.d), dtype=dtype)
    truths = []
    for k, (l, h) in enumerate(units):
        x, t = unit_keys(w, l, h)
        out[k] = x if w.fp32_keys else f32_to_bf16_bits(x)
        truths.append(t)
    return out, truths


def budget(w: Workload, ratio: float) -> int:
    """Retained count.  Sec. 3.1: |S| = ceil((1 - rho) n).  The retrieval workload is
    built explicitly as 4 sinks plus the last positions with ceil(0.3 N) retained."""
    if w.name == "retrieval":
        return int(math.ceil(0.3 * w.N))
    return int(math.ceil((1.0 - ratio) * w.N - 1e-9))


def pyramid_budgets(w: Workload, ratio: float, spread: float = 0.5) -> np.ndarray:
    """Per-layer retained counts that shrink linearly with depth, as layer-wise budget
    schedules do (the policies the repair wraps may give each layer its own budget,
    Sec. 4.1): layer l gets about mean * (1 + s * (1 - 2 l / (L - 1))), i.e.
    (1 + s) * mean at the first layer and (1 - s) * mean at the last, with s = spread
    reduced where needed so that both ends stay within [n_sink + n_recent, N].  The
    counts are integers summing to exactly L * mean: the floors, plus one for the
    layers with the largest fractional parts (lower layer first on ties).  Every head
    of a layer shares the layer's count.  Returns int64 [L]."""
    mean = budget(w, ratio)
    L, N = w.L, w.N
    if L == 1:
        return np.array([mean], np.int64)
    lo = min(N_SINK + N_RECENT, N)
    s = max(0.0, min(spread, (N - mean) / mean, (mean - lo) / mean))
    raw = np.array([mean * (1.0 + s * (1.0 - 2.0 * l / (L - 1))) for l in range(L)])
    k = np.floor(raw).astype(np.int64)
    rest = int(L * mean - k.sum())          # 0 <= rest < L: the schedule sums to L * mean
    order = np.argsort(-(raw - k), kind="stable")
    k[order[:rest]] += 1
    return np.clip(k, lo, N)


def _top_k(scores: np.ndarray, forced: np.ndarray, K: int) -> np.ndarray:
    """Retain every forced position, then the highest scores (lower index on ties)."""
    N = scores.size
    mask = np.zeros(N, dtype=np.uint8)
    mask[forced] = 1
    need = K - int(mask.sum())
    if need > 0:
        cand = np.flatnonzero(mask == 0)
        order = np.argsort(-scores[cand], kind="stable")
        mask[cand[order[:need]]] = 1
    return mask


def unit_mask(w: Workload, layer: int, head: int, ratio: float, K: int | None = None) -> np.ndarray:
    """Retained set S0 of one unit from the workload's stand-in policy (K retained;
    default the workload's uniform budget for `ratio`)."""
    N = w.N
    K = budget(w, ratio) if K is None else int(K)
    rng = _rng(w, layer, head, 1)
    protected = np.concatenate([np.arange(min(N_SINK, N)),
                                np.arange(max(N - N_RECENT, 0), N)])
    if w.name == "tiny":
        return _top_k(rng.random(N), np.zeros(0, np.int64), K)
    if w.name == "llama":
        return _top_k(rng.pareto(1.5, size=N) + 1.0, protected, K)
    if w.name == "qwen":
        logits = rng.standard_normal((32, N), dtype=np.float32)
        logits -= logits.max(axis=1, keepdims=True)
        p = np.exp(logits)
        p /= p.sum(axis=1, keepdims=True)
        forced = np.unique(np.concatenate([protected, np.arange(max(N - 32, 0), N)]))
        return _top_k(p.sum(axis=0), forced, K)
    if w.name == "retrieval":
        mask = np.zeros(N, dtype=np.uint8)
        mask[:N_SINK] = 1
        mask[N - (K - N_SINK):] = 1
        return mask
    if w.name == "long":
        return _top_k(rng.random(N), protected, K)
    raise KeyError(w.name)


def masks(w: Workload, ratio: float, units=None, schedule: str = "uniform") -> np.ndarray:
    """Retained masks [U, N] of the given units (all by default).  schedule "uniform"
    gives every unit the same budget; "pyramid" gives each layer its count from
    pyramid_budgets.  The retrieval workload keeps its explicit construction."""
    if units is None:
        units = [(l, h) for l in range(w.L) for h in range(w.H)]
    if schedule == "uniform":
        ks = {l: None for (l, _) in units}
    elif schedule == "pyramid":
        pb = pyramid_budgets(w, ratio)
        ks = {l: int(pb[l]) for (l, _) in units}
    else:
        raise ValueError(schedule)
    return np.stack([unit_mask(w, l, h, ratio, ks[l]) for (l, h) in units]).astype(np.uint8)


def random_keys(seed: int, U: int, N: int, d: int, scale: float = 1.0) -> np.ndarray:
    """Plain N(0, scale^2) keys as bf16 bits [U, N, d] (for shape sweeps)."""
    rng = np.random.default_rng([seed, U, N, d])
    return f32_to_bf16_bits(scale * rng.standard_normal((U, N, d), dtype=np.float32))


def random_masks(seed: int, U: int, N: int, K: int) -> np.ndarray:
    """Uniformly random retained sets with exactly K members per unit."""
    rng = np.random.default_rng([seed, U, N, K, 7])
    out = np.zeros((U, N), np.uint8)
    for u in range(U):
        out[u, rng.permutation(N)[:K]] = 1
    return out
