"""Brute-force allocation by enumeration (pure Python, tiny instances only).

Independent of the C oracle: it enumerates every allocation of Section 3,
Eqs. 1-5 (per class: nothing, or one SLO-feasible cell with 1 <= n <= G/tau
replicas), keeps those within the GPU budget G, and maximises the minimum
fulfilment r_i = min(lambda_i, n c) / lambda_i over classes. Fulfilment is
computed in IEEE float32 (numpy scalars), one rounding per operation.
"""

from __future__ import annotations

import itertools

import numpy as np

TP = (1, 2, 4, 8)


def f32_fulfil(n, c, lam):
    served = np.float32(n) * np.float32(c)
    r = np.float32(served / np.float32(lam))
    return np.float32(1.0) if r > np.float32(1.0) else r


def options(K, B, G, cap, tail, demand, slo):
    cap = np.asarray(cap, np.float32).reshape(K, 4, B)
    tail = np.asarray(tail, np.float32).reshape(K, 4, B)
    out = []
    for i in range(K):
        opts = []
        for j, tau in enumerate(TP):
            for b in range(B):
                if not tail[i, j, b] <= slo[i]:
                    continue
                for n in range(1, G // tau + 1):
                    f = f32_fulfil(n, cap[i, j, b], demand[i])
                    opts.append((n * tau, j, n, float(cap[i, j, b]), b, float(f)))
        out.append(opts)
    return out


def _floor_ok(combo, floor):
    """Tier 1: every critical class (floor > 0) is served at r_i >= floor_i."""
    if floor is None:
        return True
    return all(d <= 0 or (c is not None and c[5] >= np.float32(d)) for c, d in zip(combo, floor))


def best_max_min(K, B, G, cap, tail, demand, slo, floor=None):
    """Largest min_i r_i over every allocation within G that meets the critical
    floors (0 if a class must be empty, or if no allocation meets the floors)."""
    opts = options(K, B, G, cap, tail, demand, slo)
    best = 0.0
    for combo in itertools.product(*[[None] + o for o in opts]):
        cost = sum(c[0] for c in combo if c is not None)
        if cost > G or not _floor_ok(combo, floor):
            continue
        if any(c is None for c in combo):
            val = 0.0
        else:
            val = min(c[5] for c in combo)
        best = max(best, val)
    return best


def floors_met(K, B, G, cap, tail, demand, slo, floor):
    """Whether some allocation within G serves every critical class at its floor."""
    opts = options(K, B, G, cap, tail, demand, slo)
    for combo in itertools.product(*[[None] + o for o in opts]):
        if sum(c[0] for c in combo if c is not None) <= G and _floor_ok(combo, floor):
            return True
    return False


def choice_at(K, B, G, cap, tail, demand, slo, t, floor=None):
    """Per class, the preferred option covering max(t, floor_i): (cost, TP, n,
    -capacity, bin) minimal."""
    opts = options(K, B, G, cap, tail, demand, slo)
    res = []
    for i, o in enumerate(opts):
        ti = t if floor is None else max(np.float32(t), np.float32(floor[i]))
        cov = [x for x in o if x[5] >= ti]
        if not cov:
            res.append(None)
            continue
        res.append(min(cov, key=lambda x: (x[0], x[1], x[2], -x[3], x[4])))
    return res


def goodput_fx(n, c, lam):
    """rint(min(lambda, n c) 2^20): a class's served goodput (Eqs. 2, 4) in 2^-20 req/s."""
    served = np.float32(n) * np.float32(c)
    x = served if served < np.float32(lam) else np.float32(lam)
    return int(np.rint(np.float64(x) * 2.0**20))


def lexicographic(K, B, G, cap, tail, demand, slo, floor=None):
    """The four tiers of Section 3 by enumeration: among allocations within G,
    those meeting the critical floors when any does (else nothing is
    allocated), then the largest min_i r_i, then the most goodput, then the
    fewest GPUs, then class by class the option preferred by the tie rules
    (none first, then lower TP, fewer replicas, larger capacity, lower bin).
    Returns (t*, goodput_fx, gpus, per-class (tp, n, bin))."""
    opts = options(K, B, G, cap, tail, demand, slo)
    combos = [c for c in itertools.product(*[[None] + o for o in opts])
              if sum(x[0] for x in c if x is not None) <= G]
    empty = (0.0, 0, 0, [(0, 0, -1)] * K)
    if floor is not None and any(d > 0 for d in floor):
        combos = [c for c in combos if _floor_ok(c, floor)]
        if not combos:
            return empty

    def minr(c):
        return 0.0 if any(x is None for x in c) else min(x[5] for x in c)

    t = max(minr(c) for c in combos)
    pool = [c for c in combos if minr(c) == t]

    def gp(c):
        return sum(goodput_fx(x[2], x[3], demand[i]) for i, x in enumerate(c) if x is not None)

    def gpus(c):
        return sum(x[0] for x in c if x is not None)

    def tie(c):
        return tuple((-1,) if x is None else (x[1], x[2], -x[3], x[4]) for x in c)

    best = min(pool, key=lambda c: (-gp(c), gpus(c), tie(c)))
    choice = [(0, 0, -1) if x is None else (TP[x[1]], x[2], x[4]) for x in best]
    return float(t), gp(best), gpus(best), choice
