"""The counting rule behind the base solve's row table, on the CPU.

A row (capacity c, demand lambda, at most M replicas) covers a threshold t with
its smallest n such that f(n) = min(1, RN(RN(n c) / lambda)) >= t (Section 3,
Eqs. 2 and 4; a critical class covers max(t, delta)). The GPU solve does not
evaluate f for every (row, threshold): it counts how many of the row's own
values f(n0) <= ... <= f(len) lie below t, where n0 is the first n with
f(n) >= max(delta, the smallest positive float) and len the first n with
f(n) = 1 (else M), and takes n0 plus that count (no cover when every value is
below t). This checks that rule against brute force with the oracle's
fulfilment arithmetic, at thresholds taken from the row's own values, their
float neighbours and elsewhere in (0, 1].
"""

import numpy as np

import oracle

DMIN = float(np.nextafter(np.float32(0.0), np.float32(1.0)))  # smallest positive float


def _brute(t, c, lam, M):
    for n in range(1, M + 1):
        if oracle.fulfil(n, c, lam) >= t:
            return n
    return 0


def _counted(t, c, lam, M, delta):
    n0 = _brute(max(delta, DMIN), c, lam, M)
    if n0 == 0:
        return 0
    ns = _brute(1.0, c, lam, M)
    last = ns if ns else M
    vals = [oracle.fulfil(n, c, lam) for n in range(n0, last + 1)]
    q = sum(v < t for v in vals)
    return n0 + q if q < len(vals) else 0


def test_cover_by_counting_own_values_equals_brute_force():
    rng = np.random.default_rng(20)
    checked = 0
    for _ in range(300):
        M = int(rng.integers(1, 40))
        lam = float(np.float32(rng.uniform(0.5, 30.0)))
        c = float(np.float32(lam * rng.uniform(0.01, 1.5)))
        if rng.random() < 0.1:
            c = 0.0
        delta = 0.0 if rng.random() < 0.5 else float(np.float32(rng.uniform(0.0, 1.0)))
        own = [oracle.fulfil(n, c, lam) for n in range(1, M + 1)]
        ts = set()
        for v in own + [float(np.float32(rng.uniform(0, 1))) for _ in range(5)]:
            v32 = np.float32(v)
            for x in (v32, np.nextafter(v32, np.float32(2)), np.nextafter(v32, np.float32(0))):
                if 0.0 < float(x) <= 1.0:
                    ts.add(float(x))
        for t in ts:
            tc = max(t, delta)  # a critical class covers max(t, delta)
            assert _counted(tc, c, lam, M, delta) == _brute(tc, c, lam, M), (t, c, lam, M, delta)
            checked += 1
    assert checked > 5000


def test_row_length_bound():
    """A row holds at most min(M, n_sat) values, n_sat the first n with f(n) = 1.
    The library sizes the preparation's shared thresholds by the bound
    n_sat <= floor(lambda / c (1 + 2^-18)) + 3, which rests on every n >=
    lambda / c (1 + 2^-23) reaching f(n) = 1 (two RN steps lose at most 2^-24
    each). Both are checked with the oracle's fulfilment arithmetic, on ratios
    lambda / c spread over many decades and on ratios at and next to integers,
    where the rounding decides."""
    rng = np.random.default_rng(21)
    cases = []
    for _ in range(1500):
        lam = float(np.float32(10.0 ** rng.uniform(-2, 4)))
        c = float(np.float32(lam / 10.0 ** rng.uniform(-3, 4)))
        cases.append((c, lam))
    for _ in range(1500):
        lam = float(np.float32(10.0 ** rng.uniform(-2, 4)))
        k = int(rng.integers(1, 5000))
        c32 = np.float32(lam / k)
        for c in (c32, np.nextafter(c32, np.float32(0)), np.nextafter(c32, np.float32(np.inf))):
            cases.append((float(c), lam))
    for c, lam in cases:
        if c <= 0.0:
            continue
        n_tight = int(np.ceil(lam / c * (1.0 + 2.0 ** -23)))
        n_bound = int(lam / c * (1.0 + 2.0 ** -18)) + 3
        assert n_tight <= n_bound
        if n_tight > 40000:  # beyond any replica cap (M <= 32767)
            continue
        assert oracle.fulfil(n_tight, c, lam) == 1.0, (c, lam, n_tight)
        if n_tight > 1:  # and the first such n is not far below it
            assert oracle.fulfil(max(1, int(lam / c * (1.0 - 2.0 ** -20)) - 1), c, lam) < 1.0, (c, lam)
