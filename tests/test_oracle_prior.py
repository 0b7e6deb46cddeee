"""Pins of the oracle's interval refit (Section 4.1's structural prior, read as
capacity and binding tail nondecreasing in the load bin within a (class, TP)
row) and of the scores computed under it.

The paper gives no formula for its prior, so these are the properties that
fix the reading: a refit never widens an interval, the measured cell holds its
values, other rows and (under the revealed-only prior) other cells do not
move, a truth table that is monotone in the load bin stays inside every
interval whatever cells of it are measured, and measuring every cell
collapses every interval. Scores under the monotone prior keep the score
invariants and are never below the revealed-only prior's (each scenario's
gap only narrows further); scenarios equal brute force on the refit bounds.
"""

import dataclasses

import numpy as np
import pytest

import brute
from paper_2608_19659_gb300 import workloads

MONO = 1


def _random_bounds(rng, K, B, monotone_truth=False):
    shape = (K, 4, B)
    if monotone_truth:
        cap_t = np.cumsum(rng.uniform(0.0, 0.5, shape), axis=2) + 0.2
        tail_t = np.cumsum(rng.uniform(0.0, 4.0, shape), axis=2) + 5.0
    else:
        cap_t = rng.uniform(0.2, 3.0, shape)
        tail_t = rng.uniform(5.0, 40.0, shape)
    cw = rng.uniform(0.0, 1.0, (2,) + shape)
    tw = rng.uniform(0.0, 8.0, (2,) + shape)
    f = np.float32
    truth = (cap_t.astype(f).reshape(-1), tail_t.astype(f).reshape(-1))
    b = [(cap_t - cw[0]).clip(0.0).astype(f), (cap_t + cw[1]).astype(f),
         (tail_t - tw[0]).clip(0.0).astype(f), (tail_t + tw[1]).astype(f)]
    return [x.reshape(-1) for x in b], truth


@pytest.mark.parametrize("seed", range(20))
def test_refit_never_widens_and_holds_the_measurement(oracle_lib, seed):
    rng = np.random.default_rng(seed)
    K, B = 2, 6
    bounds, _ = _random_bounds(rng, K, B)
    prob = oracle_lib.Problem(K, B, 8, [1.0, 2.0], [20.0, 30.0], prior=MONO)
    for _ in range(6):
        cell = int(rng.integers(K * 4 * B))
        # measured values anywhere, also outside the cell's own interval
        c = np.float32(rng.uniform(0.0, 4.0))
        ell = np.float32(rng.uniform(0.0, 50.0))
        new = oracle_lib.refit(prob, cell, c, ell, *bounds)
        clo, chi, tlo, thi = new
        assert clo[cell] == chi[cell] == c and tlo[cell] == thi[cell] == ell
        other = np.arange(K * 4 * B) != cell
        assert np.all(clo[other] >= bounds[0][other]) and np.all(chi[other] <= bounds[1][other])
        assert np.all(tlo[other] >= bounds[2][other]) and np.all(thi[other] <= bounds[3][other])
        assert np.all(clo <= chi) and np.all(tlo <= thi)
        row = cell // B
        moved = np.nonzero([not all(new[a][x] == bounds[a][x] for a in range(4)) for x in range(K * 4 * B)])[0]
        assert np.all(moved // B == row)  # only the measured cell's row moves
        # lower-load bins only lose upper bounds, higher-load bins only gain lower bounds
        be = cell % B
        for x in moved:
            if x == cell:
                continue
            if x % B > be:
                assert chi[x] == bounds[1][x] and thi[x] == bounds[3][x]
            else:
                assert clo[x] == bounds[0][x] and tlo[x] == bounds[2][x]
        bounds = new


@pytest.mark.parametrize("seed", range(20))
def test_monotone_truth_stays_inside_every_interval(oracle_lib, seed):
    """Soundness of the prior: measuring cells of a truth that is nondecreasing in
    the load bin never cuts that truth out of any interval; measuring every cell
    collapses every interval onto it."""
    rng = np.random.default_rng(100 + seed)
    K, B = 2, 7
    bounds, (tc, tl) = _random_bounds(rng, K, B, monotone_truth=True)
    assert np.all((bounds[0] <= tc) & (tc <= bounds[1]) & (bounds[2] <= tl) & (tl <= bounds[3]))
    prob = oracle_lib.Problem(K, B, 8, [1.0, 2.0], [20.0, 30.0], prior=MONO)
    for cell in rng.permutation(K * 4 * B):
        bounds = oracle_lib.refit(prob, int(cell), tc[cell], tl[cell], *bounds)
        clo, chi, tlo, thi = bounds
        assert np.all((clo <= tc) & (tc <= chi) & (tlo <= tl) & (tl <= thi))
    assert np.array_equal(bounds[0], tc) and np.array_equal(bounds[1], tc)
    assert np.array_equal(bounds[2], tl) and np.array_equal(bounds[3], tl)


def test_revealed_only_prior_moves_one_cell(oracle_lib):
    rng = np.random.default_rng(5)
    bounds, _ = _random_bounds(rng, 2, 5)
    prob = oracle_lib.Problem(2, 5, 8, [1.0, 2.0], [20.0, 30.0])
    new = oracle_lib.refit(prob, 7, 1.5, 12.0, *bounds)
    for a in range(4):
        d = np.nonzero(new[a] != bounds[a])[0]
        assert set(d.tolist()) <= {7}
    assert new[0][7] == new[1][7] == np.float32(1.5) and new[2][7] == new[3][7] == np.float32(12.0)


def test_refit_collapses_a_neighbour_when_the_measurement_contradicts_it(oracle_lib):
    """Intervals never empty: a measured tail above a higher-load neighbour's
    interval collapses that neighbour to its upper bound."""
    K, B = 1, 3
    f = lambda *v: np.array(v * 4, np.float32)  # noqa: E731
    clo, chi = f(1.0, 1.0, 1.0), f(2.0, 2.0, 2.0)
    tlo, thi = f(10.0, 10.0, 10.0), f(20.0, 20.0, 20.0)
    prob = oracle_lib.Problem(K, B, 8, [1.0], [30.0], prior=MONO)
    nclo, nchi, ntlo, nthi = oracle_lib.refit(prob, 1, 5.0, 25.0, clo, chi, tlo, thi)
    assert (nclo[2], nchi[2], ntlo[2], nthi[2]) == (2.0, 2.0, 20.0, 20.0)  # b > b_e: raised to hi
    assert (nclo[0], nchi[0], ntlo[0], nthi[0]) == (1.0, 2.0, 10.0, 20.0)  # b < b_e: both within
    nclo, nchi, ntlo, nthi = oracle_lib.refit(prob, 1, 0.5, 5.0, clo, chi, tlo, thi)
    assert (nclo[0], nchi[0], ntlo[0], nthi[0]) == (1.0, 1.0, 10.0, 10.0)  # b < b_e: lowered to lo
    assert (nclo[2], nchi[2], ntlo[2], nthi[2]) == (1.0, 2.0, 10.0, 20.0)


def _small(seed, K=2, B=3, G=8, O=4, S=16):
    rng = np.random.default_rng(seed)
    w = workloads.random_small(rng, K, B, G)
    return dataclasses.replace(w, O=O, S=S, seed=seed, stream_id=2, round=3)


@pytest.mark.parametrize("seed", range(6))
def test_scenarios_under_the_prior_match_brute_force(oracle_lib, seed):
    w = dataclasses.replace(_small(seed), prior=MONO)
    qn = oracle_lib.triangular_table(64)
    prob = oracle_lib.Problem.of(w)
    rng = np.random.default_rng(seed)
    for _ in range(10):
        cell = int(rng.integers(0, w.cells))
        o = int(rng.integers(0, w.O))
        s = int(rng.integers(0, w.S))
        cy, ly, am, ap = oracle_lib.scenario(w, qn, cell, o, s, solver=0)
        clo, chi, tlo, thi = oracle_lib.refit(prob, cell, cy, ly, w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi)
        assert am.t_star == brute.best_max_min(w.K, w.B, w.G, clo, thi, w.demand, w.slo)
        assert ap.t_star == brute.best_max_min(w.K, w.B, w.G, chi, tlo, w.demand, w.slo)


@pytest.mark.parametrize("seed", range(6))
def test_scores_under_the_prior(oracle_lib, seed):
    """0 <= score <= Gamma_t, and per candidate at least the revealed-only score:
    the refit narrows both realisations further, so every scenario's gap is at
    most the revealed-only one for the same draw."""
    w = _small(50 + seed, K=3, B=3, G=12, O=4, S=32)
    w = dataclasses.replace(w, demand=(w.demand * np.float32(1.5)).astype(np.float32))
    qn = oracle_lib.triangular_table(4096)
    plain = oracle_lib.score(w, qn, dump=True)
    mono = oracle_lib.score(dataclasses.replace(w, prior=MONO), qn, dump=True)
    assert mono.gamma_t == plain.gamma_t
    g0 = plain.dump_t[..., 1] - plain.dump_t[..., 0]
    g1 = mono.dump_t[..., 1] - mono.dump_t[..., 0]
    assert np.all(g1 <= g0) and np.all(g1 >= 0)
    assert np.all(mono.score_fixed >= plain.score_fixed)
    assert np.all(mono.score >= 0.0) and np.all(mono.score <= mono.gamma_t)


@pytest.mark.parametrize("idx,factor,S", [(0, 3.0, 64), (1, 1.0, 96), (2, 3.0, 64)])
def test_cached_sums_equal_plain_under_the_prior(oracle_lib, idx, factor, S):
    w = workloads.make_workload(idx)
    w = dataclasses.replace(w, demand=(w.demand * np.float32(factor)).astype(np.float32), S=S, prior=MONO)
    qn = oracle_lib.triangular_table(4096)
    cand = w.candidates[:: max(1, len(w.candidates) // 6)][:6]
    ref = oracle_lib.score(w, qn, candidates=cand)
    se, gt = oracle_lib.score_sums_cached(w, qn, candidates=cand)
    assert np.array_equal(se, ref.sum_eo) and gt == ref.gamma_t
