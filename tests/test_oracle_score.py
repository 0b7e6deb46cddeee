"""Pins of the oracle's Monte-Carlo score (Section 4.3) and certificate (Section 4.2)."""

import dataclasses

import numpy as np
import pytest

import brute
from paper_2608_19659_gb300 import workloads

FRO, LIT = 1, 0


def _small(seed, K=2, B=2, G=8, O=4, S=16):
    rng = np.random.default_rng(seed)
    w = workloads.random_small(rng, K, B, G)
    return dataclasses.replace(w, O=O, S=S, seed=seed, stream_id=3, round=1)


@pytest.mark.parametrize("seed", range(6))
def test_scenarios_match_brute_force(oracle_lib, seed):
    """Each scenario: draw inside the stratum, patch cell e in both realisations, brute-force both."""
    w = _small(seed)
    qn = oracle_lib.triangular_table(64)
    W = 64 // w.O
    rng = np.random.default_rng(seed)
    for _ in range(12):
        cell = int(rng.integers(0, w.cells))
        o = int(rng.integers(0, w.O))
        s = int(rng.integers(0, w.S))
        cy, ly, am, ap = oracle_lib.scenario(w, qn, cell, o, s, solver=LIT)
        lo_c, hi_c = w.cap_lo.reshape(-1)[cell], w.cap_hi.reshape(-1)[cell]
        lo_l, hi_l = w.tail_lo.reshape(-1)[cell], w.tail_hi.reshape(-1)[cell]
        # the draw lies in the image of its outcome stratum
        assert oracle_lib.map_value(lo_c, hi_c, qn[o * W]) <= cy <= oracle_lib.map_value(lo_c, hi_c, qn[(o + 1) * W - 1])
        assert oracle_lib.map_value(lo_l, hi_l, qn[o * W]) <= ly <= oracle_lib.map_value(lo_l, hi_l, qn[(o + 1) * W - 1])
        for lo_cap, tail_b, a in ((w.cap_lo, w.tail_hi, am), (w.cap_hi, w.tail_lo, ap)):
            cap = lo_cap.reshape(-1).copy()
            tail = tail_b.reshape(-1).copy()
            cap[cell] = cy
            tail[cell] = ly
            assert a.t_star == brute.best_max_min(w.K, w.B, w.G, cap, tail, w.demand, w.slo)
        assert 0.0 <= ap.t_star - am.t_star


@pytest.mark.parametrize("seed", range(8))
def test_score_invariants_and_fixed_point(oracle_lib, seed):
    w = _small(100 + seed, K=3, B=3, G=12, O=4, S=32)
    qn = oracle_lib.triangular_table(4096)
    r = oracle_lib.score(w, qn, dump=True)
    am, ap, gt = oracle_lib.base_gap(oracle_lib.Problem.of(w), w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi)
    assert r.gamma_t == np.float32(ap.t_star - am.t_star) >= 0.0
    tm, tp = r.dump_t[..., 0], r.dump_t[..., 1]
    g = (tp - tm).astype(np.float32)
    # revealing never widens the gap: t*(A-) <= t*(A-'), t*(A+') <= t*(A+)
    assert np.all(tm >= np.float32(am.t_star)) and np.all(tp <= np.float32(ap.t_star))
    assert np.all(g >= 0) and np.all(g <= np.float32(r.gamma_t))
    # fixed-point sums: round-half-even of the exact product g * 2^40
    fixed = np.rint(g.astype(np.float64) * 2.0**40).astype(np.int64)
    assert np.array_equal(fixed.sum(axis=2), r.sum_eo)
    n = w.O * w.S
    tot = r.sum_eo.sum(axis=1)
    assert np.array_equal(r.gap, (tot.astype(np.float64) * 2.0**-40) / n)
    gfix = np.int64(np.rint(np.float64(r.gamma_t) * 2.0**40))
    assert np.array_equal(r.score_fixed, gfix * n - tot)
    assert np.all(r.score >= 0) and np.all(r.score <= r.gamma_t + 1e-12)
    assert np.all(np.abs(r.gap + r.score - np.float64(r.gamma_t)) < 2.0**-39)


def test_collapsed_bounds_give_zero(oracle_lib):
    w = _small(7, K=2, B=2, G=8)
    w = dataclasses.replace(w, cap_hi=w.cap_lo.copy(), tail_lo=w.tail_hi.copy())
    qn = oracle_lib.triangular_table(4096)
    r = oracle_lib.score(w, qn)
    assert r.gamma_t == 0.0
    assert np.all(r.sum_eo == 0) and np.all(r.score == 0) and np.all(r.gap == 0)


def test_revealed_candidate_scores_zero(oracle_lib):
    w = _small(11, K=2, B=2, G=8)
    cap_lo, cap_hi = w.cap_lo.copy(), w.cap_hi.copy()
    tail_lo, tail_hi = w.tail_lo.copy(), w.tail_hi.copy()
    cell = 5
    for a, b in ((cap_lo, cap_hi), (tail_lo, tail_hi)):
        a.reshape(-1)[cell] = b.reshape(-1)[cell]
    w = dataclasses.replace(w, cap_lo=cap_lo, cap_hi=cap_hi, tail_lo=tail_lo, tail_hi=tail_hi)
    qn = oracle_lib.triangular_table(4096)
    r = oracle_lib.score(w, qn, candidates=np.array([cell], np.int32))
    assert r.score_fixed[0] == 0 and r.score[0] == 0.0


def test_literal_and_frontier_scores_agree(oracle_lib):
    w = workloads.make_workload(0)
    qn = oracle_lib.triangular_table(4096)
    cand = w.candidates[:4]
    a = oracle_lib.score(w, qn, candidates=cand, solver=LIT, S=32)
    b = oracle_lib.score(w, qn, candidates=cand, solver=FRO, S=32)
    assert np.array_equal(a.sum_eo, b.sum_eo) and a.best == b.best


def test_argmax_ties_prefer_lower_tp_then_order(oracle_lib):
    # bounds collapsed everywhere: every score is 0, so the tie rules decide
    w = _small(5, K=2, B=2, G=8)
    w = dataclasses.replace(w, cap_hi=w.cap_lo.copy(), tail_lo=w.tail_hi.copy())
    qn = oracle_lib.triangular_table(4096)
    B = w.B
    cells = np.array([(0 * 4 + 3) * B, (1 * 4 + 1) * B + 1, (0 * 4 + 1) * B], np.int32)  # TP8, TP2, TP2
    r = oracle_lib.score(w, qn, candidates=cells)
    assert r.best == cells[1]
    assert oracle_lib.score(w, qn, candidates=cells[::-1].copy()).best == cells[2]


def test_seed_stream_round_change_draws(oracle_lib):
    def idx(seed, stream, rnd):
        return [oracle_lib.draw_index(seed, stream, rnd, 9, 4096, 8, 3, s) for s in range(32)]

    base = idx(21, 0, 0)
    for args in ((22, 0, 0), (21, 1, 0), (21, 0, 1), (21 + (1 << 32), 0, 0)):
        assert idx(*args) != base


def test_score_argument_checks(oracle_lib):
    w = _small(1)
    qn = oracle_lib.triangular_table(4096)
    with pytest.raises(ValueError):
        oracle_lib.score(w, qn, candidates=np.array([w.cells], np.int32))
    with pytest.raises(ValueError):
        oracle_lib.score(w, qn, O=3)


def test_certificate_requires_known_committed_tails(oracle_lib):
    w = _small(31, K=2, B=2, G=8)
    p = oracle_lib.Problem.of(w)
    cap, tail = w.cap_lo.copy(), w.tail_hi.copy()
    # every bound collapsed: gap 0; certificate fires only once A-'s cells are revealed
    rev = np.zeros(w.cells, np.uint8)
    st, g = oracle_lib.certificate(p, cap, cap, tail, tail, rev, 0.01)
    am = oracle_lib.solve(p, cap, tail)
    assert g == 0.0
    if am.ok:
        assert st == 0
        for i in range(w.K):
            if am.replicas[i]:
                j = [1, 2, 4, 8].index(am.tp[i])
                rev[(i * 4 + j) * w.B + am.bin[i]] = 1
        st, g = oracle_lib.certificate(p, cap, cap, tail, tail, rev, 0.01)
    assert st == 1
    # a positive gap above eps keeps it undecided
    st, g = oracle_lib.certificate(p, w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi,
                                   np.ones(w.cells, np.uint8), -1.0)
    assert st == 0


@pytest.mark.parametrize("idx,factor,n_cand,S", [(0, 3.0, 16, 256), (1, 1.0, 12, 512), (2, 3.0, 6, 384),
                                                 (3, 2.0, 3, 96)])
def test_cached_sums_equal_plain_oracle(oracle_lib, idx, factor, n_cand, S):
    """The cached scorer reuses a candidate's solves for equal (capacity position,
    tail within SLO) pairs; its sums, Gamma_t and, through or_reduce, its
    expectations, scores and argmax equal or_score's on every workload family."""
    w = workloads.make_workload(idx)
    w = dataclasses.replace(w, demand=(w.demand * np.float32(factor)).astype(np.float32), S=S)
    qn = oracle_lib.triangular_table(4096)
    rng = np.random.default_rng(idx)
    cand = np.sort(rng.choice(w.candidates, n_cand, replace=False)).astype(np.int32)
    ref = oracle_lib.score(w, qn, candidates=cand)
    se, gt = oracle_lib.score_sums_cached(w, qn, candidates=cand)
    assert gt == ref.gamma_t
    assert np.array_equal(se, ref.sum_eo)
    red = oracle_lib.reduce_sums(w, cand, se, gt)
    assert np.array_equal(red.gap, ref.gap) and np.array_equal(red.score, ref.score)
    assert np.array_equal(red.score_fixed, ref.score_fixed) and red.best == ref.best


def test_cached_sums_with_tail_gate_both_ways(oracle_lib):
    """Cells whose tail interval straddles the SLO: the cache keys on the gate, and
    scenarios with the gate open and closed at one capacity position differ."""
    rng = np.random.default_rng(7)
    w = workloads.random_small(rng, 2, 3, 10)
    L = w.slo[:, None, None] * np.ones((w.K, 4, w.B), np.float32)
    hi = np.where(np.arange(w.cells).reshape(L.shape) % 2 == 1, 1.2, 0.9) * L
    w = dataclasses.replace(w, tail_lo=(0.8 * L).astype(np.float32), tail_hi=hi.astype(np.float32),
                            demand=(3 * w.demand).astype(np.float32), O=2, S=64, seed=11)
    qn = oracle_lib.triangular_table(64)
    ref = oracle_lib.score(w, qn, solver=LIT)
    se, gt = oracle_lib.score_sums_cached(w, qn, solver=LIT)
    assert np.array_equal(se, ref.sum_eo) and gt == ref.gamma_t
    assert ref.gamma_t > 0 and np.any(ref.score_fixed > 0)
