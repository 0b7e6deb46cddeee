"""Pins of tier 1 of the objective (critical floors delta_i, Section 3) and of
the three-state certificate (Section 4.2) in the oracle.

A critical class i (delta_i > 0) must be served at r_i >= delta_i whenever
that is possible; tier 2 (max-min fulfilment) is then maximised under that
constraint. The brute force enumerates every allocation directly from that
definition, independently of the threshold rule the oracle uses.
"""

import dataclasses

import numpy as np
import pytest

import brute
from conftest import read_golden
from paper_2608_19659_gb300 import workloads

LIT, FRO = 0, 1


def _tiny(rng, K, B, G):
    w = workloads.random_small(rng, K, B, G)
    u = rng.random()
    cap = np.where(rng.random(w.cap_lo.shape) < 0.5, w.cap_lo, w.cap_hi) if u < 0.5 else w.cap_lo
    tail = w.tail_hi if u < 0.7 else w.tail_lo
    return w, cap.astype(np.float32), tail.astype(np.float32)


def _random_floors(rng, K, B, G, cap, tail, demand, slo):
    """Per class: not critical, a floor equal to one of its option values (the
    comparison r >= delta is then decided exactly at equality), just above or
    below such a value, or uniform in (0, 1]."""
    opts = brute.options(K, B, G, cap, tail, demand, slo)
    fl = np.zeros(K, np.float32)
    for i in range(K):
        u = rng.random()
        if u < 0.3 or not opts[i]:
            fl[i] = 0.0 if u < 0.3 else np.float32(rng.uniform(0.05, 1.0))
            continue
        v = np.float32(opts[i][int(rng.integers(0, len(opts[i])))][5])
        if u < 0.6:
            fl[i] = v
        elif u < 0.75:
            fl[i] = np.nextafter(v, np.float32(2.0))
        elif u < 0.85:
            fl[i] = np.nextafter(v, np.float32(0.0))
        else:
            fl[i] = np.float32(rng.uniform(0.01, 1.0))
        fl[i] = min(max(fl[i], np.float32(0.0)), np.float32(1.0))
    return fl


def _check_against_brute(oracle_lib, w, cap, tail, fl, solver):
    K, B, G = w.K, w.B, w.G
    p = oracle_lib.Problem(K, B, G, w.demand, w.slo, fl)
    a = oracle_lib.solve(p, cap, tail, solver)
    met = brute.floors_met(K, B, G, cap, tail, w.demand, w.slo, fl)
    assert a.floors_met == int(met)
    assert a.t_star == brute.best_max_min(K, B, G, cap, tail, w.demand, w.slo, fl)
    if a.ok:
        ch = brute.choice_at(K, B, G, cap, tail, w.demand, w.slo, np.float32(a.t_star), fl)
    elif met:  # tier 1 alone: the critical classes at their floors, the others empty
        ch = brute.choice_at(K, B, G, cap, tail, w.demand, w.slo, np.float32(0.0), fl)
        ch = [c if fl[i] > 0 else None for i, c in enumerate(ch)]
    else:
        ch = [None] * K
    for i in range(K):
        if ch[i] is None:
            assert (a.tp[i], a.replicas[i], a.bin[i]) == (0, 0, -1)
        else:
            cost, j, n, c, b, f = ch[i]
            assert (a.tp[i], a.replicas[i], a.bin[i]) == (brute.TP[j], n, b)
            assert a.fulfil[i] == np.float32(f)
            if fl[i] > 0:
                assert a.fulfil[i] >= fl[i]
    assert a.total_gpus == sum(x[0] for x in ch if x is not None) <= G
    return a


@pytest.mark.parametrize("seed", range(80))
def test_floors_match_brute_force(oracle_lib, seed):
    rng = np.random.default_rng(31000 + seed)
    K = 2 if seed % 3 else 3
    B = 1 + seed % 2
    G = [4, 6, 8][seed % 3] if K == 3 else [4, 8, 9][seed % 3]
    w, cap, tail = _tiny(rng, K, B, G)
    fl = _random_floors(rng, K, B, G, cap, tail, w.demand, w.slo)
    for solver in (LIT, FRO):
        _check_against_brute(oracle_lib, w, cap, tail, fl, solver)


@pytest.mark.parametrize("seed", range(150))
def test_floors_frontier_matches_literal(oracle_lib, seed):
    rng = np.random.default_rng(32000 + seed)
    K, B, G = int(rng.integers(1, 6)), int(rng.integers(1, 5)), int(rng.integers(1, 33))
    w, cap, tail = _tiny(rng, K, B, G)
    w = dataclasses.replace(w, demand=(w.demand * np.float32(rng.uniform(0.3, 3.0))).astype(np.float32))
    fl = _random_floors(rng, K, B, G, cap, tail, w.demand, w.slo)
    p = oracle_lib.Problem(K, B, G, w.demand, w.slo, fl)
    assert oracle_lib.solve(p, cap, tail, LIT) == oracle_lib.solve(p, cap, tail, FRO)


@pytest.mark.parametrize("seed", range(30))
def test_zero_floors_are_no_floors(oracle_lib, seed):
    rng = np.random.default_rng(33000 + seed)
    K, B, G = int(rng.integers(1, 6)), int(rng.integers(1, 5)), int(rng.integers(1, 33))
    w, cap, tail = _tiny(rng, K, B, G)
    p0 = oracle_lib.Problem(K, B, G, w.demand, w.slo)
    pz = oracle_lib.Problem(K, B, G, w.demand, w.slo, np.zeros(K, np.float32))
    for solver in (LIT, FRO):
        a, b = oracle_lib.solve(p0, cap, tail, solver), oracle_lib.solve(pz, cap, tail, solver)
        assert a == b and a.floors_met == 1


@pytest.mark.parametrize("seed", range(60))
def test_floor_invariants(oracle_lib, seed):
    rng = np.random.default_rng(34000 + seed)
    K, B, G = int(rng.integers(1, 5)), int(rng.integers(1, 4)), int(rng.integers(2, 30))
    w, cap, tail = _tiny(rng, K, B, G)
    fl = _random_floors(rng, K, B, G, cap, tail, w.demand, w.slo)
    plain = oracle_lib.solve(oracle_lib.Problem(K, B, G, w.demand, w.slo), cap, tail, FRO)
    p = oracle_lib.Problem(K, B, G, w.demand, w.slo, fl)
    a = oracle_lib.solve(p, cap, tail, FRO)
    # a constraint can only lower the optimum; it does not bind once the plain
    # optimum already serves every class at or above every floor
    assert a.t_star <= plain.t_star
    if plain.t_star >= fl.max():
        assert a == dataclasses.replace(plain, floors_met=1)
    # a positive t* meets the floors; unmet floors leave nothing
    if a.ok:
        assert a.floors_met == 1
    if not a.floors_met:
        assert a.t_star == 0.0 and a.total_gpus == 0 and all(r == 0 for r in a.replicas)
    # more capacity, a lower tail or more GPUs never unmeets the floors nor lowers t*
    i, j, b = rng.integers(0, K), rng.integers(0, 4), rng.integers(0, B)
    cap2 = cap.copy()
    cap2[i, j, b] *= np.float32(1.6)
    tail2 = tail.copy()
    tail2[i, j, b] *= np.float32(0.5)
    pG = oracle_lib.Problem(K, B, G + int(rng.integers(1, 8)), w.demand, w.slo, fl)
    for a2 in (oracle_lib.solve(p, cap2, tail, FRO), oracle_lib.solve(p, cap, tail2, FRO),
               oracle_lib.solve(pG, cap, tail, FRO)):
        assert a2.floors_met >= a.floors_met and a2.t_star >= a.t_star
    # a higher floor never helps
    fl2 = fl.copy()
    fl2[i] = min(np.float32(1.0), fl2[i] + np.float32(rng.uniform(0.0, 0.5)))
    a3 = oracle_lib.solve(oracle_lib.Problem(K, B, G, w.demand, w.slo, fl2), cap, tail, FRO)
    assert a3.floors_met <= a.floors_met and a3.t_star <= a.t_star


@pytest.mark.parametrize("seed", range(30))
def test_single_class_closed_form_with_floor(oracle_lib, seed):
    # K = 1: the floor holds iff the largest fulfilment any feasible row reaches
    # within G is at or above it; then t* is that fulfilment, else 0
    rng = np.random.default_rng(35000 + seed)
    B, G = int(rng.integers(1, 6)), int(rng.integers(1, 40))
    w = workloads.random_small(rng, 1, B, G)
    cap, tail = w.cap_lo, w.tail_hi
    best = 0.0
    for j, tau in enumerate(brute.TP):
        feas = [b for b in range(B) if tail[0, j, b] <= w.slo[0]]
        if G // tau >= 1 and feas:
            best = max(best, float(brute.f32_fulfil(G // tau, max(cap[0, j, b] for b in feas), w.demand[0])))
    for d in (np.float32(best), np.nextafter(np.float32(best), np.float32(2.0)), np.float32(0.5 * best)):
        if d <= 0 or d > 1:
            continue
        a = oracle_lib.solve(oracle_lib.Problem(1, B, G, w.demand, w.slo, [d]), cap, tail, FRO)
        assert a.floors_met == int(best >= d)
        assert a.t_star == (best if best >= d else 0.0)


def _table3_known(oracle_lib, lam):
    t1 = {"chat": [0.798, 1.649, 1.408], "code": [0.560, 2.779, 1.392]}
    cap = np.ones((2, 4, 1), np.float32)
    tail = np.full((2, 4, 1), 1e9, np.float32)
    for i, k in enumerate(["chat", "code"]):
        for j, tp in enumerate([2, 4, 8]):
            cap[i, j + 1, 0] = np.float32(t1[k][j] * tp)
            tail[i, j + 1, 0] = 10.0
    return np.asarray(lam, np.float32), cap, tail


def test_paper_floor_audit(oracle_lib):
    """Section 6.4: floors of 6 and 10 req/s certify; a 1000 req/s demand is
    certified infeasible (read as fractions of the 1.0x demands)."""
    rows = read_golden("critical_floors.txt")
    assert [r[0] for r in rows] == ["feasible", "infeasible"]
    for case, lc, lk, fc, fk, want in rows:
        delta = np.array([float(fc) / 12.0, float(fk) / 16.0], np.float32)
        lam, cap, tail = _table3_known(oracle_lib, [float(lc), float(lk)])
        p = oracle_lib.Problem(2, 1, 16, lam, [30.0, 30.0], delta)
        rev = np.ones(8, np.uint8)
        st, g = oracle_lib.certificate(p, cap, cap, tail, tail, rev, 0.01)
        assert st == int(want) and g == 0.0
        a = oracle_lib.solve(p, cap, tail, LIT)
        if case == "feasible":
            # the floors do not bind: the Table 3 optimum, TP4 x 2 for both classes
            assert a.floors_met == 1 and a.tp == [4, 4] and a.replicas == [2, 2] and a.t_star == 1.0
        else:
            assert a.floors_met == 0 and a.t_star == 0.0 and a.replicas == [0, 0]


def test_table3_floors_do_not_bind(oracle_lib):
    """At every demand scale of Table 3 the Chat/Code floors of Section 6.4 are
    met and leave the tier-2 allocation unchanged."""
    for r in [r for r in read_golden("table3_allocation.txt") if r[1] == "oracle"]:
        scale = float(r[0])
        lam, cap, tail = _table3_known(oracle_lib, [12.0 * scale, 16.0 * scale])
        delta = np.array([6.0 / (12.0 * scale), 10.0 / (16.0 * scale)], np.float32)
        for solver in (LIT, FRO):
            a = oracle_lib.solve(oracle_lib.Problem(2, 1, 16, lam, [30.0, 30.0], delta), cap, tail, solver)
            assert a.floors_met == 1
            assert (a.tp, a.replicas) == ([int(r[2]), int(r[3])], [int(r[4]), int(r[5])])
            assert abs(a.t_star - float(r[6])) <= 0.001


def test_certificate_states(oracle_lib):
    """Section 4.2: undecided while only A+ meets the floors, even at a zero gap."""
    rng = np.random.default_rng(36)
    w = workloads.random_small(rng, 3, 1, 12)
    clo, chi = w.cap_lo.copy(), w.cap_hi.copy()
    tlo, thi = w.tail_lo.copy(), w.tail_hi.copy()
    # class 2 is never SLO-feasible: t* = 0 on both sides, so the gap is 0
    tlo[2] = thi[2] = w.slo[2] * 3
    # class 0 is critical and can reach its floor only with the optimistic capacities
    tlo[0] = thi[0] = w.slo[0] * 0.5
    clo[0], chi[0] = 0.01, 50.0
    rev = np.zeros(w.cells, np.uint8)
    p = oracle_lib.Problem(3, 1, 12, w.demand, w.slo, [0.5, 0.0, 0.0])
    am = oracle_lib.solve(p, clo, thi)
    ap = oracle_lib.solve(p, chi, tlo)
    assert am.floors_met == 0 and ap.floors_met == 1 and am.t_star == ap.t_star == 0.0
    assert oracle_lib.certificate(p, clo, chi, tlo, thi, rev, 0.01) == (0, 0.0)
    # once the capacities are known and high, the floor holds on both sides; the
    # committed cell (class 0's floor option) must still be measured
    clo[0] = chi[0]
    st, g = oracle_lib.certificate(p, clo, chi, tlo, thi, rev, 0.01)
    a = oracle_lib.solve(p, clo, thi)
    assert st == 0 and g == 0.0 and a.floors_met == 1 and a.replicas[0] > 0 and a.t_star == 0.0
    c = (0 * 4 + [1, 2, 4, 8].index(a.tp[0])) * 1 + a.bin[0]
    rev[c] = 1
    assert oracle_lib.certificate(p, clo, chi, tlo, thi, rev, 0.01) == (1, 0.0)
    # a floor nobody can reach: certified infeasible whatever else holds
    lam = w.demand.copy()
    lam[0] = 1e6
    p_inf = oracle_lib.Problem(3, 1, 12, lam, w.slo, [1.0, 0.0, 0.0])
    assert oracle_lib.certificate(p_inf, clo, chi, tlo, thi, np.ones(w.cells, np.uint8), 0.01)[0] == 2


def test_replay_stops_certified_infeasible(oracle_lib):
    rp = workloads.make_replay(n_streams=2)
    base = rp.base
    # an unreachable floor for class 0: certified infeasible before any reveal
    base = dataclasses.replace(base, floor=np.array([1.0] + [0.0] * (base.K - 1), np.float32),
                               demand=(base.demand * np.float32(50.0)).astype(np.float32))
    rp = dataclasses.replace(rp, base=base)
    res = oracle_lib.replay_stream(rp, 0, oracle_lib.triangular_table(4096), seed=9, S=8, O=2, max_rounds=6)
    assert res.state == 2 and res.rounds == 0
    assert list(res.reveal_order[: rp.r0]) == list(rp.perm[0][: rp.r0])
