"""Pins of the oracle's allocation solvers (Section 3, Eqs. 1-5; tier 2 of the objective)."""

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


@pytest.mark.parametrize("seed", range(60))
def test_literal_matches_brute_force(oracle_lib, seed):
    rng = np.random.default_rng(1000 + seed)
    K = 2 if seed % 3 else 3
    B = 1 + seed % 2
    G = [4, 6, 8][seed % 3] if K == 3 else [4, 8, 9][seed % 3]
    w, cap, tail = _tiny(rng, K, B, G)
    p = oracle_lib.Problem.of(w)
    a = oracle_lib.solve(p, cap, tail, LIT)
    t_bf = brute.best_max_min(K, B, G, cap, tail, w.demand, w.slo)
    assert a.t_star == t_bf
    if a.ok:
        ch = brute.choice_at(K, B, G, cap, tail, w.demand, w.slo, np.float32(a.t_star))
        for i in range(K):
            cost, j, n, c, b, f = ch[i]
            assert (a.tp[i], a.replicas[i], a.bin[i]) == (brute.TP[j], n, b)
            assert a.fulfil[i] == np.float32(f)
        assert a.total_gpus == sum(x[0] for x in ch) <= G
    else:
        assert a.t_star == 0.0 and a.total_gpus == 0
        assert all(r == 0 for r in a.replicas)


@pytest.mark.parametrize("seed", range(200))
def test_frontier_matches_literal(oracle_lib, seed):
    rng = np.random.default_rng(5000 + seed)
    K = int(rng.integers(1, 5))
    B = int(rng.integers(1, 5))
    G = int(rng.integers(1, 33))
    w, cap, tail = _tiny(rng, K, B, G)
    if seed % 7 == 0:  # duplicate capacities across bins exercise the bin tie rule
        cap = np.repeat(cap[:, :, :1], B, axis=2).copy()
    p = oracle_lib.Problem.of(w)
    a = oracle_lib.solve(p, cap, tail, LIT)
    b = oracle_lib.solve(p, cap, tail, FRO)
    assert a == b


def _table3_instance(oracle_lib, scale, allowed=(2, 4, 8)):
    t1 = {"chat": [0.798, 1.649, 1.408], "code": [0.560, 2.779, 1.392]}
    lam = np.array([12.0 * scale, 16.0 * scale], np.float32)
    slo = np.array([30.0, 30.0], np.float32)
    cap = np.ones((2, 4, 1), np.float32)
    tail = np.full((2, 4, 1), 1e9, np.float32)  # TP1 was not measured: never SLO-feasible
    for i, k in enumerate(["chat", "code"]):
        for j, tp in enumerate([2, 4, 8]):
            cap[i, j + 1, 0] = np.float32(t1[k][j] * tp)
            if tp in allowed:
                tail[i, j + 1, 0] = 10.0
    return oracle_lib.Problem(2, 1, 16, lam, slo), cap, tail


def test_table3_allocation(oracle_lib):
    rows = read_golden("table3_allocation.txt")
    assert len(rows) == 12
    idx = {1: 0, 2: 1, 4: 2, 8: 3}
    for r in rows:
        scale, kind = float(r[0]), r[1]
        tps = (int(r[2]), int(r[3]))
        reps = (int(r[4]), int(r[5]))
        mm_paper, gp_paper = float(r[6]), float(r[7])
        p, cap, tail = _table3_instance(oracle_lib, scale)
        mm, gp, fits = oracle_lib.evaluate(p, cap, tail, [idx[t] for t in tps], [0, 0], reps)
        assert fits
        assert abs(mm - mm_paper) <= 0.01 and abs(gp - gp_paper) <= 0.01, r
        if kind == "oracle":
            for solver in (LIT, FRO):
                a = oracle_lib.solve(p, cap, tail, solver)
                assert (tuple(a.tp), tuple(a.replicas)) == (tps, reps)
                assert a.total_gpus == 16
                assert abs(a.t_star - mm_paper) <= 0.001
        if kind in ("fixed8", "fixed2"):
            # the solver restricted to one TP degree reproduces the fixed rows
            only = 8 if kind == "fixed8" else 2
            p2, cap2, tail2 = _table3_instance(oracle_lib, scale, allowed=(only,))
            a = oracle_lib.solve(p2, cap2, tail2, LIT)
            assert tuple(a.tp) == tps and abs(a.t_star - mm_paper) <= 0.01
            if kind == "fixed2":
                assert tuple(a.replicas) == reps


def test_table3_lower_tp_wins_equal_cost(oracle_lib):
    # 0.7x: chat TP4 x2 and TP8 x1 both cost 8 GPUs and both cover lambda = 8.4
    p, cap, tail = _table3_instance(oracle_lib, 0.7)
    a = oracle_lib.solve(p, cap, tail, LIT)
    assert oracle_lib.fulfil(1, cap[0, 3, 0], p.demand[0]) == 1.0
    assert a.tp[0] == 4 and a.replicas[0] == 2


def test_c128_tail_rejection(oracle_lib):
    rows = read_golden("c128_tail_rejection.txt")
    cells = {int(r[0]): (float(r[1]), float(r[2])) for r in rows if r[0] in ("4", "8")}
    kv = {r[0]: float(r[1]) for r in rows if r[0] in ("slo", "demand", "G")}
    cap = np.zeros((1, 4, 1), np.float32)
    tail = np.full((1, 4, 1), 1e9, np.float32)
    for tp, (c, l) in cells.items():
        j = {4: 2, 8: 3}[tp]
        cap[0, j, 0] = c
        tail[0, j, 0] = l
    for slo, want in ((kv["slo"], 8), (60.0, 4)):
        p = oracle_lib.Problem(1, 1, int(kv["G"]), [kv["demand"]], [slo])
        for solver in (LIT, FRO):
            a = oracle_lib.solve(p, cap, tail, solver)
            assert a.tp[0] == want and a.replicas[0] == 1 and a.t_star == 1.0


def test_class_without_feasible_cell_zeroes_allocation(oracle_lib):
    rng = np.random.default_rng(3)
    w = workloads.random_small(rng, 3, 2, 16)
    tail = w.tail_lo.copy()
    tail[1] = w.slo[1] * 2  # class 1 has no SLO-feasible configuration
    p = oracle_lib.Problem.of(w)
    for solver in (LIT, FRO):
        a = oracle_lib.solve(p, w.cap_hi, tail, solver)
        assert a.t_star == 0.0 and a.ok == 0 and a.total_gpus == 0
        assert a.replicas == [0, 0, 0] and a.bin == [-1, -1, -1]
        assert (a.has_option_mask >> 1) & 1 == 0


@pytest.mark.parametrize("seed", range(40))
def test_single_class_closed_form(oracle_lib, seed):
    # K = 1: any n <= floor(G/tau) fits, so t* = max over feasible rows of f(floor(G/tau), best cap)
    rng = np.random.default_rng(seed)
    B = int(rng.integers(1, 6))
    G = int(rng.integers(1, 40))
    w = workloads.random_small(rng, 1, B, G)
    cap, tail = w.cap_lo, w.tail_hi
    best = 0.0
    for j, tau in enumerate(brute.TP):
        M = G // tau
        feas = [b for b in range(B) if tail[0, j, b] <= w.slo[0]]
        if M < 1 or not feas:
            continue
        c = max(cap[0, j, b] for b in feas)
        best = max(best, float(brute.f32_fulfil(M, c, w.demand[0])))
    a = oracle_lib.solve(oracle_lib.Problem.of(w), cap, tail, FRO)
    assert a.t_star == best


@pytest.mark.parametrize("seed", range(40))
def test_monotonicity_invariants(oracle_lib, seed):
    rng = np.random.default_rng(777 + seed)
    K = int(rng.integers(1, 4))
    B = int(rng.integers(1, 4))
    G = int(rng.integers(2, 24))
    w = workloads.random_small(rng, K, B, G)
    p = oracle_lib.Problem.of(w)
    cap, tail = w.cap_lo.copy(), w.tail_hi.copy()
    t0 = oracle_lib.solve(p, cap, tail, FRO).t_star
    # conservative <= optimistic (Section 4.1)
    assert t0 <= oracle_lib.solve(p, w.cap_hi, w.tail_lo, FRO).t_star
    # nondecreasing in G
    p_more = oracle_lib.Problem(K, B, G + int(rng.integers(1, 8)), w.demand, w.slo)
    assert oracle_lib.solve(p_more, cap, tail, FRO).t_star >= t0
    # nondecreasing in any capacity, nonincreasing in any tail
    i, j, b = rng.integers(0, K), rng.integers(0, 4), rng.integers(0, B)
    cap2 = cap.copy()
    cap2[i, j, b] *= np.float32(1.5)
    assert oracle_lib.solve(p, cap2, tail, FRO).t_star >= t0
    tail2 = tail.copy()
    tail2[i, j, b] *= np.float32(0.5)
    assert oracle_lib.solve(p, cap, tail2, FRO).t_star >= t0
    # nonincreasing in demand
    lam = w.demand.copy()
    lam[i] *= np.float32(1.7)
    p_lam = oracle_lib.Problem(K, B, G, lam, w.slo)
    assert oracle_lib.solve(p_lam, cap, tail, FRO).t_star <= t0


def test_invalid_problem_rejected(oracle_lib):
    cap = np.ones(4, np.float32)
    with pytest.raises(ValueError):
        oracle_lib.solve(oracle_lib.Problem(1, 1, 0, [1.0], [1.0]), cap, cap)
    with pytest.raises(ValueError):
        oracle_lib.solve(oracle_lib.Problem(1, 1, 4, [0.0], [1.0]), cap, cap)
