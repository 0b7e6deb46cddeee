"""Critical floors (tier 1 of the objective, Section 3) and the certificate's
certified-infeasible state (Section 4.2) on the GPU, against the CPU oracle.

Every solve, scenario and score is compared bit for bit; the floors are drawn
at, just above and just below option fulfilments, so that the comparison
r >= delta is decided at equality, and some of them cannot be met.
"""

import dataclasses

import numpy as np
import pytest

import brute
from conftest import alloc_matches, load_model, read_golden
from paper_2608_19659_gb300 import workloads
from test_gpu_solve import _as_dict, _realisations, _solve_batch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def qn(oracle_lib):
    return oracle_lib.triangular_table(4096)


def _floors(rng, w, cap, tail, p_crit=0.6):
    """Per class: not critical, or the fulfilment of a random SLO-feasible option
    of (cap, tail), nudged one float up or down half of the time, or uniform."""
    K, B, G = w.K, w.B, w.G
    cap = np.asarray(cap, np.float32).reshape(K, 4, B)
    tail = np.asarray(tail, np.float32).reshape(K, 4, B)
    fl = np.zeros(K, np.float32)
    for i in range(K):
        if rng.random() >= p_crit:
            continue
        cells = [(j, b) for j in range(4) for b in range(B) if tail[i, j, b] <= w.slo[i] and G >> j >= 1]
        u = rng.random()
        if not cells or u < 0.15:
            fl[i] = np.float32(rng.uniform(0.01, 1.0))
            continue
        j, b = cells[int(rng.integers(len(cells)))]
        v = brute.f32_fulfil(int(rng.integers(1, (G >> j) + 1)), cap[i, j, b], w.demand[i])
        if u < 0.55:
            fl[i] = v
        elif u < 0.8:
            fl[i] = np.nextafter(v, np.float32(2.0))
        else:
            fl[i] = np.nextafter(v, np.float32(0.0))
        fl[i] = np.clip(fl[i], np.float32(0.0), np.float32(1.0))
    return fl


@pytest.mark.parametrize("seed", range(16))
def test_solve_batch_with_floors(fsb, cuda, oracle_lib, seed):
    rng = np.random.default_rng(60 + seed)
    K, B, G = int(rng.integers(1, 9)), int(rng.integers(1, 9)), int(rng.integers(1, 65))
    w = workloads.random_small(rng, K, B, G)
    w = dataclasses.replace(w, floor=_floors(rng, w, w.cap_hi, w.tail_lo))
    cap, tail = _realisations(rng, w, 48)
    p = oracle_lib.Problem.of(w)
    with load_model(fsb, w) as m:
        recs = _solve_batch(fsb, cuda, m, cap, tail)
    for r in range(cap.shape[0]):
        literal = r % 4 == 0 and K * B * G <= 1024
        ref = oracle_lib.solve(p, cap[r], tail[r], 0 if literal else 1)
        assert alloc_matches(_as_dict(recs[r], K), ref, K), (seed, r)


def _table3_known(lam):
    t1 = {"chat": [0.798, 1.649, 1.408], "code": [0.560, 2.779, 1.392]}
    cap = np.ones((2, 4, 1), np.float32)
    tail = np.full((2, 4, 1), 1e9, np.float32)
    for i, k in enumerate(["chat", "code"]):
        for j, tp in enumerate([2, 4, 8]):
            cap[i, j + 1, 0] = np.float32(t1[k][j] * tp)
            tail[i, j + 1, 0] = 10.0
    return workloads.Workload("table3", 2, 1, 16, np.asarray(lam, np.float32), np.array([30.0, 30.0], np.float32),
                              cap, cap, tail, tail, np.arange(8, dtype=np.int32), 1, 1, 0)


def test_paper_floor_audit(fsb, cuda, oracle_lib):
    """Section 6.4: floors of 6 and 10 req/s certify; a 1000 req/s demand is
    certified infeasible (floors read as fractions of the 1.0x demands)."""
    for case, lc, lk, fc, fk, want in read_golden("critical_floors.txt"):
        w = _table3_known([float(lc), float(lk)])
        delta = np.array([float(fc) / 12.0, float(fk) / 16.0], np.float32)
        with load_model(fsb, w) as m:
            fsb.fs_set_floors(m, delta)
            for c in range(w.cells):
                fsb.fs_reveal(m, c, float(w.cap_lo.reshape(-1)[c]), float(w.tail_lo.reshape(-1)[c]))
            assert fsb.fs_certificate(m, 0.01) == (int(want), 0.0)
            gm, gp, g = fsb.fs_solve_bounds(m)
        assert gm["floors_met"] == gp["floors_met"] == (1 if case == "feasible" else 0)
        p = oracle_lib.Problem(2, 1, 16, w.demand, w.slo, delta)
        assert alloc_matches(gm, oracle_lib.solve(p, w.cap_lo, w.tail_lo), 2)


def test_certificate_undecided_until_conservative_meets_floor(fsb, cuda, oracle_lib):
    rng = np.random.default_rng(36)
    w = workloads.random_small(rng, 3, 1, 12)
    clo, chi = w.cap_lo.copy(), w.cap_hi.copy()
    tlo, thi = w.tail_lo.copy(), w.tail_hi.copy()
    tlo[2] = thi[2] = w.slo[2] * 3  # class 2 is never feasible: t* = 0 on both sides
    tlo[0] = thi[0] = w.slo[0] * 0.5
    clo[0], chi[0] = 0.01, 50.0     # class 0 reaches its floor only optimistically
    fl = np.array([0.5, 0.0, 0.0], np.float32)
    p = oracle_lib.Problem(3, 1, 12, w.demand, w.slo, fl)
    rev = np.zeros(w.cells, np.uint8)
    with load_model(fsb, w) as m:
        fsb.fs_set_floors(m, fl)
        fsb.fs_update_bounds(m, clo, chi, tlo, thi)
        assert fsb.fs_certificate(m, 0.01) == oracle_lib.certificate(p, clo, chi, tlo, thi, rev, 0.01) == (0, 0.0)
        gm, gp, _ = fsb.fs_solve_bounds(m)
        assert (gm["floors_met"], gp["floors_met"]) == (0, 1)
        assert alloc_matches(gp, oracle_lib.solve(p, chi, tlo), 3)
        clo[0] = chi[0]
        fsb.fs_update_bounds(m, clo, chi, tlo, thi)
        gm, _, _ = fsb.fs_solve_bounds(m)
        ref = oracle_lib.solve(p, clo, thi)
        assert alloc_matches(gm, ref, 3) and ref.replicas[0] > 0 and ref.t_star == 0.0
        assert fsb.fs_certificate(m, 0.01) == (0, 0.0)
        c = [1, 2, 4, 8].index(ref.tp[0]) + ref.bin[0]
        fsb.fs_reveal(m, c, float(clo.reshape(-1)[c]), float(thi.reshape(-1)[c]))
        assert fsb.fs_certificate(m, 0.01) == (1, 0.0)
        fsb.fs_set_floors(m, None)  # without floors the class-2 hole leaves A- empty: nothing to measure
        assert fsb.fs_solve_bounds(m)[0]["replicas"] == [0, 0, 0]


def test_set_floors_rejects_bad_values(fsb, cuda):
    w = workloads.make_workload(0)
    with load_model(fsb, w) as m:
        for bad in ([float("nan"), 0.0], [1.5, 0.0], [-0.1, 0.0]):
            with pytest.raises(fsb.FleetSieveError) as ei:
                fsb.fs_set_floors(m, np.array(bad, np.float32))
            assert ei.value.code == fsb.FS_EINVAL
        fsb.fs_set_floors(m, [0.0, 1.0])
        fsb.fs_set_floors(m, None)
        fsb.fs_score_candidates(m, w.candidates, 4, 8, 0)


def _contested_with_floors(oracle_lib, rng, w):
    """Demand scaled to the widest base gap, then floors drawn around option
    values of both realisations."""
    from test_gpu_score_sweep import _contested

    w = _contested(oracle_lib, w)
    src = (w.cap_lo, w.tail_hi) if rng.random() < 0.5 else (w.cap_hi, w.tail_lo)
    return dataclasses.replace(w, floor=_floors(rng, w, *src, p_crit=0.7))


@pytest.mark.parametrize("seed", range(12))
def test_score_with_floors_random(fsb, cuda, oracle_lib, qn, seed):
    rng = np.random.default_rng(700 + seed)
    K, B, G = int(rng.integers(1, 7)), int(rng.integers(1, 7)), int(rng.integers(2, 49))
    w = _contested_with_floors(oracle_lib, rng, workloads.random_small(rng, K, B, G))
    O, S = int(2 ** rng.integers(0, 4)), int(rng.integers(1, 33))
    s, sid, rnd = int(rng.integers(0, 2**63)), int(rng.integers(0, 100)), int(rng.integers(0, 20))
    with load_model(fsb, w) as m:
        r = fsb.fs_score_candidates(m, w.candidates, O, S, s, sid, rnd)
    ref = oracle_lib.score(w, qn, seed=s, stream_id=sid, rnd=rnd, O=O, S=S)
    assert np.array_equal(r.sum_eo, ref.sum_eo) and np.array_equal(r.score, ref.score)
    assert np.array_equal(r.gap, ref.gap) and r.gamma_t == ref.gamma_t and r.best == ref.best


def test_score_with_floors_paper_scale(fsb, cuda, oracle_lib, qn):
    """The benchmark's workload with Chat critical at a floor between its
    conservative and optimistic t*: every candidate, 8 outcomes x 512 samples."""
    w = workloads.make_workload(1)
    p = oracle_lib.Problem.of(w)
    am, ap, g = oracle_lib.base_gap(p, w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi)
    d = np.float32(0.5 * (am.t_star + ap.t_star))
    w = dataclasses.replace(w, floor=np.array([d, 0.0], np.float32), S=512)
    with load_model(fsb, w) as m:
        r = fsb.fs_score_candidates(m, w.candidates, w.O, w.S, w.seed)
    ref = oracle_lib.score(w, qn)
    assert np.array_equal(r.sum_eo, ref.sum_eo) and np.array_equal(r.score, ref.score)
    assert r.gamma_t == ref.gamma_t and r.best == ref.best
    assert ref.gamma_t > g  # the conservative side misses the floor: t*(A-) drops to 0


def test_dump_records_with_floors(fsb, cuda, oracle_lib, qn):
    """Per-scenario records, including the floor-only allocations of scenarios
    where no positive threshold fits: class 2 is SLO-feasible only when its
    tails come out low, so the conservative side often has t* = 0 while the
    critical class 0 still meets its floor."""
    import torch

    rng = np.random.default_rng(5)
    found_floor_only = 0
    for attempt in range(3):
        w = workloads.random_small(rng, 3, 2, 12)
        tl, th = w.tail_lo.copy(), w.tail_hi.copy()
        tl[2], th[2] = w.slo[2] * np.float32(0.8), w.slo[2] * np.float32(1.3)
        w = dataclasses.replace(w, tail_lo=tl, tail_hi=th)
        w = _contested_with_floors(oracle_lib, rng, w)
        fl = w.floor.copy()
        fl[0] = max(fl[0], np.float32(0.3))
        fl[2] = 0.0
        w = dataclasses.replace(w, floor=fl, O=2, S=24, seed=attempt)
        with load_model(fsb, w) as m:
            stride = fsb.fs_dump_stride(m)
            n = len(w.candidates) * w.O * w.S
            dump = torch.zeros(n * stride, dtype=torch.uint8, device="cuda")
            r = fsb.fs_score_candidates(m, w.candidates, w.O, w.S, w.seed, dump_dev=dump)
        rec = dump.cpu().numpy().view(fsb.dump_dtype(w.K)).reshape(len(w.candidates), w.O, w.S)
        ref = oracle_lib.score(w, qn, dump=True)
        assert np.array_equal(rec["t_star"], ref.dump_t) and np.array_equal(r.sum_eo, ref.sum_eo)
        for e in range(0, len(w.candidates), 2):
            for o in range(w.O):
                for s in range(0, w.S, 5):
                    _, _, am, ap = oracle_lib.scenario(w, qn, int(w.candidates[e]), o, s)
                    x = rec[e, o, s]
                    for sg, a in ((0, am), (1, ap)):
                        assert x["total_gpus"][sg] == a.total_gpus
                        for i in range(w.K):
                            assert fsb.decode_choice(int(x["choice"][sg][i])) == (a.replicas[i], a.tp[i], a.bin[i])
                        found_floor_only += a.t_star == 0.0 and a.total_gpus > 0
    assert found_floor_only > 0


def test_replay_with_floors(fsb, cuda, oracle_lib, qn):
    rp = workloads.make_replay(n_streams=6)
    base = rp.base
    am, ap, _ = oracle_lib.base_gap(oracle_lib.Problem.of(base), base.cap_lo, base.cap_hi, base.tail_lo,
                                    base.tail_hi)
    base = dataclasses.replace(base, floor=np.array([0.5 * (am.t_star + ap.t_star), 0.0], np.float32))
    rp = dataclasses.replace(rp, base=base)
    with load_model(fsb, base) as m:
        res = fsb.fs_replay(m, rp.truth_cap, rp.truth_tail, rp.perm, rp.r0, rp.eps, base.O, 32, 11, rp.max_rounds)
    for k in range(6):
        ref = oracle_lib.replay_stream(rp, k, qn, seed=11, S=32)
        assert res.rounds[k] == ref.rounds and res.state[k] == ref.state
        n = len(ref.reveal_order)
        assert np.array_equal(res.reveal_order[k][:n], ref.reveal_order)
        assert np.array_equal(res.gamma_trace[k][: ref.rounds + 1], ref.gamma_trace)
    # an unreachable floor: every stream stops certified infeasible before any reveal
    bad = dataclasses.replace(base, floor=np.array([1.0, 0.0], np.float32),
                              demand=(base.demand * np.float32(50.0)).astype(np.float32))
    with load_model(fsb, bad) as m:
        res = fsb.fs_replay(m, rp.truth_cap, rp.truth_tail, rp.perm, rp.r0, rp.eps, base.O, 8, 11, 5)
    assert np.all(res.state == 2) and np.all(res.rounds == 0)
    ref = oracle_lib.replay_stream(dataclasses.replace(rp, base=bad), 0, qn, seed=11, S=8, max_rounds=5)
    assert ref.state == 2 and ref.rounds == 0


def test_table_path_with_floors(fsb, cuda, oracle_lib, qn):
    """Floors on the table path (2048 samples per outcome): the segment tables
    gate row terms by the candidate class's floor."""
    w = workloads.make_workload(1)
    p = oracle_lib.Problem.of(w)
    am, ap, _ = oracle_lib.base_gap(p, w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi)
    d = np.float32(0.5 * (am.t_star + ap.t_star))
    w = dataclasses.replace(w, floor=np.array([d, 0.0], np.float32), S=2048,
                            candidates=w.candidates[::8].copy())
    with load_model(fsb, w) as m:
        r = fsb.fs_score_candidates(m, w.candidates, w.O, w.S, w.seed)
    ref = oracle_lib.score(w, qn)
    assert np.array_equal(r.sum_eo, ref.sum_eo) and r.best == ref.best


@pytest.mark.parametrize("K,B,G", [
    (1, 2, 1000),   # row table on both realisations (7500 words)
    (1, 3, 1200),   # row table on one realisation only (6600 and 9000 words)
    (2, 3, 400),    # no row table (9752 and 8712 words): the preparation searches
    (8, 2, 64),     # eight classes, row table of 7968 words
])
def test_score_with_floors_near_row_table_limit(fsb, cuda, oracle_lib, qn, K, B, G):
    """Floors on problems at the base solve's row-table limit: the floor variants
    of the table's costs, counts and kappa walks, and of the search without it."""
    from test_gpu_score_sweep import _contested

    rng = np.random.default_rng(K * 7919 + B * 31 + G + 5)
    w = _contested(oracle_lib, workloads.random_small(rng, K, B, G))
    w = dataclasses.replace(w, floor=_floors(rng, w, w.cap_lo, w.tail_hi, p_crit=1.0))
    assert np.any(w.floor > 0)
    cells = K * 4 * B
    cand = np.sort(rng.choice(cells, size=min(16, cells), replace=False)).astype(np.int32)
    with load_model(fsb, w) as m:
        r = fsb.fs_score_candidates(m, cand, 2, 16, 91, 4, 2)
    ref = oracle_lib.score(w, qn, candidates=cand, seed=91, stream_id=4, rnd=2, O=2, S=16)
    assert np.array_equal(r.sum_eo, ref.sum_eo) and np.array_equal(r.score, ref.score)
    assert r.gamma_t == ref.gamma_t and r.best == ref.best


def test_large_workload_with_floors_sampled(fsb, cuda, oracle_lib, qn):
    """Floors on the eight-class grid at twice its demands (16,384 segments of
    512 samples: the Monte-Carlo kernel's many-segment launch shape), two
    classes critical (A- then misses a floor: Gamma_t = 1): candidates with a
    positive score and a few others, compared in full with the oracle."""
    w = workloads.make_workload(3)
    w = dataclasses.replace(w, demand=(w.demand * np.float32(2.0)).astype(np.float32), S=512)
    fl = np.zeros(w.K, np.float32)
    fl[0] = np.float32(0.5)
    fl[3] = np.float32(0.25)
    w = dataclasses.replace(w, floor=fl)
    with load_model(fsb, w) as m:
        full = fsb.fs_score_candidates(m, w.candidates, w.O, w.S, w.seed)
    pos = np.nonzero(full.score > 0)[0]
    pick = np.unique(np.concatenate([pos[:3], pos[-2:], [0, 1, len(w.candidates) // 2, len(w.candidates) - 1]]))
    se, gt = oracle_lib.score_sums_cached(w, qn, candidates=w.candidates[pick])
    assert gt == full.gamma_t
    assert np.array_equal(full.sum_eo[pick], se)
