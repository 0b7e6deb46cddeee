"""GPU allocation solver (fs_solve, fs_solve_batch, fs_solve_bounds) against the CPU oracle."""

import dataclasses

import numpy as np
import pytest

from conftest import alloc_matches, load_model, read_golden
from paper_2608_19659_gb300 import workloads

pytestmark = pytest.mark.gpu


def _realisations(rng, w, n):
    """n realisations inside the bounds, with ties, infeasible classes and extremes mixed in."""
    shape = (n,) + w.cap_lo.shape
    u = rng.random(shape).astype(np.float32)
    cap = (w.cap_lo + u * (w.cap_hi - w.cap_lo)).astype(np.float32)
    v = rng.random(shape).astype(np.float32)
    tail = (w.tail_lo + v * (w.tail_hi - w.tail_lo)).astype(np.float32)
    for r in range(n):
        kind = r % 6
        if kind == 1:
            cap[r] = w.cap_lo
            tail[r] = w.tail_hi
        elif kind == 2:
            cap[r] = w.cap_hi
            tail[r] = w.tail_lo
        elif kind == 3:  # equal capacities across bins: bin tie rule
            cap[r] = np.repeat(cap[r][:, :, :1], w.B, axis=2)
        elif kind == 4:  # a class without any SLO-feasible cell
            i = r % w.K
            tail[r][i] = w.slo[i] * 2
        elif kind == 5:  # some zero capacities
            cap[r][rng.random(cap[r].shape) < 0.3] = 0.0
    return cap.reshape(n, -1), tail.reshape(n, -1)


def _solve_batch(fsb, torch, m, cap, tail):
    n = cap.shape[0]
    dc = torch.from_numpy(cap).cuda()
    dt = torch.from_numpy(tail).cuda()
    out = torch.zeros(n * fsb.ALLOC_DTYPE.itemsize, dtype=torch.uint8, device="cuda")
    fsb.fs_solve_batch(m, n, dc, dt, out)
    fsb.fs_check(m)
    torch.cuda.synchronize()
    return out.cpu().numpy().view(fsb.ALLOC_DTYPE)


def _as_dict(rec, K):
    return {"t_star": float(rec["t_star"]), "total_gpus": int(rec["total_gpus"]), "ok": int(rec["ok"]),
            "floors_met": int(rec["floors_met"]), "has_option_mask": int(rec["has_option_mask"]), "tp": [int(x) for x in rec["tp"][:K]],
            "bin": [int(x) for x in rec["bin"][:K]], "replicas": [int(x) for x in rec["replicas"][:K]],
            "fulfil": [float(x) for x in rec["fulfil"][:K]]}


@pytest.mark.parametrize("seed", range(24))
def test_solve_batch_matches_oracle(fsb, cuda, oracle_lib, seed):
    rng = np.random.default_rng(40 + seed)
    K = int(rng.integers(1, 9))
    B = int(rng.integers(1, 9))
    G = int(rng.integers(1, 65))
    w = workloads.random_small(rng, K, B, G)
    cap, tail = _realisations(rng, w, 48)
    p = oracle_lib.Problem.of(w)
    with load_model(fsb, w) as m:
        recs = _solve_batch(fsb, cuda, m, cap, tail)
    for r in range(cap.shape[0]):
        literal = r % 4 == 0 and K * B * G <= 1024
        ref = oracle_lib.solve(p, cap[r], tail[r], 0 if literal else 1)
        assert alloc_matches(_as_dict(recs[r], K), ref, K), (seed, r)


@pytest.mark.parametrize("K,B,G", [(64, 2, 32), (8, 32, 256), (1, 1, 1), (1, 4096, 8), (3, 5, 1)])
def test_solve_batch_extreme_sizes(fsb, cuda, oracle_lib, K, B, G):
    rng = np.random.default_rng(K * 1000 + B + G)
    w = workloads.random_small(rng, K, B, G)
    cap, tail = _realisations(rng, w, 12)
    p = oracle_lib.Problem.of(w)
    with load_model(fsb, w) as m:
        recs = _solve_batch(fsb, cuda, m, cap, tail)
    for r in range(cap.shape[0]):
        assert alloc_matches(_as_dict(recs[r], K), oracle_lib.solve(p, cap[r], tail[r]), K)


def test_fs_solve_table3_and_tail_rejection(fsb, cuda, oracle_lib):
    t1 = {"chat": [0.798, 1.649, 1.408], "code": [0.560, 2.779, 1.392]}
    rows = [r for r in read_golden("table3_allocation.txt") if r[1] == "oracle"]
    for r in rows:
        scale = float(r[0])
        cap = np.ones((2, 4, 1), np.float32)
        tail = np.full((2, 4, 1), 1e9, np.float32)
        for i, k in enumerate(["chat", "code"]):
            for j, tp in enumerate([2, 4, 8]):
                cap[i, j + 1, 0] = np.float32(t1[k][j] * tp)
                tail[i, j + 1, 0] = 10.0
        lam = np.array([12.0 * scale, 16.0 * scale], np.float32)
        w = workloads.Workload("t3", 2, 1, 16, lam, np.array([30.0, 30.0], np.float32), cap, cap, tail, tail,
                               np.arange(8, dtype=np.int32), 1, 1, 0)
        with load_model(fsb, w) as m:
            a = fsb.fs_solve(m, cap, tail)
        assert a["tp"] == [int(r[2]), int(r[3])] and a["replicas"] == [int(r[4]), int(r[5])]
        assert abs(a["t_star"] - float(r[6])) <= 0.001
    rows = read_golden("c128_tail_rejection.txt")
    cap = np.zeros((1, 4, 1), np.float32)
    tail = np.full((1, 4, 1), 1e9, np.float32)
    for rr in rows:
        if rr[0] in ("4", "8"):
            j = {"4": 2, "8": 3}[rr[0]]
            cap[0, j, 0], tail[0, j, 0] = float(rr[1]), float(rr[2])
    for slo, want in ((30.0, 8), (60.0, 4)):
        w = workloads.Workload("c128", 1, 1, 8, np.array([11.27], np.float32), np.array([slo], np.float32),
                               cap, cap, tail, tail, np.arange(4, dtype=np.int32), 1, 1, 0)
        with load_model(fsb, w) as m:
            a = fsb.fs_solve(m, cap, tail)
        assert a["tp"] == [want] and a["replicas"] == [1] and a["t_star"] == 1.0


@pytest.mark.parametrize("idx", [0, 1, 2, 3])
def test_solve_bounds_matches_oracle(fsb, cuda, oracle_lib, idx):
    w = workloads.make_workload(idx)
    p = oracle_lib.Problem.of(w)
    am, ap, g = oracle_lib.base_gap(p, w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi)
    with load_model(fsb, w) as m:
        gm, gp, gg = fsb.fs_solve_bounds(m)
    assert alloc_matches(gm, am, w.K) and alloc_matches(gp, ap, w.K) and gg == g
    assert gm["t_star"] <= gp["t_star"]


def test_collapsed_bounds_have_zero_gap(fsb, cuda):
    w = workloads.make_workload(1)
    w = dataclasses.replace(w, cap_hi=w.cap_lo.copy(), tail_lo=w.tail_hi.copy())
    with load_model(fsb, w) as m:
        gm, gp, g = fsb.fs_solve_bounds(m)
    assert g == 0.0 and gm == gp


def test_reveal_and_certificate(fsb, cuda, oracle_lib):
    w = workloads.make_workload(1)
    p = oracle_lib.Problem.of(w)
    rng = np.random.default_rng(5)
    rev = np.zeros(w.cells, np.uint8)
    clo, chi = w.cap_lo.reshape(-1).copy(), w.cap_hi.reshape(-1).copy()
    tlo, thi = w.tail_lo.reshape(-1).copy(), w.tail_hi.reshape(-1).copy()
    with load_model(fsb, w) as m:
        for c in rng.permutation(w.cells)[:40]:
            vc = float(np.float32(clo[c] + 0.37 * (chi[c] - clo[c])))
            vl = float(np.float32(tlo[c] + 0.61 * (thi[c] - tlo[c])))
            fsb.fs_reveal(m, int(c), vc, vl)
            clo[c] = chi[c] = vc
            tlo[c] = thi[c] = vl
            rev[c] = 1
            for eps in (0.0, 0.05, 1.0):
                assert fsb.fs_certificate(m, eps) == oracle_lib.certificate(p, clo, chi, tlo, thi, rev, eps)
        with pytest.raises(fsb.FleetSieveError):
            fsb.fs_reveal(m, w.cells, 1.0, 1.0)
        with pytest.raises(fsb.FleetSieveError):
            fsb.fs_reveal(m, 0, float("nan"), 1.0)


def test_update_bounds(fsb, cuda, oracle_lib):
    w1 = workloads.make_workload(1)
    w3 = dataclasses.replace(w1, demand=(w1.demand * 0.5).astype(np.float32))
    p = oracle_lib.Problem.of(w1)
    with load_model(fsb, w3) as m:
        fsb.fs_update_bounds(m, w1.cap_hi, w1.cap_hi, w1.tail_lo, w1.tail_lo)
        gm, gp, g = fsb.fs_solve_bounds(m)
    ref = oracle_lib.solve(oracle_lib.Problem.of(w3), w1.cap_hi, w1.tail_lo)
    assert alloc_matches(gm, ref, w1.K) and g == 0.0
    assert p.K == 2
