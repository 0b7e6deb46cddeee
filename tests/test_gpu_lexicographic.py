"""Tiers 3-4 of the lexicographic objective (fs_set_objective) and the goodput
stage of the score (fs_score_goodput) on the GPU against the oracle.

Allocations (per class TP, bin, replicas, fulfilment), GPUs in use and
goodput must equal the oracle's tier-4 solve bit for bit; the stage-wise
certificate the oracle's; the goodput stage's int64 sums, expectations,
scores, Gamma_gp,t and argmax the oracle's.
"""

import dataclasses

import numpy as np
import pytest

from conftest import load_model
from paper_2608_19659_gb300 import workloads

pytestmark = pytest.mark.gpu

LEX = 1


@pytest.fixture(scope="module")
def qn(oracle_lib):
    return oracle_lib.triangular_table(4096)


def _same_alloc(g, a, gp_fx, K):
    assert g["t_star"] == a.t_star and g["total_gpus"] == a.total_gpus and g["floors_met"] == a.floors_met
    assert g["tp"] == a.tp and g["bin"] == a.bin and g["replicas"] == a.replicas
    assert [np.float32(x) for x in g["fulfil"]] == [np.float32(x) for x in a.fulfil]
    assert g["goodput"] == gp_fx * 2.0**-20


@pytest.mark.parametrize("seed", range(30))
def test_solve_matches_oracle(fsb, cuda, oracle_lib, seed):
    rng = np.random.default_rng(seed)
    K = int(rng.integers(1, 5))
    B = int(rng.integers(1, 4))
    G = int(rng.integers(2, 40))
    w = workloads.random_small(rng, K, B, G, p_infeasible=0.15)
    floor = None
    if seed % 3 == 0:
        floor = np.where(rng.random(K) < 0.5, rng.uniform(0.1, 0.9, K), 0.0).astype(np.float32)
    w = dataclasses.replace(w, floor=floor)
    prob = oracle_lib.Problem.of(w)
    with load_model(fsb, w) as m:
        fsb.fs_set_objective(m, LEX)
        for cap, tail in ((w.cap_lo, w.tail_hi), (w.cap_hi, w.tail_lo)):
            g = fsb.fs_solve(m, cap, tail)
            a, gp = oracle_lib.solve_lex(prob, cap, tail)
            _same_alloc(g, a, gp, K)


def test_solve_batch_and_bounds_match_oracle(fsb, cuda, oracle_lib):
    import torch

    for idx, factor in ((1, 1.0), (2, 3.0), (3, 1.0)):
        w = workloads.make_workload(idx)
        w = dataclasses.replace(w, demand=(w.demand * np.float32(factor)).astype(np.float32))
        prob = oracle_lib.Problem.of(w)
        rng = np.random.default_rng(idx)
        n = 12
        u = rng.random((2, n, w.cells)).astype(np.float32)
        cap = (w.cap_lo.reshape(-1) + u[0] * (w.cap_hi - w.cap_lo).reshape(-1)).astype(np.float32)
        tail = (w.tail_lo.reshape(-1) + u[1] * (w.tail_hi - w.tail_lo).reshape(-1)).astype(np.float32)
        with load_model(fsb, w) as m:
            fsb.fs_set_objective(m, LEX)
            out = torch.zeros(n * fsb.ALLOC_DTYPE.itemsize, dtype=torch.uint8, device="cuda")
            fsb.fs_solve_batch(m, n, torch.from_numpy(cap).cuda(), torch.from_numpy(tail).cuda(), out)
            fsb.fs_check(m)
            got = out.cpu().numpy().view(fsb.ALLOC_DTYPE)
            for r in range(n):
                a, gp = oracle_lib.solve_lex(prob, cap[r], tail[r])
                assert got[r]["total_gpus"] == a.total_gpus and got[r]["goodput"] == gp * 2.0**-20
                assert list(got[r]["replicas"][: w.K]) == a.replicas and list(got[r]["tp"][: w.K]) == a.tp
                assert list(got[r]["bin"][: w.K]) == a.bin
            am, ap, gt = fsb.fs_solve_bounds(m)
        ref = oracle_lib.base_gap_lex(prob, w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi)
        _same_alloc(am, ref[0], ref[2], w.K)
        _same_alloc(ap, ref[1], ref[3], w.K)
        assert gt == ref[4]


def test_table3_on_the_gpu(fsb, cuda, oracle_lib):
    t1 = {"chat": [0.798, 1.649, 1.408], "code": [0.560, 2.779, 1.392]}
    for scale, gp_paper in ((0.7, 19.60), (1.0, 28.00), (1.3, 33.99)):
        cap = np.ones((2, 4, 1), np.float32)
        tail = np.full((2, 4, 1), 1e9, np.float32)
        for i, k in enumerate(["chat", "code"]):
            for j, tp in enumerate([2, 4, 8]):
                cap[i, j + 1, 0] = np.float32(t1[k][j] * tp)
                tail[i, j + 1, 0] = 10.0
        lam = np.array([12.0 * scale, 16.0 * scale], np.float32)
        m = fsb.fs_load_model(cap, cap, tail, tail, [30.0, 30.0], lam, 16, 2, 1)
        with m:
            fsb.fs_set_objective(m, LEX)
            g = fsb.fs_solve(m, cap, tail)
        assert g["tp"] == [4, 4] and g["replicas"] == [2, 2] and abs(g["goodput"] - gp_paper) <= 0.01


def test_stagewise_certificate(fsb, cuda, oracle_lib):
    """No max-min gap but a goodput gap of 0.25: the max-min objective certifies,
    the lexicographic one waits until eps reaches the goodput gap."""
    from test_oracle_lexicographic import _stagewise_instance

    K, B, G, lam, slo, clo, chi, tlo, thi, rev = _stagewise_instance()
    with fsb.fs_load_model(clo, chi, tlo, thi, slo, lam, G, K, B, revealed=rev) as m:
        assert fsb.fs_certificate(m, 0.01) == (1, 0.0)
        fsb.fs_set_objective(m, LEX)
        assert fsb.fs_certificate(m, 0.01) == (0, 0.0)
        assert fsb.fs_certificate(m, 0.25) == (1, 0.0)
        am, ap, _ = fsb.fs_solve_bounds(m)
    assert (am["goodput"], ap["goodput"]) == (4.0, 6.0)
    assert am["replicas"] == [1, 4] and ap["tp"] == [8, 2] and ap["replicas"] == [1, 2]


@pytest.mark.parametrize("idx,factor,S,n_cand", [(0, 3.0, 256, None), (1, 1.0, 512, 24), (2, 3.0, 256, 12)])
def test_goodput_stage_matches_oracle(fsb, cuda, oracle_lib, qn, idx, factor, S, n_cand):
    w = workloads.make_workload(idx)
    w = dataclasses.replace(w, demand=(w.demand * np.float32(factor)).astype(np.float32), S=S)
    cand = w.candidates if n_cand is None else w.candidates[:: max(1, len(w.candidates) // n_cand)][:n_cand]
    with load_model(fsb, w) as m:
        r = fsb.fs_score_goodput(m, cand, w.O, w.S, w.seed)
    ref = oracle_lib.score_goodput(w, qn, candidates=cand)
    assert np.array_equal(r.sum_eo, ref.sum_eo), f"{int((r.sum_eo != ref.sum_eo).sum())} sums differ"
    assert np.array_equal(r.gap, ref.gap) and np.array_equal(r.score, ref.score)
    assert r.gamma_gp == ref.gamma_gp and r.best == ref.best
    assert ref.gamma_fx > 0 and np.any(ref.score_fixed != 0)


def test_goodput_stage_large_workload_sampled(fsb, cuda, oracle_lib, qn):
    """The goodput stage on the eight-class grid (G = 256: the largest programme
    over GPUs of the workloads) at twice its demands, every candidate scored:
    candidates with a positive goodput score and a few others against the
    oracle in full."""
    w = workloads.make_workload(3)
    w = dataclasses.replace(w, demand=(w.demand * np.float32(2.0)).astype(np.float32), S=64)
    with load_model(fsb, w) as m:
        full = fsb.fs_score_goodput(m, w.candidates, w.O, w.S, w.seed)
    pos = np.nonzero(full.score > 0)[0]
    assert len(pos) > 0
    pick = np.unique(np.concatenate([pos[:2], pos[-1:], [0, len(w.candidates) // 2]]))
    ref = oracle_lib.score_goodput(w, qn, candidates=w.candidates[pick])
    assert np.array_equal(full.sum_eo[pick], ref.sum_eo)
    assert np.array_equal(full.gap[pick], ref.gap) and np.array_equal(full.score[pick], ref.score)
    assert full.gamma_gp == ref.gamma_gp


@pytest.mark.parametrize("prior,floor", [(1, None), (0, (0.4, 0.0)), (1, (0.0, 0.5))])
def test_goodput_stage_with_prior_and_floors(fsb, cuda, oracle_lib, qn, prior, floor):
    w = workloads.make_workload(0)
    w = dataclasses.replace(w, demand=(w.demand * np.float32(3.0)).astype(np.float32), S=128, prior=prior,
                            floor=None if floor is None else np.array(floor, np.float32))
    with load_model(fsb, w) as m:
        r = fsb.fs_score_goodput(m, w.candidates, w.O, w.S, w.seed, 3, 2)
    ref = oracle_lib.score_goodput(w, qn, stream_id=3, rnd=2)
    assert np.array_equal(r.sum_eo, ref.sum_eo) and r.best == ref.best
    assert np.array_equal(r.score, ref.score) and r.gamma_gp == ref.gamma_gp


@pytest.mark.parametrize("K,B,G,prior,factor", [(10, 4, 40, 0, 3.0), (12, 3, 100, 1, 6.0)])
def test_goodput_stage_many_rows(fsb, cuda, oracle_lib, qn, K, B, G, prior, factor):
    """More rows than a warp has lanes (4K = 40, 48: each lane takes two rows'
    replica ranges) and more GPU counts than lanes (G + 1 = 41, 101: several
    cells per lane in each class step), without and with the prior."""
    rng = np.random.default_rng(100 + K)
    w = workloads.random_small(rng, K, B, G)
    cand = np.sort(rng.choice(len(w.candidates), 12, replace=False)).astype(np.int32)
    w = dataclasses.replace(w, candidates=cand, O=8, S=64, prior=prior,
                            demand=(w.demand * np.float32(factor)).astype(np.float32))
    with load_model(fsb, w) as m:
        r = fsb.fs_score_goodput(m, cand, w.O, w.S, w.seed)
    ref = oracle_lib.score_goodput(w, qn, candidates=cand)
    assert np.array_equal(r.sum_eo, ref.sum_eo), f"{int((r.sum_eo != ref.sum_eo).sum())} sums differ"
    assert np.array_equal(r.score, ref.score) and r.gamma_gp == ref.gamma_gp and r.best == ref.best
    assert ref.gamma_fx > 0 and np.all(ref.sum_eo != 0)


def test_goodput_stage_table_limit(fsb, cuda, oracle_lib, qn):
    """A segment's table of Q / O positions lives in shared memory: one outcome
    (Q / O = 4096 positions) is refused under the monotone prior (8192
    entries) and scored without it (4097 entries), equal to the oracle."""
    w = workloads.make_workload(0)
    w = dataclasses.replace(w, demand=(w.demand * np.float32(3.0)).astype(np.float32), O=1, S=512)
    cand = w.candidates[:4]
    with load_model(fsb, dataclasses.replace(w, prior=1)) as m:
        with pytest.raises(fsb.FleetSieveError) as ei:
            fsb.fs_score_goodput(m, cand, 1, w.S, w.seed)
        assert ei.value.code == fsb.FS_EINVAL
    with load_model(fsb, w) as m:
        r = fsb.fs_score_goodput(m, cand, 1, w.S, w.seed)
    ref = oracle_lib.score_goodput(w, qn, candidates=cand)
    assert np.array_equal(r.sum_eo, ref.sum_eo) and r.best == ref.best and r.gamma_gp == ref.gamma_gp


def test_goodput_stage_paper_scale_full(fsb, cuda):
    """The goodput stage on the paper-scale workload in full (64 candidates x
    8 outcomes x 4096 samples, the bench's configuration): every int64 sum,
    Gamma_gp,t and the argmax equal the oracle's stored values (tests/golden,
    written by the oracle alone)."""
    import sys

    from conftest import GOLDEN, read_expected_goodput

    sys.path.insert(0, GOLDEN)
    import make_expected_sums as mes

    w = workloads.make_workload(1)
    sha, gamma_fx, gamma_gp, best, cells, sums = read_expected_goodput()
    assert sha == mes.input_digest(w)
    with load_model(fsb, w) as m:
        r = fsb.fs_score_goodput(m, w.candidates, w.O, w.S, w.seed)
    assert np.array_equal(r.sum_eo, sums), f"{int((r.sum_eo != sums).sum())} sums differ"
    assert r.gamma_gp == gamma_gp and r.best == best
