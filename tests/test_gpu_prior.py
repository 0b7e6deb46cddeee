"""The monotone structural prior (Section 4.1's interval refit, fs_set_prior) on
the GPU against the oracle: each scenario's drawn outcome refits the
candidate's row in both realisations before they are solved, fs_reveal and
the batched replay refit after every reveal. Sums, scores, Gamma_t, the
argmax, dump records (draws, t*, per-class choices with bins) and replay
trajectories must equal the oracle's bit for bit.
"""

import dataclasses

import numpy as np
import pytest

from conftest import load_model
from paper_2608_19659_gb300 import workloads

pytestmark = pytest.mark.gpu

MONO = 1


@pytest.fixture(scope="module")
def qn(oracle_lib):
    return oracle_lib.triangular_table(4096)


def _w(idx, factor=1.0, **kw):
    w = workloads.make_workload(idx)
    return dataclasses.replace(w, demand=(w.demand * np.float32(factor)).astype(np.float32), prior=MONO, **kw)


def _run(fsb, w, cand=None):
    with load_model(fsb, w) as m:
        return fsb.fs_score_candidates(m, w.candidates if cand is None else cand, w.O, w.S, w.seed,
                                       w.stream_id, w.round)


def _same(r, ref, best=True):
    assert r.gamma_t == ref.gamma_t
    assert np.array_equal(r.sum_eo, ref.sum_eo), f"{int((r.sum_eo != ref.sum_eo).sum())} sums differ"
    assert np.array_equal(r.gap, ref.gap) and np.array_equal(r.score, ref.score)
    if best:
        assert r.best == ref.best


@pytest.mark.parametrize("factor", [1.0, 3.0])
def test_tiny_workload_under_the_prior(fsb, cuda, oracle_lib, qn, factor):
    """Plain path (few samples per outcome): literal oracle on every scenario."""
    w = _w(0, factor)
    r = _run(fsb, w)
    ref = oracle_lib.score(w, qn, solver=0)
    _same(r, ref)
    plain = oracle_lib.score(dataclasses.replace(w, prior=0), qn)
    assert np.all(ref.score_fixed >= plain.score_fixed)
    if factor == 3.0:
        assert ref.score.max() > 0 and np.any(ref.score_fixed > plain.score_fixed)


def test_paper_scale_workload_under_the_prior(fsb, cuda, oracle_lib, qn):
    """Table path (2W entries per segment: the closed-gate values depend on the
    position under the prior), all 64 candidates x 8 x 4096."""
    w = _w(1)
    r = _run(fsb, w)
    ref = oracle_lib.score(w, qn)
    _same(r, ref)
    assert (ref.score > 0).sum() > 0


@pytest.mark.parametrize("idx,factor,S", [(2, 3.0, 4096), (3, 2.0, 512)])
def test_larger_workloads_under_the_prior_sampled(fsb, cuda, oracle_lib, qn, idx, factor, S):
    """Four-class and eight-class grids (the latter at twice its demand, with
    contested tables longer than the shared-memory stage): candidates with a
    positive score under the prior and a few others, compared in full."""
    w = _w(idx, factor, S=S)
    full = _run(fsb, w)
    pos = np.nonzero(full.score > 0)[0]
    assert len(pos) > 0
    pick = np.unique(np.concatenate([pos[:3], pos[-2:], [0, len(w.candidates) // 2]]))
    se, gt = oracle_lib.score_sums_cached(w, qn, candidates=w.candidates[pick])
    assert gt == full.gamma_t
    assert np.array_equal(full.sum_eo[pick], se)


def test_dump_records_under_the_prior(fsb, cuda, oracle_lib, qn):
    """Per scenario: the draws, both t*, and every class's choice, including the
    bin of the candidate's refit row."""
    import torch

    w = _w(0, 3.0, S=64)
    K = w.K
    rng = np.random.default_rng(4)
    with load_model(fsb, w) as m:
        stride = fsb.fs_dump_stride(m)
        n = len(w.candidates) * w.O * w.S
        dump = torch.zeros(n * stride, dtype=torch.uint8, device="cuda")
        r = fsb.fs_score_candidates(m, w.candidates, w.O, w.S, w.seed, dump_dev=dump)
    rec = dump.cpu().numpy().view(fsb.dump_dtype(K)).reshape(len(w.candidates), w.O, w.S)
    ref = oracle_lib.score(w, qn, dump=True)
    assert np.array_equal(rec["t_star"], ref.dump_t) and np.array_equal(r.sum_eo, ref.sum_eo)
    for _ in range(200):
        e, o, s = int(rng.integers(len(w.candidates))), int(rng.integers(w.O)), int(rng.integers(w.S))
        cy, ly, am, ap = oracle_lib.scenario(w, qn, int(w.candidates[e]), o, s)
        x = rec[e, o, s]
        assert (x["c_y"], x["l_y"]) == (np.float32(cy), np.float32(ly))
        for sg, a in ((0, am), (1, ap)):
            assert x["total_gpus"][sg] == a.total_gpus
            for i in range(K):
                assert fsb.decode_choice(int(x["choice"][sg][i])) == (a.replicas[i], a.tp[i], a.bin[i])


def test_reveal_refits_the_row(fsb, cuda, oracle_lib):
    w = _w(1)
    prob = oracle_lib.Problem.of(w)
    rng = np.random.default_rng(8)
    b = [w.cap_lo.reshape(-1), w.cap_hi.reshape(-1), w.tail_lo.reshape(-1), w.tail_hi.reshape(-1)]
    with load_model(fsb, w) as m:
        for _ in range(12):
            cell = int(rng.integers(w.cells))
            c = float(np.float32(rng.uniform(0.0, 3.0)))
            ell = float(np.float32(rng.uniform(5.0, 40.0)))
            fsb.fs_reveal(m, cell, c, ell)
            b = oracle_lib.refit(prob, cell, c, ell, *b)
            got = fsb.fs_get_state(m)
            for k in range(4):
                assert np.array_equal(got[k], b[k])
        am, ap, gt = fsb.fs_solve_bounds(m)
    ref = oracle_lib.base_gap(prob, *b)
    assert gt == ref[2] and am["t_star"] == ref[0].t_star and ap["t_star"] == ref[1].t_star


def test_replay_under_the_prior(fsb, cuda, oracle_lib, qn):
    rp = workloads.make_replay(n_streams=10)
    rp = dataclasses.replace(rp, base=dataclasses.replace(rp.base, prior=MONO))
    w = rp.base
    with load_model(fsb, w) as m:
        res = fsb.fs_replay(m, rp.truth_cap, rp.truth_tail, rp.perm, rp.r0, rp.eps, w.O, 32, 2026, rp.max_rounds)
    for k in range(10):
        ref = oracle_lib.replay_stream(rp, k, qn, seed=2026, S=32)
        assert res.rounds[k] == ref.rounds and res.state[k] == ref.state
        n = len(ref.reveal_order)
        assert np.array_equal(res.reveal_order[k][:n], ref.reveal_order)
        assert res.gpu_seconds[k] == ref.gpu_seconds
        assert np.array_equal(res.gamma_trace[k][: ref.rounds + 1], ref.gamma_trace)


def test_floors_with_the_prior(fsb, cuda, oracle_lib, qn):
    w = _w(0, 3.0, S=96, floor=np.array([0.4, 0.0], np.float32))
    r = _run(fsb, w)
    _same(r, oracle_lib.score(w, qn))
