"""Loading a model with cells already measured, and checkpoint / resume of the
profiling loop (Algorithm 1) through fs_get_state.

The loop runs on the host here, one fs_score_candidates per round (candidates
in reveal-order position, Philox stream k, round r), exactly as the oracle's
replay of stream k does; it is interrupted after a few rounds, its state saved
to a file and loaded into a fresh model, and the resumed loop must reveal the
same cells, stop in the same round with the same certificate, and match the
oracle's uninterrupted replay.
"""

import numpy as np
import pytest

from paper_2608_19659_gb300 import workloads

pytestmark = pytest.mark.gpu

S = 64


def _loop(fsb, m, rp, k, start_round, stop_after=None):
    """Rounds of Algorithm 1 from start_round; returns (revealed cells, state, last round)."""
    w = rp.base
    perm = rp.perm[k]
    tc, tl = rp.truth_cap[k], rp.truth_tail[k]
    order = []
    r = start_round
    while True:
        state, _ = fsb.fs_certificate(m, rp.eps)
        if state != 0:
            return order, state, r
        rev = fsb.fs_get_state(m)[4]
        cand = np.array([c for c in perm if not rev[c]], np.int32)
        if len(cand) == 0 or (stop_after is not None and r >= stop_after):
            return order, 0, r
        res = fsb.fs_score_candidates(m, cand, w.O, S, 2026, k, r)
        fsb.fs_reveal(m, res.best, float(tc[res.best]), float(tl[res.best]))
        order.append(res.best)
        r += 1


def _fresh(fsb, rp, k):
    w = rp.base
    clo, chi = w.cap_lo.reshape(-1).copy(), w.cap_hi.reshape(-1).copy()
    tlo, thi = w.tail_lo.reshape(-1).copy(), w.tail_hi.reshape(-1).copy()
    rev = np.zeros(w.cells, np.uint8)
    for c in rp.perm[k][: rp.r0]:  # the common initial design, measured before round 0
        clo[c] = chi[c] = rp.truth_cap[k][c]
        tlo[c] = thi[c] = rp.truth_tail[k][c]
        rev[c] = 1
    return fsb.fs_load_model(clo, chi, tlo, thi, w.slo, w.demand, w.G, w.K, w.B, revealed=rev)


@pytest.mark.parametrize("k", [2, 7])  # streams that take 7 and 9 rounds at this sample size
def test_checkpoint_resume_equals_uninterrupted_loop_and_oracle(fsb, cuda, oracle_lib, tmp_path, k):
    rp = workloads.make_replay(n_streams=8)
    w = rp.base
    with _fresh(fsb, rp, k) as m:
        full_order, full_state, full_rounds = _loop(fsb, m, rp, k, 0)
    assert full_state == 1 and full_rounds >= 4
    with _fresh(fsb, rp, k) as m:
        first, st, r = _loop(fsb, m, rp, k, 0, stop_after=3)
        assert st == 0 and r == 3
        path = str(tmp_path / "state.npz")
        fsb.save_state(m, path, round=r)
    m2, r2, _ = fsb.load_state(path, w.slo, w.demand)
    with m2:
        assert r2 == 3
        rest, st2, rounds2 = _loop(fsb, m2, rp, k, r2)
    assert first + rest == full_order and st2 == full_state and rounds2 == full_rounds
    ref = oracle_lib.replay_stream(rp, k, oracle_lib.triangular_table(4096), seed=2026, S=S)
    assert ref.state == full_state and ref.rounds == full_rounds
    assert list(ref.reveal_order[rp.r0:]) == full_order


def test_loaded_revealed_flags_drive_the_certificate(fsb, cuda, oracle_lib):
    """The same collapsed bounds certify only when their cells are loaded as revealed."""
    rp = workloads.make_replay(n_streams=4)
    w = rp.base
    with _fresh(fsb, rp, 3) as m:
        _loop(fsb, m, rp, 3, 0)
        clo, chi, tlo, thi, rev = fsb.fs_get_state(m)
        st, gt = fsb.fs_certificate(m, rp.eps)
    assert st == 1 and rev.sum() > rp.r0
    ref_st, ref_gt = oracle_lib.certificate(oracle_lib.Problem.of(w), clo, chi, tlo, thi, rev, rp.eps)
    assert (ref_st, ref_gt) == (st, gt)
    with fsb.fs_load_model(clo, chi, tlo, thi, w.slo, w.demand, w.G, w.K, w.B, revealed=rev) as m:
        assert fsb.fs_certificate(m, rp.eps) == (st, gt)
        assert np.array_equal(fsb.fs_get_state(m)[4], rev)
    with fsb.fs_load_model(clo, chi, tlo, thi, w.slo, w.demand, w.G, w.K, w.B) as m:
        st0, gt0 = fsb.fs_certificate(m, rp.eps)
    ref0 = oracle_lib.certificate(oracle_lib.Problem.of(w), clo, chi, tlo, thi, np.zeros_like(rev), rp.eps)
    assert (st0, gt0) == ref0 and st0 == 0 and gt0 == gt
