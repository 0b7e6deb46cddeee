"""Pins of the oracle's profiling loop (Algorithm 1) on the replay workload."""

import numpy as np
import pytest

from paper_2608_19659_gb300 import workloads


@pytest.fixture(scope="module")
def replay():
    return workloads.make_replay(n_streams=6)


@pytest.mark.parametrize("k", range(6))
def test_replay_stream_invariants(oracle_lib, replay, k):
    qn = oracle_lib.triangular_table(4096)
    r = oracle_lib.replay_stream(replay, k, qn, seed=2026, S=32)
    w = replay.base
    cells = w.cells
    order = r.reveal_order
    # the common initial design comes first, then one reveal per round
    assert np.array_equal(order[: replay.r0], replay.perm[k][: replay.r0])
    assert len(order) == replay.r0 + r.rounds
    assert len(set(order.tolist())) == len(order)
    # GPU-seconds: 300 s per cell x TP degree (Section 5)
    tp = np.array([1, 2, 4, 8])[(order // w.B) % 4]
    assert r.gpu_seconds == pytest.approx(300.0 * tp.sum())
    # collapsing an interval to a point inside it never widens the gap
    assert np.all(np.diff(r.gamma_trace) <= 0)
    # the loop stops on the certificate (Section 4.2)
    assert r.state == 1 and r.gamma_trace[-1] <= replay.eps
    rev = np.zeros(cells, np.uint8)
    rev[order] = 1
    clo, chi = w.cap_lo.reshape(-1).copy(), w.cap_hi.reshape(-1).copy()
    tlo, thi = w.tail_lo.reshape(-1).copy(), w.tail_hi.reshape(-1).copy()
    for c in order:
        clo[c] = chi[c] = replay.truth_cap[k][c]
        tlo[c] = thi[c] = replay.truth_tail[k][c]
    st, g = oracle_lib.certificate(oracle_lib.Problem.of(w), clo, chi, tlo, thi, rev, replay.eps)
    assert st == 1 and g == r.gamma_trace[-1]
    am = oracle_lib.solve(oracle_lib.Problem.of(w), clo, thi)
    assert am == r.final_minus


def test_replay_with_every_cell_revealed_certifies_at_once(oracle_lib, replay):
    qn = oracle_lib.triangular_table(4096)
    import dataclasses

    full = dataclasses.replace(replay, r0=replay.base.cells)
    r = oracle_lib.replay_stream(full, 0, qn, seed=1, S=8)
    assert r.rounds == 0 and r.state == 1 and r.gamma_trace[0] == 0.0


def test_replay_round_cap(oracle_lib, replay):
    qn = oracle_lib.triangular_table(4096)
    import dataclasses

    never = dataclasses.replace(replay, eps=-1.0)
    r = oracle_lib.replay_stream(never, 1, qn, seed=1, S=8, max_rounds=3)
    assert r.rounds == 3 and r.state == 0


@pytest.mark.parametrize("k", [0, 2, 7, 13])
def test_cached_replay_equals_plain(oracle_lib, k):
    """The replay scored by the cached scorer reveals the same cells in the same
    rounds with the same traces as the one scored scenario by scenario."""
    rp = workloads.make_replay(n_streams=16)
    qn = oracle_lib.triangular_table(4096)
    a = oracle_lib.replay_stream(rp, k, qn, seed=2026, S=96)
    b = oracle_lib.replay_stream(rp, k, qn, seed=2026, S=96, cached=True)
    assert (a.rounds, a.state, a.gpu_seconds) == (b.rounds, b.state, b.gpu_seconds)
    assert np.array_equal(a.reveal_order, b.reveal_order) and np.array_equal(a.gamma_trace, b.gamma_trace)


def test_expected_replay_file(oracle_lib):
    """The stored replay of all 200 reveal orders: the generator's inputs today,
    every stream certified, traces nonincreasing to at most eps, and two streams
    recomputed by the oracle."""
    import sys

    from conftest import GOLDEN, read_expected_replay

    sys.path.insert(0, GOLDEN)
    import make_expected_sums as mes

    rp = workloads.make_replay()
    sha, exp = read_expected_replay()
    assert sha == mes.replay_digest(rp) and sorted(exp) == list(range(200))
    for k, (rounds, state, gs, order, trace) in exp.items():
        assert state == 1 and len(trace) == rounds + 1 and trace[-1] <= rp.eps
        assert len(order) == rp.r0 + rounds and np.all(np.diff(trace) <= 0)
    qn = oracle_lib.triangular_table(4096)
    short = [k for k in range(200) if exp[k][0] <= 2][:2]
    for k in short:
        r = oracle_lib.replay_stream(rp, k, qn, seed=mes.REPLAY_SEED, cached=True)
        rounds, state, gs, order, trace = exp[k]
        assert (r.rounds, r.state, r.gpu_seconds) == (rounds, state, gs)
        assert np.array_equal(r.reveal_order, order) and np.array_equal(r.gamma_trace, trace)
