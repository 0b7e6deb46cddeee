"""Batched profiling loop (fs_replay, Algorithm 1) against the oracle's per-stream replay."""

import numpy as np
import pytest

from conftest import load_model
from paper_2608_19659_gb300 import workloads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def qn(oracle_lib):
    return oracle_lib.triangular_table(4096)


def _gpu_replay(fsb, rp, S, seed, max_rounds=None):
    w = rp.base
    mr = rp.max_rounds if max_rounds is None else max_rounds
    with load_model(fsb, w) as m:
        return fsb.fs_replay(m, rp.truth_cap, rp.truth_tail, rp.perm, rp.r0, rp.eps, w.O, S, seed, mr)


def _compare(fsb, res, rp, k, ref, K):
    assert res.rounds[k] == ref.rounds and res.state[k] == ref.state
    assert res.gpu_seconds[k] == ref.gpu_seconds
    n = len(ref.reveal_order)
    assert np.array_equal(res.reveal_order[k][:n], ref.reveal_order)
    assert np.all(res.reveal_order[k][n:] == -1)
    assert np.array_equal(res.gamma_trace[k][: ref.rounds + 1], ref.gamma_trace)
    f = res.final_minus[k]
    a = ref.final_minus
    assert float(f["t_star"]) == a.t_star and int(f["total_gpus"]) == a.total_gpus
    assert [int(x) for x in f["tp"][:K]] == a.tp and [int(x) for x in f["bin"][:K]] == a.bin
    assert [int(x) for x in f["replicas"][:K]] == a.replicas


def test_replay_small_samples_matches_oracle(fsb, cuda, oracle_lib, qn):
    rp = workloads.make_replay(n_streams=12)
    res = _gpu_replay(fsb, rp, S=32, seed=2026)
    for k in range(12):
        ref = oracle_lib.replay_stream(rp, k, qn, seed=2026, S=32)
        _compare(fsb, res, rp, k, ref, rp.base.K)


def test_replay_round_cap_and_full_initial_design(fsb, cuda, oracle_lib, qn):
    import dataclasses

    rp = dataclasses.replace(workloads.make_replay(n_streams=3), eps=-1.0)
    res = _gpu_replay(fsb, rp, S=8, seed=1, max_rounds=4)
    for k in range(3):
        ref = oracle_lib.replay_stream(rp, k, qn, seed=1, S=8, max_rounds=4)
        assert res.rounds[k] == 4 and res.state[k] == 0
        _compare(fsb, res, rp, k, ref, rp.base.K)
    full = dataclasses.replace(workloads.make_replay(n_streams=2), r0=64)
    res = _gpu_replay(fsb, full, S=8, seed=1)
    assert np.all(res.rounds == 0) and np.all(res.state == 1) and np.all(res.gamma_trace[:, 0] == 0)


def test_replay_full_size(fsb, cuda, oracle_lib, qn):
    """The replay workload in full: 200 reveal orders x (unrevealed x 8 x 4096)
    per round; every stream's rounds, state, GPU-seconds, reveal order and
    Gamma_t trace equal the oracle's stored replay (tests/golden, oracle only),
    and stream 0 is also replayed by the oracle here."""
    import sys

    from conftest import GOLDEN, read_expected_replay

    sys.path.insert(0, GOLDEN)
    import make_expected_sums as mes

    rp = workloads.make_replay()
    sha, exp = read_expected_replay()
    assert sha == mes.replay_digest(rp)
    res = _gpu_replay(fsb, rp, S=4096, seed=mes.REPLAY_SEED)
    assert np.all(res.state == 1)
    for k in range(200):
        rounds, state, gs, order, trace = exp[k]
        assert res.rounds[k] == rounds and res.state[k] == state and res.gpu_seconds[k] == gs, k
        assert np.array_equal(res.reveal_order[k][: len(order)], order) and np.all(res.reveal_order[k][len(order):] == -1)
        assert np.array_equal(res.gamma_trace[k][: rounds + 1], trace), k
    ref = oracle_lib.replay_stream(rp, 0, qn, seed=2026, S=4096)
    _compare(fsb, res, rp, 0, ref, rp.base.K)


def test_replay_rejects_bad_specs(fsb, cuda):
    rp = workloads.make_replay(n_streams=2)
    bad = rp.perm.copy()
    bad[1, 3] = bad[1, 4]
    w = rp.base
    with load_model(fsb, w) as m:
        with pytest.raises(fsb.FleetSieveError):
            fsb.fs_replay(m, rp.truth_cap, rp.truth_tail, bad, 6, 0.01, 8, 16, 1, 64)
        with pytest.raises(fsb.FleetSieveError):
            fsb.fs_replay(m, rp.truth_cap, rp.truth_tail, rp.perm, 6, 0.01, 3, 16, 1, 64)


def test_fixed_order_policies_match_oracle(fsb, cuda, oracle_lib, qn):
    """Section 6.2's fixed-order baselines (uniform random, fixed grid order) on the
    GPU replay: same stop, state, order, GPU-seconds and final allocation as the oracle."""
    from paper_2608_19659_gb300 import compare

    rp = workloads.make_replay(n_streams=10)
    w = rp.base
    for perm in (rp.perm, compare.grid_order(rp.perm, rp.r0)):
        with load_model(fsb, w) as m:
            res = fsb.fs_replay(m, rp.truth_cap, rp.truth_tail, perm, rp.r0, rp.eps, w.O, 16, 3,
                                rp.max_rounds, policy=1)
        for k in range(10):
            ref = oracle_lib.replay_stream(rp, k, qn, seed=3, S=16, policy=1, perm=perm[k])
            _compare(fsb, res, rp, k, ref, w.K)


def test_policy_comparison_runs(fsb, cuda):
    from paper_2608_19659_gb300 import compare

    rp = workloads.make_replay(n_streams=8)
    w = rp.base
    with load_model(fsb, w) as m:
        runs = compare.run_policies(m, rp, 4, 32, 7)
        with pytest.raises(fsb.FleetSieveError):
            fsb.fs_replay(m, rp.truth_cap, rp.truth_tail, rp.perm, rp.r0, rp.eps, 4, 32, 7, 10, policy=2)
    assert set(runs) == {"fleetsieve", "uniform_random", "fixed_grid"}
    for r in runs.values():
        assert np.all(r.state == 1)
        assert np.allclose(r.class_seconds.sum(axis=1), r.gpu_seconds)
    s = compare.summarise(runs["fleetsieve"], runs["uniform_random"], n_boot=200)
    lo, hi = s["ci95"]
    assert lo <= s["advantage"] <= hi and len(s["per_class"]) == w.K
