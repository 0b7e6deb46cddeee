"""Host-side statistics of the acquisition comparison (Section 6.2) and the
oracle's fixed-order replay."""

import numpy as np
import pytest

from paper_2608_19659_gb300 import compare, workloads


def test_grid_order_keeps_the_initial_design():
    rng = np.random.default_rng(1)
    perm = np.stack([rng.permutation(40).astype(np.int32) for _ in range(5)])
    g = compare.grid_order(perm, 6)
    for k in range(5):
        assert list(g[k, :6]) == list(perm[k, :6])
        assert sorted(g[k]) == list(range(40))
        assert list(g[k, 6:]) == sorted(g[k, 6:])


def test_class_gpu_seconds():
    K, B = 2, 3  # cells: class i, TP index j, bin b -> (i*4 + j)*3 + b
    order = np.array([[0, 3, 13, 23, -1], [14, -1, -1, -1, -1]], np.int32)
    s = compare.class_gpu_seconds(order, K, B)
    # cell 0: class 0 TP1; 3: class 0 TP2; 13: class 1 TP1 (13 = (4+0)*3+1); 23: class 1 TP8 ((4+3)*3+2)
    assert np.array_equal(s, [[300.0 + 600.0, 300.0 + 2400.0], [0.0, 300.0]])


def test_ratio_of_means_and_bootstrap():
    base = np.array([10.0, 20.0, 30.0, 40.0])
    ours = 0.9 * base
    assert compare.ratio_of_means_advantage(ours, base) == pytest.approx(0.1)
    # a constant ratio in every pair: every resample gives the same statistic
    lo, hi = compare.paired_bootstrap_ci(ours, base, n_boot=500, seed=3)
    assert lo == pytest.approx(0.1) and hi == pytest.approx(0.1)
    rng = np.random.default_rng(0)
    b = rng.uniform(10, 20, 200)
    o = b * rng.uniform(0.8, 1.05, 200)
    pt = compare.ratio_of_means_advantage(o, b)
    lo, hi = compare.paired_bootstrap_ci(o, b, n_boot=2000, seed=5)
    assert lo < pt < hi and hi - lo < 0.05
    assert (lo, hi) == compare.paired_bootstrap_ci(o, b, n_boot=2000, seed=5)


def test_summarise_per_class():
    K = 2
    base = compare.PolicyRun("b", np.array([10.0, 20.0]), np.array([[4.0, 6.0], [12.0, 8.0]]),
                             np.ones(2, np.int32), np.zeros(2, np.int32))
    ours = compare.PolicyRun("o", np.array([8.0, 20.0]), np.array([[2.0, 6.0], [10.0, 10.0]]),
                             np.ones(2, np.int32), np.zeros(2, np.int32))
    s = compare.summarise(ours, base, n_boot=200)
    assert s["advantage"] == pytest.approx(1 - 14.0 / 15.0) and s["fewer_share"] == 0.5
    assert [c["advantage"] for c in s["per_class"]] == pytest.approx([1 - 6.0 / 8.0, 1 - 8.0 / 7.0])


@pytest.fixture(scope="module")
def replay():
    return workloads.make_replay(n_streams=4)


@pytest.mark.parametrize("k", [0, 1, 2, 3])
def test_oracle_fixed_order_stops_at_the_first_certified_prefix(oracle_lib, replay, k):
    """Policy 1 reveals perm in order; it must stop exactly at the first prefix of
    perm whose revealed state the certificate (Section 4.2) decides."""
    qn = oracle_lib.triangular_table(4096)
    for perm in (replay.perm[k], compare.grid_order(replay.perm, replay.r0)[k]):
        r = oracle_lib.replay_stream(replay, k, qn, seed=1, S=8, policy=1, perm=perm)
        w = replay.base
        p = oracle_lib.Problem.of(w)
        clo, chi = w.cap_lo.reshape(-1).copy(), w.cap_hi.reshape(-1).copy()
        tlo, thi = w.tail_lo.reshape(-1).copy(), w.tail_hi.reshape(-1).copy()
        rev = np.zeros(w.cells, np.uint8)
        stop, state = None, 0
        for j, c in enumerate(perm):
            clo[c] = chi[c] = replay.truth_cap[k][c]
            tlo[c] = thi[c] = replay.truth_tail[k][c]
            rev[c] = 1
            if j + 1 < replay.r0:
                continue
            st, _ = oracle_lib.certificate(p, clo, chi, tlo, thi, rev, replay.eps)
            if st != 0:
                stop, state = j + 1, st
                break
        assert stop is not None
        assert r.state == state and r.rounds == stop - replay.r0
        assert list(r.reveal_order) == list(perm[:stop])
        tp = 1 << ((np.asarray(perm[:stop]) // w.B) % 4)
        assert r.gpu_seconds == 300.0 * tp.sum()
