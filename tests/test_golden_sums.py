"""The stored expected sums of the large workloads against the oracle (CPU).

tests/golden/make_expected_sums.py writes them with the oracle alone; here a
few candidates of each file are recomputed (the argmax, candidates with a
positive score, candidates without) and the inputs are checked to be the ones
the generator makes today, so that the GPU parity tests that read these files
compare against the oracle's values for the right inputs.
"""

import os
import sys

import numpy as np
import pytest

from conftest import GOLDEN, read_expected_sums

sys.path.insert(0, GOLDEN)
import make_expected_sums as mes  # noqa: E402


@pytest.mark.parametrize("name", sorted(mes.WORKLOADS))
def test_expected_sums_reproduce(oracle_lib, name):
    w = mes.workload(name)
    sha, gamma_t, best, cells, sums = read_expected_sums(mes.WORKLOADS[name][2])
    assert sha == mes.input_digest(w)
    assert np.array_equal(cells, w.candidates) and sums.shape == (len(w.candidates), w.O)
    qn = oracle_lib.triangular_table(4096)
    am, ap, gt = oracle_lib.base_gap(oracle_lib.Problem.of(w), w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi)
    assert gt == gamma_t
    red = oracle_lib.reduce_sums(w, w.candidates, sums, gamma_t)
    assert red.best == best
    pos = np.nonzero(red.score_fixed > 0)[0]
    zero = np.nonzero(red.score_fixed == 0)[0]
    assert len(pos) > 0 and len(zero) > 0
    e_best = int(np.nonzero(w.candidates == best)[0][0])
    pick = np.unique([e_best, pos[0], pos[-1], zero[0], zero[len(zero) // 2]])
    se, g2 = oracle_lib.score_sums_cached(w, qn, candidates=w.candidates[pick])
    assert g2 == gamma_t
    assert np.array_equal(se, sums[pick])
    # the estimator's invariants hold for every stored candidate: 0 <= score <= Gamma_t
    assert np.all(red.score >= 0.0) and np.all(red.score <= gamma_t)


def test_expected_goodput_sums_reproduce(oracle_lib):
    """The stored goodput-stage sums of the paper-scale workload: the inputs,
    the base goodput gap, and the argmax candidate plus four others recomputed
    by the oracle. Sums are nonnegative (a scenario's goodput gap is an
    absolute difference; unlike the max-min gap it has no upper bound in
    Gamma_gp,t, since tier 3 is taken at each realisation's own t*)."""
    from conftest import read_expected_goodput
    from paper_2608_19659_gb300 import workloads

    w = workloads.make_workload(1)
    sha, gamma_fx, gamma_gp, best, cells, sums = read_expected_goodput()
    assert sha == mes.input_digest(w)
    assert np.array_equal(cells, w.candidates) and sums.shape == (len(w.candidates), w.O)
    assert np.all(sums >= 0)
    qn = oracle_lib.triangular_table(4096)
    e_best = int(np.nonzero(w.candidates == best)[0][0])
    pick = np.unique([0, e_best, 17, 40, len(cells) - 1])
    r = oracle_lib.score_goodput(w, qn, candidates=w.candidates[pick])
    assert np.array_equal(r.sum_eo, sums[pick])
    assert r.gamma_fx == gamma_fx and r.gamma_gp == gamma_gp
