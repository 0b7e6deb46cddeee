"""Full-size scoring launches against the oracle's stored sums.

The 8-class workload (1024 candidates x 16 outcomes x 16384 samples, the
largest single-GPU scoring workload) and the 4-class workload at three times
its demands (256 x 8 x 16384) are scored in one fs_score_candidates call each,
in the launch configuration the benchmark times, and every candidate's int64
sum per outcome, its expectation and score, Gamma_t and the argmax must equal
the oracle's (tests/golden/*_sums.txt, written by make_expected_sums.py from
the oracle alone) bit for bit. At its nominal demands the 4-class workload has
spare capacity: Gamma_t = 0 and every score is exactly 0.
"""

import os
import sys

import numpy as np
import pytest

from conftest import GOLDEN, load_model, read_expected_sums
from paper_2608_19659_gb300 import workloads

sys.path.insert(0, GOLDEN)
import make_expected_sums as mes  # noqa: E402

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name", ["large", "mid_x3"])
def test_full_launch_equals_oracle_sums(fsb, cuda, oracle_lib, name):
    w = mes.workload(name)
    sha, gamma_t, best, cells, sums = read_expected_sums(mes.WORKLOADS[name][2])
    assert sha == mes.input_digest(w) and np.array_equal(cells, w.candidates)
    with load_model(fsb, w) as m:
        r = fsb.fs_score_candidates(m, w.candidates, w.O, w.S, w.seed, w.stream_id, w.round)
    assert r.gamma_t == gamma_t
    assert np.array_equal(r.sum_eo, sums), f"{int((r.sum_eo != sums).sum())} sums differ"
    ref = oracle_lib.reduce_sums(w, w.candidates, sums, gamma_t)
    assert np.array_equal(r.gap, ref.gap) and np.array_equal(r.score, ref.score)
    assert r.best == best == ref.best
    assert (ref.score > 0).sum() > 0


def test_mid_workload_nominal_demand_has_no_gap(fsb, cuda, oracle_lib):
    w = workloads.make_workload(2)
    am, ap, gt = oracle_lib.base_gap(oracle_lib.Problem.of(w), w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi)
    assert gt == 0.0 and am.t_star == ap.t_star == 1.0
    with load_model(fsb, w) as m:
        r = fsb.fs_score_candidates(m, w.candidates, w.O, w.S, w.seed)
    full = np.int64(np.rint(np.float64(r.gamma_t) * 2.0**40)) * w.S
    assert r.gamma_t == 0.0 and np.all(r.score == 0.0) and np.all(r.sum_eo == full)
    # every score ties at 0: the argmax is the first TP-1 candidate in the list
    assert r.best == int(w.candidates[(w.candidates // w.B) % 4 == 0][0])
