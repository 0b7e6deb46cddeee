"""The allocation-free scoring entry point against the allocating one.

fs_score_candidates_noalloc exists for callers that cannot allocate device
memory while they run (memory already handed out by their own pool, or no
room for cudaMalloc's device-wide synchronisation on their path). It keeps all
intermediates in the library's fixed device array, so these tests check that
two calls in a row (the second reusing whatever the first left in the array)
give exactly the allocating entry point's results, and that a call too large
for the array is refused cleanly. This file is collected last on purpose.
"""

import dataclasses

import numpy as np
import pytest

from conftest import load_model
from paper_2608_19659_gb300 import workloads

pytestmark = pytest.mark.gpu


def _device_inputs(torch, w):
    bounds = np.concatenate([w.cap_lo.reshape(-1), w.cap_hi.reshape(-1), w.tail_lo.reshape(-1),
                             w.tail_hi.reshape(-1)]).astype(np.float32)
    return (torch.from_numpy(bounds).cuda(), torch.from_numpy(w.slo.copy()).cuda(),
            torch.from_numpy(w.demand.copy()).cuda(), torch.from_numpy(w.candidates.copy()).cuda())


@pytest.mark.parametrize("idx,factor", [(1, 1.0), (2, 3.0)])
def test_noalloc_matches_allocating_entry_point_on_two_calls(fsb, cuda, idx, factor):
    torch = cuda
    w = workloads.make_workload(idx)
    w = dataclasses.replace(w, demand=(w.demand * factor).astype(np.float32), S=min(w.S, 4096))
    bounds, slo, lam, cand = _device_inputs(torch, w)
    n = len(w.candidates)
    stream = torch.cuda.current_stream()
    with load_model(fsb, w) as m:
        for rnd in (0, 1):  # two calls in a row through the shared array
            ref = fsb.fs_score_candidates(m, w.candidates, w.O, w.S, w.seed, 0, rnd)
            gap = torch.full((n,), float("nan"), dtype=torch.float64, device="cuda")
            score = torch.full((n,), float("nan"), dtype=torch.float64, device="cuda")
            gt = torch.full((1,), float("nan"), dtype=torch.float32, device="cuda")
            best = torch.full((1,), -7, dtype=torch.int32, device="cuda")
            fsb.fs_score_candidates_noalloc(w.K, w.B, w.G, bounds, slo, lam, cand, w.O, w.S, w.seed, 0, rnd,
                                            gap_dev=gap, score_dev=score, gamma_t_dev=gt, best_dev=best,
                                            stream=stream)
            # the fixed-point sums make both paths bit-identical: tolerance zero
            assert np.array_equal(gap.cpu().numpy(), ref.gap)
            assert np.array_equal(score.cpu().numpy(), ref.score)
            assert float(gt.item()) == ref.gamma_t and int(best.item()) == ref.best
    if factor != 1.0:
        assert ref.score.max() > 0


def test_noalloc_refuses_calls_beyond_its_array(fsb, cuda):
    torch = cuda
    w = workloads.make_workload(3)  # 1024 candidates x 2 tables of 16 + 3 * 4096 floats: ~100 MB
    bounds, slo, lam, cand = _device_inputs(torch, w)
    with pytest.raises(fsb.FleetSieveError) as ei:
        fsb.fs_score_candidates_noalloc(w.K, w.B, w.G, bounds, slo, lam, cand, w.O, w.S, w.seed)
    assert ei.value.code == fsb.FS_EINVAL and "scratch" in str(ei.value)
    # a smaller slice of the same problem fits and matches the allocating path
    sub = cand[:8]
    gap = torch.zeros(8, dtype=torch.float64, device="cuda")
    fsb.fs_score_candidates_noalloc(w.K, w.B, w.G, bounds, slo, lam, sub, w.O, 64, w.seed, gap_dev=gap)
    with load_model(fsb, w) as m:
        ref = fsb.fs_score_candidates(m, w.candidates[:8], w.O, 64, w.seed)
    assert np.array_equal(gap.cpu().numpy(), ref.gap)
