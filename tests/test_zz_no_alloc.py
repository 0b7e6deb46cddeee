"""The allocation-free scoring entry point against the allocating one and the oracle.

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


def test_noalloc_matches_oracle(fsb, cuda, oracle_lib):
    """The allocation-free entry point against the oracle directly: the tiny
    workload at 3x demand (nonzero scores), two rounds through the shared
    array; gap, score, Gamma_t and the argmax equal the oracle's bit for bit."""
    torch = cuda
    w = workloads.make_workload(0)
    w = dataclasses.replace(w, demand=(w.demand * np.float32(3.0)).astype(np.float32))
    bounds, slo, lam, cand = _device_inputs(torch, w)
    n = len(w.candidates)
    qn = oracle_lib.triangular_table(4096)
    stream = torch.cuda.current_stream()
    for rnd in (0, 1):
        ref = oracle_lib.score(w, qn, rnd=rnd)
        gap = torch.full((n,), float("nan"), dtype=torch.float64, device="cuda")
        score = torch.full((n,), float("nan"), dtype=torch.float64, device="cuda")
        gt = torch.full((1,), float("nan"), dtype=torch.float32, device="cuda")
        best = torch.full((1,), -7, dtype=torch.int32, device="cuda")
        fsb.fs_score_candidates_noalloc(w.K, w.B, w.G, bounds, slo, lam, cand, w.O, w.S, w.seed, 0, rnd,
                                        gap_dev=gap, score_dev=score, gamma_t_dev=gt, best_dev=best, stream=stream)
        assert np.array_equal(gap.cpu().numpy(), ref.gap) and np.array_equal(score.cpu().numpy(), ref.score)
        assert float(gt.item()) == ref.gamma_t and int(best.item()) == ref.best
        assert ref.score.max() > 0


def _scratch_bytes(K, G, O, Q, n, builtin_table=True):
    """The scratch a call takes, as the header states it: pieces rounded up to 256 bytes."""
    up = lambda x: (x + 255) // 256 * 256  # noqa: E731
    T = K * ((G >> 0) + (G >> 1) + (G >> 2) + (G >> 3))
    P = 4
    while P < T + 1:
        P *= 2
    W = Q // O
    I = 2 * (20 + 3 * P) + O * (4 + 4 * ((W + 3) // 4))
    n = max(n, 1)
    parts = [4, 32, 1024] + ([4 * Q] if builtin_table else []) + [8 * T, 8, 32 * K, 32 * K, 1216, 65536,
                                                                   4 * n * I, 8 * n * O]
    return sum(up(p) for p in parts)


def test_noalloc_limit_is_the_stated_formula(fsb, cuda):
    """The largest call the header's formula allows runs (and matches the
    allocating path); one candidate more is refused without running."""
    torch = cuda
    w = workloads.make_workload(1)
    n = 1
    while _scratch_bytes(w.K, w.G, w.O, 4096, n + 1) <= 16 << 20:
        n += 1
    assert n == 913  # the figure the header quotes for this grid
    cells = np.resize(w.candidates, n + 1).astype(np.int32)
    bounds, slo, lam, _ = _device_inputs(torch, w)
    cand = torch.from_numpy(cells).cuda()
    gap = torch.zeros(n, dtype=torch.float64, device="cuda")
    best = torch.zeros(1, dtype=torch.int32, device="cuda")
    fsb.fs_score_candidates_noalloc(w.K, w.B, w.G, bounds, slo, lam, cand[:n], w.O, 8, w.seed,
                                    gap_dev=gap, best_dev=best)
    with load_model(fsb, w) as m:
        ref = fsb.fs_score_candidates(m, cells[:n], w.O, 8, w.seed)
    assert np.array_equal(gap.cpu().numpy(), ref.gap) and int(best.item()) == ref.best
    with pytest.raises(fsb.FleetSieveError) as ei:
        fsb.fs_score_candidates_noalloc(w.K, w.B, w.G, bounds, slo, lam, cand, w.O, 8, w.seed, gap_dev=gap)
    assert ei.value.code == fsb.FS_EINVAL and "scratch" in str(ei.value)


@pytest.mark.parametrize("idx", [1, 3])
def test_noalloc_negative_zero_capacities(fsb, cuda, idx):
    """Device bounds are not canonicalised by this entry point: capacities of
    -0.0 (which the rules accept as 0) must score exactly as the allocating
    path, which stores them as +0. The 8-class workload runs the preparation
    without a row table (too many rows x thresholds), the paper-scale one with."""
    torch = cuda
    w = workloads.make_workload(idx)
    w = dataclasses.replace(w, demand=(w.demand * np.float32(2.0)).astype(np.float32), S=64)
    clo = w.cap_lo.copy().reshape(w.K, 4, w.B)
    chi = w.cap_hi.copy().reshape(w.K, 4, w.B)
    clo[0, 1, :] = np.float32(-0.0)  # class 0, TP 2: lower capacity -0 in every bin
    chi[0, 1, : w.B // 2] = np.float32(-0.0)  # and a collapsed [-0, -0] interval in half of them
    w = dataclasses.replace(w, cap_lo=clo.reshape(w.cap_lo.shape), cap_hi=chi.reshape(w.cap_hi.shape))
    cand_np = np.arange(w.B, 2 * w.B, dtype=np.int32)  # every cell of that row
    cand_np = np.concatenate([cand_np, w.candidates[:: max(1, len(w.candidates) // 16)]]).astype(np.int32)
    bounds, slo, lam, _ = _device_inputs(torch, w)
    assert bool(torch.signbit(bounds[w.B]).item())  # the device holds -0.0
    n = len(cand_np)
    gap = torch.zeros(n, dtype=torch.float64, device="cuda")
    score = torch.zeros(n, dtype=torch.float64, device="cuda")
    gt = torch.zeros(1, dtype=torch.float32, device="cuda")
    best = torch.zeros(1, dtype=torch.int32, device="cuda")
    fsb.fs_score_candidates_noalloc(w.K, w.B, w.G, bounds, slo, lam, torch.from_numpy(cand_np).cuda(), w.O, w.S,
                                    w.seed, gap_dev=gap, score_dev=score, gamma_t_dev=gt, best_dev=best)
    with load_model(fsb, w) as m:
        ref = fsb.fs_score_candidates(m, cand_np, w.O, w.S, w.seed)
    assert np.array_equal(gap.cpu().numpy(), ref.gap) and np.array_equal(score.cpu().numpy(), ref.score)
    assert float(gt.item()) == ref.gamma_t and int(best.item()) == ref.best


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
