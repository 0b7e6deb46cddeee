"""GPU Monte-Carlo scorer (fs_score_candidates) against the CPU oracle.

Fixed-point sums, E[Gamma_{t+1} | e], scores, Gamma_t and the argmax must be
bit-identical to the oracle; per-scenario draws, t* and allocation choices are
compared record by record through the dump mode.
"""

import dataclasses

import numpy as np
import pytest

from conftest import load_model
from paper_2608_19659_gb300 import workloads

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def qn(oracle_lib):
    return oracle_lib.triangular_table(4096)


def stressed(idx, factor=3.0, **kw):
    w = workloads.make_workload(idx)
    return dataclasses.replace(w, demand=(w.demand * factor).astype(np.float32), **kw)


def assert_same(r, ref, cand=None):
    assert np.array_equal(r.sum_eo, ref.sum_eo)
    assert np.array_equal(r.gap, ref.gap)
    assert np.array_equal(r.score, ref.score)
    assert r.gamma_t == ref.gamma_t
    if cand is None:
        assert r.best == ref.best


def run(fsb, w, cand=None, **kw):
    with load_model(fsb, w, kw.pop("quantile", None)) as m:
        return fsb.fs_score_candidates(m, w.candidates if cand is None else cand, kw.pop("O", w.O),
                                       kw.pop("S", w.S), kw.pop("seed", w.seed), kw.pop("stream_id", w.stream_id),
                                       kw.pop("rnd", w.round))


@pytest.mark.parametrize("factor", [1.0, 3.0])
def test_tiny_workload_full(fsb, cuda, oracle_lib, qn, factor):
    w = stressed(0, factor)
    r = run(fsb, w)
    ref = oracle_lib.score(w, qn, solver=0)  # literal solver on every scenario
    assert_same(r, ref)
    if factor == 3.0:
        assert ref.gamma_t > 0 and ref.score.max() > 0


def test_paper_scale_workload_full(fsb, cuda, oracle_lib, qn):
    """64 candidates x 8 outcomes x 4096 samples, the benchmark's workload, in full."""
    w = workloads.make_workload(1)
    r = run(fsb, w)
    ref = oracle_lib.score(w, qn)
    assert_same(r, ref)
    assert ref.gamma_t > 0 and (ref.score > 0).sum() > 0


@pytest.mark.parametrize("S", [4093, 4094])
def test_paper_scale_table_path_ragged_samples(fsb, cuda, oracle_lib, qn, S):
    """The table path with a ragged last Philox call in every segment (S mod 4
    samples of its four words), all 64 candidates in full."""
    w = dataclasses.replace(workloads.make_workload(1), S=S)
    r = run(fsb, w)
    ref = oracle_lib.score(w, qn)
    assert_same(r, ref)
    assert ref.gamma_t > 0


def test_large_workload_ragged_samples_sampled(fsb, cuda, oracle_lib, qn):
    """The eight-class workload at S = 16,383: one problem's many-segment launch
    (one chunk a segment) whose segments end with a call serving three
    samples; candidates with a positive score and a few others in full."""
    w = dataclasses.replace(workloads.make_workload(3), S=16383)
    full = run(fsb, w)
    pos = np.nonzero(full.score > 0)[0]
    assert len(pos) > 0
    pick = np.unique(np.concatenate([pos[:3], pos[-2:], [0, len(w.candidates) - 1]]))
    se, gt = oracle_lib.score_sums_cached(w, qn, candidates=w.candidates[pick])
    assert gt == full.gamma_t
    assert np.array_equal(full.sum_eo[pick], se)


@pytest.mark.parametrize("factor", [1.0, 3.0])
def test_mid_workload_sampled_candidates(fsb, cuda, oracle_lib, qn, factor):
    w = stressed(2, factor)
    with load_model(fsb, w) as m:
        full = fsb.fs_score_candidates(m, w.candidates, w.O, w.S, w.seed)
    # the oracle scores a few candidates in full (all 8 x 16384 scenarios each)
    pick = np.array([16, 37, 200], np.int32)
    ref = oracle_lib.score(w, qn, candidates=w.candidates[pick])
    assert np.array_equal(full.sum_eo[pick], ref.sum_eo)
    assert np.array_equal(full.score[pick], ref.score) and full.gamma_t == ref.gamma_t
    # argmax consistent with the tie rules over the GPU's own exact sums
    sc = np.rint(np.float64(full.gamma_t) * 2.0**40).astype(np.int64) * (w.O * w.S) - full.sum_eo.sum(axis=1)
    j = (w.candidates // w.B) % 4
    order = np.lexsort((np.arange(len(sc)), j, -sc))
    assert full.best == w.candidates[order[0]]


def _check_dump(fsb, oracle_lib, w, qn, m, cand, n_check, rng):
    import torch

    K = w.K
    stride = fsb.fs_dump_stride(m)
    n = len(cand) * w.O * w.S
    dump = torch.zeros(n * stride, dtype=torch.uint8, device="cuda")
    r = fsb.fs_score_candidates(m, cand, w.O, w.S, w.seed, w.stream_id, w.round, dump_dev=dump)
    rec = dump.cpu().numpy().view(fsb.dump_dtype(K)).reshape(len(cand), w.O, w.S)
    # fixed-point sums recomputed from the per-scenario t*
    g = (rec["t_star"][..., 1] - rec["t_star"][..., 0]).astype(np.float32)
    assert np.array_equal(np.rint(g.astype(np.float64) * 2.0**40).astype(np.int64).sum(axis=2), r.sum_eo)
    for _ in range(n_check):
        e = int(rng.integers(len(cand)))
        o = int(rng.integers(w.O))
        s = int(rng.integers(w.S))
        cy, ly, am, ap = oracle_lib.scenario(w, qn, int(cand[e]), o, s)
        x = rec[e, o, s]
        assert (x["c_y"], x["l_y"]) == (np.float32(cy), np.float32(ly))
        for sg, a in ((0, am), (1, ap)):
            assert x["t_star"][sg] == np.float32(a.t_star)
            assert x["total_gpus"][sg] == a.total_gpus
            for i in range(K):
                n_, tp, b = fsb.decode_choice(int(x["choice"][sg][i]))
                assert (n_, tp, b) == (a.replicas[i], a.tp[i], a.bin[i])
    return r, rec


def test_dump_records_match_oracle_tiny(fsb, cuda, oracle_lib, qn):
    w = stressed(0, 3.0, S=256)
    rng = np.random.default_rng(0)
    with load_model(fsb, w) as m:
        r, rec = _check_dump(fsb, oracle_lib, w, qn, m, w.candidates, 300, rng)
    ref = oracle_lib.score(w, qn, dump=True)
    assert np.array_equal(rec["t_star"], ref.dump_t)


def test_large_workload_full_launch_and_dump_sample(fsb, cuda, oracle_lib, qn):
    """The 8-class workload at full size; the oracle checks sampled scenarios one by one."""
    w = workloads.make_workload(3)
    with load_model(fsb, w) as m:
        full = fsb.fs_score_candidates(m, w.candidates, w.O, w.S, w.seed)
        assert full.gamma_t == oracle_lib.base_gap(oracle_lib.Problem.of(w), w.cap_lo, w.cap_hi,
                                                   w.tail_lo, w.tail_hi)[2]
        pos = np.nonzero(full.score > 0)[0]
        assert len(pos) > 0
        pick = np.unique(np.concatenate([pos[:2], pos[-1:], [0, 511]])).astype(np.int64)
        sub, _ = _check_dump(fsb, oracle_lib, w, qn, m, w.candidates[pick], 120, np.random.default_rng(3))
    # scoring a subset reproduces the full launch's sums for those candidates
    assert np.array_equal(sub.sum_eo, full.sum_eo[pick])
    assert np.array_equal(sub.score, full.score[pick])
    assert np.all(full.score >= 0) and np.all(full.score <= full.gamma_t)


def test_long_tables_read_from_global_memory(fsb, cuda, oracle_lib, qn):
    """The 8-class workload at twice its demand has contested threshold ranges of up
    to ~300 entries, longer than the 256 the scorer stages in shared memory: those
    scenarios search their tables in global memory. Every candidate, few samples;
    then denser sampling on candidates with a positive score."""
    w = stressed(3, 2.0, O=2, S=8)
    r = run(fsb, w)
    ref = oracle_lib.score(w, qn)
    assert_same(r, ref)
    pos = np.nonzero(ref.score > 0)[0]
    assert len(pos) > 0
    w2 = dataclasses.replace(w, S=96)
    cand = w.candidates[pos[:: max(1, len(pos) // 4)][:4]]
    r2 = run(fsb, w2, cand=cand)
    assert_same(r2, oracle_lib.score(w2, qn, candidates=cand), cand=cand)


@pytest.mark.parametrize("cap", [0.0, 1e-20])
def test_row_term_outside_markstein_range(fsb, cuda, oracle_lib, qn, cap):
    """A row whose capacities under A- are zero or below 2^-60: the row-term
    quotient of its candidates cannot use Markstein's method and goes through the
    IEEE division; every cell is a candidate."""
    w = stressed(0, 3.0, O=4, S=128)
    cap_lo = w.cap_lo.copy().reshape(w.K, 4, w.B)
    cap_lo[0, 0, :] = cap  # class 0, TP 1, every bin
    w = dataclasses.replace(w, cap_lo=cap_lo.reshape(w.cap_lo.shape),
                            candidates=np.arange(w.K * 4 * w.B, dtype=np.int32))
    r = run(fsb, w)
    ref = oracle_lib.score(w, qn)
    assert_same(r, ref)
    assert ref.gamma_t > 0


@pytest.mark.parametrize("O,S", [(1, 7), (4, 1), (4096, 3), (16, 33), (2, 2)])
def test_outcome_and_sample_edge_cases(fsb, cuda, oracle_lib, qn, O, S):
    w = stressed(0, 3.0, O=O, S=S)
    r = run(fsb, w)
    assert_same(r, oracle_lib.score(w, qn))


def test_seed_stream_round_and_duplicates(fsb, cuda, oracle_lib, qn):
    w = stressed(0, 3.0, S=32, seed=(7 << 32) | 11, stream_id=5, round=9)
    cand = np.array([3, 3, 60, 0, 17, 3], np.int32)
    r = run(fsb, w, cand=cand)
    ref = oracle_lib.score(w, qn, candidates=cand)
    assert_same(r, ref)
    assert np.array_equal(r.sum_eo[0], r.sum_eo[1])


def test_no_candidates(fsb, cuda, oracle_lib):
    w = workloads.make_workload(1)
    with load_model(fsb, w) as m:
        r = fsb.fs_score_candidates(m, np.zeros(0, np.int32), 8, 16, 1)
    assert r.best == -1 and r.gap.size == 0
    p = oracle_lib.Problem.of(w)
    assert r.gamma_t == oracle_lib.base_gap(p, w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi)[2]


def test_revealed_candidates_and_collapsed_bounds(fsb, cuda, oracle_lib, qn):
    w = workloads.make_workload(1)
    with load_model(fsb, w) as m:
        fsb.fs_reveal(m, 5, float(w.cap_lo.reshape(-1)[5]), float(w.tail_hi.reshape(-1)[5]))
        r = fsb.fs_score_candidates(m, np.array([5, 6], np.int32), 8, 64, 1)
        assert r.score[0] == 0.0 and r.sum_eo[0].sum() == np.rint(np.float64(r.gamma_t) * 2**40) * 8 * 64
        fsb.fs_update_bounds(m, w.cap_lo, w.cap_lo, w.tail_hi, w.tail_hi)
        z = fsb.fs_score_candidates(m, w.candidates, 8, 64, 1)
    assert z.gamma_t == 0.0 and np.all(z.score == 0) and np.all(z.sum_eo == 0)


def test_single_class_and_custom_quantiles(fsb, cuda, oracle_lib):
    rng = np.random.default_rng(77)
    w = workloads.random_small(rng, 1, 6, 24)
    w = dataclasses.replace(w, demand=(w.demand * 8).astype(np.float32), O=8, S=64, seed=3)
    uni = ((np.arange(256) + 0.5) / 256).astype(np.float32)
    r = run(fsb, w, quantile=uni)
    ref = oracle_lib.score(w, uni)
    assert_same(r, ref)


def test_async_matches_sync_and_launches_kernels(fsb, cuda, oracle_lib, qn):
    torch = cuda
    w = workloads.make_workload(1)
    n = len(w.candidates)
    with load_model(fsb, w) as m:
        ref = fsb.fs_score_candidates(m, w.candidates, w.O, w.S, w.seed)
        st = torch.cuda.Stream()
        cand = torch.from_numpy(w.candidates).cuda()
        gap = torch.zeros(n, dtype=torch.float64, device="cuda")
        score = torch.zeros(n, dtype=torch.float64, device="cuda")
        gt = torch.zeros(1, dtype=torch.float32, device="cuda")
        best = torch.zeros(1, dtype=torch.int32, device="cuda")
        sums = torch.zeros((n, w.O), dtype=torch.int64, device="cuda")
        c0 = fsb.fs_launch_count()
        with torch.cuda.stream(st):
            fsb.fs_score_candidates_async(m, cand, w.O, w.S, w.seed, gap_dev=gap, score_dev=score,
                                          gamma_t_dev=gt, best_dev=best, sum_eo_dev=sums, stream=st)
        fsb.fs_check(m, st)
        assert fsb.fs_launch_count() - c0 == 4
    assert np.array_equal(gap.cpu().numpy(), ref.gap) and np.array_equal(score.cpu().numpy(), ref.score)
    assert np.array_equal(sums.cpu().numpy(), ref.sum_eo)
    assert float(gt.item()) == ref.gamma_t and int(best.item()) == ref.best


@pytest.mark.parametrize("bad", ["O3", "Obig", "S0", "cand", "OS"])
def test_score_rejects_bad_plans(fsb, cuda, bad):
    w = workloads.make_workload(0)
    O, S, cand = 4, 16, w.candidates
    if bad == "O3":
        O = 3
    elif bad == "Obig":
        O = 8192
    elif bad == "S0":
        S = 0
    elif bad == "cand":
        cand = np.array([0, w.cells], np.int32)
    elif bad == "OS":
        O, S = 4096, 4096
    with load_model(fsb, w) as m:
        with pytest.raises(fsb.FleetSieveError) as ei:
            fsb.fs_score_candidates(m, cand, O, S, 0)
        assert ei.value.code == fsb.FS_EINVAL
        fsb.fs_score_candidates(m, w.candidates, 4, 8, 0)  # the model stays usable


def test_watchdog_times_out_cleanly(fsb, cuda):
    assert fsb.fs_watchdog_selftest(2_000_000) == fsb.FS_ETIMEOUT
    w = workloads.make_workload(0)
    with load_model(fsb, w) as m:
        fsb.fs_score_candidates(m, w.candidates, 4, 8, 0)


def test_draw_floor_measures_both_modes(fsb, cuda):
    """The measurement floor of the table path's draws runs at least the calls
    asked for in both modes and leaves the context usable."""
    for mode in (0, 1):
        ms, done = fsb.fs_draw_floor(mode, 8, 1 << 20, 3)
        assert ms > 0.0 and done >= 1 << 20
    w = workloads.make_workload(0)
    with load_model(fsb, w) as m:
        fsb.fs_score_candidates(m, w.candidates, 4, 8, 0)


def test_staged_bounds_reach_every_later_call(fsb, cuda, oracle_lib, qn):
    """fs_update_bounds only stages: a synchronous score reads the staged bounds,
    every device-side call after it (asynchronous scoring on another stream,
    bounds solves) sees them too."""
    torch = cuda
    w1 = stressed(0, 3.0, S=64)
    w2 = stressed(0, 2.0, S=64, cap_lo=(workloads.make_workload(0).cap_lo * 0.9).astype(np.float32))
    n = len(w1.candidates)
    cand = torch.from_numpy(w1.candidates).cuda()
    side = torch.cuda.Stream()

    def score_async(m):
        gap = torch.zeros(n, dtype=torch.float64, device="cuda")
        sums = torch.zeros((n, w1.O), dtype=torch.int64, device="cuda")
        with torch.cuda.stream(side):
            fsb.fs_score_candidates_async(m, cand, w1.O, w1.S, w1.seed, gap_dev=gap, sum_eo_dev=sums, stream=side)
        fsb.fs_check(m, side)
        return sums.cpu().numpy()

    ref1 = oracle_lib.score(w1, qn)
    w2s = dataclasses.replace(w2, demand=w1.demand)
    ref2 = oracle_lib.score(w2s, qn)
    with load_model(fsb, w1) as m:
        fsb.fs_update_bounds(m, w2.cap_lo, w2.cap_hi, w2.tail_lo, w2.tail_hi)
        assert np.array_equal(score_async(m), ref2.sum_eo)           # straight after the update
        fsb.fs_update_bounds(m, w1.cap_lo, w1.cap_hi, w1.tail_lo, w1.tail_hi)
        r = fsb.fs_score_candidates(m, w1.candidates, w1.O, w1.S, w1.seed)  # reads the staging
        assert np.array_equal(r.sum_eo, ref1.sum_eo)
        assert np.array_equal(score_async(m), ref1.sum_eo)           # the device copy followed
        fsb.fs_update_bounds(m, w2.cap_lo, w2.cap_hi, w2.tail_lo, w2.tail_hi)
        gm, gp, g = fsb.fs_solve_bounds(m)
        assert g == oracle_lib.base_gap(oracle_lib.Problem.of(w2s), w2.cap_lo, w2.cap_hi, w2.tail_lo, w2.tail_hi)[2]
        r = fsb.fs_score_candidates(m, w1.candidates, w1.O, w1.S, w1.seed)
        assert np.array_equal(r.sum_eo, ref2.sum_eo)


def test_table_path_with_long_tables(fsb, cuda, oracle_lib, qn):
    """The table path on the 8-class workload at twice its demand, where some
    candidates' contested ranges exceed the 256 entries staged in shared memory,
    so their segment tables are built from global memory."""
    w = stressed(3, 2.0, O=16, S=512)
    probe = stressed(3, 2.0, O=2, S=8)
    ref0 = oracle_lib.score(probe, qn)
    pos = np.nonzero(ref0.score > 0)[0]
    cand = probe.candidates[pos[:: max(1, len(pos) // 3)][:3]]
    r = run(fsb, w, cand=cand)
    assert_same(r, oracle_lib.score(w, qn, candidates=cand), cand=cand)


def test_split_reduction_keeps_candidate_order(fsb, cuda, oracle_lib, qn):
    """More than 256 candidates: the reduction is split over several blocks and
    the argmax is merged from their results. Every cell appears several times,
    so equal scores must still resolve to the earliest position of the list."""
    w = stressed(0, 3.0, O=4, S=64)
    rng = np.random.default_rng(12)
    cand = rng.permutation(np.tile(np.arange(w.cells, dtype=np.int32), 10))[:600].astype(np.int32)
    r = run(fsb, w, cand=cand)
    ref = oracle_lib.score(w, qn, candidates=cand)
    assert_same(r, ref)
    assert r.best == ref.best and np.sum(cand == r.best) > 1


def test_repeated_arrays_read_at_every_call(fsb, cuda, oracle_lib, qn):
    """The binding reuses the addresses of arrays passed again; their contents
    are still read at every call (bounds and candidates changed in place)."""
    w = stressed(0, 3.0, S=64)
    cl, ch, tl, th = (np.ascontiguousarray(getattr(w, k).reshape(-1)).copy()
                      for k in ("cap_lo", "cap_hi", "tail_lo", "tail_hi"))
    cand = w.candidates.copy()
    n = len(cand)
    outs = (np.zeros(n), np.zeros(n), np.zeros(1, np.float32), np.zeros(1, np.int32), np.zeros((n, w.O), np.int64))
    with load_model(fsb, w) as m:
        fsb.fs_update_bounds(m, cl, ch, tl, th)
        r = fsb.fs_score_candidates(m, cand, w.O, w.S, w.seed, outputs=outs)
        assert np.array_equal(r.sum_eo, oracle_lib.score(w, qn).sum_eo)
        cl *= np.float32(0.9)  # in place: same arrays, new contents
        cand[:] = cand[::-1]
        fsb.fs_update_bounds(m, cl, ch, tl, th)
        r = fsb.fs_score_candidates(m, cand, w.O, w.S, w.seed, outputs=outs)
    w2 = dataclasses.replace(w, cap_lo=cl.reshape(w.cap_lo.shape).copy(), candidates=cand.copy())
    ref = oracle_lib.score(w2, qn)
    assert np.array_equal(r.sum_eo, ref.sum_eo) and r.best == ref.best


def test_models_of_different_sizes_used_alternately(fsb, cuda, oracle_lib, qn):
    """Kernels' shared-memory limits belong to the kernels, not to a model: a
    smaller model scored between two calls of a larger one leaves the larger
    one's launches valid."""
    big, small = stressed(2, S=64), stressed(0, S=64)
    big = dataclasses.replace(big, candidates=big.candidates[::16].copy())
    with load_model(fsb, big) as mb:
        first = fsb.fs_score_candidates(mb, big.candidates, big.O, big.S, big.seed)
        with load_model(fsb, small) as ms:
            r = fsb.fs_score_candidates(ms, small.candidates, small.O, small.S, small.seed)
        again = fsb.fs_score_candidates(mb, big.candidates, big.O, big.S, big.seed)
        fsb.fs_solve_bounds(mb)
    assert np.array_equal(r.sum_eo, oracle_lib.score(small, qn).sum_eo)
    assert np.array_equal(first.sum_eo, again.sum_eo)
    assert np.array_equal(again.sum_eo, oracle_lib.score(big, qn).sum_eo)


def test_table_work_counted_by_the_library(fsb, cuda, oracle_lib, qn):
    """The table path builds W gap-table entries in each segment whose tail
    gate is open at some position of its stratum, and none where it is closed at
    every position (all entries are the closed-gate value); an entry evaluates a
    realisation's t* only where its capacity lies above that realisation's
    Cexcl (the best SLO-feasible capacity of the candidate's row without its
    bin; at or below it t* is the closed-gate one). Only the scenarios of strata
    whose tails lie on both sides of the SLO test their gate. The library's
    counts, which the benchmark's algorithmic work uses, must say exactly that."""
    w = workloads.make_workload(1)
    W = 4096 // w.O
    lo, hi = w.tail_lo.reshape(-1), w.tail_hi.reshape(-1)
    clo, chi = w.cap_lo.reshape(-1), w.cap_hi.reshape(-1)
    L = np.repeat(w.slo, 4 * w.B)

    def cexcl(c, sigma):  # A- (cap_lo, tail_hi) or A+ (cap_hi, tail_lo)
        cap, tail = (chi, lo) if sigma else (clo, hi)
        row = c - c % w.B
        feas = [cap[x] for x in range(row, row + w.B) if x != c and tail[x] <= L[x]]
        return max(feas) if feas else 0.0
    # the smallest and largest tail values of stratum o map its first and last quantile
    first = [[oracle_lib.map_value(lo[c], hi[c], qn[o * W]) <= L[c] for o in range(w.O)] for c in w.candidates]
    last = [[oracle_lib.map_value(lo[c], hi[c], qn[(o + 1) * W - 1]) <= L[c] for o in range(w.O)]
            for c in w.candidates]
    open_segments = sum(f for row in first for f in row)
    mixed = sum(f and not g for fr, lr in zip(first, last) for f, g in zip(fr, lr))
    assert 0 < open_segments < len(w.candidates) * w.O and mixed > 0
    evals = 0
    for c, row in zip(w.candidates, first):
        cx = (cexcl(c, 0), cexcl(c, 1))
        for o in range(w.O):
            if row[o]:
                cy = [oracle_lib.map_value(clo[c], chi[c], qn[o * W + k]) for k in range(W)]
                evals += sum(int(y > cx[0]) + int(y > cx[1]) for y in cy)
    assert 0 < evals < 2 * open_segments * W
    with load_model(fsb, w) as m:
        fsb.fs_timing_enable(m, 1)
        r = fsb.fs_score_candidates(m, w.candidates, w.O, w.S, w.seed)
        r = fsb.fs_score_candidates(m, w.candidates, w.O, w.S, w.seed)
        _, n, _, (entries, gated) = fsb.fs_timing_read(m, with_entries=True)
        assert n == 2 and entries == 2 * evals and gated == 2 * mixed * w.S
        assert fsb.fs_timing_read(m, with_entries=True)[3] == (0, 0)
    assert np.array_equal(r.sum_eo, oracle_lib.score(w, qn).sum_eo)
