"""Monte-Carlo scorer (fs_score_candidates) against the CPU oracle across many
random small problems and at the extreme sizes the model accepts.

Every case compares the fixed-point sums, E[Gamma_{t+1} | e], the scores,
Gamma_t and the argmax bit for bit. The random cases vary K, B, G, demands,
outcomes O, samples S (ragged last Philox call), seed, stream id, round and,
for a quarter of them, the quantile table.
"""

import dataclasses

import numpy as np
import pytest

from conftest import load_model
from paper_2608_19659_gb300 import workloads

pytestmark = pytest.mark.gpu


def _score_both(fsb, oracle_lib, w, qn, cand, O, S, seed, stream_id, rnd, quantile=None):
    with load_model(fsb, w, quantile) as m:
        r = fsb.fs_score_candidates(m, cand, O, S, seed, stream_id, rnd)
    ref = oracle_lib.score(w, qn, candidates=cand, seed=seed, stream_id=stream_id, rnd=rnd, O=O, S=S)
    return r, ref


def _assert_same(r, ref):
    assert np.array_equal(r.sum_eo, ref.sum_eo)
    assert np.array_equal(r.gap, ref.gap)
    assert np.array_equal(r.score, ref.score)
    assert r.gamma_t == ref.gamma_t
    assert r.best == ref.best


def _contested(oracle_lib, w):
    """w with its demand scaled by the power of sqrt(2) that gives the widest
    base gap Gamma_t (the oracle's), so that scores are not all zero."""
    best_g, best_w = -1.0, w
    for k in range(-8, 37):
        x = dataclasses.replace(w, demand=(w.demand * np.float32(2.0 ** (k / 2))).astype(np.float32))
        g = oracle_lib.base_gap(oracle_lib.Problem.of(x), x.cap_lo, x.cap_hi, x.tail_lo, x.tail_hi)[2]
        if g > best_g:
            best_g, best_w = g, x
    return best_w


def _random_quantiles(rng, Q):
    """A nondecreasing table in [0, 1] with repeated values and both ends."""
    v = np.sort(rng.random(Q).astype(np.float32))
    v[: Q // 16] = v[0]
    v[0], v[-1] = np.float32(0.0), np.float32(1.0)
    return np.sort(v)


@pytest.mark.parametrize("seed", range(16))
def test_random_small_problems(fsb, cuda, oracle_lib, seed):
    rng = np.random.default_rng(900 + seed)
    K, B, G = int(rng.integers(1, 9)), int(rng.integers(1, 9)), int(rng.integers(1, 65))
    w = workloads.random_small(rng, K, B, G)
    if seed % 3:  # one case in three keeps its raw demand (often Gamma_t = 0 or 1)
        w = _contested(oracle_lib, w)
    O, S = int(2 ** rng.integers(0, 4)), int(rng.integers(1, 41))
    s, sid, rnd = int(rng.integers(0, 2**63)), int(rng.integers(0, 1000)), int(rng.integers(0, 50))
    if seed % 4 == 0:
        qn = _random_quantiles(rng, int(2 ** rng.integers(4, 11)))
        O = min(O, qn.size)
        r, ref = _score_both(fsb, oracle_lib, w, qn, w.candidates, O, S, s, sid, rnd, quantile=qn)
    else:
        qn = oracle_lib.triangular_table(4096)
        r, ref = _score_both(fsb, oracle_lib, w, qn, w.candidates, O, S, s, sid, rnd)
    _assert_same(r, ref)


@pytest.mark.parametrize("K,B,G,n_cand", [
    (64, 2, 128, 24),   # 64 classes, 15360 thresholds
    (1, 4096, 8, 24),   # 16384 cells
    (1, 1, 1, 4),       # one GPU, one bin
    (1, 6, 1, 24),      # one GPU, six bins
    (3, 5, 1, 60),      # one GPU for three classes: t* = 0 on both sides
    (1, 2, 8738, 8),    # 16383 thresholds, within one of the most a model holds
    (1, 2, 1000, 16),   # 1875 thresholds: row table of 7500 words, several passes per count
    (1, 3, 1200, 16),   # row table on one realisation only (6600 and 9000 words)
    (8, 2, 64, 24),     # eight classes, row table of 7968 words
    (2, 3, 69, 24),     # theta_cap = 256: the preparation loads its row words with their count
    (2, 3, 70, 24),     # theta_cap = 260: it reads the count first
])
def test_extreme_sizes(fsb, cuda, oracle_lib, K, B, G, n_cand):
    rng = np.random.default_rng(K * 7919 + B * 31 + G)
    w = _contested(oracle_lib, workloads.random_small(rng, K, B, G))
    cells = K * 4 * B
    cand = np.sort(rng.choice(cells, size=min(n_cand, cells), replace=False)).astype(np.int32)
    qn = oracle_lib.triangular_table(4096)
    r, ref = _score_both(fsb, oracle_lib, w, qn, cand, 2, 16, 77, 3, 1)
    _assert_same(r, ref)


@pytest.mark.parametrize("seed", range(8))
def test_table_path_random_problems(fsb, cuda, oracle_lib, seed):
    """Enough samples per outcome that the scorer tabulates each segment's
    values of rint(Gamma' 2^40) (W = 4096 / O entries) and only draws indices;
    a subset of candidates, sums compared bit for bit."""
    rng = np.random.default_rng(1700 + seed)
    K, B, G = int(rng.integers(1, 7)), int(rng.integers(1, 7)), int(rng.integers(2, 49))
    w = _contested(oracle_lib, workloads.random_small(rng, K, B, G))
    O = int(rng.choice([4, 8, 16]))
    S = int(rng.integers(800, 2600))
    cand = np.sort(rng.choice(w.cells, size=min(6, w.cells), replace=False)).astype(np.int32)
    s, sid, rnd = int(rng.integers(0, 2**63)), int(rng.integers(0, 100)), int(rng.integers(0, 20))
    qn = oracle_lib.triangular_table(4096)
    r, ref = _score_both(fsb, oracle_lib, w, qn, cand, O, S, s, sid, rnd)
    _assert_same(r, ref)


def test_sixty_four_classes_over_every_cell(fsb, cuda, oracle_lib):
    """64 classes (the most a model takes) with every one of their 1,024 cells a
    candidate: 2,048 preparation blocks, so the launch takes 64-thread blocks,
    whose threads just cover the classes' demands, and with 15,360 thresholds
    no row table (the joint search with two probe groups a block). Sampled
    candidates are compared with the oracle in full."""
    rng = np.random.default_rng(4242)
    w = _contested(oracle_lib, workloads.random_small(rng, 64, 4, 128))
    qn = oracle_lib.triangular_table(4096)
    cand = np.arange(w.K * 4 * w.B, dtype=np.int32)
    with load_model(fsb, w) as m:
        r = fsb.fs_score_candidates(m, cand, 2, 64, 7)
    pick = np.arange(0, cand.size, 97)
    se, gt = oracle_lib.score_sums_cached(w, qn, candidates=cand[pick], O=2, S=64, seed=7)
    assert gt == r.gamma_t > 0
    assert np.array_equal(r.sum_eo[pick], se)
