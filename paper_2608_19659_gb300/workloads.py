"""Seeded synthetic workloads for the decision-gap scorer.

This module only makes inputs: per-cell capacity and tail-latency bounds,
SLOs, demands, candidate lists, and (for the replay workload) a hidden true
value per cell plus a reveal order. It holds none of the method's
arithmetic (no fulfilment, no solver, no sampler), so both the CUDA path and
the CPU oracle can be fed from it.

The paper's measured H100 grid and the Azure traces are not available, so
these generators stand in for them. They keep the paper's structure: classes
with a demand and an SLO, a TP degree in {1, 2, 4, 8} and a load bin per cell,
and a GPU budget G (Section 3, Eqs. 1-5; Section 5 and the 16-GPU allocation
of Table 3).

Recipe (all draws from ``numpy.random.default_rng(seed)``, in float64, then
rounded to float32):
  * capacity of cell (i, tau, b): two draws exp(ln(0.5 * tau**0.8) + sigma_c z)
    req/s per replica; lo / hi are their min / max;
  * binding tail of cell (i, tau, b): two draws
    exp(ln(12) + b ln(1.15) + sigma_l z) seconds; lo / hi are min / max;
  * the straddle rule of the 8-class workload moves tail bounds so that exactly
    round(0.1 * cells) cells have lo <= SLO < hi.
"""

from __future__ import annotations

import dataclasses
import math

import numpy as np

TP_DEGREES = (1, 2, 4, 8)
T = len(TP_DEGREES)


@dataclasses.dataclass
class Workload:
    """One scoring problem: bounds, policy, candidates and sample plan."""

    name: str
    K: int
    B: int
    G: int
    demand: np.ndarray  # [K] float32, req/s
    slo: np.ndarray  # [K] float32, seconds
    cap_lo: np.ndarray  # [K, 4, B] float32, req/s per replica
    cap_hi: np.ndarray
    tail_lo: np.ndarray  # [K, 4, B] float32, seconds
    tail_hi: np.ndarray
    candidates: np.ndarray  # [n_cand] int32 cell ids, cell = (i*4 + j)*B + b
    O: int  # outcomes (quantile strata)
    S: int  # samples per (candidate, outcome)
    seed: int
    stream_id: int = 0
    round: int = 0
    floor: np.ndarray | None = None  # [K] float32 critical floors delta_i in [0, 1] (0 = not critical)
    prior: int = 0  # interval refit after a measurement: 0 revealed cell only, 1 monotone in load bin

    @property
    def cells(self) -> int:
        return self.K * T * self.B

    @property
    def scenarios(self) -> int:
        return int(len(self.candidates)) * self.O * self.S

    def flat(self, name: str) -> np.ndarray:
        return np.ascontiguousarray(getattr(self, name).reshape(-1), dtype=np.float32)


@dataclasses.dataclass
class Replay:
    """Many independent reveal orders over one prior grid (Algorithm 1 loop)."""

    base: Workload
    truth_cap: np.ndarray  # [n_streams, cells] float32
    truth_tail: np.ndarray  # [n_streams, cells] float32
    perm: np.ndarray  # [n_streams, cells] int32, reveal order / tie order
    r0: int  # cells of perm revealed before the first round
    eps: float  # stopping tolerance on the gap
    max_rounds: int


def _bounds(rng, K, B, sigma_c, sigma_l):
    shape = (K, T, B)
    tau = np.array(TP_DEGREES, dtype=np.float64)[None, :, None]
    b = np.arange(B, dtype=np.float64)[None, None, :]
    mu_c = np.log(0.5 * tau**0.8) + np.zeros(shape)
    mu_l = np.log(12.0) + b * np.log(1.15) + np.zeros(shape)
    z = rng.standard_normal((4,) + shape)
    c1 = np.exp(mu_c + sigma_c * z[0])
    c2 = np.exp(mu_c + sigma_c * z[1])
    l1 = np.exp(mu_l + sigma_l * z[2])
    l2 = np.exp(mu_l + sigma_l * z[3])
    cap_lo = np.minimum(c1, c2).astype(np.float32)
    cap_hi = np.maximum(c1, c2).astype(np.float32)
    tail_lo = np.minimum(l1, l2).astype(np.float32)
    tail_hi = np.maximum(l1, l2).astype(np.float32)
    return cap_lo, cap_hi, tail_lo, tail_hi


def _straddle(rng, tail_lo, tail_hi, slo, frac, sigma_l):
    """Make exactly round(frac * cells) cells straddle their class SLO."""
    K, _, B = tail_lo.shape
    cells = K * T * B
    n_str = int(round(frac * cells))
    chosen = np.zeros(cells, dtype=bool)
    chosen[rng.choice(cells, size=n_str, replace=False)] = True
    chosen = chosen.reshape(K, T, B)
    lo = tail_lo.astype(np.float64)
    hi = tail_hi.astype(np.float64)
    L = slo.astype(np.float64)[:, None, None] + np.zeros((K, T, B))
    z = np.abs(rng.standard_normal((2, K, T, B)))
    s_lo = L * np.exp(-z[0] * sigma_l - 0.01)
    s_hi = L * np.exp(z[1] * sigma_l + 0.01)
    mid = np.sqrt(lo * hi)
    below = np.where(mid < L, 0.99 * L / hi, 1.0)
    above = np.where(mid >= L, 1.01 * L / lo, 1.0)
    crosses = (lo <= L) & (L < hi)
    scale = np.where(crosses, np.where(mid < L, below, above), 1.0)
    lo2 = np.where(chosen, s_lo, lo * scale)
    hi2 = np.where(chosen, s_hi, hi * scale)
    lo32 = lo2.astype(np.float32)
    hi32 = hi2.astype(np.float32)
    L32 = np.broadcast_to(slo.astype(np.float32)[:, None, None], lo32.shape)
    st = (lo32 <= L32) & (L32 < hi32)
    assert int(st.sum()) == n_str and bool((st == chosen).all())
    return lo32, hi32


def make_workload(idx: int) -> Workload:
    """The five synthetic workloads: 0 tiny, 1 paper-scale, 2 mid, 3 large.

    Index 4 (the replay) is built by :func:`make_replay`.
    """
    if idx == 0:
        rng = np.random.default_rng(0)
        K, B, G = 2, 8, 16
        cap_lo, cap_hi, tail_lo, tail_hi = _bounds(rng, K, B, 0.3, 0.4)
        cand = np.sort(rng.permutation(K * T * B)[:16]).astype(np.int32)
        return Workload("tiny: K=2 B=8 G=16, 16 cand x 4 outcomes x 256 samples",
                        K, B, G, np.array([3.0, 2.0], np.float32),
                        np.array([30.0, 30.0], np.float32),
                        cap_lo, cap_hi, tail_lo, tail_hi, cand, 4, 256, 0)
    if idx == 1:
        rng = np.random.default_rng(1)
        K, B, G = 2, 8, 16
        cap_lo, cap_hi, tail_lo, tail_hi = _bounds(rng, K, B, 0.3, 0.4)
        cand = np.arange(K * T * B, dtype=np.int32)
        return Workload("paper-scale: K=2 B=8 G=16, 64 cand x 8 outcomes x 4096 samples",
                        K, B, G, np.array([6.0, 4.0], np.float32),
                        np.array([30.0, 20.0], np.float32),
                        cap_lo, cap_hi, tail_lo, tail_hi, cand, 8, 4096, 1)
    if idx == 2:
        rng = np.random.default_rng(2)
        K, B, G = 4, 16, 64
        lam = rng.uniform(1.0, 10.0, K).astype(np.float32)
        slo = rng.choice(np.array([10.0, 20.0, 30.0, 60.0]), K).astype(np.float32)
        cap_lo, cap_hi, tail_lo, tail_hi = _bounds(rng, K, B, 0.3, 0.5)
        cand = np.arange(K * T * B, dtype=np.int32)
        return Workload("mid: K=4 B=16 G=64, 256 cand x 8 outcomes x 16384 samples",
                        K, B, G, lam, slo, cap_lo, cap_hi, tail_lo, tail_hi,
                        cand, 8, 16384, 2)
    if idx == 3:
        rng = np.random.default_rng(3)
        K, B, G = 8, 32, 256
        lam = rng.uniform(0.5, 20.0, K).astype(np.float32)
        slo = rng.choice(np.array([10.0, 20.0, 30.0, 60.0]), K).astype(np.float32)
        cap_lo, cap_hi, tail_lo, tail_hi = _bounds(rng, K, B, 0.3, 0.4)
        tail_lo, tail_hi = _straddle(rng, tail_lo, tail_hi, slo, 0.1, 0.4)
        cand = np.arange(K * T * B, dtype=np.int32)
        return Workload("large: K=8 B=32 G=256, 1024 cand x 16 outcomes x 16384 samples",
                        K, B, G, lam, slo, cap_lo, cap_hi, tail_lo, tail_hi,
                        cand, 16, 16384, 3)
    raise ValueError(f"no workload {idx}")


def make_replay(n_streams: int = 200, S: int = 4096, O: int = 8, r0: int = 6,
                eps: float = 0.01, first_seed: int = 100) -> Replay:
    """Independent reveal orders over the paper-scale grid.

    Stream k draws, from ``default_rng(first_seed + k)``, a hidden true
    (capacity, tail) per cell uniformly inside its bounds and a random
    permutation of the cells. The first ``r0`` cells of the permutation form
    the common initial design; the permutation position also breaks exact
    score ties.
    """
    base = make_workload(1)
    base = dataclasses.replace(base, O=O, S=S,
                               name=f"replay: {n_streams} streams over the paper-scale grid, "
                                    f"unrevealed cand x {O} outcomes x {S} samples per round")
    cells = base.cells
    lo_c = base.cap_lo.reshape(-1).astype(np.float64)
    hi_c = base.cap_hi.reshape(-1).astype(np.float64)
    lo_l = base.tail_lo.reshape(-1).astype(np.float64)
    hi_l = base.tail_hi.reshape(-1).astype(np.float64)
    tc = np.empty((n_streams, cells), np.float32)
    tl = np.empty((n_streams, cells), np.float32)
    perm = np.empty((n_streams, cells), np.int32)
    for k in range(n_streams):
        rng = np.random.default_rng(first_seed + k)
        u = rng.random((2, cells))
        c = np.clip((lo_c + u[0] * (hi_c - lo_c)).astype(np.float32),
                    base.cap_lo.reshape(-1), base.cap_hi.reshape(-1))
        l = np.clip((lo_l + u[1] * (hi_l - lo_l)).astype(np.float32),
                    base.tail_lo.reshape(-1), base.tail_hi.reshape(-1))
        tc[k] = c
        tl[k] = l
        perm[k] = rng.permutation(cells).astype(np.int32)
    return Replay(base, tc, tl, perm, r0, eps, cells)


def random_small(rng: np.random.Generator, K: int, B: int, G: int,
                 p_infeasible: float = 0.2) -> Workload:
    """A random small instance for brute-force and property tests.

    Capacities are drawn so that the interesting range of fulfilment (about
    0.2 to 1.5 of demand per full budget) is hit; a share of cells gets a tail
    above its SLO.
    """
    lam = rng.uniform(0.5, 6.0, K).astype(np.float32)
    slo = rng.choice(np.array([10.0, 20.0, 30.0]), K).astype(np.float32)
    shape = (K, T, B)
    base = rng.uniform(0.1, 3.0, shape)
    w = rng.uniform(0.0, 0.6, shape)
    cap_lo = base.astype(np.float32)
    cap_hi = (base * (1.0 + w)).astype(np.float32)
    cap_hi = np.maximum(cap_hi, cap_lo)
    L = slo[:, None, None].astype(np.float64)
    t_mid = L * rng.uniform(0.3, 1.2, shape)
    bad = rng.random(shape) < p_infeasible
    t_mid = np.where(bad, L * rng.uniform(1.3, 3.0, shape), t_mid)
    span = rng.uniform(0.0, 0.5, shape)
    tail_lo = (t_mid * (1.0 - 0.5 * span)).astype(np.float32)
    tail_hi = (t_mid * (1.0 + 0.5 * span)).astype(np.float32)
    tail_hi = np.maximum(tail_hi, tail_lo)
    cand = np.arange(K * T * B, dtype=np.int32)
    return Workload(f"random K={K} B={B} G={G}", K, B, G, lam, slo,
                    cap_lo, cap_hi, tail_lo, tail_hi, cand, 2, 8,
                    int(rng.integers(0, 2**31)))


def log2_exact(x: int) -> int:
    v = int(round(math.log2(x)))
    if 1 << v != x:
        raise ValueError(f"{x} is not a power of two")
    return v
