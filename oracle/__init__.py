"""ctypes front end of the CPU oracle (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
leg use this package. It builds ``liboracle.so`` with gcc on first use.
"""

from __future__ import annotations

import ctypes as C
import dataclasses

import numpy as np

from . import build as _build

OR_KMAX = 64
SOLVER_LITERAL = 0
SOLVER_FRONTIER = 1


class _Problem(C.Structure):
    _fields_ = [("K", C.c_int), ("B", C.c_int), ("G", C.c_int),
                ("demand", C.POINTER(C.c_float)), ("slo", C.POINTER(C.c_float)),
                ("floor", C.POINTER(C.c_float)), ("prior", C.c_int)]


class _Alloc(C.Structure):
    _fields_ = [("t_star", C.c_float), ("total_gpus", C.c_int32), ("ok", C.c_int32),
                ("floors_met", C.c_int32), ("has_option_mask", C.c_uint64),
                ("tp", C.c_int32 * OR_KMAX), ("bin", C.c_int32 * OR_KMAX),
                ("replicas", C.c_int32 * OR_KMAX), ("fulfil", C.c_float * OR_KMAX)]


@dataclasses.dataclass
class Allocation:
    t_star: float
    total_gpus: int
    ok: int
    has_option_mask: int
    tp: list
    bin: list
    replicas: list
    fulfil: list
    floors_met: int = 1

    @staticmethod
    def of(a: _Alloc, K: int) -> "Allocation":
        return Allocation(float(a.t_star), int(a.total_gpus), int(a.ok), int(a.has_option_mask),
                          [int(a.tp[i]) for i in range(K)], [int(a.bin[i]) for i in range(K)],
                          [int(a.replicas[i]) for i in range(K)],
                          [float(np.float32(a.fulfil[i])) for i in range(K)], int(a.floors_met))


_lib = None


def lib():
    global _lib
    if _lib is None:
        _lib = C.CDLL(_build.build())
        fp = C.POINTER(C.c_float)
        ip = C.POINTER(C.c_int32)
        _lib.or_philox4x32_10.argtypes = [C.POINTER(C.c_uint32), C.POINTER(C.c_uint32),
                                          C.POINTER(C.c_uint32)]
        _lib.or_triangular_table.argtypes = [C.c_int, fp]
        _lib.or_draw_index.argtypes = [C.c_uint64, C.c_uint32, C.c_uint32, C.c_int32, C.c_int,
                                       C.c_int, C.c_int, C.c_int, ip, ip]
        _lib.or_map.argtypes = [C.c_float, C.c_float, C.c_float]
        _lib.or_map.restype = C.c_float
        _lib.or_fulfil.argtypes = [C.c_int, C.c_float, C.c_float]
        _lib.or_fulfil.restype = C.c_float
        for name in ("or_solve_literal", "or_solve_frontier"):
            getattr(_lib, name).argtypes = [C.POINTER(_Problem), fp, fp, C.POINTER(_Alloc)]
        _lib.or_evaluate.argtypes = [C.POINTER(_Problem), fp, fp, ip, ip, ip,
                                     C.POINTER(C.c_double), C.POINTER(C.c_double)]
        _lib.or_base_gap.argtypes = [C.POINTER(_Problem), fp, fp, fp, fp, C.c_int,
                                     C.POINTER(_Alloc), C.POINTER(_Alloc), fp]
        _lib.or_scenario.argtypes = [C.POINTER(_Problem), fp, fp, fp, fp, fp, C.c_int,
                                     C.c_uint64, C.c_uint32, C.c_uint32, C.c_int32,
                                     C.c_int, C.c_int, C.c_int, C.c_int,
                                     fp, fp, C.POINTER(_Alloc), C.POINTER(_Alloc)]
        _lib.or_score.argtypes = [C.POINTER(_Problem), fp, fp, fp, fp, fp, C.c_int,
                                  C.c_uint64, C.c_uint32, C.c_uint32, C.c_int, ip, C.c_int,
                                  C.c_int, C.c_int, C.POINTER(C.c_int64), C.POINTER(C.c_double),
                                  C.POINTER(C.c_double), C.POINTER(C.c_int64), fp, ip, fp]
        _lib.or_score_cached.argtypes = [C.POINTER(_Problem), fp, fp, fp, fp, fp, C.c_int,
                                         C.c_uint64, C.c_uint32, C.c_uint32, C.c_int, ip, C.c_int,
                                         C.c_int, C.c_int, C.POINTER(C.c_int64), fp]
        i64p = C.POINTER(C.c_int64)
        _lib.or_goodput_fx.argtypes = [C.c_int, C.c_float, C.c_float]
        _lib.or_goodput_fx.restype = C.c_int64
        _lib.or_solve_lex.argtypes = [C.POINTER(_Problem), fp, fp, C.c_int, C.POINTER(_Alloc), i64p]
        _lib.or_base_gap_lex.argtypes = [C.POINTER(_Problem), fp, fp, fp, fp, C.c_int,
                                         C.POINTER(_Alloc), C.POINTER(_Alloc), i64p, i64p, fp,
                                         C.POINTER(C.c_double)]
        _lib.or_certificate_lex.argtypes = [C.POINTER(_Problem), fp, fp, fp, fp,
                                            C.POINTER(C.c_uint8), C.c_float, C.c_int,
                                            C.POINTER(C.c_int), fp, C.POINTER(C.c_double)]
        _lib.or_score_goodput.argtypes = [C.POINTER(_Problem), fp, fp, fp, fp, fp, C.c_int,
                                          C.c_uint64, C.c_uint32, C.c_uint32, C.c_int, ip, C.c_int,
                                          C.c_int, C.c_int, i64p, C.POINTER(C.c_double),
                                          C.POINTER(C.c_double), i64p, i64p,
                                          C.POINTER(C.c_double), ip]
        _lib.or_refit.argtypes = [C.POINTER(_Problem), C.c_int, C.c_int32, C.c_float, C.c_float,
                                  fp, fp, fp, fp]
        _lib.or_reduce.argtypes = [C.POINTER(_Problem), C.c_int, ip, C.c_int, C.c_int, C.c_float,
                                   C.POINTER(C.c_int64), C.POINTER(C.c_double),
                                   C.POINTER(C.c_double), C.POINTER(C.c_int64), ip]
        _lib.or_certificate.argtypes = [C.POINTER(_Problem), fp, fp, fp, fp,
                                        C.POINTER(C.c_uint8), C.c_float, C.c_int,
                                        C.POINTER(C.c_int), fp]
        _lib.or_replay_stream.argtypes = [C.POINTER(_Problem), fp, fp, fp, fp, fp, fp, ip,
                                          C.c_int, C.c_float, fp, C.c_int, C.c_uint64,
                                          C.c_uint32, C.c_int, C.c_int, C.c_int, C.c_int, C.c_int,
                                          ip, ip, ip, C.POINTER(C.c_double), ip,
                                          C.POINTER(_Alloc), fp]
        _lib.or_replay_stream_cached.argtypes = [C.POINTER(_Problem), fp, fp, fp, fp, fp, fp, ip,
                                          C.c_int, C.c_float, fp, C.c_int, C.c_uint64,
                                          C.c_uint32, C.c_int, C.c_int, C.c_int, C.c_int, C.c_int,
                                          ip, ip, ip, C.POINTER(C.c_double), ip,
                                          C.POINTER(_Alloc), fp]
    return _lib


def _f32(a) -> np.ndarray:
    return np.ascontiguousarray(np.asarray(a, dtype=np.float32).reshape(-1))


def _ptr(a: np.ndarray, ctype):
    return a.ctypes.data_as(C.POINTER(ctype))


PRIOR_REVEALED = 0
PRIOR_MONOTONE = 1


class Problem:
    """K classes, B bins, budget G, demands, SLOs and optional critical floors
    delta_i in [0, 1] (0 = not critical) (Section 3); the interval prior used
    when a cell is measured (PRIOR_REVEALED or PRIOR_MONOTONE, Section 4.1)."""

    def __init__(self, K, B, G, demand, slo, floor=None, prior=PRIOR_REVEALED):
        self.K, self.B, self.G = int(K), int(B), int(G)
        self.demand = _f32(demand)
        self.slo = _f32(slo)
        self.floor = None if floor is None else _f32(floor)
        assert self.demand.size == self.K and self.slo.size == self.K
        assert self.floor is None or self.floor.size == self.K
        self.prior = int(prior)
        self._s = _Problem(self.K, self.B, self.G, _ptr(self.demand, C.c_float),
                           _ptr(self.slo, C.c_float),
                           None if self.floor is None else _ptr(self.floor, C.c_float), self.prior)

    @staticmethod
    def of(w) -> "Problem":
        return Problem(w.K, w.B, w.G, w.demand, w.slo, getattr(w, "floor", None),
                       getattr(w, "prior", PRIOR_REVEALED))

    @property
    def cells(self) -> int:
        return self.K * 4 * self.B


def philox4x32_10(ctr, key):
    c = np.ascontiguousarray(ctr, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    out = np.zeros(4, np.uint32)
    lib().or_philox4x32_10(_ptr(c, C.c_uint32), _ptr(k, C.c_uint32), _ptr(out, C.c_uint32))
    return out


def triangular_table(Q: int = 4096) -> np.ndarray:
    out = np.zeros(Q, np.float32)
    lib().or_triangular_table(Q, _ptr(out, C.c_float))
    return out


def draw_index(seed, stream_id, rnd, cell, Q, O, o, s):
    kc, kl = C.c_int32(), C.c_int32()
    rc = lib().or_draw_index(seed, stream_id, rnd, cell, Q, O, o, s, C.byref(kc), C.byref(kl))
    if rc:
        raise ValueError("invalid draw arguments")
    return kc.value, kl.value


def map_value(lo, hi, q) -> float:
    return float(np.float32(lib().or_map(lo, hi, q)))


def fulfil(n, c, lam) -> float:
    return float(np.float32(lib().or_fulfil(n, c, lam)))


def solve(prob: Problem, cap, tail, solver: int = SOLVER_FRONTIER) -> Allocation:
    cap = _f32(cap)
    tail = _f32(tail)
    assert cap.size == prob.cells and tail.size == prob.cells
    a = _Alloc()
    fn = lib().or_solve_literal if solver == SOLVER_LITERAL else lib().or_solve_frontier
    rc = fn(C.byref(prob._s), _ptr(cap, C.c_float), _ptr(tail, C.c_float), C.byref(a))
    if rc:
        raise ValueError(f"oracle solve failed ({rc})")
    return Allocation.of(a, prob.K)


def evaluate(prob: Problem, cap, tail, tp_index, bins, replicas):
    cap = _f32(cap)
    tail = _f32(tail)
    ti = np.ascontiguousarray(tp_index, np.int32)
    bi = np.ascontiguousarray(bins, np.int32)
    ri = np.ascontiguousarray(replicas, np.int32)
    mm, gp = C.c_double(), C.c_double()
    rc = lib().or_evaluate(C.byref(prob._s), _ptr(cap, C.c_float), _ptr(tail, C.c_float),
                           _ptr(ti, C.c_int32), _ptr(bi, C.c_int32), _ptr(ri, C.c_int32),
                           C.byref(mm), C.byref(gp))
    if rc < 0:
        raise ValueError("bad problem")
    return mm.value, gp.value, rc == 0


def _bounds(w):
    return [_f32(w.cap_lo), _f32(w.cap_hi), _f32(w.tail_lo), _f32(w.tail_hi)]


def base_gap(prob: Problem, cap_lo, cap_hi, tail_lo, tail_hi, solver=SOLVER_FRONTIER):
    arrs = [_f32(x) for x in (cap_lo, cap_hi, tail_lo, tail_hi)]
    am, ap = _Alloc(), _Alloc()
    g = C.c_float()
    rc = lib().or_base_gap(C.byref(prob._s), *[_ptr(x, C.c_float) for x in arrs], solver,
                           C.byref(am), C.byref(ap), C.byref(g))
    if rc:
        raise ValueError("oracle base gap failed")
    return Allocation.of(am, prob.K), Allocation.of(ap, prob.K), float(np.float32(g.value))


def scenario(w, qn, cell, o, s, solver=SOLVER_FRONTIER, seed=None, stream_id=None, rnd=None):
    prob = Problem.of(w)
    b = _bounds(w)
    qn = _f32(qn)
    cy, ly = C.c_float(), C.c_float()
    am, ap = _Alloc(), _Alloc()
    rc = lib().or_scenario(C.byref(prob._s), *[_ptr(x, C.c_float) for x in b],
                           _ptr(qn, C.c_float), qn.size,
                           w.seed if seed is None else seed,
                           w.stream_id if stream_id is None else stream_id,
                           w.round if rnd is None else rnd, cell, w.O, o, s, solver,
                           C.byref(cy), C.byref(ly), C.byref(am), C.byref(ap))
    if rc:
        raise ValueError("oracle scenario failed")
    return (float(np.float32(cy.value)), float(np.float32(ly.value)),
            Allocation.of(am, prob.K), Allocation.of(ap, prob.K))


@dataclasses.dataclass
class ScoreResult:
    sum_eo: np.ndarray  # [n_cand, O] int64
    gap: np.ndarray  # [n_cand] float64, E[Gamma_{t+1} | e]
    score: np.ndarray  # [n_cand] float64
    score_fixed: np.ndarray  # [n_cand] int64
    gamma_t: float
    best: int
    dump_t: np.ndarray | None  # [n_cand, O, S, 2] float32 (t*-, t*+)


def score(w, qn, candidates=None, solver=SOLVER_FRONTIER, dump=False, seed=None,
          stream_id=None, rnd=None, O=None, S=None) -> ScoreResult:
    prob = Problem.of(w)
    b = _bounds(w)
    qn = _f32(qn)
    cand = np.ascontiguousarray(w.candidates if candidates is None else candidates, np.int32)
    O = w.O if O is None else O
    S = w.S if S is None else S
    n = cand.size
    sum_eo = np.zeros((n, O), np.int64)
    gap = np.zeros(n, np.float64)
    sc = np.zeros(n, np.float64)
    scf = np.zeros(n, np.int64)
    gt = C.c_float()
    best = C.c_int32()
    dt = np.zeros((n, O, S, 2), np.float32) if dump else None
    rc = lib().or_score(C.byref(prob._s), *[_ptr(x, C.c_float) for x in b],
                        _ptr(qn, C.c_float), qn.size,
                        w.seed if seed is None else seed,
                        w.stream_id if stream_id is None else stream_id,
                        w.round if rnd is None else rnd, n, _ptr(cand, C.c_int32), O, S,
                        solver, _ptr(sum_eo, C.c_int64), _ptr(gap, C.c_double),
                        _ptr(sc, C.c_double), _ptr(scf, C.c_int64), C.byref(gt), C.byref(best),
                        _ptr(dt, C.c_float) if dump else None)
    if rc:
        raise ValueError(f"oracle score failed ({rc})")
    return ScoreResult(sum_eo, gap, sc, scf, float(np.float32(gt.value)), int(best.value), dt)


def score_sums_cached(w, qn, candidates=None, solver=SOLVER_FRONTIER, seed=None,
                      stream_id=None, rnd=None, O=None, S=None):
    """Fixed-point sums [n_cand, O] of :func:`score` and Gamma_t, with each
    candidate's solves cached by (capacity position, tail within SLO); the
    same values as :func:`score`, for workloads too large for it."""
    prob = Problem.of(w)
    b = _bounds(w)
    qn = _f32(qn)
    cand = np.ascontiguousarray(w.candidates if candidates is None else candidates, np.int32)
    O = w.O if O is None else O
    S = w.S if S is None else S
    sum_eo = np.zeros((cand.size, O), np.int64)
    gt = C.c_float()
    rc = lib().or_score_cached(C.byref(prob._s), *[_ptr(x, C.c_float) for x in b],
                               _ptr(qn, C.c_float), qn.size,
                               w.seed if seed is None else seed,
                               w.stream_id if stream_id is None else stream_id,
                               w.round if rnd is None else rnd, cand.size, _ptr(cand, C.c_int32),
                               O, S, solver, _ptr(sum_eo, C.c_int64), C.byref(gt))
    if rc:
        raise ValueError(f"oracle cached score failed ({rc})")
    return sum_eo, float(np.float32(gt.value))


def reduce_sums(w, candidates, sum_eo, gamma_t, O=None, S=None) -> ScoreResult:
    """E[Gamma_{t+1} | e], scores and the argmax from fixed-point sums."""
    prob = Problem.of(w)
    cand = np.ascontiguousarray(candidates, np.int32)
    se = np.ascontiguousarray(sum_eo, np.int64)
    O = w.O if O is None else O
    S = w.S if S is None else S
    assert se.shape == (cand.size, O)
    n = cand.size
    gap = np.zeros(n, np.float64)
    sc = np.zeros(n, np.float64)
    scf = np.zeros(n, np.int64)
    best = C.c_int32()
    rc = lib().or_reduce(C.byref(prob._s), n, _ptr(cand, C.c_int32), O, S, gamma_t,
                         _ptr(se, C.c_int64), _ptr(gap, C.c_double), _ptr(sc, C.c_double),
                         _ptr(scf, C.c_int64), C.byref(best))
    if rc:
        raise ValueError("oracle reduce failed")
    return ScoreResult(se.copy(), gap, sc, scf, float(np.float32(gamma_t)), int(best.value), None)


def refit(prob: Problem, cell, c, l, cap_lo, cap_hi, tail_lo, tail_hi, prior=None):
    """The four bound arrays after measuring (c, l) at cell under the prior
    (the problem's when None); returns new arrays."""
    arrs = [_f32(x).copy() for x in (cap_lo, cap_hi, tail_lo, tail_hi)]
    rc = lib().or_refit(C.byref(prob._s), prob.prior if prior is None else int(prior), int(cell),
                        float(c), float(l), *[_ptr(x, C.c_float) for x in arrs])
    if rc:
        raise ValueError("oracle refit failed")
    return arrs


def goodput_fx(n, c, lam) -> int:
    return int(lib().or_goodput_fx(int(n), float(c), float(lam)))


def solve_lex(prob: Problem, cap, tail, solver: int = SOLVER_FRONTIER):
    """Tiers 1-4 of the lexicographic objective: (Allocation, goodput in 2^-20 req/s)."""
    cap = _f32(cap)
    tail = _f32(tail)
    a = _Alloc()
    g = C.c_int64()
    rc = lib().or_solve_lex(C.byref(prob._s), _ptr(cap, C.c_float), _ptr(tail, C.c_float), solver,
                            C.byref(a), C.byref(g))
    if rc:
        raise ValueError(f"oracle lexicographic solve failed ({rc})")
    return Allocation.of(a, prob.K), int(g.value)


def base_gap_lex(prob: Problem, cap_lo, cap_hi, tail_lo, tail_hi, solver=SOLVER_FRONTIER):
    """(A-, A+, GP-, GP+, max-min gap, goodput gap) with both solved to tier 4."""
    arrs = [_f32(x) for x in (cap_lo, cap_hi, tail_lo, tail_hi)]
    am, ap = _Alloc(), _Alloc()
    gm, gp = C.c_int64(), C.c_int64()
    gmm = C.c_float()
    ggp = C.c_double()
    rc = lib().or_base_gap_lex(C.byref(prob._s), *[_ptr(x, C.c_float) for x in arrs], solver,
                               C.byref(am), C.byref(ap), C.byref(gm), C.byref(gp), C.byref(gmm),
                               C.byref(ggp))
    if rc:
        raise ValueError("oracle lexicographic base gap failed")
    return (Allocation.of(am, prob.K), Allocation.of(ap, prob.K), int(gm.value), int(gp.value),
            float(np.float32(gmm.value)), float(ggp.value))


def certificate_lex(prob: Problem, cap_lo, cap_hi, tail_lo, tail_hi, revealed, eps,
                    solver=SOLVER_FRONTIER):
    arrs = [_f32(x) for x in (cap_lo, cap_hi, tail_lo, tail_hi)]
    rev = np.ascontiguousarray(revealed, np.uint8).reshape(-1)
    st = C.c_int()
    gmm = C.c_float()
    ggp = C.c_double()
    rc = lib().or_certificate_lex(C.byref(prob._s), *[_ptr(x, C.c_float) for x in arrs],
                                  _ptr(rev, C.c_uint8), eps, solver, C.byref(st), C.byref(gmm),
                                  C.byref(ggp))
    if rc:
        raise ValueError("oracle lexicographic certificate failed")
    return int(st.value), float(np.float32(gmm.value)), float(ggp.value)


@dataclasses.dataclass
class GoodputScore:
    sum_eo: np.ndarray  # [n_cand, O] int64, sums of |GP+' - GP-'| in 2^-20 req/s
    gap: np.ndarray  # [n_cand] E[Gamma_gp,t+1 | e] (fraction of total demand)
    score: np.ndarray
    score_fixed: np.ndarray
    gamma_fx: int  # |GP+ - GP-| at the bounds, 2^-20 req/s
    gamma_gp: float
    best: int


def score_goodput(w, qn, candidates=None, solver=SOLVER_FRONTIER, seed=None, stream_id=None,
                  rnd=None, O=None, S=None) -> GoodputScore:
    prob = Problem.of(w)
    b = _bounds(w)
    qn = _f32(qn)
    cand = np.ascontiguousarray(w.candidates if candidates is None else candidates, np.int32)
    O = w.O if O is None else O
    S = w.S if S is None else S
    n = cand.size
    sum_eo = np.zeros((n, O), np.int64)
    gap = np.zeros(n, np.float64)
    sc = np.zeros(n, np.float64)
    scf = np.zeros(n, np.int64)
    gfx = C.c_int64()
    ggp = C.c_double()
    best = C.c_int32()
    rc = lib().or_score_goodput(C.byref(prob._s), *[_ptr(x, C.c_float) for x in b],
                                _ptr(qn, C.c_float), qn.size,
                                w.seed if seed is None else seed,
                                w.stream_id if stream_id is None else stream_id,
                                w.round if rnd is None else rnd, n, _ptr(cand, C.c_int32), O, S, solver,
                                _ptr(sum_eo, C.c_int64), _ptr(gap, C.c_double), _ptr(sc, C.c_double),
                                _ptr(scf, C.c_int64), C.byref(gfx), C.byref(ggp), C.byref(best))
    if rc:
        raise ValueError(f"oracle goodput score failed ({rc})")
    return GoodputScore(sum_eo, gap, sc, scf, int(gfx.value), float(ggp.value), int(best.value))


def certificate(prob: Problem, cap_lo, cap_hi, tail_lo, tail_hi, revealed, eps,
                solver=SOLVER_FRONTIER):
    arrs = [_f32(x) for x in (cap_lo, cap_hi, tail_lo, tail_hi)]
    rev = np.ascontiguousarray(revealed, np.uint8).reshape(-1)
    st = C.c_int()
    g = C.c_float()
    rc = lib().or_certificate(C.byref(prob._s), *[_ptr(x, C.c_float) for x in arrs],
                              _ptr(rev, C.c_uint8), eps, solver, C.byref(st), C.byref(g))
    if rc:
        raise ValueError("oracle certificate failed")
    return int(st.value), float(np.float32(g.value))


@dataclasses.dataclass
class ReplayResult:
    rounds: int
    reveal_order: np.ndarray
    gpu_seconds: float
    state: int
    final_minus: Allocation
    gamma_trace: np.ndarray


def replay_stream(rp, k: int, qn, seed: int, S=None, O=None, max_rounds=None,
                  solver=SOLVER_FRONTIER, policy: int = 0, perm=None, cached: bool = False) -> ReplayResult:
    """Algorithm 1 on stream k of the replay ``rp``. policy 0: reveal the
    best-scored cell; 1: the next unrevealed cell of ``perm`` (default: the
    stream's own permutation). cached: each round scored by the cached scorer
    (the same sums and argmax)."""
    w = rp.base
    prob = Problem.of(w)
    b = _bounds(w)
    qn = _f32(qn)
    cells = w.cells
    tc = _f32(rp.truth_cap[k])
    tl = _f32(rp.truth_tail[k])
    perm = np.ascontiguousarray(rp.perm[k] if perm is None else perm, np.int32)
    order = np.full(cells, -1, np.int32)
    mr = rp.max_rounds if max_rounds is None else max_rounds
    trace = np.zeros(mr + 1, np.float32)
    rounds, nrev, st = C.c_int32(), C.c_int32(), C.c_int32()
    gs = C.c_double()
    am = _Alloc()
    fn = lib().or_replay_stream_cached if cached else lib().or_replay_stream
    rc = fn(C.byref(prob._s), *[_ptr(x, C.c_float) for x in b],
                                _ptr(tc, C.c_float), _ptr(tl, C.c_float), _ptr(perm, C.c_int32),
                                rp.r0, rp.eps, _ptr(qn, C.c_float), qn.size, seed, k,
                                w.O if O is None else O, w.S if S is None else S, mr, solver, policy,
                                C.byref(rounds), _ptr(order, C.c_int32), C.byref(nrev),
                                C.byref(gs), C.byref(st), C.byref(am), _ptr(trace, C.c_float))
    if rc:
        raise ValueError("oracle replay failed")
    r = int(rounds.value)
    return ReplayResult(r, order[: nrev.value].copy(), float(gs.value), int(st.value),
                        Allocation.of(am, prob.K), trace[: r + 1].copy())
