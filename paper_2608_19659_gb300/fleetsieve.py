"""ctypes binding of ``libfleetsieve.so`` (the C ABI of include/fleetsieve.h).

Argument marshalling only: every step of the computation runs in the CUDA
library. Host arrays are numpy arrays; device buffers and streams are torch
tensors and ``torch.cuda.Stream`` handles (PyTorch is used for device memory
and streams, nothing else). Every call raises :class:`FleetSieveError` on a
non-zero status, with the library's message. Loading fails loudly when the
library has not been built; there is no fallback.
"""

from __future__ import annotations

import ctypes as C
import dataclasses
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libfleetsieve.so")

FS_OK, FS_EINVAL, FS_ENOMEM, FS_ECUDA, FS_ETIMEOUT, FS_EDEVICE = 0, -1, -2, -3, -4, -5
FS_MAX_CLASSES = 64
EXPORTS = ("fs_load_model", "fs_update_bounds", "fs_set_floors", "fs_dump_stride", "fs_score_candidates",
           "fs_score_candidates_async", "fs_solve", "fs_solve_batch", "fs_solve_bounds",
           "fs_reveal", "fs_set_prior", "fs_set_objective", "fs_score_goodput", "fs_get_state",
           "fs_certificate", "fs_replay", "fs_check", "fs_launch_count",
           "fs_watchdog_selftest", "fs_free_model", "fs_last_error", "fs_score_candidates_noalloc",
           "fs_timing_enable",
           "fs_timing_read", "fs_draw_floor")


class FleetSieveError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"{msg} (status {code})")
        self.code = code


class fs_bounds(C.Structure):
    _fields_ = [("K", C.c_int32), ("B", C.c_int32), ("cap_lo", C.POINTER(C.c_float)),
                ("cap_hi", C.POINTER(C.c_float)), ("tail_lo", C.POINTER(C.c_float)),
                ("tail_hi", C.POINTER(C.c_float)), ("revealed", C.c_void_p),
                ("quantile", C.POINTER(C.c_float)), ("Q", C.c_int32), ("reserved", C.c_int32)]


class fs_samples(C.Structure):
    _fields_ = [("seed", C.c_uint64), ("stream_id", C.c_uint32), ("round", C.c_uint32),
                ("n_cand", C.c_int32), ("O", C.c_int32), ("S", C.c_int32),
                ("reserved", C.c_int32), ("cand", C.c_void_p)]


class fs_allocation(C.Structure):
    _fields_ = [("t_star", C.c_float), ("total_gpus", C.c_int32),
                ("has_option_mask", C.c_uint64), ("ok", C.c_int32), ("floors_met", C.c_int32),
                ("tp", C.c_int8 * FS_MAX_CLASSES), ("bin", C.c_int16 * FS_MAX_CLASSES),
                ("replicas", C.c_int16 * FS_MAX_CLASSES), ("fulfil", C.c_float * FS_MAX_CLASSES),
                ("goodput", C.c_double)]


class fs_replay_spec(C.Structure):
    _fields_ = [("n_streams", C.c_int32), ("r0", C.c_int32), ("eps", C.c_float),
                ("O", C.c_int32), ("S", C.c_int32), ("max_rounds", C.c_int32),
                ("policy", C.c_int32), ("seed", C.c_uint64), ("truth_cap", C.POINTER(C.c_float)),
                ("truth_tail", C.POINTER(C.c_float)), ("perm", C.POINTER(C.c_int32))]


ALLOC_DTYPE = np.dtype({"names": ["t_star", "total_gpus", "has_option_mask", "ok", "floors_met",
                                  "tp", "bin", "replicas", "fulfil", "goodput"],
                        "formats": [np.float32, np.int32, np.uint64, np.int32, np.int32,
                                    (np.int8, 64), (np.int16, 64), (np.int16, 64), (np.float32, 64),
                                    np.float64],
                        "offsets": [0, 4, 8, 16, 20, 24, 88, 216, 344, 600], "itemsize": 608})

_lib = None


def lib():
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise FleetSieveError(FS_ECUDA, f"{LIB_PATH} is not built; run __graft_entry__.build()")
        L = C.CDLL(LIB_PATH)
        fp = C.POINTER(C.c_float)
        L.fs_load_model.argtypes = [C.POINTER(fs_bounds), fp, fp, C.c_int32, C.c_void_p,
                                    C.POINTER(C.c_void_p)]
        L.fs_update_bounds.argtypes = [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]
        L.fs_set_floors.argtypes = [C.c_void_p, C.c_void_p]
        L.fs_dump_stride.argtypes = [C.c_void_p]
        L.fs_dump_stride.restype = C.c_int32
        L.fs_score_candidates.argtypes = [C.c_void_p, C.POINTER(fs_samples), C.c_void_p, C.c_void_p,
                                          C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]
        L.fs_score_candidates_async.argtypes = [C.c_void_p, C.POINTER(fs_samples), C.c_void_p,
                                                C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                                C.c_void_p, C.c_void_p]
        L.fs_score_candidates_noalloc.argtypes = [C.c_int32, C.c_int32, C.c_int32, C.c_void_p,
                                                  C.c_void_p, C.c_void_p, C.c_void_p, C.c_int32,
                                                  C.POINTER(fs_samples), C.c_void_p, C.c_void_p,
                                                  C.c_void_p, C.c_void_p, C.c_void_p]
        L.fs_solve.argtypes = [C.c_void_p, fp, fp, C.POINTER(fs_allocation)]
        L.fs_solve_batch.argtypes = [C.c_void_p, C.c_int32, C.c_void_p, C.c_void_p, C.c_void_p,
                                     C.c_void_p]
        L.fs_solve_bounds.argtypes = [C.c_void_p, C.POINTER(fs_allocation),
                                      C.POINTER(fs_allocation), fp]
        L.fs_reveal.argtypes = [C.c_void_p, C.c_int32, C.c_float, C.c_float]
        L.fs_set_prior.argtypes = [C.c_void_p, C.c_int32]
        L.fs_set_objective.argtypes = [C.c_void_p, C.c_int32]
        L.fs_score_goodput.argtypes = [C.c_void_p, C.POINTER(fs_samples), C.c_void_p, C.c_void_p,
                                       C.c_void_p, C.c_void_p, C.c_void_p]
        L.fs_get_state.argtypes = [C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p,
                                   C.c_void_p]
        L.fs_certificate.argtypes = [C.c_void_p, C.c_float, C.POINTER(C.c_int32), fp]
        L.fs_replay.argtypes = [C.c_void_p, C.POINTER(fs_replay_spec), C.c_void_p, C.c_void_p,
                                C.c_void_p, C.c_void_p, C.c_void_p, C.c_void_p]
        L.fs_check.argtypes = [C.c_void_p, C.c_void_p]
        L.fs_launch_count.restype = C.c_uint64
        L.fs_timing_enable.argtypes = [C.c_void_p, C.c_int32]
        L.fs_timing_read.argtypes = [C.c_void_p, C.POINTER(C.c_double), C.POINTER(C.c_int32),
                                     C.c_void_p, C.c_void_p]
        L.fs_watchdog_selftest.argtypes = [C.c_int64]
        L.fs_draw_floor.argtypes = [C.c_int32, C.c_int32, C.c_int64, C.c_int32, C.POINTER(C.c_double),
                                    C.POINTER(C.c_int64)]
        L.fs_free_model.argtypes = [C.c_void_p]
        L.fs_free_model.restype = None
        L.fs_last_error.restype = C.c_char_p
        _lib = L
    return _lib


def _check(rc: int) -> int:
    if rc != FS_OK:
        raise FleetSieveError(rc, lib().fs_last_error().decode(errors="replace"))
    return rc


def _f32(a) -> np.ndarray:
    if isinstance(a, np.ndarray) and a.dtype == np.float32 and a.flags.c_contiguous:
        return a
    return np.ascontiguousarray(np.asarray(a, dtype=np.float32).reshape(-1))


def _fp(a: np.ndarray):
    return a.ctypes.data_as(C.POINTER(C.c_float))


def _vp(a) -> int | None:
    """Address of a numpy array or torch tensor for a void* argument (None passes NULL)."""
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        try:  # a writable array: a third of the cost of building the array interface
            return C.addressof(C.c_char.from_buffer(a))
        except (TypeError, ValueError):
            return a.__array_interface__["data"][0]
    return a.data_ptr()


def _stream(s) -> C.c_void_p | None:
    if s is None:
        return None
    return C.c_void_p(s.cuda_stream if hasattr(s, "cuda_stream") else int(s))


class Model:
    """Owning handle of an ``fs_model*`` (freed by :func:`fs_free_model` or on collection)."""

    def __init__(self, handle: int, K: int, B: int, G: int, Q: int):
        self.handle = C.c_void_p(handle)
        self.K, self.B, self.G, self.Q = K, B, G, Q
        self.cells = K * 4 * B
        # the arrays of the last call and their addresses: a caller that passes
        # the same arrays again skips taking them (the references held here keep
        # those arrays alive and stop numpy from resizing them in place)
        self._bounds_args = None
        self._score_args = None

    def __del__(self):
        try:
            fs_free_model(self)
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *a):
        fs_free_model(self)


def fs_load_model(cap_lo, cap_hi, tail_lo, tail_hi, slo, demand, G: int, K: int, B: int,
                  quantile=None, stream=None, revealed=None) -> Model:
    """revealed: optional [K*4*B] flags of cells already measured (bounds collapsed)."""
    arrs = [_f32(x) for x in (cap_lo, cap_hi, tail_lo, tail_hi)]
    q = _f32(quantile) if quantile is not None else None
    rv = np.ascontiguousarray(np.asarray(revealed).reshape(-1) != 0, np.uint8) if revealed is not None else None
    if rv is not None and rv.size != K * 4 * B:
        raise ValueError(f"revealed has {rv.size} flags for {K * 4 * B} cells")
    b = fs_bounds(K, B, *[_fp(x) for x in arrs], _vp(rv), _fp(q) if q is not None else None,
                  q.size if q is not None else 0, 0)
    s_ = _f32(slo)
    d_ = _f32(demand)
    out = C.c_void_p()
    _check(lib().fs_load_model(C.byref(b), _fp(s_), _fp(d_), int(G), _stream(stream), C.byref(out)))
    return Model(out.value, K, B, G, q.size if q is not None else 4096)


def fs_update_bounds(m: Model, cap_lo, cap_hi, tail_lo, tail_hi) -> None:
    c = m._bounds_args
    if (c is not None and cap_lo is c[0] and cap_hi is c[1] and tail_lo is c[2] and tail_hi is c[3]):
        addrs = c[4]
    else:
        given = (cap_lo, cap_hi, tail_lo, tail_hi)
        arrs = [_f32(x) for x in given]
        addrs = [_vp(x) for x in arrs]
        # cached only when no conversion was needed (the addresses are the caller's)
        m._bounds_args = (*given, addrs) if all(a is g for a, g in zip(arrs, given)) else None
    _check(lib().fs_update_bounds(m.handle, *addrs))


def fs_set_floors(m: Model, floor=None) -> None:
    """Critical floors delta_i in [0, 1] per class (0: not critical); None clears them."""
    f = _f32(floor) if floor is not None else None
    if f is not None and f.size != m.K:
        raise ValueError(f"floor has {f.size} values for K = {m.K} classes")
    _check(lib().fs_set_floors(m.handle, _vp(f) if f is not None else None))


def fs_dump_stride(m: Model) -> int:
    return int(lib().fs_dump_stride(m.handle))


@dataclasses.dataclass
class ScoreResult:
    gap: np.ndarray  # [n_cand] E[Gamma_{t+1} | e]
    score: np.ndarray  # [n_cand]
    gamma_t: float
    best: int
    sum_eo: np.ndarray  # [n_cand, O] int64


def _samples(seed, stream_id, rnd, n, O, S, cand_addr) -> fs_samples:
    return fs_samples(int(seed) & (2**64 - 1), int(stream_id), int(rnd), int(n), int(O), int(S), 0,
                      cand_addr)


def fs_score_candidates(m: Model, cand, O: int, S: int, seed: int, stream_id: int = 0,
                        rnd: int = 0, dump_dev=None, outputs=None) -> ScoreResult:
    """Synchronous scoring with host inputs and outputs (``outputs`` reuses arrays)."""
    c = m._score_args
    key = (seed, stream_id, rnd, O, S)
    if c is not None and cand is c[0] and outputs is not None and outputs is c[1] and dump_dev is None:
        smp, addrs = c[2], c[3]
        if c[4] != key:
            smp = _samples(seed, stream_id, rnd, smp.n_cand, O, S, smp.cand)
            m._score_args = (cand, outputs, smp, addrs, key)
    else:
        given = cand
        cand = np.ascontiguousarray(cand, dtype=np.int32)
        n = cand.size
        reuse = outputs is not None and dump_dev is None and cand is given
        if outputs is None:
            outputs = (np.zeros(n, np.float64), np.zeros(n, np.float64), np.zeros(1, np.float32),
                       np.zeros(1, np.int32), np.zeros((n, O), np.int64))
        smp = _samples(seed, stream_id, rnd, n, O, S, _vp(cand) if n else None)
        addrs = [_vp(x) for x in outputs] + [_vp(dump_dev)]
        m._score_args = (cand, outputs, smp, addrs, key) if reuse else None
    gap, score, gt, best, sums = outputs
    _check(lib().fs_score_candidates(m.handle, C.byref(smp), *addrs))
    return ScoreResult(gap, score, float(gt[0]), int(best[0]), sums)


def fs_score_candidates_noalloc(K: int, B: int, G: int, bounds_dev, slo_dev, demand_dev, cand_dev,
                                O: int, S: int, seed: int, stream_id: int = 0, rnd: int = 0,
                                gap_dev=None, score_dev=None, gamma_t_dev=None, best_dev=None,
                                quantile_dev=None, stream=None) -> None:
    """Scoring that allocates no device memory (every buffer is the caller's device tensor).

    For callers that cannot allocate while they run (device memory handed out
    by their own pool, or no room for cudaMalloc's device-wide synchronisation
    on their path). bounds_dev: float32 [4 * K * 4 * B] (cap_lo, cap_hi,
    tail_lo, tail_hi); slo_dev, demand_dev: float32 [K]; cand_dev: int32.
    Intermediates use the library's fixed 16 MiB device array; larger calls
    raise FS_EINVAL. Returns after the work on ``stream`` has finished.
    """
    n = int(cand_dev.numel())
    smp = _samples(seed, stream_id, rnd, n, O, S, cand_dev.data_ptr() if n else None)
    Q = int(quantile_dev.numel()) if quantile_dev is not None else 0
    _check(lib().fs_score_candidates_noalloc(int(K), int(B), int(G), _vp(bounds_dev), _vp(slo_dev),
                                             _vp(demand_dev), _vp(quantile_dev), Q, C.byref(smp),
                                             _vp(gap_dev), _vp(score_dev), _vp(gamma_t_dev),
                                             _vp(best_dev), _stream(stream)))


def fs_score_candidates_async(m: Model, cand_dev, O: int, S: int, seed: int, stream_id: int = 0,
                              rnd: int = 0, gap_dev=None, score_dev=None, gamma_t_dev=None,
                              best_dev=None, sum_eo_dev=None, dump_dev=None, stream=None) -> None:
    """Device-pointer scoring enqueued on ``stream`` (torch tensors for every buffer)."""
    n = int(cand_dev.numel())
    smp = _samples(seed, stream_id, rnd, n, O, S, cand_dev.data_ptr() if n else None)
    _check(lib().fs_score_candidates_async(m.handle, C.byref(smp), _vp(gap_dev), _vp(score_dev),
                                           _vp(gamma_t_dev), _vp(best_dev), _vp(sum_eo_dev),
                                           _vp(dump_dev), _stream(stream)))


def alloc_to_dict(a: fs_allocation, K: int) -> dict:
    return {"t_star": float(np.float32(a.t_star)), "total_gpus": int(a.total_gpus),
            "has_option_mask": int(a.has_option_mask), "ok": int(a.ok), "floors_met": int(a.floors_met),
            "tp": [int(a.tp[i]) for i in range(K)], "bin": [int(a.bin[i]) for i in range(K)],
            "replicas": [int(a.replicas[i]) for i in range(K)],
            "fulfil": [float(np.float32(a.fulfil[i])) for i in range(K)], "goodput": float(a.goodput)}


def fs_solve(m: Model, cap, tail) -> dict:
    out = fs_allocation()
    c, t = _f32(cap), _f32(tail)
    _check(lib().fs_solve(m.handle, _fp(c), _fp(t), C.byref(out)))
    return alloc_to_dict(out, m.K)


def fs_solve_batch(m: Model, n: int, cap_dev, tail_dev, out_dev, stream=None) -> None:
    """out_dev: a torch uint8 tensor of n * 608 bytes (view it with :data:`ALLOC_DTYPE`)."""
    _check(lib().fs_solve_batch(m.handle, int(n), _vp(cap_dev), _vp(tail_dev), _vp(out_dev),
                                _stream(stream)))


def fs_solve_bounds(m: Model):
    am, ap = fs_allocation(), fs_allocation()
    g = C.c_float()
    _check(lib().fs_solve_bounds(m.handle, C.byref(am), C.byref(ap), C.byref(g)))
    return alloc_to_dict(am, m.K), alloc_to_dict(ap, m.K), float(np.float32(g.value))


def fs_reveal(m: Model, cell: int, cap: float, tail: float) -> None:
    _check(lib().fs_reveal(m.handle, int(cell), float(cap), float(tail)))


FS_PRIOR_REVEALED, FS_PRIOR_MONOTONE = 0, 1


def fs_set_prior(m: Model, prior: int) -> None:
    """How a measurement refits the intervals: FS_PRIOR_REVEALED (the measured
    cell only) or FS_PRIOR_MONOTONE (also its row, nondecreasing in load)."""
    _check(lib().fs_set_prior(m.handle, int(prior)))


FS_OBJECTIVE_MAXMIN, FS_OBJECTIVE_LEXICOGRAPHIC = 0, 1


def fs_set_objective(m: Model, objective: int) -> None:
    """FS_OBJECTIVE_MAXMIN (tiers 1-2) or FS_OBJECTIVE_LEXICOGRAPHIC (tiers 1-4) for
    the model's solves and certificate."""
    _check(lib().fs_set_objective(m.handle, int(objective)))


@dataclasses.dataclass
class GoodputScore:
    gap: np.ndarray  # [n_cand] E[Gamma_gp,t+1 | e] (fraction of total demand)
    score: np.ndarray  # [n_cand]
    gamma_gp: float
    best: int
    sum_eo: np.ndarray  # [n_cand, O] int64, 2^-20 req/s


def fs_score_goodput(m: Model, cand, O: int, S: int, seed: int, stream_id: int = 0, rnd: int = 0) -> GoodputScore:
    """The goodput stage of the Monte-Carlo score (host inputs and outputs)."""
    cand = np.ascontiguousarray(cand, dtype=np.int32)
    n = cand.size
    gap = np.zeros(n, np.float64)
    score = np.zeros(n, np.float64)
    gg = np.zeros(1, np.float64)
    best = np.zeros(1, np.int32)
    sums = np.zeros((n, O), np.int64)
    smp = _samples(seed, stream_id, rnd, n, O, S, _vp(cand) if n else None)
    _check(lib().fs_score_goodput(m.handle, C.byref(smp), _vp(gap), _vp(score), _vp(gg), _vp(best), _vp(sums)))
    return GoodputScore(gap, score, float(gg[0]), int(best[0]), sums)


def fs_get_state(m: Model):
    """(cap_lo, cap_hi, tail_lo, tail_hi, revealed) of the model now, each [K*4*B]."""
    out = [np.zeros(m.cells, np.float32) for _ in range(4)] + [np.zeros(m.cells, np.uint8)]
    _check(lib().fs_get_state(m.handle, *[_vp(x) for x in out]))
    return tuple(out)


def save_state(m: Model, path: str, round: int = 0, **extra) -> None:
    """Checkpoint of the profiling loop: the model's bounds and revealed flags,
    its K, B, G and the next round number (the draws are counter-based, so a
    resumed loop repeats an uninterrupted one exactly), plus caller arrays."""
    clo, chi, tlo, thi, rev = fs_get_state(m)
    np.savez(path, cap_lo=clo, cap_hi=chi, tail_lo=tlo, tail_hi=thi, revealed=rev,
             dims=np.array([m.K, m.B, m.G, int(round)], np.int64), **extra)


def load_state(path: str, slo, demand, quantile=None, stream=None):
    """A model rebuilt from :func:`save_state`'s file, its next round and the file's arrays."""
    z = dict(np.load(path))
    K, B, G, rnd = (int(x) for x in z.pop("dims"))
    m = fs_load_model(z.pop("cap_lo"), z.pop("cap_hi"), z.pop("tail_lo"), z.pop("tail_hi"), slo, demand,
                      G, K, B, quantile=quantile, stream=stream, revealed=z.pop("revealed"))
    return m, rnd, z


def fs_certificate(m: Model, eps: float):
    st = C.c_int32()
    g = C.c_float()
    _check(lib().fs_certificate(m.handle, float(eps), C.byref(st), C.byref(g)))
    return int(st.value), float(np.float32(g.value))


@dataclasses.dataclass
class ReplayResult:
    rounds: np.ndarray
    state: np.ndarray
    gpu_seconds: np.ndarray
    reveal_order: np.ndarray  # [n, cells], -1 padded
    gamma_trace: np.ndarray  # [n, max_rounds + 1]
    final_minus: np.ndarray  # [n] ALLOC_DTYPE


def fs_replay(m: Model, truth_cap, truth_tail, perm, r0: int, eps: float, O: int, S: int,
              seed: int, max_rounds: int, policy: int = 0) -> ReplayResult:
    """policy 0: reveal the best-scored cell each round; 1: the next unrevealed cell of perm."""
    tc = _f32(truth_cap)
    tl = _f32(truth_tail)
    pm = np.ascontiguousarray(perm, dtype=np.int32).reshape(-1)
    n = pm.size // m.cells
    spec = fs_replay_spec(n, int(r0), float(eps), int(O), int(S), int(max_rounds), int(policy),
                          int(seed) & (2**64 - 1), _fp(tc), _fp(tl),
                          pm.ctypes.data_as(C.POINTER(C.c_int32)))
    rounds = np.zeros(n, np.int32)
    state = np.zeros(n, np.int32)
    gs = np.zeros(n, np.float64)
    order = np.zeros((n, m.cells), np.int32)
    trace = np.zeros((n, max_rounds + 1), np.float32)
    final = np.zeros(n, ALLOC_DTYPE)
    _check(lib().fs_replay(m.handle, C.byref(spec), _vp(rounds), _vp(state), _vp(gs), _vp(order),
                           _vp(trace), _vp(final)))
    return ReplayResult(rounds, state, gs, order, trace, final)


def fs_check(m: Model, stream=None) -> None:
    _check(lib().fs_check(m.handle, _stream(stream)))


def fs_timing_enable(m: Model, mode: int) -> None:
    """0 off, 1 Monte-Carlo kernel only, 2 every phase of a scoring call."""
    _check(lib().fs_timing_enable(m.handle, int(mode)))


def fs_timing_read(m: Model, with_entries: bool = False):
    """(Monte-Carlo kernel ms, timed calls, [solve, prep, Monte-Carlo, reduction] ms) since the last
    read; with_entries adds the work counts since then: (t* evaluated in gap-table builds,
    scenarios that tested their tail gate)."""
    ms = C.c_double()
    n = C.c_int32()
    ph = np.zeros(4, np.float64)
    wc = np.zeros(2, np.uint64)
    _check(lib().fs_timing_read(m.handle, C.byref(ms), C.byref(n), _vp(ph), _vp(wc) if with_entries else None))
    if with_entries:
        return float(ms.value), int(n.value), ph, (int(wc[0]), int(wc[1]))
    return float(ms.value), int(n.value), ph


def fs_launch_count() -> int:
    return int(lib().fs_launch_count())


def fs_draw_floor(mode: int, w: int, calls: int, reps: int = 10):
    """Measurement floor of the table path's draws (mode 0: Philox alone; 1:
    with the per-sample lookup): (median ms per launch, calls per launch)."""
    ms = C.c_double(0.0)
    done = C.c_int64(0)
    _check(lib().fs_draw_floor(int(mode), int(w), int(calls), int(reps), C.byref(ms), C.byref(done)))
    return float(ms.value), int(done.value)


def fs_watchdog_selftest(timeout_ns: int) -> int:
    """Returns the status code (FS_ETIMEOUT when the watchdog works)."""
    return int(lib().fs_watchdog_selftest(int(timeout_ns)))


def fs_free_model(m: Model) -> None:
    if m is not None and m.handle and m.handle.value:
        lib().fs_free_model(m.handle)
        m.handle = C.c_void_p()


def fs_last_error() -> str:
    return lib().fs_last_error().decode(errors="replace")


def dump_dtype(K: int) -> np.dtype:
    """numpy view of one dump record (fs_scenario_head + choice[2][K])."""
    return np.dtype([("c_y", np.float32), ("l_y", np.float32), ("t_star", np.float32, 2),
                     ("total_gpus", np.int32, 2), ("choice", np.uint32, (2, K))])


def decode_choice(code: int):
    """(replicas, TP degree, bin) of one packed dump choice; (0, 0, -1) when empty."""
    n = code & 0xFFFF
    if n == 0:
        return 0, 0, -1
    return n, 1 << ((code >> 16) & 3), (code >> 18) & 0x1FFF
