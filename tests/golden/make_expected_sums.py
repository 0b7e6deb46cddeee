"""Write the oracle's expected fixed-point sums of the large scoring workloads.

Calls only the CPU oracle (``oracle/``) and the seeded input generator
(``paper_2608_19659_gb300/workloads.py``, inputs only). For every candidate e
and outcome o of a workload the oracle's Monte-Carlo estimator (Section 4.3:
draws, patched conservative and optimistic realisations, both allocations
solved, g = rint(Gamma' 2^40) summed in int64) gives sum_eo[e][o];
``or_score_cached`` computes the same values as ``or_score`` scenario for
scenario, reusing a candidate's solves for repeated (capacity position, tail
within SLO) pairs. Candidates are split into contiguous ranges, one
single-threaded oracle process per range; the sums do not depend on the split.

Usage: python tests/golden/make_expected_sums.py [--procs N] [name ...]
with names from WORKLOADS below, "replay" and "goodput" (default: all). Each sums file records:
  * the sha256 of the workload's inputs (bounds, demands, SLOs, candidates),
  * Gamma_t and the argmax cell,
  * per candidate the deficits d[e][o] = S rint(Gamma_t 2^40) - sum_eo[e][o]
    (the fixed-point score of each outcome stratum; 0 for a candidate that
    cannot change either allocation), so that sum_eo = S rint(Gamma_t 2^40) - d.

"goodput" writes the goodput stage of the score (every scenario's two
realisations solved to tier 4) on the paper-scale workload in full: per
candidate and outcome the int64 sum, with Gamma_gp,t in 2^-20 units and the
argmax.

"replay" writes the replay workload (Algorithm 1 over 200 reveal orders of
the paper-scale grid, 8 x 4096 samples per candidate and round, seed 2026):
per stream its rounds, final certificate state, GPU-seconds, reveal order and
Gamma_t trace, from the oracle's replay with each round scored by the cached
scorer (held equal to the plain one by the tests).
"""

from __future__ import annotations

import argparse
import dataclasses
import hashlib
import multiprocessing as mp
import os
import sys
import time

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(os.path.dirname(HERE))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

# name -> (workload index, demand factor, output file)
WORKLOADS = {
    "large": (3, 1.0, "large_workload_sums.txt"),
    "mid_x3": (2, 3.0, "mid_workload_x3_sums.txt"),
}


def workload(name):
    from paper_2608_19659_gb300 import workloads

    idx, factor, _ = WORKLOADS[name]
    w = workloads.make_workload(idx)
    if factor != 1.0:
        w = dataclasses.replace(w, demand=(w.demand * np.float32(factor)).astype(np.float32))
    return w


def input_digest(w) -> str:
    h = hashlib.sha256()
    for a in (w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi, w.demand, w.slo):
        h.update(np.ascontiguousarray(a, np.float32).tobytes())
    h.update(np.ascontiguousarray(w.candidates, np.int32).tobytes())
    h.update(np.array([w.K, w.B, w.G, w.O, w.S, w.seed, w.stream_id, w.round], np.int64).tobytes())
    return h.hexdigest()


def _range_sums(args):
    name, lo, hi = args
    import oracle

    w = workload(name)
    qn = oracle.triangular_table(4096)
    se, gt = oracle.score_sums_cached(w, qn, candidates=w.candidates[lo:hi])
    return lo, se, gt


def compute(name, procs):
    import oracle

    w = workload(name)
    n = len(w.candidates)
    step = max(1, (n + 4 * procs - 1) // (4 * procs))
    jobs = [(name, lo, min(n, lo + step)) for lo in range(0, n, step)]
    sums = np.zeros((n, w.O), np.int64)
    gts = set()
    with mp.get_context("spawn").Pool(procs) as pool:
        for lo, se, gt in pool.imap_unordered(_range_sums, jobs):
            sums[lo:lo + se.shape[0]] = se
            gts.add(gt)
    assert len(gts) == 1
    gamma_t = gts.pop()
    res = oracle.reduce_sums(w, w.candidates, sums, gamma_t)
    return w, sums, res


def write(name, w, sums, res):
    _, _, fname = WORKLOADS[name]
    full = np.int64(w.S) * np.int64(np.rint(np.float64(np.float32(res.gamma_t)) * 2.0**40))
    d = full - sums
    with open(os.path.join(HERE, fname), "w") as f:
        f.write(f"# Expected fixed-point sums of the oracle's decision-gap estimator (Section 4.3)\n")
        f.write(f"# workload: {w.name}, demands x{WORKLOADS[name][1]}\n")
        f.write(f"# written by tests/golden/make_expected_sums.py {name} (oracle/ only)\n")
        f.write(f"# inputs_sha256 {input_digest(w)}\n")
        f.write(f"# columns: cell, then O deficits d[o] = S rint(Gamma_t 2^40) - sum_eo[o]\n")
        f.write(f"gamma_t {np.float32(res.gamma_t).view(np.uint32):08x} {res.gamma_t!r}\n")
        f.write(f"best {res.best}\n")
        f.write(f"shape {len(w.candidates)} {w.O} {w.S}\n")
        for e, cell in enumerate(w.candidates):
            f.write(f"{int(cell)} " + " ".join(str(int(x)) for x in d[e]) + "\n")


GOODPUT_FILE = "goodput_paper_scale_sums.txt"


def write_goodput():
    """The goodput stage of the score (Section 4.3 with both realisations of
    every scenario solved to tier 4 of Section 3's objective) on the
    paper-scale workload in full: 64 candidates x 8 outcomes x 4096 samples,
    one oracle call."""
    import oracle
    from paper_2608_19659_gb300 import workloads

    w = workloads.make_workload(1)
    qn = oracle.triangular_table(4096)
    r = oracle.score_goodput(w, qn)
    with open(os.path.join(HERE, GOODPUT_FILE), "w") as f:
        f.write("# Expected int64 sums of the oracle's goodput stage (Section 4.3, tiers 1-4 of Section 3)\n")
        f.write(f"# workload: {w.name}\n")
        f.write("# written by tests/golden/make_expected_sums.py goodput (oracle/ only)\n")
        f.write(f"# inputs_sha256 {input_digest(w)}\n")
        f.write("# columns: cell, then O sums of rint(|GP(A+') - GP(A-')| 2^20) over the outcome's samples\n")
        f.write(f"gamma_fx {r.gamma_fx}\n")
        f.write(f"gamma_gp {r.gamma_gp!r}\n")
        f.write(f"best {r.best}\n")
        f.write(f"shape {len(w.candidates)} {w.O} {w.S}\n")
        for e, cell in enumerate(w.candidates):
            f.write(f"{int(cell)} " + " ".join(str(int(x)) for x in r.sum_eo[e]) + "\n")
    return w, r


REPLAY_FILE = "replay_200_streams.txt"
REPLAY_SEED = 2026


def _replay_stream(k):
    import oracle
    from paper_2608_19659_gb300 import workloads

    rp = workloads.make_replay()
    qn = oracle.triangular_table(4096)
    r = oracle.replay_stream(rp, k, qn, seed=REPLAY_SEED, cached=True)
    return k, r


def replay_digest(rp) -> str:
    h = hashlib.sha256()
    h.update(input_digest(rp.base).encode())
    for a in (rp.truth_cap, rp.truth_tail):
        h.update(np.ascontiguousarray(a, np.float32).tobytes())
    h.update(np.ascontiguousarray(rp.perm, np.int32).tobytes())
    h.update(np.array([rp.r0, rp.max_rounds], np.int64).tobytes())
    h.update(np.float32(rp.eps).tobytes())
    return h.hexdigest()


def write_replay(procs):
    from paper_2608_19659_gb300 import workloads

    rp = workloads.make_replay()
    n = len(rp.perm)
    res = [None] * n
    with mp.get_context("spawn").Pool(procs) as pool:
        for k, r in pool.imap_unordered(_replay_stream, range(n)):
            res[k] = r
    with open(os.path.join(HERE, REPLAY_FILE), "w") as f:
        f.write("# Expected replay of the oracle: Algorithm 1 on 200 reveal orders of the paper-scale grid\n")
        f.write(f"# {rp.base.O} outcomes x {rp.base.S} samples per candidate and round, eps {rp.eps}, "
                f"seed {REPLAY_SEED}, stream k = Philox stream id k\n")
        f.write("# written by tests/golden/make_expected_sums.py replay (oracle/ only)\n")
        f.write(f"# inputs_sha256 {replay_digest(rp)}\n")
        f.write("# per stream: k rounds state gpu_seconds | reveal order | Gamma_t trace (float32 bits)\n")
        for k, r in enumerate(res):
            trace = " ".join(f"{np.float32(x).view(np.uint32):08x}" for x in r.gamma_trace)
            order = " ".join(str(int(c)) for c in r.reveal_order)
            f.write(f"{k} {r.rounds} {r.state} {r.gpu_seconds!r} | {order} | {trace}\n")
    return res


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("names", nargs="*", default=list(WORKLOADS) + ["replay", "goodput"])
    ap.add_argument("--procs", type=int, default=len(os.sched_getaffinity(0)))
    a = ap.parse_args()
    for name in a.names:
        t0 = time.time()
        if name == "goodput":
            w, r = write_goodput()
            print(f"goodput: {len(w.candidates)} candidates, gamma_fx {r.gamma_fx}, best {r.best}, "
                  f"{time.time() - t0:.0f} s")
            continue
        if name == "replay":
            res = write_replay(a.procs)
            print(f"replay: {len(res)} streams, {sum(r.rounds for r in res)} rounds, "
                  f"{time.time() - t0:.0f} s on {a.procs} processes")
            continue
        w, sums, res = compute(name, a.procs)
        write(name, w, sums, res)
        print(f"{name}: {len(w.candidates)} candidates, Gamma_t {res.gamma_t}, best {res.best}, "
              f"{int((res.score > 0).sum())} with a positive score, {time.time() - t0:.0f} s "
              f"on {a.procs} processes")


if __name__ == "__main__":
    main()
