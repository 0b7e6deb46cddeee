"""Benchmark of the GB300 decision-gap scorer.

One step = one fs_score_candidates pass over the largest single-GPU scoring
workload (8 classes, TP in {1,2,4,8}, G = 256, 32 load bins; 1024 candidates x
16 outcomes x 16384 samples = 268,435,456 scenarios, each solving the
allocation under both realisations): base solves, per-candidate tables, the
Monte-Carlo kernel and the reduction. Inputs are resident in HBM when the
timed region starts; L2 is flushed (256 MiB write) between timed steps. The
paper-scale and 4-class workloads are reported beside it, and the replay
workload (Algorithm 1 over 200 reveal orders) is timed wall-clock. Prints one
JSON line.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload I] [--impl reference]

--impl reference times the CPU oracle (single-threaded C) on a bounded
sample of the same workload. Under torchrun (N > 1) every rank scores its own
independent problem (stream id = rank): weak scaling, no collective on the
data path.
"""

from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

from paper_2608_19659_gb300 import workloads  # noqa: E402

METRIC = "scenario allocation-solves/s"
UNIT = "allocation-solves/s"
ISSUE_PER_SM_CLK = 4 * 32  # 4 schedulers x 32 lanes, one warp instruction each per clock

# Algorithmic thread-operations of the Monte-Carlo kernel. Plain path, per
# scenario (the parametric re-solve):
#   a quarter of one Philox4x32-10 call (10 rounds x (2 wide multiplies +
#   2 three-input XORs), four samples per call)                          10
#   capacity position (the word's top w bits), its address, the lookup    3
#   tail gate (mask, compare) and the gated capacity                      3
#   the two patched row capacities (max with Cexcl)                       2
#   two table searches: loop test, address, read of the reached threshold 6
#   Gamma' = t*(A+') - t*(A-')                                             1
#   exact fixed-point accumulation of rint(Gamma' 2^40)                   7
# Table path (a segment's W + 1 values of rint(Gamma' 2^40) tabulated once):
# per scenario the Philox share (10), capacity position (1), the entry's load
# (1) and its 64-bit sum (two 32-bit adds: 2) = 14, plus the tail gate's test (mask,
# compare, index select: 3) in the scenarios of strata whose tails lie on both
# sides of the SLO (elsewhere the gate is the same at every position); per
# table entry with both t* evaluated the two patched capacities (2), two table
# searches (6), Gamma' (1), the fixed-point conversion (5) and the store (1) =
# 15, counted as 7.5 per t* evaluated (an entry with one t* evaluated, the
# other taken from the closed-gate value because its capacity is at or below
# that realisation's Cexcl, then counts 7.5 of its 11). A segment whose tail
# gate is closed at every position of its stratum evaluates nothing (every
# entry equals the closed-gate value, from the preparation). The library
# counts the t* evaluated and the scenarios that tested their gate. Search
# probes beyond the first (3 each) and row-term fulfilments are not counted:
# lower bounds.
OPS_PER_SCENARIO = 32
OPS_PER_SCENARIO_TABLE = 14
OPS_PER_GATE_TEST = 3
OPS_PER_TSTAR_EVAL = 7.5  # half of a fully evaluated table entry's 15
Q_TABLE = 4096  # quantile table size of the built-in triangular table


def table_path(O: int, S: int) -> bool:
    """Whether a launch of O outcomes x S samples takes the table path: the
    scorer's rule (W = Q/O entries at most 4096, and 3 (W + 1) at most twice
    the smaller of S and a minimum chunk of 2048 samples)."""
    W = Q_TABLE // O
    return W <= 4096 and 3 * (W + 1) <= 2 * min(S, 2048)


def draw_floors(w, kernel_ms: float, reps: int = 10):
    """The Monte-Carlo kernel against measured floors of its draws: the same
    number of Philox4x32-10 calls (counters as the scorer's) on the table
    path's 128-thread grid, timed alone and with the table path's per-sample
    lookup and sum (fs_draw_floor; no chunks, staging, table builds or
    barriers), scaled to the workload's calls. Table path only."""
    import math

    from paper_2608_19659_gb300 import fleetsieve as fsb

    if not table_path(w.O, w.S):
        return None
    calls = len(w.candidates) * w.O * ((w.S + 3) // 4)
    wbits = int(math.log2(Q_TABLE // w.O))
    out = {"calls_per_launch": calls, "kernel_ms": kernel_ms}
    for mode, key in ((0, "philox_only_ms"), (1, "philox_and_lookup_ms")):
        ms, done = fsb.fs_draw_floor(mode, wbits, calls, reps)
        out[key] = ms * calls / done
    out["frac_of_philox_only"] = out["philox_only_ms"] / kernel_ms
    out["frac_of_philox_and_lookup"] = out["philox_and_lookup_ms"] / kernel_ms
    out["basis"] = ("median of %d launches each (after 3 untimed) of fs_draw_floor mode 0 (draws alone) and "
                    "mode 1 (draws + position, entry load and 64-bit sum from a %d-entry shared table), "
                    "scaled from the calls one launch made to the workload's" % (reps, (Q_TABLE // w.O) + 1))
    return out


def algorithmic_ops(w, tstar_evals_per_launch=None, gated_per_launch=None) -> float:
    """Algorithmic thread-operations of one Monte-Carlo launch over workload w:
    on the table path, with the t* its gap-table builds evaluated and the
    scenarios that tested their tail gate (as the library counted them; None:
    both t* of W entries and a gate test in every segment)."""
    if table_path(w.O, w.S):
        W = Q_TABLE // w.O
        if tstar_evals_per_launch is None:
            tstar_evals_per_launch = 2.0 * len(w.candidates) * w.O * W
        if gated_per_launch is None:
            gated_per_launch = float(w.scenarios)
        return (float(OPS_PER_SCENARIO_TABLE) * w.scenarios + OPS_PER_GATE_TEST * float(gated_per_launch)
                + OPS_PER_TSTAR_EVAL * float(tstar_evals_per_launch))
    return float(OPS_PER_SCENARIO) * w.scenarios

# ncu summaries with the DRAM bytes of one k_score launch, per workload; used
# for roofline.traffic only while the scorer source is the one profiled.
PROFILES = {1: "k_score_paper_scale.md", 3: "k_score_large.md"}  # sha-checked below


def _env_int(name, default):
    try:
        return int(os.environ.get(name, default))
    except ValueError:
        return default


def _profile_text(workload: int):
    """The committed ncu summary of this workload's k_score launch, or None
    when there is none or the scorer source changed since it was taken (its
    sha256 prefix is recorded in the summary)."""
    import hashlib
    import re

    name = PROFILES.get(workload)
    if not name:
        return None
    try:
        text = open(os.path.join(ROOT, "profiles", name)).read()
        src = open(os.path.join(ROOT, "paper_2608_19659_gb300", "csrc", "fs_score.cu"), "rb").read()
    except OSError:
        return None
    m = re.search(r"sha256 prefix `([0-9a-f]+)`", text)
    if not m or not hashlib.sha256(src).hexdigest().startswith(m.group(1)):
        return None
    return text


def _profiled_traffic(workload: int):
    """DRAM bytes (read + write) of one k_score launch from the committed ncu summary."""
    import re

    text = _profile_text(workload)
    m = re.search(r"dram__bytes_read\.sum \+ dram__bytes_write\.sum \| ([0-9,]+) B \+ ([0-9,]+) B", text or "")
    if not m:
        return None
    return float(m.group(1).replace(",", "")) + float(m.group(2).replace(",", ""))


def _profiled_pipes(workload: int):
    """The busiest execution units of one k_score launch from the committed ncu
    summary (fractions of their peak): the integer multiplier (fmaheavy pipe,
    the unit Philox4x32-10's 32x32->64 products run on), the ALU pipe and the
    issue slots. None when the summary is missing or stale."""
    import re

    text = _profile_text(workload)
    if not text:
        return None
    out = {}
    m = re.search(r"sm__pipe_fmaheavy_cycles_active \(of peak, elapsed\) \| ([0-9.]+) %", text)
    if m:
        out["fmaheavy_busy"] = float(m.group(1)) / 100.0
    m = re.search(r"sm__inst_executed_pipe_alu / _fma / _lsu \(of peak, active\) \| ([0-9.]+) %", text)
    if m:
        out["alu_busy"] = float(m.group(1)) / 100.0
    m = re.search(r"smsp__issue_active \(of peak, active\) \| ([0-9.]+) %", text)
    if m:
        out["issue_active"] = float(m.group(1)) / 100.0
    if not out:
        return None
    out["source"] = f"ncu, profiles/{PROFILES[workload]}"
    busiest = max(("integer multiplier (fmaheavy)", out.get("fmaheavy_busy", 0.0)),
                  ("ALU", out.get("alu_busy", 0.0)), ("issue", out.get("issue_active", 0.0)), key=lambda x: x[1])
    out["binding"] = busiest[0] if busiest[1] >= 0.5 else "latency (no unit half busy)"
    return out


def _measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f)
    except OSError:
        return {}


class ClockSampler:
    """nvidia-smi clock / throttle samples during the timed region."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = str(gpu_index)
        try:  # name the GPU by UUID: CUDA and nvidia-smi may number devices differently
            import torch

            u = str(torch.cuda.get_device_properties(gpu_index).uuid)
            self.gpu = u if u.startswith("GPU-") else "GPU-" + u
        except Exception:
            pass
        self.proc = None
        self.path = None

    def __enter__(self):
        fd, self.path = tempfile.mkstemp(prefix="fs_clocks_", suffix=".csv")
        os.close(fd)
        try:
            self.out = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.out, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *a):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
        self.out.close()

    def summary(self):
        try:
            lines = [ln.split(",") for ln in open(self.path).read().strip().splitlines() if ln.strip()]
            os.unlink(self.path)
        except OSError:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for f in lines:
            f = [x.strip() for x in f]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def dist_setup(n_gpus: int):
    world = _env_int("WORLD_SIZE", 1)
    rank = _env_int("RANK", 0)
    local = _env_int("LOCAL_RANK", 0)
    if world > 1:
        import torch.distributed as dist

        backend = "nccl" if os.environ.get("FS_BENCH_BACKEND", "nccl") == "nccl" else "gloo"
        dist.init_process_group(backend=backend)
        return dist, rank, world, local
    return None, 0, 1, 0


def max_over_ranks(dist, value: float, device=None) -> float:
    if dist is None:
        return value
    import torch

    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(dist, value: float, device=None) -> float:
    if dist is None:
        return value
    import torch

    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


def config_of(w, extra=None):
    c = {"workload": w.name, "classes": w.K, "load_bins": w.B, "gpu_budget": w.G,
         "candidates": int(len(w.candidates)), "outcomes": w.O, "samples": w.S,
         "scenarios_per_step": w.scenarios, "solves_per_scenario": 2,
         "l2": "flushed between timed steps (256 MiB write)"}
    if extra:
        c.update(extra)
    return c


def other_workload(idx: int, steps: int, warmup: int, alu_peak: float, stream_id: int = 0,
                   demand_factor: float = 1.0):
    """The same device-resident measurement on another synthetic workload (the
    mid and large ones): step time with the L2 flushed between steps, the
    Monte-Carlo kernel's own duration, and its roofline fraction. demand_factor
    scales the demands (the mid workload at its nominal demands has spare
    capacity, so its gap is 0; at three times them it is not)."""
    import dataclasses

    import torch

    from paper_2608_19659_gb300 import fleetsieve as fsb

    w = workloads.make_workload(idx)
    if demand_factor != 1.0:
        w = dataclasses.replace(w, name=f"{w.name}, demands x{demand_factor:g}",
                                demand=(w.demand * np.float32(demand_factor)).astype(np.float32))
    stream = torch.cuda.current_stream()
    m = fsb.fs_load_model(w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi, w.slo, w.demand, w.G, w.K, w.B,
                          stream=stream)
    n = len(w.candidates)
    cand = torch.from_numpy(w.candidates).cuda()
    gap = torch.zeros(n, dtype=torch.float64, device="cuda")
    score = torch.zeros(n, dtype=torch.float64, device="cuda")
    gt = torch.zeros(1, dtype=torch.float32, device="cuda")
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device="cuda")

    def step():
        fsb.fs_score_candidates_async(m, cand, w.O, w.S, w.seed, stream_id, 0, gap_dev=gap, score_dev=score,
                                      gamma_t_dev=gt, stream=stream)

    for _ in range(warmup):
        flush.zero_()
        step()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for a, b in ev:
        flush.zero_()
        a.record(stream)
        step()
        b.record(stream)
    torch.cuda.synchronize()
    step_ms = statistics.median(a.elapsed_time(b) for a, b in ev)
    fsb.fs_timing_read(m)
    fsb.fs_timing_enable(m, 1)
    for _ in range(steps):
        flush.zero_()
        step()
    torch.cuda.synchronize()
    kernel_ms, kernel_n, _, (evals, gated) = fsb.fs_timing_read(m, with_entries=True)
    fsb.fs_timing_enable(m, 0)
    fsb.fs_check(m, stream)
    fsb.fs_free_model(m)
    kern_s = kernel_ms / 1000.0 / max(kernel_n, 1)
    achieved = algorithmic_ops(w, evals / max(kernel_n, 1), gated / max(kernel_n, 1)) / kern_s
    gamma_t = float(gt.item())
    return {"workload": w.name, "ms_per_step": step_ms, "scenarios_per_s": w.scenarios / (step_ms / 1000.0),
            "gamma_t": gamma_t,
            "note": ("Gamma_t = 0 at these demands (spare capacity): every score is exactly 0, and the "
                     "Monte-Carlo kernel's tables are empty" if gamma_t == 0.0 else ""),
            "allocation_solves_per_s": 2.0 * w.scenarios / (step_ms / 1000.0),
            "candidate_scores_per_s": n / (step_ms / 1000.0),
            "kernel_ms_per_launch": kern_s * 1000.0,
            "roofline": {"bound": "alu", "achieved": achieved / 1e12, "peak": alu_peak / 1e12,
                         "unit": "Tops/s (32-bit thread operations)", "frac": achieved / alu_peak,
                         "traffic": _profiled_traffic(idx), "pipes": _profiled_pipes(idx)}}


def oracle_prefix(w, seconds_target: float):
    """A deterministic prefix of workload w's scenarios sized to about
    seconds_target of one core: the first n candidates, every outcome, and
    samples 0 .. S' - 1 of each (a subset of the workload's own scenarios;
    S' = S once whole candidates fit). Returns (n, S')."""
    import oracle

    qn = oracle.triangular_table(4096)
    s1 = min(w.S, 32)
    t0 = time.perf_counter()
    oracle.score(w, qn, candidates=w.candidates[:1], S=s1)
    per_scen = (time.perf_counter() - t0) / (w.O * s1)
    s_fit = int(seconds_target / max(per_scen * w.O, 1e-9))
    if s_fit < w.S:
        return 1, max(1, s_fit)
    n = int(max(1, min(len(w.candidates), seconds_target / max(per_scen * w.O * w.S, 1e-9))))
    return n, w.S


def _sample_text(w, n, s_pref):
    if s_pref == w.S:
        return f"first {n} of {len(w.candidates)} candidates, all {w.O}x{w.S} scenarios each"
    return (f"first {n} of {len(w.candidates)} candidates, all {w.O} outcomes, samples 0..{s_pref - 1} of "
            f"{w.S} per outcome (a prefix of the workload's scenarios; the rate extrapolates to the "
            f"whole workload, which the oracle would take {len(w.candidates) * w.S / (n * s_pref):.0f}x as long for)")


def cpu_baseline(w, seconds_target: float = 15.0):
    """The oracle, single-threaded, on a deterministic prefix of the workload."""
    import oracle

    qn = oracle.triangular_table(4096)
    n, s_pref = oracle_prefix(w, seconds_target)
    t0 = time.perf_counter()
    oracle.score(w, qn, candidates=w.candidates[:n], S=s_pref)
    dt = time.perf_counter() - t0
    scen = n * w.O * s_pref
    return {"value": 2 * scen / dt, "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"{_sample_text(w, n, s_pref)} ({scen} scenarios, {dt:.1f} s)",
            "candidate_scores_per_s": scen / dt / (w.O * w.S), "prefix": [n, s_pref]}


def _oracle_worker(widx, lo, hi, s_pref, reps, barrier, out):
    """One oracle instance on candidates [lo, hi) of workload widx (samples
    0 .. s_pref - 1 of every outcome), `reps` passes, timed from a barrier
    shared with the other instances."""
    import oracle

    w = workloads.make_workload(widx)
    qn = oracle.triangular_table(4096)
    oracle.score(w, qn, candidates=w.candidates[lo:lo + 1], S=1)  # the library is loaded before the start
    barrier.wait(timeout=600)
    t0 = time.monotonic()
    for _ in range(reps):
        oracle.score(w, qn, candidates=w.candidates[lo:hi], S=s_pref)
    out.put((t0, time.monotonic()))


def cpu_baseline_all_cores(widx: int, w, seconds_per_scenario: float, seconds_target: float = 10.0):
    """Independent oracle instances, one process per core this process may use,
    over contiguous candidate ranges of the same workload: the harness's
    parallelism (the oracle itself stays single-threaded). Each instance takes
    the same prefix of samples per outcome as the single-core run, sized so
    that the run lasts about seconds_target. Processes are spawned, not forked
    (the CUDA context exists by now)."""
    import multiprocessing as mp
    import queue

    n_all = len(w.candidates)
    k = max(1, min(len(os.sched_getaffinity(0)), n_all))
    s_fit = int(seconds_target / max(seconds_per_scenario * w.O, 1e-9))
    if s_fit < w.S:  # one candidate per process, a prefix of its samples
        s_pref, n = max(1, s_fit), k
        reps = 1
    else:
        s_pref, n = w.S, n_all
        per = (n + k - 1) // k
        reps = max(1, int(round(seconds_target / max(seconds_per_scenario * per * w.O * w.S, 1e-9))))
    bounds = [(i * n // k, (i + 1) * n // k) for i in range(k)]
    ctx = mp.get_context("spawn")
    barrier, out = ctx.Barrier(k), ctx.Queue()
    procs = [ctx.Process(target=_oracle_worker, args=(widx, lo, hi, s_pref, reps, barrier, out), daemon=True)
             for lo, hi in bounds]
    for p in procs:
        p.start()
    try:
        spans = [out.get(timeout=900) for _ in procs]
    except queue.Empty:
        return {"unavailable": "an oracle process did not report within 900 s"}
    finally:
        for p in procs:
            p.join(timeout=60)
    wall = max(e for _, e in spans) - min(b for b, _ in spans)
    scen = n * w.O * s_pref * reps
    return {"value": 2 * scen / wall, "unit": UNIT, "cores": k, "kind": "oracle",
            "sample": f"{_sample_text(w, n, s_pref)}, x {reps} passes, {k} processes over contiguous "
                      f"candidate ranges ({wall:.4g} s)",
            "candidate_scores_per_s": scen / wall / (w.O * w.S)}


def mode_entries(stream, steps: int, warmup: int, alu_peak: float):
    """The paper-scale workload under the other modes of the method, each
    device-resident with the L2 flushed between steps: the monotone
    structural prior (Section 4.1's interval refit in every scenario; the
    table path keeps 2W entries a segment), and the goodput stage of the
    score (every scenario solved to tier 4 of the lexicographic objective in
    both realisations; fs_score_goodput is synchronous, so its time is the
    call's wall clock), the latter also on the large workload."""
    import torch

    from paper_2608_19659_gb300 import fleetsieve as fsb

    w = workloads.make_workload(1)
    n = len(w.candidates)
    out = []
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device="cuda")
    # monotone prior, asynchronous scoring as in the headline step
    m = fsb.fs_load_model(w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi, w.slo, w.demand, w.G, w.K, w.B,
                          stream=stream)
    fsb.fs_set_prior(m, fsb.FS_PRIOR_MONOTONE)
    cand = torch.from_numpy(w.candidates).cuda()
    gap = torch.zeros(n, dtype=torch.float64, device="cuda")
    score = torch.zeros(n, dtype=torch.float64, device="cuda")

    def step():
        fsb.fs_score_candidates_async(m, cand, w.O, w.S, w.seed, 0, 0, gap_dev=gap, score_dev=score, stream=stream)

    for _ in range(warmup):
        flush.zero_()
        step()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for a, b in ev:
        flush.zero_()
        a.record(stream)
        step()
        b.record(stream)
    torch.cuda.synchronize()
    fsb.fs_check(m, stream)
    ms = statistics.median(a.elapsed_time(b) for a, b in ev)
    fsb.fs_free_model(m)
    out.append({"mode": "monotone structural prior (row refit per scenario)", "workload": w.name,
                "ms_per_step": ms, "allocation_solves_per_s": 2.0 * w.scenarios / (ms / 1000.0),
                "candidate_scores_per_s": n / (ms / 1000.0)})
    # goodput stage (tiers 1-4 per realisation), synchronous host API, on the
    # paper-scale workload and on the large one
    for wg in (w, workloads.make_workload(3)):
        m = fsb.fs_load_model(wg.cap_lo, wg.cap_hi, wg.tail_lo, wg.tail_hi, wg.slo, wg.demand, wg.G, wg.K, wg.B,
                              stream=stream)
        for _ in range(warmup):
            fsb.fs_score_goodput(m, wg.candidates, wg.O, wg.S, wg.seed)
        walls = []
        for _ in range(max(3, min(steps, 10))):
            flush.zero_()
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            r = fsb.fs_score_goodput(m, wg.candidates, wg.O, wg.S, wg.seed)
            walls.append(time.perf_counter() - t0)
        fsb.fs_free_model(m)
        wall = statistics.median(walls)
        ng = len(wg.candidates)
        out.append({"mode": "goodput stage (both realisations of every scenario to tier 4), host API wall clock",
                    "workload": wg.name, "ms_per_step": wall * 1000.0,
                    "allocation_solves_per_s": 2.0 * wg.scenarios / wall, "candidate_scores_per_s": ng / wall,
                    "gamma_gp": r.gamma_gp})
    return out


def replay_entry(stream, alu_peak):
    """The replay workload: Algorithm 1 on 200 independent reveal orders of the
    paper-scale grid, each round scoring every unrevealed candidate with 8 x
    4096 samples, until the certificate fires: fs_replay batches all streams'
    rounds into one launch sequence per round. Wall-clock per whole replay (a
    synchronous call, timed on the host after a synchronize), and the oracle
    on the first rounds of stream 0."""
    import torch

    import oracle
    from paper_2608_19659_gb300 import fleetsieve as fsb

    rp = workloads.make_replay()
    w = rp.base
    seed = 2026
    m = fsb.fs_load_model(w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi, w.slo, w.demand, w.G, w.K, w.B,
                          stream=stream)
    res = fsb.fs_replay(m, rp.truth_cap, rp.truth_tail, rp.perm, rp.r0, rp.eps, w.O, w.S, seed, rp.max_rounds)
    walls = []
    for _ in range(3):
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        res = fsb.fs_replay(m, rp.truth_cap, rp.truth_tail, rp.perm, rp.r0, rp.eps, w.O, w.S, seed,
                            rp.max_rounds)
        walls.append(time.perf_counter() - t0)
    fsb.fs_free_model(m)
    wall = statistics.median(walls)
    cells = w.cells
    # scenarios scored: stream k's round r scores its cells - r0 - r unrevealed candidates
    cand_rounds = sum(sum(cells - rp.r0 - r for r in range(int(res.rounds[k]))) for k in range(len(res.rounds)))
    scen = cand_rounds * w.O * w.S
    # the oracle: the first two rounds of stream 0 (same seed, same samples)
    qn = oracle.triangular_table(4096)
    t0 = time.perf_counter()
    oracle.replay_stream(rp, 0, qn, seed=seed, S=w.S, max_rounds=2)
    odt = time.perf_counter() - t0
    o_scen = sum(cells - rp.r0 - r for r in range(2)) * w.O * w.S
    return {"workload": f"replay: 200 reveal orders of the paper-scale grid, unrevealed candidates x "
                        f"{w.O} x {w.S} per round, eps {rp.eps}, seeds 100-299",
            "wall_s_per_replay": wall, "wall_s_runs": walls,
            "streams_per_s": len(res.rounds) / wall, "rounds_total": int(res.rounds.sum()),
            "certified": int((res.state == 1).sum()), "candidate_scores": int(cand_rounds),
            "scenarios": int(scen), "allocation_solves_per_s": 2.0 * scen / wall,
            "candidate_scores_per_s": cand_rounds / wall,
            "roofline": {"bound": "alu", "achieved": OPS_PER_SCENARIO_TABLE * scen / wall / 1e12,
                         "peak": alu_peak / 1e12, "unit": "Tops/s (32-bit thread operations)",
                         "frac": OPS_PER_SCENARIO_TABLE * scen / wall / alu_peak,
                         "basis": "14 thread-operations per scenario (the table path's per-scenario count; "
                                  "table builds, gate tests and every other phase of the round loop not "
                                  "counted: a lower bound) over the whole replay's wall clock"},
            "cpu_baseline": {"value": 2.0 * o_scen / odt, "unit": UNIT, "cores": 1, "kind": "oracle",
                             "sample": f"stream 0, rounds 0-1 ({o_scen} scenarios, {odt:.1f} s)"}}


def run_reference(args, w, rank):
    if rank != 0:
        return 0
    import oracle

    qn = oracle.triangular_table(4096)
    # a bounded sample per step: a prefix of the workload's scenarios for about 0.5 s of CPU work
    n, s_pref = oracle_prefix(w, 0.5)
    for _ in range(args.warmup):
        oracle.score(w, qn, candidates=w.candidates[:n], S=s_pref)
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        oracle.score(w, qn, candidates=w.candidates[:n], S=s_pref)
        times.append(time.perf_counter() - t0)
    total = sum(times)
    scen = n * w.O * s_pref
    value = 2 * scen * args.steps / total
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * total / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
            "data": "synthetic", "config": config_of(w, {"reference_sample": [n, s_pref]}),
            "candidate_scores_per_s": scen * args.steps / total / (w.O * w.S),
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle",
                             "sample": f"{_sample_text(w, n, s_pref)}, per step"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def step_ms_of(starts, ends):
    return [a.elapsed_time(b) for a, b in zip(starts, ends)]


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--workload", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-all-cores", action="store_true", help="skip the all-cores oracle run")
    ap.add_argument("--no-other-workloads", action="store_true")
    ap.add_argument("--no-replay", action="store_true", help="skip the replay workload")
    ap.add_argument("--kernel-pass-s", type=float, default=1.0,
                    help="least duration of the kernel-timing pass (0: --steps steps)")
    ap.add_argument("--no-e2e", action="store_true", help="skip the end-to-end pass (profiling runs)")
    ap.add_argument("--no-floors", action="store_true", help="skip the draw-floor measurement (profiling runs)")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        args.warmup = 3

    dist, rank, world, local = dist_setup(args.gpus)
    w = workloads.make_workload(args.workload)
    if args.impl == "reference":
        rc = run_reference(args, w, rank)
        if dist is not None:
            dist.destroy_process_group()
        return rc

    import torch

    from paper_2608_19659_gb300 import fleetsieve as fsb

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    fsb.lib()
    stream = torch.cuda.current_stream()
    n = len(w.candidates)
    model = fsb.fs_load_model(w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi, w.slo, w.demand, w.G, w.K, w.B,
                              stream=stream)
    cand = torch.from_numpy(w.candidates).to(dev)
    gap = torch.zeros(n, dtype=torch.float64, device=dev)
    score = torch.zeros(n, dtype=torch.float64, device=dev)
    gt = torch.zeros(1, dtype=torch.float32, device=dev)
    best = torch.zeros(1, dtype=torch.int32, device=dev)
    flush = torch.empty(64 * 1024 * 1024, dtype=torch.float32, device=dev)  # 256 MiB > 129 MB L2
    stream_id = rank

    def step():
        fsb.fs_score_candidates_async(model, cand, w.O, w.S, w.seed, stream_id, 0, gap_dev=gap,
                                      score_dev=score, gamma_t_dev=gt, best_dev=best, stream=stream)

    for _ in range(args.warmup):
        flush.zero_()
        step()
    fsb.fs_check(model, stream)
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    fsb.fs_timing_enable(model, 0)
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    launches0 = fsb.fs_launch_count()
    with ClockSampler(local) as clocks:
        # pass 1, the measured steps: no events inside a step, so each kernel can
        # start while its predecessor drains (programmatic dependent launch)
        for k in range(args.steps):
            flush.zero_()
            starts[k].record(stream)
            step()
            ends[k].record(stream)
        torch.cuda.synchronize()
        launches = fsb.fs_launch_count() - launches0
        if dist is not None:
            dist.barrier()
        fsb.fs_check(model, stream)
        # pass 2, the same steps with events around the Monte-Carlo kernel on its
        # stream, for the kernel's own duration (the roofline)
        # (at least about a second of them, so that the clock samples taken
        # every 200 ms see the GPU under this load)
        fsb.fs_timing_read(model)
        fsb.fs_timing_enable(model, 1)  # (also zeroes the library's work counts)
        per_step_s = max(sum(step_ms_of(starts, ends)) / 1000.0 / args.steps, 1e-6)
        n2 = max(args.steps, min(4000, int(args.kernel_pass_s / per_step_s)))
        for k in range(n2):
            flush.zero_()
            step()
            if (k + 1) % 1000 == 0:  # the library keeps up to 4096 timed calls
                torch.cuda.synchronize()
        torch.cuda.synchronize()
        kernel_ms, kernel_n, _, (evals, gated) = fsb.fs_timing_read(model, with_entries=True)
        fsb.fs_timing_enable(model, 0)
    step_ms = step_ms_of(starts, ends)
    total_ms = max_over_ranks(dist, sum(step_ms), dev)
    scen_all = sum_over_ranks(dist, float(w.scenarios) * args.steps, dev)
    value = 2.0 * scen_all / (total_ms / 1000.0)

    # end to end through the public host API: bounds in from pinned host memory,
    # scores out to host memory, every step
    pinned = {k: torch.from_numpy(getattr(w, k).reshape(-1).copy()).pin_memory().numpy()
              for k in ("cap_lo", "cap_hi", "tail_lo", "tail_hi")}
    cand_h = torch.from_numpy(w.candidates.copy()).pin_memory().numpy()
    outs = (torch.zeros(n, dtype=torch.float64).pin_memory().numpy(),
            torch.zeros(n, dtype=torch.float64).pin_memory().numpy(),
            torch.zeros(1, dtype=torch.float32).pin_memory().numpy(),
            torch.zeros(1, dtype=torch.int32).pin_memory().numpy(), None)

    def e2e_step():
        fsb.fs_update_bounds(model, pinned["cap_lo"], pinned["cap_hi"], pinned["tail_lo"], pinned["tail_hi"])
        return fsb.fs_score_candidates(model, cand_h, w.O, w.S, w.seed, stream_id, 0, outputs=outs)

    e2e_value, e2e_best = None, None
    if not args.no_e2e:
        for _ in range(args.warmup):
            e2e_step()
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            res = e2e_step()
        torch.cuda.synchronize()
        e2e_s = max_over_ranks(dist, time.perf_counter() - t0, dev)
        e2e_value = 2.0 * scen_all / e2e_s
        e2e_best = int(res.best)
    h2d = 16 * w.cells + w.cells + 4 * n
    d2h = 8 * n + 8 * n + 4 + 4

    peaks = _measured_peaks()
    clk = clocks.summary()
    sm_max = float(peaks.get("sm_max_mhz", 2070.0))
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    alu_peak = sms * ISSUE_PER_SM_CLK * sm_max * 1e6  # thread-ops/s at the maximum SM clock
    kern_s = kernel_ms / 1000.0 / max(kernel_n, 1)
    evals_per_launch = evals / max(kernel_n, 1)
    gated_per_launch = gated / max(kernel_n, 1)
    ops = algorithmic_ops(w, evals_per_launch, gated_per_launch)
    achieved = ops / kern_s if kernel_n else None
    roofline = {"bound": "alu", "kernel": "k_score (Monte-Carlo sampler + parametric re-solve)",
                "achieved": achieved / 1e12 if achieved else None,
                "peak": alu_peak / 1e12, "unit": "Tops/s (32-bit thread operations)",
                "frac": (achieved / alu_peak) if achieved else None,
                "traffic": _profiled_traffic(args.workload), "traffic_unit": "DRAM bytes per launch (ncu)",
                "algorithmic_bytes": 0, "kernel_ms_per_launch": kern_s * 1000.0,
                "ops_per_scenario": ops / w.scenarios,
                "tstar_evaluations_per_launch": evals_per_launch,
                "gate_tested_scenarios_per_launch": gated_per_launch,
                "path": "table" if table_path(w.O, w.S) else "plain",
                "peak_basis": f"{sms} SMs x 4 issue slots x 32 lanes x {sm_max:.0f} MHz (max SM clock)",
                "kernel_share_of_step": (kern_s * 1000.0 / (sum(step_ms) / len(step_ms))) if kernel_n else None,
                "pipes": _profiled_pipes(args.workload)}
    if kernel_n and not args.no_floors:
        # the binding unit's floor: the integer multiplier serves Philox's products
        roofline["draw_floors"] = draw_floors(w, kern_s * 1000.0)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w)
        if not args.no_all_cores:
            per_scen = 1.0 / (cpu["value"] / 2.0)
            cpu["all_cores"] = cpu_baseline_all_cores(args.workload, w, per_scen)
    # the other scoring workloads beside the headline (not the headline), and the replay
    others = []
    if world == 1 and not args.no_other_workloads:
        others = [other_workload(i, max(3, min(args.steps, 10)), args.warmup, alu_peak)
                  for i in (1, 2, 3) if i != args.workload]
        # the mid workload at three times its demands: a nonzero gap (its oracle
        # sums are stored in tests/golden/mid_workload_x3_sums.txt)
        others.append(other_workload(2, max(3, min(args.steps, 10)), args.warmup, alu_peak, demand_factor=3.0))
    replay = None
    if world == 1 and not args.no_replay:
        replay = replay_entry(stream, alu_peak)
    modes = None
    if world == 1 and not args.no_other_workloads:
        modes = mode_entries(stream, max(3, min(args.steps, 10)), args.warmup, alu_peak)
    line = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": total_ms / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": config_of(w, {"parallelism": f"replicas x{world} (independent problems)"}),
            "candidate_scores_per_s": len(w.candidates) * args.steps * world / (total_ms / 1000.0),
            "scenarios_per_s": scen_all / (total_ms / 1000.0),
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "api": "fs_update_bounds + fs_score_candidates (pinned host buffers; inputs and results cross through mapped page-locked memory the kernels read and write)",
                    "best": e2e_best},
            "gpu_launches": int(launches), "roofline": roofline, "clocks": clk,
            "cpu_baseline": cpu, "other_workloads": others, "replay": replay, "other_modes": modes}
    if rank == 0:
        print(json.dumps(line))
    fsb.fs_free_model(model)
    if dist is not None:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
