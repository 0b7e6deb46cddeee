"""Acquisition comparison on the replay (Section 6.2).

GPU-seconds to the common certificate (Section 4.2) under FleetSieve's scored
reveals and under fixed reveal orders, over many independent reveal orders,
summarised the way Section 6.2 reports them: the ratio-of-means advantage of
FleetSieve over a baseline, a 95% paired bootstrap interval for it, and the
share of orders on which FleetSieve uses fewer GPU-seconds; overall and per
class (the GPU-seconds spent on each class's cells).

Baselines, all started from the same initial design (the first r0 cells of
each stream's permutation) and stopped by the same certificate:
  uniform random  the stream's random permutation;
  fixed grid      the grid in cell-id order (class, then TP degree, then load
                  bin) after the initial design.

Every replay runs on the GPU through :func:`fleetsieve.fs_replay`; this module
only arranges reveal orders and summarises the results (host-side statistics).
"""

from __future__ import annotations

import dataclasses

import numpy as np

from . import fleetsieve as fsb

SECONDS_PER_CELL = 300.0  # Section 5: each measurement takes 300 s on TP GPUs


def grid_order(perm: np.ndarray, r0: int) -> np.ndarray:
    """Per stream: the first r0 cells of perm, then every other cell by ascending id."""
    perm = np.asarray(perm, np.int32)
    out = np.empty_like(perm)
    for k in range(perm.shape[0]):
        head = perm[k, :r0]
        rest = np.setdiff1d(np.arange(perm.shape[1], dtype=np.int32), head, assume_unique=True)
        out[k, :r0] = head
        out[k, r0:] = rest
    return out


def class_gpu_seconds(reveal_order: np.ndarray, K: int, B: int) -> np.ndarray:
    """[streams, K]: GPU-seconds spent on each class's cells (300 s x TP per cell;
    reveal_order is -1 padded)."""
    ro = np.asarray(reveal_order)
    out = np.zeros((ro.shape[0], K), np.float64)
    valid = ro >= 0
    c = np.where(valid, ro, 0)
    cls = c // (4 * B)
    tp = 1 << ((c // B) % 4)
    sec = np.where(valid, SECONDS_PER_CELL * tp, 0.0)
    for i in range(K):
        out[:, i] = (sec * (cls == i)).sum(axis=1)
    return out


def ratio_of_means_advantage(ours: np.ndarray, base: np.ndarray) -> float:
    """1 - mean(ours) / mean(base): the share of the baseline's mean GPU-seconds saved."""
    return float(1.0 - np.mean(ours) / np.mean(base))


def paired_bootstrap_ci(ours: np.ndarray, base: np.ndarray, n_boot: int = 10000, level: float = 0.95,
                        seed: int = 0) -> tuple[float, float]:
    """Percentile interval of the ratio-of-means advantage over n_boot resamples
    of the streams (with replacement; a stream keeps its pair of values)."""
    ours = np.asarray(ours, np.float64)
    base = np.asarray(base, np.float64)
    n = ours.size
    rng = np.random.default_rng(seed)
    idx = rng.integers(0, n, size=(n_boot, n))
    stat = 1.0 - ours[idx].mean(axis=1) / base[idx].mean(axis=1)
    a = (1.0 - level) / 2.0
    lo, hi = np.quantile(stat, [a, 1.0 - a])
    return float(lo), float(hi)


@dataclasses.dataclass
class PolicyRun:
    name: str
    gpu_seconds: np.ndarray      # [streams]
    class_seconds: np.ndarray    # [streams, K]
    state: np.ndarray            # [streams] certificate state at the stop
    rounds: np.ndarray           # [streams]


def summarise(ours: PolicyRun, base: PolicyRun, n_boot: int = 10000, seed: int = 0) -> dict:
    """Section 6.2's statistics of ours against one baseline, overall and per class."""
    out = {"baseline": base.name, "mean_gpu_seconds": float(ours.gpu_seconds.mean()),
           "baseline_mean_gpu_seconds": float(base.gpu_seconds.mean()),
           "advantage": ratio_of_means_advantage(ours.gpu_seconds, base.gpu_seconds),
           "ci95": paired_bootstrap_ci(ours.gpu_seconds, base.gpu_seconds, n_boot, 0.95, seed),
           "fewer_share": float(np.mean(ours.gpu_seconds < base.gpu_seconds)), "per_class": []}
    for i in range(ours.class_seconds.shape[1]):
        a, b = ours.class_seconds[:, i], base.class_seconds[:, i]
        if b.mean() > 0:
            out["per_class"].append({"class": i, "advantage": ratio_of_means_advantage(a, b),
                                     "ci95": paired_bootstrap_ci(a, b, n_boot, 0.95, seed + 1 + i),
                                     "fewer_share": float(np.mean(a < b))})
    return out


def run_policies(model, rp, O: int, S: int, seed: int, max_rounds: int | None = None) -> dict[str, PolicyRun]:
    """FleetSieve, uniform random and fixed grid order on every stream of the
    replay ``rp`` (a :class:`workloads.Replay`), each as one batched fs_replay."""
    w = rp.base
    mr = rp.max_rounds if max_rounds is None else max_rounds
    orders = {"fleetsieve": (rp.perm, 0), "uniform_random": (rp.perm, 1),
              "fixed_grid": (grid_order(rp.perm, rp.r0), 1)}
    runs = {}
    for name, (perm, policy) in orders.items():
        r = fsb.fs_replay(model, rp.truth_cap, rp.truth_tail, perm, rp.r0, rp.eps, O, S, seed, mr, policy=policy)
        runs[name] = PolicyRun(name, r.gpu_seconds.copy(), class_gpu_seconds(r.reveal_order, w.K, w.B),
                               r.state.copy(), r.rounds.copy())
    return runs


def main(argv=None) -> None:
    """The Section 6.2 comparison on the replay workload: 200 reveal orders over
    the paper-scale grid by default; one JSON line per baseline."""
    import argparse
    import json

    import torch

    from . import workloads

    ap = argparse.ArgumentParser(description=main.__doc__)
    ap.add_argument("--streams", type=int, default=200)
    ap.add_argument("--samples", type=int, default=4096)
    ap.add_argument("--outcomes", type=int, default=8)
    ap.add_argument("--seed", type=int, default=2026)
    ap.add_argument("--boot", type=int, default=10000)
    a = ap.parse_args(argv)
    if not torch.cuda.is_available():
        raise SystemExit("the comparison runs the replay on a CUDA device")
    rp = workloads.make_replay(n_streams=a.streams, S=a.samples, O=a.outcomes)
    w = rp.base
    with fsb.fs_load_model(w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi, w.slo, w.demand, w.G, w.K, w.B) as m:
        runs = run_policies(m, rp, a.outcomes, a.samples, a.seed)
    for name in ("uniform_random", "fixed_grid"):
        line = summarise(runs["fleetsieve"], runs[name], a.boot, a.seed)
        line.update({"streams": a.streams, "samples": a.samples, "outcomes": a.outcomes,
                     "certified_share": {k: float(np.mean(r.state == 1)) for k, r in runs.items()}})
        print(json.dumps(line))


if __name__ == "__main__":
    main()
