"""Host logic of bench.py: rank aggregation over gloo (world size 2) and the reference arm."""

import json
import os
import socket
import subprocess
import sys

import pytest

from conftest import ROOT


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


CHILD = r"""
import os, sys
sys.path.insert(0, {root!r})
import bench
dist, rank, world, local = bench.dist_setup(2)
assert world == 2 and dist is not None
mx = bench.max_over_ranks(dist, 10.0 * (rank + 1))
sm = bench.sum_over_ranks(dist, float(rank + 1))
print(f"rank={{rank}} max={{mx}} sum={{sm}}")
dist.destroy_process_group()
"""


def test_rank_aggregation_gloo_world2():
    port = _free_port()
    procs = []
    for rank in range(2):
        env = dict(os.environ, RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE="2",
                   MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), FS_BENCH_BACKEND="gloo")
        procs.append(subprocess.Popen([sys.executable, "-c", CHILD.format(root=ROOT)], env=env,
                                      stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True))
    outs = []
    for p in procs:
        out, err = p.communicate(timeout=120)
        assert p.returncode == 0, err
        outs.append(out.strip())
    for o in outs:
        assert "max=20.0" in o and "sum=3.0" in o


def test_reference_arm_prints_one_json_line():
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "2",
                        "--warmup", "3", "--workload", "0"], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0 and d["unit"] == "allocation-solves/s"
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] == 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["steps"] == 2


def test_reference_arm_non_zero_ranks_exit_quietly():
    port = _free_port()
    procs = []
    for rank in range(2):
        env = dict(os.environ, RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE="2",
                   MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), FS_BENCH_BACKEND="gloo")
        procs.append(subprocess.Popen([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                                       "--steps", "1", "--warmup", "3", "--workload", "0", "--gpus", "2"],
                                      env=env, stdout=subprocess.PIPE, stderr=subprocess.PIPE, text=True))
    outs = [p.communicate(timeout=300) for p in procs]
    assert all(p.returncode == 0 for p in procs), [o[1] for o in outs]
    assert len([ln for ln in outs[0][0].splitlines() if ln.strip()]) == 1
    assert outs[1][0].strip() == ""


def test_roofline_traffic_only_for_the_profiled_source(tmp_path, monkeypatch):
    """roofline.traffic comes from an ncu summary of the bench's workload while
    the scorer source has the sha256 the summary records, and is null otherwise."""
    import hashlib
    import re

    sys.path.insert(0, ROOT)
    import bench

    # the committed summaries carry a source hash and a parsable DRAM line
    for name in bench.PROFILES.values():
        text = open(os.path.join(ROOT, "profiles", name)).read()
        assert re.search(r"sha256 prefix `[0-9a-f]{16}`", text)
        assert re.search(r"dram__bytes_read\.sum \+ dram__bytes_write\.sum \| [0-9,]+ B \+ [0-9,]+ B", text)
    # a tree whose summary matches its scorer source, then a changed source
    (tmp_path / "profiles").mkdir()
    csrc = tmp_path / "paper_2608_19659_gb300" / "csrc"
    csrc.mkdir(parents=True)
    src = b"// scorer source\n"
    (csrc / "fs_score.cu").write_bytes(src)
    h = hashlib.sha256(src).hexdigest()[:16]
    (tmp_path / "profiles" / bench.PROFILES[1]).write_text(
        f"Source: fs_score.cu, sha256 prefix `{h}`.\n"
        "| dram__bytes_read.sum + dram__bytes_write.sum | 1,237,760 B + 512 B per launch |\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench._profiled_traffic(1) == 1237760.0 + 512.0
    assert bench._profiled_traffic(2) is None  # no summary for that workload
    (csrc / "fs_score.cu").write_bytes(src + b"\n")
    assert bench._profiled_traffic(1) is None


def _passes_and_wall(r):
    reps = int(r["sample"].split(", x ")[1].split()[0])
    wall = float(r["sample"].rsplit("(", 1)[1].split(" s")[0])
    return reps, wall


def test_all_cores_oracle_baseline_counts_every_scenario():
    """The all-cores CPU baseline: one spawned oracle process per usable core
    over contiguous candidate ranges; its rate counts every scenario of every
    pass once. Whole candidates when they fit the time target; else one
    candidate per process with the same prefix of samples per outcome."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2608_19659_gb300 import workloads

    w = workloads.make_workload(0)
    k = min(len(os.sched_getaffinity(0)), len(w.candidates))
    r = bench.cpu_baseline_all_cores(0, w, seconds_per_scenario=1e-6, seconds_target=0.2)
    assert "unavailable" not in r, r
    assert r["cores"] == k and r["kind"] == "oracle" and r["value"] > 0
    reps, wall = _passes_and_wall(r)
    assert reps >= 1 and wall > 0
    assert abs(r["value"] - 2 * len(w.candidates) * w.O * w.S * reps / wall) <= 0.06 * r["value"]
    # a prefix of 16 samples per outcome: one candidate per process
    r = bench.cpu_baseline_all_cores(0, w, seconds_per_scenario=0.2 / (w.O * 16), seconds_target=0.2)
    reps, wall = _passes_and_wall(r)
    assert "samples 0..15 of 256" in r["sample"] and reps == 1
    assert abs(r["value"] - 2 * k * w.O * 16 / wall) <= 0.06 * r["value"]


def test_oracle_prefix_is_a_prefix_of_the_workload():
    """The single-core sample: whole candidates when they fit, else the first
    candidate with samples 0 .. S' - 1 of every outcome."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2608_19659_gb300 import workloads

    n, s = bench.oracle_prefix(workloads.make_workload(0), 0.5)
    assert s == 256 and 1 <= n <= 16
    w3 = workloads.make_workload(3)
    n, s = bench.oracle_prefix(w3, 0.2)
    assert n == 1 and 1 <= s < w3.S


def test_algorithmic_counts_of_the_scorer_paths():
    """The roofline's algorithmic thread-operations: 14 per scenario, 3 per tail-gate
    test and 7.5 per t* evaluated in a table build on the table path (at most two per entry, W entries
    per segment; 15 per fully evaluated entry), 32 per scenario on
    the plain path; the path rule mirrors the scorer's (3 (W + 1) at most twice
    the smaller of S and 2048)."""
    sys.path.insert(0, ROOT)
    import bench
    from paper_2608_19659_gb300 import workloads

    w1, w3, w0 = workloads.make_workload(1), workloads.make_workload(3), workloads.make_workload(0)
    assert bench.table_path(w1.O, w1.S) and bench.table_path(w3.O, w3.S) and not bench.table_path(w0.O, w0.S)
    assert abs(bench.algorithmic_ops(w1) / w1.scenarios - (17 + 15 * 512 / 4096)) < 1e-12
    assert abs(bench.algorithmic_ops(w3) / w3.scenarios - (17 + 15 * 256 / 16384)) < 1e-12
    # with the library's counts: 14 per scenario, 3 per gate test, 7.5 per t* evaluated
    assert bench.algorithmic_ops(w3, 1000.0, 500.0) == 14.0 * w3.scenarios + 3.0 * 500.0 + 7.5 * 1000.0
    assert bench.algorithmic_ops(w0) == 32 * w0.scenarios
    # the rule's edges: W = 512 needs 769 samples (3 * 513 <= 2 * 769), W = 4096 at most
    assert bench.table_path(8, 770) and not bench.table_path(8, 769)
    assert not bench.table_path(1, 1 << 20)  # W = 4096: 3 * 4097 > 2 * 2048
