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
    """roofline.traffic comes from the committed ncu summary while the scorer
    source is the profiled one, and is null once that source changes."""
    import shutil

    sys.path.insert(0, ROOT)
    import bench

    got = bench._profiled_traffic(1)
    assert got is not None and got > 0
    assert bench._profiled_traffic(2) is None  # no summary for that workload
    # a copy of the tree whose scorer source differs by one byte
    (tmp_path / "profiles").mkdir()
    shutil.copy(os.path.join(ROOT, "profiles", bench.PROFILES[1]), tmp_path / "profiles")
    csrc = tmp_path / "paper_2608_19659_gb300" / "csrc"
    csrc.mkdir(parents=True)
    src = open(os.path.join(ROOT, "paper_2608_19659_gb300", "csrc", "fs_score.cu"), "rb").read()
    (csrc / "fs_score.cu").write_bytes(src)
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench._profiled_traffic(1) == got
    (csrc / "fs_score.cu").write_bytes(src + b"\n")
    assert bench._profiled_traffic(1) is None
