import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

GOLDEN = os.path.join(ROOT, "tests", "golden")


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (sm_103a) and the built library")


def read_golden(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append(line.split())
    return rows


@pytest.fixture(scope="session")
def oracle_lib():
    import oracle

    oracle.lib()
    return oracle


@pytest.fixture(scope="session")
def fsb():
    """The ctypes binding of the CUDA library (built in-tree first)."""
    from paper_2608_19659_gb300 import _build

    _build.build()
    from paper_2608_19659_gb300 import fleetsieve

    fleetsieve.lib()
    return fleetsieve


@pytest.fixture(scope="session")
def cuda():
    import torch

    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    torch.cuda.set_device(0)
    return torch


def load_model(fsb, w, quantile=None):
    m = fsb.fs_load_model(w.cap_lo, w.cap_hi, w.tail_lo, w.tail_hi, w.slo, w.demand, w.G, w.K, w.B,
                          quantile=quantile)
    if getattr(w, "floor", None) is not None:
        fsb.fs_set_floors(m, w.floor)
    if getattr(w, "prior", 0):
        fsb.fs_set_prior(m, w.prior)
    return m


def alloc_matches(gpu: dict, ref, K: int) -> bool:
    """GPU allocation dict equals an oracle Allocation field by field (bit-exact floats)."""
    import numpy as np

    return (gpu["t_star"] == ref.t_star and gpu["total_gpus"] == ref.total_gpus and gpu["ok"] == ref.ok
            and gpu["floors_met"] == ref.floors_met
            and gpu["has_option_mask"] == ref.has_option_mask and gpu["tp"] == ref.tp
            and gpu["bin"] == ref.bin and gpu["replicas"] == ref.replicas
            and [np.float32(x) for x in gpu["fulfil"]] == [np.float32(x) for x in ref.fulfil])


def read_expected_sums(name):
    """An expected-sums file written by tests/golden/make_expected_sums.py:
    (inputs_sha256, gamma_t, best, cells [n], sum_eo [n, O])."""
    import numpy as np

    sha = None
    gamma_t = best = None
    cells, deficits = [], []
    S = None
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            if line.startswith("# inputs_sha256"):
                sha = line.split()[2]
                continue
            if not line.strip() or line.startswith("#"):
                continue
            t = line.split()
            if t[0] == "gamma_t":
                gamma_t = float(np.uint32(int(t[1], 16)).view(np.float32))
            elif t[0] == "best":
                best = int(t[1])
            elif t[0] == "shape":
                S = int(t[3])
            else:
                cells.append(int(t[0]))
                deficits.append([int(x) for x in t[1:]])
    full = np.int64(S) * np.int64(np.rint(np.float64(np.float32(gamma_t)) * 2.0**40))
    return sha, gamma_t, best, np.array(cells, np.int32), full - np.array(deficits, np.int64)


def read_expected_goodput():
    """The goodput-stage sums file written by tests/golden/make_expected_sums.py:
    (inputs_sha256, gamma_fx, gamma_gp, best, cells [n], sum_eo [n, O])."""
    import numpy as np

    sha = None
    gamma_fx = gamma_gp = best = None
    cells, sums = [], []
    with open(os.path.join(GOLDEN, "goodput_paper_scale_sums.txt")) as f:
        for line in f:
            if line.startswith("# inputs_sha256"):
                sha = line.split()[2]
                continue
            if not line.strip() or line.startswith("#"):
                continue
            t = line.split()
            if t[0] == "gamma_fx":
                gamma_fx = int(t[1])
            elif t[0] == "gamma_gp":
                gamma_gp = float(t[1])
            elif t[0] == "best":
                best = int(t[1])
            elif t[0] == "shape":
                continue
            else:
                cells.append(int(t[0]))
                sums.append([int(x) for x in t[1:]])
    return sha, gamma_fx, gamma_gp, best, np.array(cells, np.int32), np.array(sums, np.int64)


def read_expected_replay():
    """The expected replay file written by tests/golden/make_expected_sums.py:
    (inputs_sha256, {stream: (rounds, state, gpu_seconds, reveal order, Gamma_t trace)})."""
    import numpy as np

    sha, out = None, {}
    with open(os.path.join(GOLDEN, "replay_200_streams.txt")) as f:
        for line in f:
            if line.startswith("# inputs_sha256"):
                sha = line.split()[2]
                continue
            if not line.strip() or line.startswith("#"):
                continue
            head, order, trace = line.split("|")
            k, rounds, state, gs = head.split()
            out[int(k)] = (int(rounds), int(state), float(gs), np.array([int(x) for x in order.split()], np.int32),
                           np.array([int(x, 16) for x in trace.split()], np.uint32).view(np.float32))
    return sha, out
