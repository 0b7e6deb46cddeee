"""The C ABI library builds, loads and exports what include/fleetsieve.h declares (no GPU needed)."""

import ctypes
import os
import re

import numpy as np
import pytest

from conftest import ROOT


def declared_functions():
    text = open(os.path.join(ROOT, "include", "fleetsieve.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(fs_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("fs_load_model", "fs_score_candidates", "fs_solve", "fs_solve_batch",
                     "fs_solve_bounds", "fs_reveal", "fs_certificate", "fs_free_model",
                     "fs_last_error", "fs_replay"):
        assert required in names


def test_library_exports_every_declared_symbol(fsb):
    L = fsb.lib()
    for name in declared_functions():
        assert hasattr(L, name), name
    assert set(declared_functions()) == set(fsb.EXPORTS)
    assert os.path.dirname(fsb.LIB_PATH) == os.path.join(ROOT, "paper_2608_19659_gb300")


def test_binding_refuses_a_missing_library(fsb, monkeypatch):
    monkeypatch.setattr(fsb, "_lib", None)
    monkeypatch.setattr(fsb, "LIB_PATH", os.path.join(ROOT, "does-not-exist.so"))
    with pytest.raises(fsb.FleetSieveError):
        fsb.lib()


def test_allocation_layout(fsb):
    assert ctypes.sizeof(fsb.fs_allocation) == 608 == fsb.ALLOC_DTYPE.itemsize
    assert fsb.fs_allocation.fulfil.offset == 344 and fsb.fs_allocation.bin.offset == 88
    assert fsb.fs_allocation.goodput.offset == 600


def _good(K=2, B=3):
    n = K * 4 * B
    lo = np.full(n, 1.0, np.float32)
    hi = np.full(n, 2.0, np.float32)
    return lo, hi, lo * 5, hi * 5, np.full(K, 30.0, np.float32), np.full(K, 3.0, np.float32)


@pytest.mark.parametrize("case", ["nan", "neg", "lo_gt_hi", "K0", "K65", "B0", "G0", "theta",
                                  "slo0", "demand0", "qn_bad", "qn_size", "revealed_open"])
def test_load_model_rejects_bad_input(fsb, case):
    K, B, G = 2, 3, 16
    clo, chi, tlo, thi, slo, lam = _good(K, B)
    q = None
    if case == "nan":
        clo = clo.copy(); clo[3] = np.nan
    elif case == "neg":
        tlo = tlo.copy(); tlo[0] = -1.0
    elif case == "lo_gt_hi":
        chi = chi.copy(); chi[5] = 0.5
    elif case == "K0":
        K = 0
    elif case == "K65":
        K = 65
    elif case == "B0":
        B = 0
    elif case == "G0":
        G = 0
    elif case == "theta":
        G = 10000  # K * (G + G/2 + G/4 + G/8) > 16384
    elif case == "slo0":
        slo = slo.copy(); slo[1] = 0.0
    elif case == "demand0":
        lam = lam.copy(); lam[0] = -2.0
    elif case == "qn_bad":
        q = np.linspace(1.0, 0.0, 16, dtype=np.float32)
    elif case == "qn_size":
        q = np.linspace(0.0, 1.0, 12, dtype=np.float32)
    rev = None
    if case == "revealed_open":  # a measured cell must have collapsed bounds
        rev = np.zeros(K * 4 * B, np.uint8)
        rev[4] = 1
    with pytest.raises(fsb.FleetSieveError) as ei:
        fsb.fs_load_model(clo, chi, tlo, thi, slo, lam, G, K, B, quantile=q, revealed=rev)
    assert ei.value.code == fsb.FS_EINVAL
    assert fsb.fs_last_error()


@pytest.mark.parametrize("args", [(2, 8, 1024, 10), (0, 13, 1024, 10), (1, -1, 1024, 10), (0, 8, 0, 10),
                                  (1, 8, 1 << 40, 10), (0, 8, 1024, 0), (1, 8, 1024, 1001)])
def test_draw_floor_rejects_bad_arguments(fsb, args):
    """The measurement floor checks its arguments before touching a device."""
    with pytest.raises(fsb.FleetSieveError) as ei:
        fsb.fs_draw_floor(*args)
    assert ei.value.code == fsb.FS_EINVAL
