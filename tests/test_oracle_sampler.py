"""Pins of the oracle's sampler: Philox known answers, quantile CDF, strata."""

import numpy as np
import pytest

from conftest import read_golden


def test_philox_known_answers(oracle_lib):
    rows = read_golden("philox4x32_10_kat.txt")
    assert len(rows) == 3
    for r in rows:
        v = [int(x, 16) for x in r]
        out = oracle_lib.philox4x32_10(v[0:4], v[4:6])
        assert [int(x) for x in out] == v[6:10]


@pytest.mark.parametrize("Q", [1, 2, 16, 4096])
def test_triangular_table_matches_closed_form_cdf(oracle_lib, Q):
    qn = oracle_lib.triangular_table(Q).astype(np.float64)
    u = (np.arange(Q) + 0.5) / Q
    # CDF of the symmetric triangular law on [0, 1]
    F = np.where(qn <= 0.5, 2.0 * qn * qn, 1.0 - 2.0 * (1.0 - qn) ** 2)
    # one float rounding of u/2 and of the sqrt, then the CDF slope (<= 2)
    assert np.max(np.abs(F - u)) < 4e-7
    assert np.all(np.diff(qn) > 0)
    assert np.all((qn > 0) & (qn < 1))
    # symmetry of the law about 1/2
    assert np.max(np.abs(qn + qn[::-1] - 1.0)) < 2e-7


def test_triangular_table_moments(oracle_lib):
    qn = oracle_lib.triangular_table(4096).astype(np.float64)
    # mean 1/2, variance 1/24 for the symmetric triangular law on [0, 1]
    assert abs(qn.mean() - 0.5) < 1e-7
    assert abs(qn.var() - 1.0 / 24.0) < 1e-6


@pytest.mark.parametrize("O", [1, 4, 8, 16, 4096])
def test_draw_indices_stay_in_their_stratum(oracle_lib, O):
    Q = 4096
    W = Q // O
    for o in range(0, O, max(1, O // 4)):
        for s in range(64):
            kc, kl = oracle_lib.draw_index(12345, 7, 3, 17, Q, O, o, s)
            assert o * W <= kc < (o + 1) * W
            assert o * W <= kl < (o + 1) * W


def test_draw_indices_uniform_within_stratum(oracle_lib):
    Q, O = 64, 4
    W = Q // O
    counts = np.zeros((2, W), np.int64)
    n = 4000
    for s in range(n):
        kc, kl = oracle_lib.draw_index(99, 0, 0, 5, Q, O, 2, s)
        counts[0, kc - 2 * W] += 1
        counts[1, kl - 2 * W] += 1
    exp = n / W
    chi2 = ((counts - exp) ** 2 / exp).sum(axis=1)
    # 15 degrees of freedom: the 99.99% quantile is about 44
    assert np.all(chi2 < 44.0)
    # capacity and tail positions are not the same stream
    assert not np.array_equal(counts[0], counts[1])


def test_draw_arguments_validated(oracle_lib):
    with pytest.raises(ValueError):
        oracle_lib.draw_index(0, 0, 0, 0, 4096, 3, 0, 0)  # O does not divide Q
    with pytest.raises(ValueError):
        oracle_lib.draw_index(0, 0, 0, 0, 96, 8, 0, 0)  # Q/O not a power of two
    with pytest.raises(ValueError):
        oracle_lib.draw_index(0, 0, 0, 0, 4096, 8, 8, 0)  # outcome out of range
    with pytest.raises(ValueError):
        oracle_lib.draw_index(0, 0, 0, 0, 1 << 17, 1, 0, 0)  # more than 2^16 positions per stratum
    assert 0 <= oracle_lib.draw_index(0, 0, 0, 0, 1 << 16, 1, 0, 5)[0] < (1 << 16)


def test_four_samples_share_one_philox_call(oracle_lib):
    """Samples 4m..4m+3 read the four words of the call with counter m (16-bit halves)."""
    Q, O, o, cell, seed, stream, rnd = 4096, 16, 5, 33, (3 << 32) | 9, 2, 7
    W = Q // O
    for m in (0, 1, 77):
        x = oracle_lib.philox4x32_10([m, o, cell, rnd], [seed & 0xFFFFFFFF, (seed >> 32) ^ stream])
        for h in range(4):
            kc, kl = oracle_lib.draw_index(seed, stream, rnd, cell, Q, O, o, 4 * m + h)
            word = int(x[h])
            assert kc == o * W + ((word >> 16) >> 8) and kl == o * W + ((word & 0xFFFF) >> 8)


def test_map_is_affine_clamped_and_monotone(oracle_lib):
    assert oracle_lib.map_value(2.5, 2.5, 0.7) == np.float32(2.5)
    assert oracle_lib.map_value(1.0, 3.0, 0.0) == np.float32(1.0)
    assert oracle_lib.map_value(1.0, 3.0, 1.0) == np.float32(3.0)
    assert oracle_lib.map_value(1.0, 3.0, 0.5) == np.float32(2.0)
    qs = np.linspace(0, 1, 257, dtype=np.float32)
    vals = [oracle_lib.map_value(0.3, 7.9, float(q)) for q in qs]
    assert all(a <= b for a, b in zip(vals, vals[1:]))
    assert all(np.float32(0.3) <= v <= np.float32(7.9) for v in vals)
