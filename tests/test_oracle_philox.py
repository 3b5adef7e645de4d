"""Pins of the oracle's Philox4x32-10 and its DP normal draws."""
import math
import os

import numpy as np
import pytest
import scipy.stats

import oracle
import synth
from conftest import GOLDEN


def _kat():
    rows = []
    with open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                rows.append([int(t, 16) for t in line.split()])
    return rows


@pytest.mark.parametrize("row", _kat())
def test_known_answers(row):
    out = oracle.philox(tuple(np.uint64(v) for v in row[:4]), (row[4], row[5]))
    assert [int(v) for v in out] == row[6:]


@pytest.mark.parametrize("row", _kat())
def test_input_generator_matches_known_answers(row):
    # the shared input generator is a separate implementation; pin it too
    out = synth.philox4x32_10(*[np.array([v], np.uint64) for v in row[:4]], row[4], row[5])
    assert [int(v[0]) for v in out] == row[6:]


def test_weyl_constants_from_their_definition():
    # key increments: first 32 fractional bits of the golden ratio and of sqrt(3) - 1
    s = math.isqrt(5 << 128)                       # floor(sqrt(5) * 2^64)
    golden_frac = ((1 << 64) + s) // 2 - (1 << 64)  # floor((phi - 1) * 2^64)
    assert golden_frac >> 32 == oracle.PHILOX_W[0]
    s3 = math.isqrt(3 << 128) - (1 << 64)          # floor((sqrt(3) - 1) * 2^64)
    assert s3 >> 32 == oracle.PHILOX_W[1]


def _inverse_round(c, k0, k1):
    m0inv = pow(oracle.PHILOX_M[0], -1, 1 << 32)
    m1inv = pow(oracle.PHILOX_M[1], -1, 1 << 32)
    o0, o1, o2, o3 = c
    x0 = (o3 * m0inv) & 0xFFFFFFFF
    x2 = (o1 * m1inv) & 0xFFFFFFFF
    hi0 = (x0 * oracle.PHILOX_M[0]) >> 32
    hi1 = (x2 * oracle.PHILOX_M[1]) >> 32
    return [x0, o0 ^ hi1 ^ k0, x2, o2 ^ hi0 ^ k1]


def test_rounds_are_a_bijection():
    rng = np.random.default_rng(1)
    for _ in range(20):
        c = [int(v) for v in rng.integers(0, 1 << 32, 4, dtype=np.uint64)]
        k = [int(v) for v in rng.integers(0, 1 << 32, 2, dtype=np.uint64)]
        out = [int(v) for v in oracle.philox(tuple(np.uint64(v) for v in c), k)]
        keys = [((k[0] + r * oracle.PHILOX_W[0]) & 0xFFFFFFFF, (k[1] + r * oracle.PHILOX_W[1]) & 0xFFFFFFFF)
                for r in range(10)]
        x = out
        for r in reversed(range(10)):
            x = _inverse_round(x, *keys[r])
        assert x == c


def test_dp_normals_are_standard_normal():
    z = oracle.dp_normals(seed=7, k=3, rows=2000, cols=500).ravel()
    n = z.size
    assert abs(z.mean()) < 4.0 / math.sqrt(n)
    assert abs(z.var() - 1.0) < 4.0 * math.sqrt(2.0 / n)
    assert scipy.stats.kstest(z, "norm").pvalue > 1e-4


def test_dp_normals_layout():
    # column c of row i uses block (c//4, i, k); pairs (x0,x1) and (x2,x3)
    seed, k = 0x123456789, 11
    z = oracle.dp_normals(seed, k, rows=3, cols=10)
    x = synth.philox4x32_10(np.array([2], np.uint64), np.array([1], np.uint64),
                            np.array([k], np.uint64), np.array([oracle.TAG_DP], np.uint64),
                            seed & 0xFFFFFFFF, seed >> 32)
    # row 1, columns 8 and 9: block q = 2, first pair (x0, x1)
    u1 = ((int(x[0][0]) >> 8) + 1) * 2.0 ** -24
    u2 = (int(x[1][0]) >> 8) * 2.0 ** -24
    r = math.sqrt(-2 * math.log(u1))
    assert z[1, 8] == pytest.approx(r * math.cos(2 * math.pi * u2), rel=1e-14)
    assert z[1, 9] == pytest.approx(r * math.sin(2 * math.pi * u2), rel=1e-14)
    z2 = oracle.dp_normals(seed, k, rows=3, cols=12)
    u1 = ((int(x[2][0]) >> 8) + 1) * 2.0 ** -24
    u2 = (int(x[3][0]) >> 8) * 2.0 ** -24
    r = math.sqrt(-2 * math.log(u1))
    assert z2[1, 10] == pytest.approx(r * math.cos(2 * math.pi * u2), rel=1e-14)
    assert z2[1, 11] == pytest.approx(r * math.sin(2 * math.pi * u2), rel=1e-14)
    np.testing.assert_array_equal(z2[:, :10], z)
    # different steps and rows draw different noise
    assert not np.allclose(oracle.dp_normals(seed, k + 1, 3, 10), z)
    assert not np.allclose(z[0], z[1])
