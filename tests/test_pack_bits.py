"""The host layout of bit-packed binary features (vfl_bind_host_data_bits): row r of a [n, d] 0 / 1
matrix is ceil(d / 32) 32-bit words, feature c in bit c mod 32 of word c // 32.  Host logic only."""
import numpy as np
import pytest

from paper_2510_12494_gb300 import pack_bits


@pytest.mark.parametrize("d", [1, 11, 12, 31, 32, 33, 1000, 1024])
def test_pack_bits_layout(d):
    rng = np.random.default_rng(d)
    x = (rng.random((9, d)) < 0.3).astype(np.float32)
    w = pack_bits(x)
    assert w.dtype == np.int32 and w.shape == (9, (d + 31) // 32) and w.flags.c_contiguous
    u = w.view(np.uint32)
    for r in range(9):
        for c in range(d):
            assert (int(u[r, c // 32]) >> (c % 32)) & 1 == int(x[r, c])
        # bits past d in the last word are zero
        tail = d % 32
        if tail:
            assert int(u[r, -1]) >> tail == 0


def test_pack_bits_single_features():
    x = np.zeros((3, 70), np.float32)
    x[0, 0] = x[1, 31] = x[2, 69] = 1
    u = pack_bits(x).view(np.uint32)
    assert u[0].tolist() == [1, 0, 0]
    assert u[1].tolist() == [1 << 31, 0, 0]
    assert u[2].tolist() == [0, 0, 1 << 5]


def test_pack_bits_rejects_non_binary():
    with pytest.raises(ValueError):
        pack_bits(np.array([[0.0, 0.5]]))
