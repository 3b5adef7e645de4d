"""The oracle's staleness schedules: bounded, realisable (versions never move
backwards), and reproducible from the seed."""
import numpy as np
import pytest

import oracle


def test_sync_and_max():
    tp, ta = oracle.make_schedule(0, 3, oracle.SCHED_SYNC, 10)
    assert not tp.any() and not ta.any()
    tp, ta = oracle.make_schedule(0, 3, oracle.SCHED_MAX, 10)
    np.testing.assert_array_equal(tp, [0, 1, 2, 3, 3, 3, 3, 3, 3, 3])
    np.testing.assert_array_equal(ta, tp)


@pytest.mark.parametrize("S", [0, 1, 2, 4])
@pytest.mark.parametrize("seed", [0, 1, 2 ** 40 + 3])
def test_seeded_is_bounded_and_realisable(S, seed):
    n = 600
    for tau in oracle.make_schedule(seed, S, oracle.SCHED_SEEDED, n):
        assert tau.dtype == np.int32 and tau[0] == 0
        k = np.arange(n)
        assert (tau >= 0).all() and (tau <= np.minimum(k, S)).all()
        v = k - tau
        assert (np.diff(v) >= 0).all()          # the version consumed never decreases
        if S:
            assert set(np.unique(tau)) == set(range(S + 1))


def test_seeded_depends_on_seed_and_party():
    a = oracle.make_schedule(0, 4, oracle.SCHED_SEEDED, 200)
    b = oracle.make_schedule(1, 4, oracle.SCHED_SEEDED, 200)
    assert not np.array_equal(a[0], b[0])
    assert not np.array_equal(a[0], a[1])
    c = oracle.make_schedule(0, 4, oracle.SCHED_SEEDED, 120)
    np.testing.assert_array_equal(c[0], a[0][:120])


def test_invalid():
    with pytest.raises(ValueError):
        oracle.make_schedule(0, -1, oracle.SCHED_SYNC, 3)
    with pytest.raises(ValueError):
        oracle.make_schedule(0, 1, 7, 3)
