"""The seeded input generators: row-addressable, deterministic, and with the
distributions each workload recipe states."""
import numpy as np
import pytest

import synth


@pytest.mark.parametrize("cid", [1, 2, 3, 4, 5])
def test_row_ranges_are_consistent(cid):
    p = synth.preset(cid)
    a = synth.make_dataset(p, rows=(0, 300))
    b = synth.make_dataset(p, rows=(120, 300), chunk=50)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x[120:], y)
    assert a[0].shape == (300, p.d_passive) and a[1].shape == (300, p.d_active)
    assert a[0].dtype == np.float32 and a[2].dtype == np.int32


def test_recipes():
    xp, xa, y = synth.make_dataset(synth.preset(1))
    x = np.concatenate([xp, xa], 1)
    assert abs(x.mean()) < 0.03 and abs(x.std() - 1) < 0.03 and set(np.unique(y)) == {0, 1}
    xp, xa, y = synth.make_dataset(synth.preset(2))
    assert abs(y.mean() - 0.22) < 0.001
    cat = np.concatenate([xp[:, 7:], xa[:, 7:]], 1)
    assert set(np.unique(cat)) == set(range(7))
    xp, xa, y = synth.make_dataset(synth.preset(3), rows=(0, 5000))
    x = np.concatenate([xp, xa], 1)
    np.testing.assert_array_equal(x[:, 10:14].sum(1), 1)
    np.testing.assert_array_equal(x[:, 14:].sum(1), 1)
    assert set(np.unique(y)) <= set(range(7)) and len(np.unique(y)) >= 5
    xp, xa, y = synth.make_dataset(synth.preset(4), rows=(0, 2000))
    assert abs(np.concatenate([xp, xa], 1).mean() - 0.05) < 0.002
    assert abs(y.mean() - 0.5) < 0.1
    xp, xa, y = synth.make_dataset(synth.preset(5), rows=(0, 2000))
    x = np.concatenate([xp, xa], 1)
    assert x.min() >= 0 and x.max() <= 1 and np.bincount(y, minlength=10).min() > 50


@pytest.mark.parametrize("cid", [1, 2, 3, 4, 5])
def test_init_params(cid):
    p = synth.preset(cid)
    params = synth.init_params(p)
    assert len(params) == len(p.passive) + len(p.active) + len(p.top)
    for (party, l, out, fin) in synth.layer_shapes(p):
        W, b = params[(party, l)]
        assert W.shape == (out, fin) and b.shape == (out,)
        bound = 1 / np.sqrt(fin)
        assert np.abs(W).max() <= bound and np.abs(b).max() <= bound
    assert synth.layer_shapes(p)[len(p.passive) + len(p.active)][3] == p.e_active + p.e_passive


def test_custom_shape_recipe():
    """cid 0: any widths; N(0, 1) features, labels within the classes of the loss."""
    p = synth.preset(1).with_(cid=0, d_passive=37, d_active=5, n_rows=3000, top=(8, 5), loss="ce")
    xp, xa, y = synth.make_dataset(p)
    assert xp.shape == (3000, 37) and xa.shape == (3000, 5)
    x = np.concatenate([xp, xa], 1)
    assert abs(x.mean()) < 0.03 and abs(x.std() - 1) < 0.03
    assert set(np.unique(y)) == set(range(5))
    a = synth.make_dataset(p, rows=(1000, 1200))
    for u, v in zip(a, (xp[1000:1200], xa[1000:1200], y[1000:1200])):
        np.testing.assert_array_equal(u, v)
    _, _, yb = synth.make_dataset(p.with_(loss="bce", top=(8, 1)))
    assert set(np.unique(yb)) == {0, 1}
