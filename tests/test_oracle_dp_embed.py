"""Pins of the oracle's DP mechanism on the published embedding (App. C, Eq. 25):
the identity and clipping reductions, the noise statistics, the
straight-through backward against torch autograd with the clip factor held
constant, and the noise-multiplier formula."""
import math

import numpy as np
import pytest
import torch

import oracle
from _torch_ref import F64, leaves, mono_loss

from test_oracle_model import one_step, rand_data, rand_params, tiny_cfg


def emb_cfg(**kw):
    c = tiny_cfg(**{k: v for k, v in kw.items() if k != "dp_target"})
    c.dp_target = kw.get("dp_target", "emb")
    return c


def test_embedding_dp_without_noise_or_clipping_is_identity():
    rng = np.random.default_rng(21)
    base = tiny_cfg()
    params = rand_params(base, rng)
    data = rand_data(base, 8, rng)
    _, r0 = one_step(base, params, *data)
    _, r1 = one_step(emb_cfg(dp_clip=1e30, dp_sigma=0.0), params, *data)
    np.testing.assert_array_equal(r1.zp, r0.zp)
    np.testing.assert_array_equal(r1.dzp, r0.dzp)
    for key in params:
        np.testing.assert_allclose(r1.grads[key][0], r0.grads[key][0], rtol=1e-15)
        np.testing.assert_allclose(r1.grads[key][1], r0.grads[key][1], rtol=1e-15)


def test_embedding_clipping_bounds_published_rows_and_keeps_direction():
    rng = np.random.default_rng(22)
    cfg = emb_cfg(dp_clip=2.0, dp_sigma=0.0)
    params = rand_params(cfg, rng, 1.5)
    data = rand_data(cfg, 8, rng)
    _, rec = one_step(cfg, params, *data)
    _, ref = one_step(tiny_cfg(), params, *data)
    norms = np.linalg.norm(rec.zp, axis=1)
    raw = np.linalg.norm(ref.zp, axis=1)
    assert (norms <= 2.0 * (1 + 1e-12)).all()
    assert (raw > 2.0).any() and (raw <= 2.0).any()        # both branches are exercised
    for i in range(8):
        if raw[i] <= 2.0:
            np.testing.assert_array_equal(rec.zp[i], ref.zp[i])
        else:
            np.testing.assert_allclose(rec.zp[i] / norms[i], ref.zp[i] / raw[i], rtol=1e-12)


def test_embedding_noise_statistics():
    # with a clip far below every row norm the published embedding is C z/|z| + sigma C xi
    rng = np.random.default_rng(23)
    cfg = emb_cfg(passive=(6, 64), active=(4, 3), top=(4, 1), dp_clip=1e-3, dp_sigma=2.0, batch=256)
    params = rand_params(cfg, rng, 0.6)
    data = rand_data(cfg, 256, rng)
    _, rec = one_step(cfg, params, *data, dp_seed=77)
    _, ref = one_step(tiny_cfg(passive=(6, 64), active=(4, 3), top=(4, 1), batch=256), params, *data)
    zc = ref.zp * np.minimum(1.0, 1e-3 / np.maximum(np.linalg.norm(ref.zp, axis=1, keepdims=True), 1e-300))
    noise = ((rec.zp - zc) / (2.0 * 1e-3)).ravel()
    assert abs(noise.mean()) < 4 / np.sqrt(noise.size)
    assert abs(noise.std() - 1) < 0.02
    # the embedding's draws are independent of the gradient mechanism's (another counter tag)
    g = oracle.dp_normals(77, 0, 256, 64, oracle.TAG_DP).ravel()
    assert abs(np.corrcoef(noise, g)[0, 1]) < 4 / np.sqrt(noise.size)


@pytest.mark.parametrize("loss,top", [("bce", (5, 1)), ("ce", (5, 3))])
@pytest.mark.parametrize("sigma", [0.0, 0.7])
def test_straight_through_backward_matches_autograd(loss, top, sigma):
    """Every gradient of one step equals torch autograd of the split model in
    which the published embedding is c * z^p + sigma C xi with c (and the noise)
    held constant: the straight-through reading of the mechanism's backward."""
    rng = np.random.default_rng(24)
    cfg = emb_cfg(top=top, loss=loss, dp_clip=0.5, dp_sigma=sigma, batch=8)
    params = rand_params(cfg, rng, 1.2)
    xp, xa, y = rand_data(cfg, 8, rng)
    _, rec = one_step(cfg, params, xp, xa, y, dp_seed=5)

    t = leaves(params)
    h = torch.as_tensor(xp, dtype=F64)
    for l in range(len(cfg.passive)):
        W, b = t[(0, l)]
        h = torch.relu(h @ W.T + b)
    zp = h
    c = torch.clamp(0.5 / zp.detach().norm(dim=1), max=1.0)
    xi = torch.as_tensor(oracle.dp_normals(5, 0, 8, zp.shape[1], oracle.TAG_DPE), dtype=F64)
    zt = zp * c[:, None] + sigma * 0.5 * xi
    ha = torch.as_tensor(xa, dtype=F64)
    for l in range(len(cfg.active)):
        W, b = t[(1, l)]
        ha = torch.relu(ha @ W.T + b)
    s = torch.cat([ha, zt], dim=1)
    for l in range(len(cfg.top)):
        W, b = t[(2, l)]
        s = s @ W.T + b
        if l < len(cfg.top) - 1:
            s = torch.relu(s)
    mono_loss(s, y, loss).backward()
    np.testing.assert_allclose(rec.zp, zt.detach().numpy(), rtol=1e-12, atol=1e-14)
    for key, (W, b) in t.items():
        np.testing.assert_allclose(rec.grads[key][0], W.grad.numpy(), rtol=1e-9, atol=1e-13)
        np.testing.assert_allclose(rec.grads[key][1], b.grad.numpy(), rtol=1e-9, atol=1e-13)


def test_gradient_target_is_unchanged_by_the_embedding_option():
    rng = np.random.default_rng(25)
    params = rand_params(tiny_cfg(), rng)
    data = rand_data(tiny_cfg(), 8, rng)
    _, a = one_step(tiny_cfg(dp_clip=0.05, dp_sigma=0.5), params, *data, dp_seed=3)
    _, b = one_step(emb_cfg(dp_clip=0.05, dp_sigma=0.5, dp_target="grad"), params, *data, dp_seed=3)
    np.testing.assert_array_equal(a.dzp, b.dzp)
    np.testing.assert_array_equal(a.zp, b.zp)


def test_gdp_sigma_follows_eq25():
    # Eq. 25: sigma ~ N_m sqrt(K) / (mu N): linear in the minibatch and in 1/mu, sqrt in the queries,
    # inverse in the dataset size
    base = oracle.gdp_sigma(1.0, 1024, 30000, 150)
    assert base > 0 and math.isfinite(base)
    assert oracle.gdp_sigma(1.0, 1024, 60000, 150) == pytest.approx(base / 2)
    assert oracle.gdp_sigma(0.5, 1024, 30000, 150) == pytest.approx(2 * oracle.gdp_sigma(1.0, 1024, 30000, 150))
    assert oracle.gdp_sigma(1.0, 1024, 30000, 600) == pytest.approx(2 * oracle.gdp_sigma(1.0, 1024, 30000, 150))
    assert oracle.gdp_sigma(1.0, 2048, 30000, 150) == pytest.approx(2 * oracle.gdp_sigma(1.0, 1024, 30000, 150))
