"""Pins of the oracle's forward, backward, loss, update and staleness model
against things other than itself: finite differences, a monolithic torch model
with autograd, torch.optim.SGD, brute-force delayed SGD and closed forms."""
import itertools
from types import SimpleNamespace

import numpy as np
import pytest
import torch

import oracle
from _torch_ref import leaves, mono_logits, mono_loss, to_numpy


def tiny_cfg(passive=(4, 3), active=(4, 2), top=(5, 1), loss="bce", d_p=3, d_a=2, batch=8,
             lr=0.05, S=0, dtype="fp32", dp_clip=0.0, dp_sigma=0.0):
    return SimpleNamespace(d_passive=d_p, d_active=d_a, passive=tuple(passive), active=tuple(active),
                           top=tuple(top), loss=loss, batch=batch, lr=lr, staleness=S, dtype=dtype,
                           dp_clip=dp_clip, dp_sigma=dp_sigma, seed=0)


def rand_params(cfg, rng, scale=0.8):
    params = {}
    for party, d_in, widths in ((0, cfg.d_passive, cfg.passive), (1, cfg.d_active, cfg.active),
                                (2, cfg.active[-1] + cfg.passive[-1], cfg.top)):
        for l, w in enumerate(widths):
            params[(party, l)] = (rng.normal(0, scale, (w, d_in)), rng.normal(0, 0.3, w))
            d_in = w
    return params


def rand_data(cfg, n, rng):
    xp = rng.normal(size=(n, cfg.d_passive))
    xa = rng.normal(size=(n, cfg.d_active))
    if cfg.loss == "bce":
        y = rng.integers(0, 2, n).astype(np.int32)
    else:
        y = rng.integers(0, cfg.top[-1], n).astype(np.int32)
    return xp, xa, y


def batch_loss(cfg, params, xp, xa, y):
    """Loss of one batch through the oracle's forward pieces only."""
    P = [params[(0, l)] for l in range(len(cfg.passive))]
    A = [params[(1, l)] for l in range(len(cfg.active))]
    T = [params[(2, l)] for l in range(len(cfg.top))]
    zp = oracle.mlp_forward(P, xp, True, "fp32")[-1]
    za = oracle.mlp_forward(A, xa, True, "fp32")[-1]
    s = oracle.mlp_forward(T, np.concatenate([za, zp], 1), False, "fp32")[-1]
    return oracle.loss_and_dlogits(s, y, cfg.loss)[0], zp, za


def min_abs_preact(cfg, params, xp, xa):
    """Smallest |pre-activation| over all ReLU units (FD needs to stay off the kinks)."""
    m = np.inf
    for party, x, n in ((0, xp, len(cfg.passive)), (1, xa, len(cfg.active))):
        h = x
        for l in range(n):
            W, b = params[(party, l)]
            pre = h @ W.T + b
            m = min(m, np.abs(pre).min())
            h = np.maximum(pre, 0)
    return m


def one_step(cfg, params, xp, xa, y, **kw):
    o = oracle.Oracle(cfg, xp, xa, y, params, **kw)
    return o, o.step(0, 0, record=True)


@pytest.mark.parametrize("loss,top", [("bce", (5, 1)), ("ce", (5, 3)), ("ce", (4, 6, 4))])
def test_gradients_match_finite_differences(loss, top):
    cfg = tiny_cfg(loss=loss, top=top)
    rng = np.random.default_rng(3)
    for _ in range(50):
        params = rand_params(cfg, rng)
        xp, xa, y = rand_data(cfg, 8, rng)
        if min_abs_preact(cfg, params, xp, xa) > 1e-3:
            break
    _, rec = one_step(cfg, params, xp, xa, y)
    h = 1e-6
    for key, (W, b) in params.items():
        for arr, gi in ((W, 0), (b, 1)):
            fd = np.zeros_like(arr)
            for idx in np.ndindex(arr.shape):
                old = arr[idx]
                arr[idx] = old + h
                lp = batch_loss(cfg, params, xp, xa, y)[0]
                arr[idx] = old - h
                lm = batch_loss(cfg, params, xp, xa, y)[0]
                arr[idx] = old
                fd[idx] = (lp - lm) / (2 * h)
            got = rec.grads[key][gi]
            np.testing.assert_allclose(got, fd, rtol=1e-6, atol=1e-8 * max(1.0, np.abs(fd).max()),
                                       err_msg=f"{key} {'W' if gi == 0 else 'b'}")
    # the published gradient is dLoss/dz^p: perturb z^p directly at the top's input
    T = [params[(2, l)] for l in range(len(cfg.top))]
    _, zp, za = batch_loss(cfg, params, xp, xa, y)
    fd = np.zeros_like(zp)
    for idx in np.ndindex(zp.shape):
        for sgn in (1, -1):
            z = zp.copy()
            z[idx] += sgn * h
            s = oracle.mlp_forward(T, np.concatenate([za, z], 1), False, "fp32")[-1]
            fd[idx] += sgn * oracle.loss_and_dlogits(s, y, loss)[0] / (2 * h)
    np.testing.assert_allclose(rec.dzp, fd, rtol=1e-6, atol=1e-9)


@pytest.mark.parametrize("shape", [
    dict(passive=(6, 4), active=(5, 3), top=(4, 1), loss="bce"),            # tiny / credit-like
    dict(passive=(6, 6, 4), active=(5, 5, 4), top=(6, 7), loss="ce"),        # multiclass-like
    dict(passive=(8, 6, 6, 3), active=(5, 4), top=(6, 10), loss="ce"),       # heterogeneous depth
])
def test_split_equals_blockdiagonal_monolithic(shape):
    cfg = tiny_cfg(d_p=7, d_a=5, **shape)
    rng = np.random.default_rng(5)
    params = rand_params(cfg, rng)
    xp, xa, y = rand_data(cfg, 8, rng)
    _, rec = one_step(cfg, params, xp, xa, y)
    tp = leaves(params)
    logits = mono_logits(tp, xp, xa)
    loss = mono_loss(logits, y, cfg.loss)
    loss.backward()
    assert rec.loss == pytest.approx(loss.item(), rel=1e-13)
    np.testing.assert_allclose(rec.logits, logits.detach().numpy(), rtol=1e-12, atol=1e-14)
    for key, (W, b) in tp.items():
        np.testing.assert_allclose(rec.grads[key][0], W.grad.numpy(), rtol=1e-11, atol=1e-14)
        np.testing.assert_allclose(rec.grads[key][1], b.grad.numpy(), rtol=1e-11, atol=1e-14)


@pytest.mark.parametrize("loss,top,n", [("bce", (5, 1), 29), ("ce", (5, 4), 21)])
def test_zero_staleness_is_synchronous_sgd(loss, top, n):
    cfg = tiny_cfg(loss=loss, top=top, batch=8, lr=0.1, S=2)
    rng = np.random.default_rng(9)
    params = rand_params(cfg, rng, 0.6)
    xp, xa, y = rand_data(cfg, n, rng)
    nb = -(-n // cfg.batch)
    steps = 2 * nb + 1                                  # crosses epochs and the partial batch
    o = oracle.Oracle(cfg, xp, xa, y, params)
    tau = np.zeros(steps, np.int32)
    losses, _ = o.run(tau, tau, steps)
    tp = leaves(params)
    opt = torch.optim.SGD([t for pair in tp.values() for t in pair], lr=cfg.lr)
    ref = []
    for k in range(steps):
        j = k % nb
        r0, r1 = j * cfg.batch, min(n, (j + 1) * cfg.batch)
        opt.zero_grad()
        l = mono_loss(mono_logits(tp, xp[r0:r1], xa[r0:r1]), y[r0:r1], loss)
        l.backward()
        opt.step()
        ref.append(l.item())
    np.testing.assert_allclose(losses, ref, rtol=1e-12)
    got = o.current_params()
    for key, (W, b) in to_numpy(tp).items():
        np.testing.assert_allclose(got[key][0], W, rtol=1e-11, atol=1e-13)
        np.testing.assert_allclose(got[key][1], b, rtol=1e-11, atol=1e-13)


def _realisable(S, n):
    """Every tau sequence with tau(0)=0, tau(k) <= min(k, S) and tau(k) <= tau(k-1)+1."""
    seqs = [[0]]
    for k in range(1, n):
        seqs = [s + [t] for s in seqs for t in range(0, min(k, S, s[-1] + 1) + 1)]
    return seqs


def _delayed_sgd_torch(cfg, params, xp, xa, y, tau_p, tau_a):
    """theta_{k+1} = theta_k - eta g(theta at the stale versions), by brute force:
    every version kept, gradients from torch autograd on the monolithic model."""
    n = xp.shape[0]
    nb = -(-n // cfg.batch)
    versions = [{k: (W.copy(), b.copy()) for k, (W, b) in params.items()}]
    for k in range(len(tau_p)):
        j = k % nb
        r0, r1 = j * cfg.batch, min(n, (j + 1) * cfg.batch)
        tpas = leaves({key: v for key, v in versions[k - tau_p[k]].items() if key[0] == 0})
        tact = leaves({key: v for key, v in versions[k - tau_a[k]].items() if key[0] != 0})
        l = mono_loss(mono_logits(tpas, xp[r0:r1], xa[r0:r1], tp_active=tact), y[r0:r1], cfg.loss)
        l.backward()
        grads = {**{k_: (W.grad.numpy(), b.grad.numpy()) for k_, (W, b) in tpas.items()},
                 **{k_: (W.grad.numpy(), b.grad.numpy()) for k_, (W, b) in tact.items()}}
        versions.append({key: (W - cfg.lr * grads[key][0], b - cfg.lr * grads[key][1])
                         for key, (W, b) in versions[k].items()})
    return versions[-1]


@pytest.mark.parametrize("S,n", [(1, 5), (2, 4)])
def test_every_realisable_schedule_matches_brute_force_delayed_sgd(S, n):
    cfg = tiny_cfg(passive=(3, 2), active=(3, 2), top=(3, 1), batch=4, lr=0.3, S=S)
    rng = np.random.default_rng(11)
    params = rand_params(cfg, rng, 0.7)
    xp, xa, y = rand_data(cfg, 10, rng)
    seqs = _realisable(S, n)
    for tp_seq, ta_seq in itertools.product(seqs, seqs):
        o = oracle.Oracle(cfg, xp, xa, y, params)
        o.run(tp_seq, ta_seq, n)
        ref = _delayed_sgd_torch(cfg, params, xp, xa, y, tp_seq, ta_seq)
        got = o.current_params()
        for key in params:
            np.testing.assert_allclose(got[key][0], ref[key][0], rtol=1e-11, atol=1e-13)
            np.testing.assert_allclose(got[key][1], ref[key][1], rtol=1e-11, atol=1e-13)


def test_staleness_outside_bound_is_rejected():
    cfg = tiny_cfg(S=1)
    rng = np.random.default_rng(0)
    o = oracle.Oracle(cfg, *rand_data(cfg, 16, rng), rand_params(cfg, rng))
    with pytest.raises(ValueError):
        o.step(1, 0)          # k = 0 cannot read version -1
    o.step(0, 0)
    with pytest.raises(ValueError):
        o.step(0, 2)          # beyond S


def test_top_gradient_is_logistic_regression_gradient():
    # a single-layer top with BCE is logistic regression on the features [z^a | z^p]
    cfg = tiny_cfg(top=(1,))
    rng = np.random.default_rng(2)
    params = rand_params(cfg, rng)
    xp, xa, y = rand_data(cfg, 8, rng)
    _, rec = one_step(cfg, params, xp, xa, y)
    z = np.concatenate([rec.za, rec.zp], 1)
    w, b = params[(2, 0)]
    r = 1.0 / (1.0 + np.exp(-(z @ w[0] + b[0]))) - y
    np.testing.assert_allclose(rec.grads[(2, 0)][0][0], z.T @ r / 8, rtol=1e-12)
    np.testing.assert_allclose(rec.grads[(2, 0)][1][0], r.mean(), rtol=1e-12)
    np.testing.assert_allclose(rec.dzp, np.outer(r, w[0, rec.za.shape[1]:]) / 8, rtol=1e-12)


def test_zero_learning_rate_makes_staleness_irrelevant():
    cfg = tiny_cfg(S=2, lr=0.0, batch=4)
    rng = np.random.default_rng(4)
    params = rand_params(cfg, rng)
    data = rand_data(cfg, 14, rng)
    tp, ta = oracle.make_schedule(5, 2, oracle.SCHED_SEEDED, 9)
    assert tp.max() > 0 and ta.max() > 0
    a = oracle.Oracle(cfg, *data, params).run(tp, ta, 9)[0]
    z = np.zeros(9, np.int32)
    b = oracle.Oracle(cfg, *data, params).run(z, z, 9)[0]
    np.testing.assert_array_equal(a, b)


def test_dp_without_noise_or_clipping_is_identity():
    rng = np.random.default_rng(6)
    base = tiny_cfg()
    params = rand_params(base, rng)
    data = rand_data(base, 8, rng)
    _, r0 = one_step(base, params, *data)
    _, r1 = one_step(tiny_cfg(dp_clip=1e30, dp_sigma=0.0), params, *data)
    np.testing.assert_allclose(r1.dzp, r0.dzp, rtol=1e-15)
    for key in params:
        np.testing.assert_allclose(r1.grads[key][0], r0.grads[key][0], rtol=1e-15)


def test_dp_clipping_bounds_published_row_norms():
    rng = np.random.default_rng(8)
    cfg = tiny_cfg(dp_clip=0.05, dp_sigma=0.0, batch=8)
    params = rand_params(cfg, rng, 1.5)
    data = rand_data(cfg, 8, rng)
    _, rec = one_step(cfg, params, *data)
    norms = np.linalg.norm(rec.dzp, axis=1)
    assert (norms <= 0.05 / 8 * (1 + 1e-12)).all()
    _, ref = one_step(tiny_cfg(), params, *data)
    raw = np.linalg.norm(ref.dzp, axis=1)
    # rows under the bound are untouched, rows over it keep their direction
    for i in range(8):
        if raw[i] * 8 <= 0.05:
            np.testing.assert_allclose(rec.dzp[i], ref.dzp[i], rtol=1e-14)
        else:
            np.testing.assert_allclose(rec.dzp[i] / norms[i], ref.dzp[i] / raw[i], rtol=1e-12)


def test_dp_noise_statistics_on_published_gradient():
    # with clip -> 0 the published gradient is pure noise: sigma C xi / B
    rng = np.random.default_rng(10)
    cfg = tiny_cfg(passive=(6, 64), active=(4, 3), top=(4, 1), dp_clip=1e-3, dp_sigma=2.0, batch=256)
    params = rand_params(cfg, rng, 0.3)
    data = rand_data(cfg, 256, rng)
    _, rec = one_step(cfg, params, *data, dp_seed=99)
    noise = rec.dzp * 256 / (2.0 * 1e-3)
    z = noise.ravel()
    assert abs(z.mean()) < 4 / np.sqrt(z.size)
    assert abs(z.std() - 1) < 0.02


@pytest.mark.parametrize("values", [
    np.array([1.0, -1.0, 0.0, -0.0, 1.00390625, 1.01171875, 1.0078125 + 2 ** -9, 3.4e38, -3.4e38,
              1e-40, -1e-42, np.inf, -np.inf, 65504.0, 1 / 3, 2 / 3, 1.00390625 + 2 ** -30]),
    np.random.default_rng(12).normal(0, 100, 100000),
    np.random.default_rng(13).normal(0, 1e-39, 1000),
])
def test_bf16_rounding_matches_torch(values):
    got = oracle.bf16_round(values)
    ref = torch.tensor(values.astype(np.float32)).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(got, ref)
    assert np.isnan(oracle.bf16_round(np.array([np.nan]))).all()


def test_bf16_preset_rounds_at_the_stated_points():
    cfg = tiny_cfg(dtype="bf16", passive=(6, 4), active=(5, 3), top=(4, 3), loss="ce")
    rng = np.random.default_rng(14)
    params = rand_params(cfg, rng)
    data = rand_data(cfg, 8, rng)
    _, rec = one_step(cfg, params, *data)
    for t in (rec.zp, rec.za, rec.dzp, rec.dza):
        np.testing.assert_array_equal(t, oracle.bf16_round(t))
    assert not np.array_equal(rec.logits, oracle.bf16_round(rec.logits))
    # against the fp32 run: close but not equal
    _, ref = one_step(tiny_cfg(passive=(6, 4), active=(5, 3), top=(4, 3), loss="ce"), params, *data)
    assert rec.loss == pytest.approx(ref.loss, rel=2e-2)
    assert rec.loss != ref.loss
