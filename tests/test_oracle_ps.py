"""Pins of the oracle's intra-party semi-asynchronous parameter server (Sec.
4.2, Eq. 5, Algorithm 1): the synchronisation interval against values worked
out by hand, one worker reducing to plain SGD, and W replicas against a torch
brute force (independent models trained with autograd on their own steps,
averaged at the end of the epochs Eq. 5 selects)."""
import numpy as np
import pytest
import torch

import oracle
from _torch_ref import leaves, mono_logits, mono_loss

from test_oracle_model import rand_data, rand_params, tiny_cfg


def ps_cfg(workers, dt0, **kw):
    c = tiny_cfg(**kw)
    c.workers = workers
    c.ps_dt0 = dt0
    return c


def test_eq5_interval_and_aggregation_epochs():
    # Delta T_0 = 5: 2.5 tanh(0.4 t - 2) + 2.5 rounded up, worked out by hand for t = 0..10
    assert [oracle.ps_interval(t, 5) for t in range(11)] == [1, 1, 1, 1, 2, 3, 4, 5, 5, 5, 5]
    assert [t for t in range(1, 11) if oracle.ps_aggregates_after(t, 5)] == [1, 2, 3, 4, 10]
    # Delta T_0 = 1: 0.5 tanh(2 t - 2) + 0.5 is in (0, 1] for t >= 1: every epoch
    assert all(oracle.ps_aggregates_after(t, 1) for t in range(1, 20))
    # Delta T_0 = 2: tanh(t - 2) + 1 -> 0.24, 1, 1.76, 1.96 -> intervals 1, 1, 2, 2
    assert [t for t in range(1, 5) if oracle.ps_aggregates_after(t, 2)] == [1, 2, 4]


def test_one_worker_is_plain_sgd():
    rng = np.random.default_rng(31)
    base = tiny_cfg(batch=8)
    params = rand_params(base, rng)
    data = rand_data(base, 8 * 5, rng)
    z = np.zeros(15, np.int32)
    a = oracle.Oracle(base, *data, params)
    la = a.run(z, z, 15)[0]
    cfg = ps_cfg(1, 2, batch=8)
    b = oracle.Oracle(cfg, *data, params)
    lb = b.run(z, z, 15)[0]
    np.testing.assert_array_equal(la, lb)
    for key, (W, bias) in a.current_params().items():
        np.testing.assert_array_equal(W, b.current_params()[key][0])
        np.testing.assert_array_equal(bias, b.current_params()[key][1])


def test_staleness_is_rejected_in_parameter_server_mode():
    rng = np.random.default_rng(32)
    cfg = ps_cfg(2, 1, S=1)
    with pytest.raises(ValueError):
        oracle.Oracle(cfg, *rand_data(cfg, 16, rng), rand_params(cfg, rng))


# epochs 1..4 after which the replicas are averaged, worked out by hand from Eq. 5 (see above)
AGGREGATION_EPOCHS = {1: {1, 2, 3, 4}, 2: {1, 2, 4}, 5: {1, 2, 3, 4}}


@pytest.mark.parametrize("workers,dt0", [(2, 1), (3, 1), (2, 2), (3, 5)])
def test_replicas_match_torch_brute_force(workers, dt0):
    rng = np.random.default_rng(33 + workers + dt0)
    cfg = ps_cfg(workers, dt0, batch=6, lr=0.1)
    n = 6 * 4 + 3                        # 5 batches per epoch, the last one ragged
    params = rand_params(cfg, rng)
    xp, xa, y = rand_data(cfg, n, rng)
    nb = -(-n // 6)
    epochs = 4
    steps = nb * epochs
    z = np.zeros(steps, np.int32)
    o = oracle.Oracle(cfg, xp, xa, y, params)
    losses = o.run(z, z, steps)[0]

    reps = [leaves(params) for _ in range(workers)]
    ref_losses = []
    for k in range(steps):
        t = reps[k % workers]
        j = k % nb
        r0, r1 = j * 6, min(n, (j + 1) * 6)
        loss = mono_loss(mono_logits(t, xp[r0:r1], xa[r0:r1]), y[r0:r1], cfg.loss)
        loss.backward()
        ref_losses.append(loss.item())
        with torch.no_grad():
            for W, b in t.values():
                W -= cfg.lr * W.grad
                b -= cfg.lr * b.grad
                W.grad = None
                b.grad = None
        epoch = (k + 1) // nb
        if (k + 1) % nb == 0 and epoch in AGGREGATION_EPOCHS[dt0]:
            with torch.no_grad():
                for key in params:
                    for i in range(2):
                        avg = sum(r[key][i] for r in reps) / workers
                        for r in reps:
                            r[key][i].copy_(avg)
    np.testing.assert_allclose(losses, ref_losses, rtol=1e-10)
    for w in range(workers):
        got = o.replica_params(w)
        for key, (W, b) in reps[w].items():
            np.testing.assert_allclose(got[key][0], W.detach().numpy(), rtol=1e-9, atol=1e-12)
            np.testing.assert_allclose(got[key][1], b.detach().numpy(), rtol=1e-9, atol=1e-12)
