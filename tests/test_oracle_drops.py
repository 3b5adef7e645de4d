"""Pins of the oracle's waiting-deadline / buffer-overflow drops (Sec. 4.1,
Algorithm 1's subscriber branch): the seeded drop draws, a dropped step leaving
every parameter unchanged and handing its batch to the next step, against
brute forces that replay the reassigned batches (delayed SGD with every
version kept, and independent replicas for the parameter-server mode)."""
import numpy as np
import pytest
import torch

import oracle
from _torch_ref import leaves, mono_logits, mono_loss

from test_oracle_model import rand_data, rand_params, tiny_cfg


def test_drop_draws_rate_bounds_and_nesting():
    n = 20000
    assert not oracle.make_drops(5, 0.0, n).any()
    assert oracle.make_drops(5, 1.0, n).all()
    lo, hi = oracle.make_drops(5, 0.05, n), oracle.make_drops(5, 0.2, n)
    for d, r in ((lo, 0.05), (hi, 0.2)):
        assert abs(d.mean() - r) < 4 * np.sqrt(r * (1 - r) / n)
    # one uniform per step compared against a threshold: a lower rate drops a subset of the steps
    assert not (lo & ~hi).any()
    assert (oracle.make_drops(6, 0.2, n) != hi).any()
    # the draws do not depend on how many steps are asked for
    np.testing.assert_array_equal(oracle.make_drops(5, 0.2, 100), hi[:100])
    with pytest.raises(ValueError):
        oracle.make_drops(5, 1.5, 10)


def test_dropped_step_changes_nothing_and_records_nan():
    rng = np.random.default_rng(41)
    cfg = tiny_cfg(S=1)
    params = rand_params(cfg, rng)
    data = rand_data(cfg, 24, rng)
    o = oracle.Oracle(cfg, *data, params)
    o.step(0, 0)
    before = o.current_params()
    rec = o.step(1, 0, record=True, drop=True)
    assert rec.dropped and np.isnan(rec.loss) and rec.batch == 1
    for key, (W, b) in o.current_params().items():
        np.testing.assert_array_equal(W, before[key][0])
        np.testing.assert_array_equal(b, before[key][1])
    assert o.step(0, 0).batch == 1                 # the dropped batch goes to the next step


@pytest.mark.parametrize("n_rows", [24, 29])
def test_zero_staleness_drops_only_shift_the_batches(n_rows):
    # with S = 0 every trained step reads the latest parameters, so the steps that were not dropped
    # are exactly a drop-free run over the same batch sequence
    rng = np.random.default_rng(42)
    cfg = tiny_cfg(batch=6)
    params = rand_params(cfg, rng)
    data = rand_data(cfg, n_rows, rng)
    n = 23
    drops = np.zeros(n, np.uint8)
    drops[[0, 3, 4, 11, 22]] = 1
    z = np.zeros(n, np.int32)
    a = oracle.Oracle(cfg, *data, params)
    la = a.run(z, z, n, drops=drops)[0]
    b = oracle.Oracle(cfg, *data, params)
    lb = b.run(z, z, n - int(drops.sum()))[0]
    assert np.isnan(la[drops == 1]).all()
    np.testing.assert_array_equal(la[drops == 0], lb)
    for key, (W, bias) in a.current_params().items():
        np.testing.assert_array_equal(W, b.current_params()[key][0])
        np.testing.assert_array_equal(bias, b.current_params()[key][1])


def _delayed_sgd_with_drops(cfg, params, xp, xa, y, tau_p, tau_a, drops):
    """Every version kept; a dropped step copies version k forward and the next step trains its batch."""
    n = xp.shape[0]
    nb = -(-n // cfg.batch)
    versions = [{k: (W.copy(), b.copy()) for k, (W, b) in params.items()}]
    done = 0
    for k in range(len(tau_p)):
        if drops[k]:
            versions.append(versions[k])
            continue
        j = done % nb
        done += 1
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


@pytest.mark.parametrize("S,seed", [(1, 3), (2, 4), (3, 5)])
def test_drops_with_staleness_match_brute_force(S, seed):
    cfg = tiny_cfg(passive=(3, 2), active=(3, 2), top=(3, 1), batch=4, lr=0.3, S=S)
    rng = np.random.default_rng(43)
    params = rand_params(cfg, rng, 0.7)
    xp, xa, y = rand_data(cfg, 10, rng)
    n = 14
    tp, ta = oracle.make_schedule(seed, S, oracle.SCHED_SEEDED, n)
    drops = oracle.make_drops(seed, 0.3, n)
    assert 0 < drops.sum() < n
    o = oracle.Oracle(cfg, xp, xa, y, params)
    o.run(tp, ta, n, drops=drops)
    ref = _delayed_sgd_with_drops(cfg, params, xp, xa, y, tp, ta, drops)
    for key in params:
        np.testing.assert_allclose(o.current_params()[key][0], ref[key][0], rtol=1e-11, atol=1e-13)
        np.testing.assert_allclose(o.current_params()[key][1], ref[key][1], rtol=1e-11, atol=1e-13)


# epochs after which the replicas are averaged, from Eq. 5 by hand: Delta T_0 = 2 gives 1, 2, 4
AGGREGATION_EPOCHS = {2: {1, 2, 4}}


def test_parameter_server_epochs_count_trained_batches():
    """Drops shift the epoch ends: the replicas are averaged after the step that
    trains the last batch of an aggregated epoch, whichever step index that is."""
    rng = np.random.default_rng(44)
    workers, dt0 = 3, 2
    cfg = tiny_cfg(batch=6, lr=0.1)
    cfg.workers, cfg.ps_dt0 = workers, dt0
    n = 6 * 3 + 2                        # 4 batches per epoch, the last one ragged
    nb = 4
    params = rand_params(cfg, rng)
    xp, xa, y = rand_data(cfg, n, rng)
    steps = 21
    drops = np.zeros(steps, np.uint8)
    drops[[2, 3, 8, 13]] = 1
    assert (steps - drops.sum()) // nb == 4
    z = np.zeros(steps, np.int32)
    o = oracle.Oracle(cfg, xp, xa, y, params)
    losses = o.run(z, z, steps, drops=drops)[0]

    reps = [leaves(params) for _ in range(workers)]
    ref = []
    done = 0
    for k in range(steps):
        if drops[k]:
            ref.append(np.nan)
            continue
        t = reps[k % workers]
        j = done % nb
        done += 1
        r0, r1 = j * 6, min(n, (j + 1) * 6)
        loss = mono_loss(mono_logits(t, xp[r0:r1], xa[r0:r1]), y[r0:r1], cfg.loss)
        loss.backward()
        ref.append(loss.item())
        with torch.no_grad():
            for W, b in t.values():
                W -= cfg.lr * W.grad
                b -= cfg.lr * b.grad
                W.grad = None
                b.grad = None
        if j == nb - 1 and done // nb in AGGREGATION_EPOCHS[dt0]:
            with torch.no_grad():
                for key in params:
                    for i in range(2):
                        avg = sum(r[key][i] for r in reps) / workers
                        for r in reps:
                            r[key][i].copy_(avg)
    np.testing.assert_allclose(losses, ref, rtol=1e-10)
    for w in range(workers):
        for key, (W, b) in reps[w].items():
            np.testing.assert_allclose(o.replica_params(w)[key][0], W.detach().numpy(), rtol=1e-9, atol=1e-12)
            np.testing.assert_allclose(o.replica_params(w)[key][1], b.detach().numpy(), rtol=1e-9, atol=1e-12)
