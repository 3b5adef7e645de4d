"""The library's seeded parameter initialisation and its epoch call: the
initial parameters equal the input generator's bit for bit (the same Philox
stream), and vfl_train_epoch runs the epoch's steps and returns the mean loss
per sample over the steps it trained, against the oracle."""
import numpy as np
import pytest

import oracle
import synth
from _parity import new_context, schedule, setup

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def vfl():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2510_12494_gb300 import build
    build.build()
    import paper_2510_12494_gb300 as v
    return v


@pytest.mark.parametrize("cid,seed", [(1, 0), (2, 7), (5, 123456789012)])
def test_init_params_equal_the_generator(vfl, cid, seed):
    p = synth.preset(cid).with_(n_rows=4096)
    ctx = vfl.Context(p, p.n_rows)
    ctx.init_params(seed)
    want = synth.init_params(p, seed)
    for key, (W, b) in ctx.get_params().items():
        np.testing.assert_array_equal(W, want[key][0])
        np.testing.assert_array_equal(b, want[key][1])


@pytest.mark.parametrize("with_drops", [False, True])
def test_train_epoch_mean_loss(vfl, with_drops):
    q, xp, xa, y, params = setup(synth.preset(2), 3 * 1024 + 304)
    nb = q.steps_per_epoch
    tp, ta = schedule(q, 2 * nb)
    drops = None
    if with_drops:
        drops = np.zeros(2 * nb, np.uint8)
        drops[[1, nb + 2]] = 1
    ctx = new_context(vfl, q, xp, xa, y, params)
    got = [ctx.train_epoch(e, tp, ta, drops) for e in range(2)]
    o = oracle.Oracle(q, xp, xa, y, params, dp_seed=q.seed)
    for e in range(2):
        losses, recs = o.run(tp, ta, nb, record_steps=range(e * nb, (e + 1) * nb), drops=drops)
        rows = np.array([0 if r.dropped else r.rows[1] - r.rows[0] for r in (recs[k] for k in sorted(recs))])
        want = np.nansum(losses * rows) / rows.sum()
        assert abs(got[e] - want) / abs(want) < 1e-5
        mine = ctx.read_losses(e * nb, nb)
        assert np.isnan(mine).sum() == (0 if drops is None else int(drops[e * nb:(e + 1) * nb].sum()))


@pytest.mark.parametrize("cid", [2, 3])
def test_uniform_order_and_graph_updates(vfl, cid):
    """The uniform dependency order computes exactly what the overlapping order does, and in it one
    graph updated in place per epoch (vfl_graph_update) replays every epoch of a seeded schedule."""
    rows = {2: 4 * 1024 + 304, 3: 2 * 4096 + 288}[cid]
    q, xp, xa, y, params = setup(synth.preset(cid), rows)
    nb = q.steps_per_epoch
    n = 4 * nb
    tp, ta = schedule(q, n)
    ref = new_context(vfl, q, xp, xa, y, params)
    ref.train_steps(0, n, tp, ta)
    uni = new_context(vfl, q, xp, xa, y, params)
    uni.set_order(True)
    uni.train_steps(0, n, tp, ta)
    np.testing.assert_array_equal(uni.read_losses(0, n), ref.read_losses(0, n))
    ctx = new_context(vfl, q, xp, xa, y, params)
    ctx.set_order(True)
    # a window's shape also depends on which worker stream its first step lands on: one graph per
    # first worker, each updated in place for every later window that starts on that worker
    graphs = {}
    for e in range(4):
        w = (e * nb) % q.workers
        if w in graphs:
            assert ctx.update_graph(graphs[w], e * nb, nb, tp, ta), f"epoch {e} did not fit its graph"
        else:
            graphs[w] = ctx.capture(e * nb, nb, tp, ta)
        ctx.launch_graph(graphs[w])
    ctx.synchronize()
    np.testing.assert_array_equal(ctx.read_losses(0, n), ref.read_losses(0, n))
    for key, (W, b) in ctx.get_params().items():
        np.testing.assert_array_equal(W, ref.get_params()[key][0])
        np.testing.assert_array_equal(b, ref.get_params()[key][1])
    assert vfl.lib().vfl_set_order(ctx.h, 2) == vfl.VFL_E_INVAL


@pytest.mark.parametrize("cid", [3, 4])
def test_per_layer_path_headers_ride_in_the_kernels(vfl, cid):
    """On the per-layer path the payload's last writer publishes the channel header and the first reader
    checks it: no header kernels run unless a DP kernel writes the payload (wide-dp perturbs the gradient),
    and the published headers are the steps' own."""
    rows = {3: 2 * 4096 + 288, 4: 8192 + 576}[cid]
    q, xp, xa, y, params = setup(synth.preset(cid), rows)
    ctx = new_context(vfl, q, xp, xa, y, params)
    tp, ta = schedule(q, 4)
    ctx.profile(True)
    ctx.train_steps(0, 4, tp, ta)
    ctx.profile(False)
    used = {k: v[0] for k, v in ctx.profile_summary().items()}
    assert used.get("channel_header", 0) == (4 if cid == 4 else 0), used
    ctx.check_channel(0, 3)
    ctx.check_channel(1, 3)


def test_exchange_bytes_count_the_published_payloads(vfl):
    q, xp, xa, y, params = setup(synth.preset(2), 3 * 1024 + 304)
    ctx = new_context(vfl, q, xp, xa, y, params)
    n = 2 * q.steps_per_epoch
    tp, ta = schedule(q, n)
    drops = np.zeros(n, np.uint8)
    drops[3] = 1
    ctx.train_steps(0, n, tp, ta, drops)
    rows = sum(ctx.batch_rows(k)[1] - ctx.batch_rows(k)[0] for k in range(n))
    rows_kept = sum(ctx.batch_rows(k)[1] - ctx.batch_rows(k)[0] for k in range(n) if not drops[k])
    assert ctx.exchange_bytes() == (rows * q.e_passive * 4, rows_kept * q.e_passive * 4)


def test_graph_update_refuses_another_shape_and_keeps_the_graph(vfl):
    """A window whose graph has another shape (here: a dropped step) is refused by vfl_graph_update, and the
    graph still replays the window it holds."""
    q, xp, xa, y, params = setup(synth.preset(2), 4 * 1024 + 304)
    nb = q.steps_per_epoch
    n = 2 * nb
    tp, ta = schedule(q, n)
    ref = new_context(vfl, q, xp, xa, y, params)
    ref.set_order(True)
    ref.train_steps(0, n, tp, ta)
    ctx = new_context(vfl, q, xp, xa, y, params)
    ctx.set_order(True)
    g = ctx.capture(0, nb, tp, ta)
    drops = np.zeros(n, np.uint8)
    drops[1] = 1
    assert not ctx.update_graph(g, 0, nb, tp, ta, drops)
    ctx.launch_graph(g)
    ctx.train_steps(nb, nb, tp, ta)
    ctx.synchronize()
    np.testing.assert_array_equal(ctx.read_losses(0, n), ref.read_losses(0, n))


@pytest.mark.parametrize("cid", [2, 3])
def test_train_epoch_as_updated_graphs(vfl, cid):
    """In the uniform order vfl_train_epoch replays each epoch as a graph it keeps and updates in place;
    the epochs equal direct enqueue in the overlapping order bit for bit."""
    rows = {2: 4 * 1024 + 304, 3: 2 * 4096 + 288}[cid]
    q, xp, xa, y, params = setup(synth.preset(cid), rows)
    nb = q.steps_per_epoch
    n = 5 * nb
    tp, ta = schedule(q, n)
    ref = new_context(vfl, q, xp, xa, y, params)
    ref.train_steps(0, n, tp, ta)
    ctx = new_context(vfl, q, xp, xa, y, params)
    ctx.set_order(True)
    launches = []
    for e in range(5):
        l0 = ctx.launches
        ctx.train_epoch(e, tp, ta, mean_loss=(e == 4))
        launches.append(ctx.launches - l0)
    ctx.synchronize()
    np.testing.assert_array_equal(ctx.read_losses(0, n), ref.read_losses(0, n))
    for key, (W, b) in ctx.get_params().items():
        np.testing.assert_array_equal(W, ref.get_params()[key][0])
    assert len(set(launches)) == 1, launches      # every epoch's graph runs the same kernels


def test_planner_calibration_tool(vfl):
    """The calibration tool fits Eq. 7-8's constants from a synchronous run on this GPU and Algorithm 2
    picks a candidate of the search space."""
    from paper_2510_12494_gb300 import calibrate as planner
    p = synth.preset(1)
    model, meas = planner.calibrate(vfl, p, [128, 256, 512], steps=6, warmup=2)
    assert sorted(meas) == [128, 256, 512]
    assert all(v > 0 for b in meas for v in meas[b].values())
    assert model["lambda_a"] > 0 and model["lambda_p"] > 0 and model["phi_p"] > 0
    wa, wp, b, o = vfl.plan(vfl.plan_model(**model), (1, 2), (1, 2), [128, 256, 512])
    assert (wa, wp) == (1, 1) and b in (128, 256, 512) and o > 0
