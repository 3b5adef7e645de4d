"""GPU parity of the waiting-deadline / buffer-overflow drops (Sec. 4.1,
Algorithm 1's subscriber branch): a dropped step trains nothing, records a NaN
loss, carries both parties' versions forward and hands its batch to the next
step.  Against the oracle step by step (with and without the dropped step's
publish, with staleness, in the parameter-server mode, bf16), the whole-DAG
enqueue and graph replay against one step at a time bit for bit, host-resident
data, checkpoint / restore, the enqueue guards, and a deadline made on the host
(the publisher never enqueued, the bounded device wait giving up)."""
import numpy as np
import pytest

import oracle
import synth
from _parity import new_context, run_sequential, schedule, setup

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


def assert_parity(vfl, q, steps, drops, **kw):
    assert 0 < drops[:steps].sum() < steps
    worst, failures = run_sequential(vfl, q, q.n_rows, steps=steps, drops=drops, **kw)
    assert not failures, f"{q.name}: {failures[:3]}; worst {sorted(worst.items(), key=lambda t: -t[1])[:6]}"


@pytest.mark.parametrize("path", ["fused", "generic"])
@pytest.mark.parametrize("publish", [True, False])
def test_drops_fp32(vfl, path, publish, monkeypatch):
    """S = 2 seeded, 3 worker streams, a ragged last batch, one drop in five."""
    if path == "generic":
        monkeypatch.setenv("VFL_DISABLE_FUSED", "1")
    q = synth.preset(1).with_(n_rows=3 * 256 + 37, staleness=2, schedule="seeded", workers=3)
    steps = 14
    drops = oracle.make_drops(11, 0.2, steps)
    assert_parity(vfl, q, steps, drops, publish_dropped=publish)


def test_drops_consecutive_and_first(vfl):
    q = synth.preset(2).with_(n_rows=3 * 1024 + 304)
    drops = np.zeros(12, np.uint8)
    drops[[0, 4, 5, 6, 11]] = 1
    assert_parity(vfl, q, 12, drops)


def test_drops_parameter_server(vfl):
    """Epochs count trained batches: drops move the averaging steps."""
    q = synth.preset(1).with_(n_rows=3 * 256 + 37, staleness=0, schedule="sync", workers=3, ps_dt0=2)
    drops = np.zeros(19, np.uint8)
    drops[[2, 3, 9, 15]] = 1
    assert_parity(vfl, q, 19, drops)


def test_drops_bf16(vfl):
    q = synth.preset(3).with_(n_rows=2 * 4096 + 288)
    drops = np.zeros(6, np.uint8)
    drops[[1, 3]] = 1
    assert_parity(vfl, q, 6, drops)


def run_all(vfl, q, steps, drops, mode, host=False):
    import torch
    q2, xp, xa, y, params = setup(q, q.n_rows)
    tp, ta = schedule(q2, steps)
    if host:
        ctx = vfl.Context(q2, q2.n_rows)
        ctx.set_params(params)
        pins = [torch.from_numpy(a).pin_memory() for a in (xp, xa, y)]
        loss = torch.full((steps,), 0.0, dtype=torch.float32).pin_memory()
        ctx.bind_host_data(*pins, loss_out=loss)
    else:
        ctx = new_context(vfl, q2, xp, xa, y, params)
        loss = None
    if mode == "phases":
        for k in range(steps):
            ctx.passive_forward(k, int(tp[k]))
            if drops[k]:
                ctx.drop_step(k)
            else:
                ctx.active_step(k, int(ta[k]))
            ctx.passive_backward(k)
    elif mode == "train_steps":
        ctx.train_steps(0, steps, tp, ta, drops)
    else:
        ctx.train_steps(0, 2, tp, ta, drops)
        k = 2
        while k < steps:
            m = min(ctx.nb, steps - k)
            ctx.launch_graph(ctx.capture(k, m, tp, ta, drops))
            k += m
    ctx.synchronize()
    return ctx, loss


@pytest.mark.parametrize("cid,workers,ps", [(1, 2, 0), (2, 2, 0), (2, 3, 4), (3, 1, 0)])
def test_concurrent_enqueue_with_drops_equals_sequential(vfl, cid, workers, ps):
    rows = {1: 3 * 256 + 37, 2: 4 * 1024 + 304, 3: 2 * 4096 + 288}[cid]
    q = synth.preset(cid).with_(n_rows=rows, workers=workers)
    if ps:
        q = q.with_(ps_dt0=ps, staleness=0, schedule="sync")
    steps = 3 * (-(-rows // q.batch)) + 2
    drops = oracle.make_drops(cid, 0.25, steps)
    ref, _ = run_all(vfl, q, steps, drops, "phases")
    want = ref.read_losses(0, steps)
    assert np.isnan(want[drops == 1]).all() and not np.isnan(want[drops == 0]).any()
    get = (lambda c: c.get_replica(0)) if ps else (lambda c: c.get_params())
    for mode in ("train_steps", "graphs"):
        ctx, _ = run_all(vfl, q, steps, drops, mode)
        np.testing.assert_array_equal(ctx.read_losses(0, steps), want, err_msg=mode)
        for key, (W, b) in get(ctx).items():
            np.testing.assert_array_equal(W, get(ref)[key][0], err_msg=f"{mode} {key}")
            np.testing.assert_array_equal(b, get(ref)[key][1], err_msg=f"{mode} {key}")
    ctx, loss = run_all(vfl, q, steps, drops, "train_steps", host=True)
    np.testing.assert_array_equal(loss.numpy(), want)
    for key, (W, b) in get(ctx).items():
        np.testing.assert_array_equal(W, get(ref)[key][0], err_msg=f"host data {key}")


def test_checkpoint_restore_keeps_the_batch_sequence(vfl):
    q = synth.preset(2).with_(n_rows=3 * 1024 + 304)
    q2, xp, xa, y, params = setup(q, q.n_rows)
    n = 9
    tp, ta = schedule(q2, 2 * n)
    drops = np.zeros(2 * n, np.uint8)
    drops[[2, 5, 6, 12]] = 1
    a = new_context(vfl, q2, xp, xa, y, params)
    a.train_steps(0, n, tp, ta, drops)
    ck = a.checkpoint()
    assert ck[3] == 3
    a.train_steps(n, n, tp, ta, drops)
    b = new_context(vfl, q2, xp, xa, y, params)
    b.restore(ck)
    b.train_steps(n, n, tp, ta, drops)
    np.testing.assert_array_equal(b.read_losses(n, n), a.read_losses(n, n))
    for key, (W, bias) in a.get_params().items():
        np.testing.assert_array_equal(b.get_params()[key][0], W)


def test_drop_guards(vfl):
    """A drop must be decided before the next step is published (whose batch it
    changes); a graph replays only from the drop count it was captured at."""
    q = synth.preset(2).with_(n_rows=3 * 1024 + 304)       # S = 2
    q2, xp, xa, y, params = setup(q, q.n_rows)
    tp, ta = schedule(q2, 12)
    ctx = new_context(vfl, q2, xp, xa, y, params)
    ctx.passive_forward(0, 0)
    ctx.active_step(0, 0)
    ctx.passive_backward(0)
    ctx.passive_forward(1, 0)
    ctx.passive_forward(2, 1)            # version 1 exists: step 2 publishes ahead of step 1's subscriber
    with pytest.raises(vfl.VflError):
        ctx.drop_step(1)
    ctx.active_step(1, 0)
    ctx.active_step(2, 0)
    ctx.passive_backward(1)
    ctx.passive_backward(2)
    zero = np.zeros(12, np.int32)
    g = ctx.capture(3, 4, zero, zero)
    ctx.passive_forward(3, 0)
    ctx.drop_step(3)
    ctx.passive_backward(3)
    ctx.synchronize()
    assert ctx.drops() == 1
    ctx.set_cursor(3)                    # back to step 3, but with one drop counted
    ctx.set_drops(1)
    with pytest.raises(vfl.VflError):
        ctx.launch_graph(g)
    ctx.set_drops(0)
    ctx.launch_graph(g)
    ctx.synchronize()


def test_deadline_from_a_missing_publish(vfl):
    """The publisher of step 3 is never enqueued: the subscriber's bounded device
    wait gives up (VFL_E_TIMEOUT, context usable), the step is dropped, and
    training continues as the oracle's run with step 3 dropped."""
    q = synth.preset(2).with_(n_rows=3 * 1024 + 304, staleness=0, schedule="sync")
    q2, xp, xa, y, params = setup(q, q.n_rows)
    n = 8
    tp, ta = schedule(q2, n)
    drops = np.zeros(n, np.uint8)
    drops[3] = 1
    ctx = new_context(vfl, q2, xp, xa, y, params)
    ctx.train_steps(0, 3, tp, ta)
    with pytest.raises(vfl.VflError) as e:
        ctx.wait_channel(0, 3, 20000)
    assert e.value.status == vfl.VFL_E_TIMEOUT
    ctx.drop_step(3)
    ctx.passive_backward(3)
    ctx.train_steps(4, n - 4, tp, ta)
    o = oracle.Oracle(q2, xp, xa, y, params, dp_seed=q2.seed)
    ref = o.run(tp, ta, n, drops=drops)[0]
    got = ctx.read_losses(0, n)
    assert np.isnan(got[3]) and np.isnan(ref[3])
    keep = drops == 0
    assert np.abs(got[keep] - ref[keep]).max() / np.abs(ref[keep]).max() < 1e-5


@pytest.mark.parametrize("target", ["grad", "emb"])
def test_drops_with_dp(vfl, target):
    """Drops with either DP mechanism: the noise of a step is keyed by its step index, so the draws of the
    steps after a drop are the oracle's."""
    q = synth.preset(1).with_(n_rows=3 * 256 + 37, staleness=1, schedule="seeded", dp_clip=1.0, dp_sigma=0.7,
                              dp_target=target)
    drops = np.zeros(10, np.uint8)
    drops[[2, 7]] = 1
    assert_parity(vfl, q, 10, drops)


def test_drops_at_the_largest_staleness_bound(vfl):
    """S = 15 (16 version slots) with three worker streams and a drop in four."""
    q = synth.preset(1).with_(n_rows=5 * 256 + 37, staleness=15, schedule="seeded", workers=3)
    drops = oracle.make_drops(5, 0.25, 30)
    assert_parity(vfl, q, 30, drops)
