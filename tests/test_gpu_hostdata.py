"""Host-resident data (vfl_bind_host_data): every step copies its own rows from
pinned host memory into the staging ring and its loss back out.  Training this
way is bit-identical to training on the device-resident dataset, directly
enqueued or replayed from CUDA graphs, across epochs (ring slots reused) and
with several worker streams."""
import numpy as np
import pytest

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


def host_context(vfl, q, xp, xa, y, params, cap, bf16_host=False):
    """A context that never loads the dataset: its resident copy stays zero.  With
    bf16_host the features are bound as bf16 (vfl_bind_host_data_bf16)."""
    import torch
    ctx = vfl.Context(q, q.n_rows)
    ctx.set_params(params)
    pins = [torch.from_numpy(a).pin_memory() for a in (xp, xa, y)]
    if bf16_host:
        pins[0] = pins[0].to(torch.bfloat16).pin_memory()
        pins[1] = pins[1].to(torch.bfloat16).pin_memory()
    loss = torch.full((cap,), float("nan"), dtype=torch.float32).pin_memory()
    ctx.bind_host_data(*pins, loss_out=loss)
    return ctx, loss


def assert_same_state(a, b):
    for key, (W, bias) in a.get_params().items():
        W2, b2 = b.get_params()[key]
        np.testing.assert_array_equal(W, W2)
        np.testing.assert_array_equal(bias, b2)


@pytest.mark.parametrize("cid,workers", [(1, 0), (2, 0), (2, 3), (3, 0)])
def test_host_data_equals_resident(vfl, cid, workers):
    p = synth.preset(cid)
    if workers:
        p = p.with_(workers=workers)
    rows = {1: 4096 - 100, 2: 4 * 1024 + 304, 3: 2 * 4096 + 288}[cid]
    q, xp, xa, y, params = setup(p, rows)
    n = 2 * q.steps_per_epoch + 3
    tp, ta = schedule(q, n)
    ref = new_context(vfl, q, xp, xa, y, params)
    ref.train_steps(0, n, tp, ta)
    ctx, loss = host_context(vfl, q, xp, xa, y, params, cap=n)
    ctx.train_steps(0, n, tp, ta)
    ctx.synchronize()
    np.testing.assert_array_equal(ctx.read_losses(0, n), ref.read_losses(0, n))
    np.testing.assert_array_equal(loss.numpy(), ref.read_losses(0, n))
    assert_same_state(ctx, ref)


@pytest.mark.parametrize("cid", [2, 3])
def test_host_data_graph_replay(vfl, cid):
    """Graphs captured under the binding carry the copies: replaying windows
    gives the same losses and weights as direct enqueue on resident data."""
    p = synth.preset(cid)
    rows = {2: 4 * 1024 + 304, 3: 2 * 4096 + 288}[cid]
    q, xp, xa, y, params = setup(p, rows)
    nb = q.steps_per_epoch
    n = 2 * nb + 3
    tp, ta = schedule(q, n)
    ref = new_context(vfl, q, xp, xa, y, params)
    ref.train_steps(0, n, tp, ta)
    ctx, loss = host_context(vfl, q, xp, xa, y, params, cap=n)
    ctx.train_steps(0, 2, tp, ta)                  # a direct prefix, then graphs
    k = 2
    while k < n:
        m = min(nb, n - k)
        g = ctx.capture(k, m, tp, ta)
        ctx.launch_graph(g)
        k += m
    ctx.synchronize()
    np.testing.assert_array_equal(loss.numpy(), ref.read_losses(0, n))
    assert_same_state(ctx, ref)


def test_unbind_returns_to_resident_data(vfl):
    q, xp, xa, y, params = setup(synth.preset(2), 2 * 1024 + 304)
    n = 7
    tp, ta = schedule(q, 2 * n)
    ref = new_context(vfl, q, xp, xa, y, params)
    ref.train_steps(0, 2 * n, tp, ta)
    ctx, loss = host_context(vfl, q, xp, xa, y, params, cap=n)
    ctx.train_steps(0, n, tp, ta)
    ctx.bind_host_data(None, None, None)
    ctx.load_data(xp, xa, y)
    ctx.train_steps(n, n, tp, ta)
    np.testing.assert_array_equal(ctx.read_losses(0, 2 * n), ref.read_losses(0, 2 * n))
    assert_same_state(ctx, ref)


def test_fetch_loss_copies_each_step_loss(vfl):
    """vfl_fetch_loss: an asynchronous copy of one step's mean loss into pinned
    host memory, valid once the step's active worker stream passes it."""
    import torch
    q, xp, xa, y, params = setup(synth.preset(2), 2 * 1024 + 304)
    n = 6
    tp, ta = schedule(q, n)
    ctx = new_context(vfl, q, xp, xa, y, params)
    out = torch.full((n,), float("nan"), dtype=torch.float32).pin_memory()
    ctx.train_steps(0, n, tp, ta)
    for k in range(n):
        ctx.fetch_loss(k, out.data_ptr() + 4 * k)
    ctx.synchronize()
    np.testing.assert_array_equal(out.numpy(), ctx.read_losses(0, n))


def test_host_data_uniform_order_graph_updates(vfl):
    """The end-to-end path: host-resident rows, the uniform dependency order, one graph per epoch updated
    in place -- the same losses and weights as direct enqueue on resident data."""
    p = synth.preset(2)
    rows = 4 * 1024 + 304
    q, xp, xa, y, params = setup(p, rows)
    nb = q.steps_per_epoch
    n = 4 * nb
    tp, ta = schedule(q, n)
    ref = new_context(vfl, q, xp, xa, y, params)
    ref.train_steps(0, n, tp, ta)
    ctx, loss = host_context(vfl, q, xp, xa, y, params, cap=n)
    ctx.set_order(True)
    graphs = {}
    for e in range(4):
        w = (e * nb) % q.workers
        if w not in graphs:
            graphs[w] = ctx.capture(e * nb, nb, tp, ta)
        else:
            assert ctx.update_graph(graphs[w], e * nb, nb, tp, ta)
        ctx.launch_graph(graphs[w])
    ctx.synchronize()
    np.testing.assert_array_equal(loss.numpy(), ref.read_losses(0, n))
    assert_same_state(ctx, ref)


@pytest.mark.parametrize("cid,workers", [(3, 0), (3, 3), (4, 0)])
def test_bf16_host_data_equals_resident(vfl, cid, workers):
    """bf16 host arrays (round to nearest even of the fp32 features, as the
    resident load rounds them) reach the staging ring by the copy engines;
    training on them is bit-identical to training on the resident dataset,
    directly enqueued and replayed from graphs."""
    p = synth.preset(cid)
    if workers:
        p = p.with_(workers=workers)
    rows = {3: 2 * 4096 + 288, 4: 2 * 8192 + 520}[cid]
    q, xp, xa, y, params = setup(p, rows)
    nb = q.steps_per_epoch
    n = 2 * nb + 1
    tp, ta = schedule(q, n)
    ref = new_context(vfl, q, xp, xa, y, params)
    ref.train_steps(0, n, tp, ta)
    ctx, loss = host_context(vfl, q, xp, xa, y, params, cap=n, bf16_host=True)
    ctx.train_steps(0, nb, tp, ta)
    ctx.launch_graph(ctx.capture(nb, n - nb, tp, ta))
    ctx.synchronize()
    np.testing.assert_array_equal(ctx.read_losses(0, n), ref.read_losses(0, n))
    np.testing.assert_array_equal(loss.numpy(), ref.read_losses(0, n))
    assert_same_state(ctx, ref)


def test_bf16_host_data_needs_bf16_context(vfl):
    import torch
    q, xp, xa, y, params = setup(synth.preset(1), 1024)
    ctx = vfl.Context(q, q.n_rows)
    pins = [torch.from_numpy(a).pin_memory() for a in (xp, xa, y)]
    with pytest.raises(vfl.VflError):
        ctx.bind_host_data(pins[0].to(torch.bfloat16).pin_memory(), pins[1].to(torch.bfloat16).pin_memory(), pins[2])
    ctx.close()


def bits_context(vfl, q, xp, xa, y, params, cap):
    """A context bound to bit-packed copies of binary features (vfl_bind_host_data_bits)."""
    import torch
    ctx = vfl.Context(q, q.n_rows)
    ctx.set_params(params)
    pins = [torch.from_numpy(a).pin_memory() for a in (vfl.pack_bits(xp), vfl.pack_bits(xa), y)]
    loss = torch.full((cap,), float("nan"), dtype=torch.float32).pin_memory()
    ctx.bind_host_bits(*pins, loss_out=loss)
    return ctx, loss


@pytest.mark.parametrize("cid,workers,binarize", [(4, 0, False), (4, 3, False), (1, 0, True)])
def test_bits_host_data_equals_resident(vfl, cid, workers, binarize):
    """Binary features bit-packed on the host (wide-dp's own Bernoulli columns, d = 1000 = 31 words and a
    partial one; and the credit-shaped fp32 context on 0 / 1 features, d = 12 / 11 in one partial word):
    the staging kernel's 0 / 1 values are exact, so training is bit-identical to training on the resident
    dataset, directly enqueued and replayed from graphs."""
    p = synth.preset(cid)
    if workers:
        p = p.with_(workers=workers)
    rows = {1: 4096 - 100, 4: 2 * 8192 + 520}[cid]
    q, xp, xa, y, params = setup(p, rows)
    if binarize:
        xp = (xp > 0).astype(np.float32)
        xa = (xa > 0).astype(np.float32)
    nb = q.steps_per_epoch
    n = 2 * nb + 1
    tp, ta = schedule(q, n)
    ref = new_context(vfl, q, xp, xa, y, params)
    ref.train_steps(0, n, tp, ta)
    ctx, loss = bits_context(vfl, q, xp, xa, y, params, cap=n)
    ctx.train_steps(0, nb, tp, ta)
    ctx.launch_graph(ctx.capture(nb, n - nb, tp, ta))
    ctx.synchronize()
    np.testing.assert_array_equal(ctx.read_losses(0, n), ref.read_losses(0, n))
    np.testing.assert_array_equal(loss.numpy(), ref.read_losses(0, n))
    assert_same_state(ctx, ref)
