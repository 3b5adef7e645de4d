"""GPU parity: the CUDA path through the C ABI against the oracle, on the same
seeded inputs, step by step (taps, gradients, updated weights) and over whole
epochs.  fp32 presets within 1e-5 per step and 1e-3 on the epoch loss; bf16
presets within 2e-2 per step."""
import numpy as np
import pytest

import oracle
from _parity import EPOCH_LOSS_TOL, TOL, compare_step, new_context, rel_err, run_sequential, schedule, setup

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


# Rows per preset: at least two full batches plus a ragged last batch, with the
# full per-step shapes (batch, layer widths) of each workload.
CASES = {
    1: 4096 - 100,            # 16 steps, last batch 156 rows
    2: 2 * 1024 + 304,        # full batch 1024 and the 304-row tail of the 30000-row set
    3: 2 * 4096 + 288,
    4: 8192 + 576,
    5: 2 * 2048 + 1344,
}


@pytest.mark.parametrize("cid", [1, 2, 3, 4, 5])
def test_step_parity(vfl, cid):
    worst, failures = run_sequential(vfl, cid, CASES[cid])
    print(f"preset {cid}: worst {sorted(worst.items(), key=lambda t: -t[1])[:8]}")
    assert not failures, f"preset {cid}: {failures[:3]}; worst {sorted(worst.items(), key=lambda t: -t[1])[:6]}"


def test_step_parity_worker_streams(vfl):
    """Several worker streams per party: each step's buffers and gradient
    partials live with its worker (k mod W), and every step still matches."""
    worst, failures = run_sequential(vfl, 2, CASES[2], workers=3)
    assert not failures, f"{failures[:3]}; worst {sorted(worst.items(), key=lambda t: -t[1])[:6]}"


@pytest.mark.parametrize("cid", [1, 2])
def test_worker_streams_equal_one_stream(vfl, cid):
    """With W worker streams per party the steps that the schedule's staleness
    allows run concurrently; the result is bit-identical to one stream."""
    import synth
    q, xp, xa, y, params = setup(synth.preset(cid), CASES[cid] if cid == 1 else 4 * 1024 + 304)
    n = 2 * q.steps_per_epoch + 1
    tp, ta = schedule(q, n)
    one = new_context(vfl, q.with_(workers=1), xp, xa, y, params)
    one.train_steps(0, n, tp, ta)
    for w in (2, 3):
        many = new_context(vfl, q.with_(workers=w), xp, xa, y, params)
        many.train_steps(0, n, tp, ta)
        np.testing.assert_array_equal(many.read_losses(0, n), one.read_losses(0, n))
        for key, (W, b) in one.get_params().items():
            W2, b2 = many.get_params()[key]
            np.testing.assert_array_equal(W, W2)
            np.testing.assert_array_equal(b, b2)


@pytest.mark.parametrize("cid", [1, 2])
def test_fp32_epoch_loss_and_dag_equals_sequential(vfl, cid):
    """The whole-DAG enqueue (vfl_train_steps, parties overlapping on their
    streams) gives exactly the result of phase-by-phase execution, and the
    full-size fp32 workloads match the oracle's epoch losses within 1e-3."""
    import synth
    p = synth.preset(cid)
    q, xp, xa, y, params = setup(p)
    n_steps = q.steps_per_epoch * q.epochs
    tp, ta = schedule(q, n_steps)
    dag = new_context(vfl, q, xp, xa, y, params)
    dag.train_steps(0, n_steps, tp, ta)
    losses = dag.read_losses(0, n_steps)
    o = oracle.Oracle(q, xp, xa, y, params)
    ref, _ = o.run(tp, ta, n_steps)
    nb = q.steps_per_epoch
    for e in range(q.epochs):
        got = o.epoch_loss(losses[e * nb:(e + 1) * nb], e * nb)
        want = o.epoch_loss(ref[e * nb:(e + 1) * nb], e * nb)
        assert abs(got - want) <= EPOCH_LOSS_TOL * abs(want), (e, got, want)
    gp = dag.get_params()
    for key, (W, b) in gp.items():
        assert rel_err(W, o.current_params()[key][0]) < 1e-3
    # sequential phase-by-phase run of the first epoch: identical bits
    seq = new_context(vfl, q, xp, xa, y, params)
    for k in range(nb):
        seq.passive_forward(k, int(tp[k]))
        seq.active_step(k, int(ta[k]))
        seq.passive_backward(k)
    dag2 = new_context(vfl, q, xp, xa, y, params)
    dag2.train_steps(0, nb, tp, ta)
    np.testing.assert_array_equal(seq.read_losses(0, nb), dag2.read_losses(0, nb))
    for key, (W, b) in seq.get_params().items():
        W2, b2 = dag2.get_params()[key]
        np.testing.assert_array_equal(W, W2)
        np.testing.assert_array_equal(b, b2)


def test_full_size_in_the_bench_configuration(vfl):
    """The credit-shaped workload at full size as bench.py times it: the whole
    training run (five epochs) as one CUDA graph, captured then replayed, two
    worker streams per party; epoch losses within 1e-3 of the oracle and the
    final weights within 1e-3."""
    import synth
    q, xp, xa, y, params = setup(synth.preset(2))
    nb = q.steps_per_epoch
    n_steps = nb * q.epochs
    tp, ta = schedule(q, n_steps)
    ctx = new_context(vfl, q, xp, xa, y, params)
    ctx.launch_graph(ctx.capture(0, n_steps, tp, ta))
    ctx.synchronize()
    losses = ctx.read_losses(0, n_steps)
    o = oracle.Oracle(q, xp, xa, y, params)
    ref, _ = o.run(tp, ta, n_steps)
    for e in range(q.epochs):
        got = o.epoch_loss(losses[e * nb:(e + 1) * nb], e * nb)
        want = o.epoch_loss(ref[e * nb:(e + 1) * nb], e * nb)
        assert abs(got - want) <= EPOCH_LOSS_TOL * abs(want), (e, got, want)
    for key, (W, b) in ctx.get_params().items():
        assert rel_err(W, o.current_params()[key][0]) < 1e-3
        assert rel_err(b, o.current_params()[key][1]) < 1e-3


@pytest.mark.parametrize("cid", [3, 4, 5])
def test_bf16_free_running_epoch_loss(vfl, cid):
    """Without teacher forcing, a whole bf16 epoch stays within 2e-2 of the
    oracle's per-step losses and weights."""
    import synth
    p = synth.preset(cid)
    q, xp, xa, y, params = setup(p, CASES[cid])
    n = q.steps_per_epoch + 1
    tp, ta = schedule(q, n)
    ctx = new_context(vfl, q, xp, xa, y, params)
    ctx.train_steps(0, n, tp, ta)
    o = oracle.Oracle(q, xp, xa, y, params)
    ref, _ = o.run(tp, ta, n)
    got = ctx.read_losses(0, n)
    assert np.abs(got - ref).max() <= TOL["bf16"] * np.abs(ref).max()
    for key, (W, b) in ctx.get_params().items():
        assert rel_err(W, o.current_params()[key][0]) < TOL["bf16"]


@pytest.mark.parametrize("cid", [2, 5])
def test_checkpoint_restore_is_bit_exact(vfl, cid):
    """Train k1 steps, checkpoint, restore into a fresh context, continue: the
    result equals an uninterrupted run bit for bit."""
    import synth
    p = synth.preset(cid)
    q, xp, xa, y, params = setup(p, CASES[cid] if cid != 2 else 4 * 1024 + 304)
    n1, n2 = 3, 4
    tp, ta = schedule(q, n1 + n2)
    a = new_context(vfl, q, xp, xa, y, params)
    a.train_steps(0, n1, tp, ta)
    ck = a.checkpoint()
    a.train_steps(n1, n2, tp, ta)
    b = new_context(vfl, q, xp, xa, y, params)
    b.restore(ck)
    b.train_steps(n1, n2, tp, ta)
    np.testing.assert_array_equal(a.read_losses(n1, n2), b.read_losses(n1, n2))
    pa, pb = a.get_params(), b.get_params()
    for key in pa:
        np.testing.assert_array_equal(pa[key][0], pb[key][0])
        np.testing.assert_array_equal(pa[key][1], pb[key][1])


@pytest.mark.parametrize("cid", [1, 2])
def test_step_parity_generic_kernels(vfl, cid, monkeypatch):
    """The fp32 presets run the fused one-launch-per-phase kernels by default;
    the per-layer kernels they would otherwise use must match the oracle too."""
    monkeypatch.setenv("VFL_DISABLE_FUSED", "1")
    worst, failures = run_sequential(vfl, cid, CASES[cid])
    assert not failures, f"preset {cid}: {failures[:3]}"


@pytest.mark.parametrize("cid", [3, 5])
def test_step_parity_generic_head(vfl, cid, monkeypatch):
    """The bf16 presets fold g's output layer and the loss into one kernel by
    default; the per-layer GEMMs and loss kernel it replaces must match the
    oracle too."""
    monkeypatch.setenv("VFL_DISABLE_HEAD", "1")
    worst, failures = run_sequential(vfl, cid, CASES[cid], steps=4)
    assert not failures, f"preset {cid}: {failures[:3]}"


@pytest.mark.parametrize("cid", [3, 4, 5])
def test_head_kernel_runs(vfl, cid):
    """The bf16 presets' active step runs the folded output-layer kernel once
    per step, and no separate loss kernel."""
    import synth
    q, xp, xa, y, params = setup(synth.preset(cid), CASES[cid])
    ctx = new_context(vfl, q, xp, xa, y, params)
    tp, ta = schedule(q, 3)
    ctx.profile(True)
    ctx.train_steps(0, 3, tp, ta)
    ctx.profile(False)
    summ = ctx.profile_summary()
    assert summ["head_loss"][0] == 3
    assert summ.get("loss", (0,))[0] == 0


@pytest.mark.parametrize("cid,workers", [(2, 0), (2, 3), (3, 0)])
def test_graph_replay_equals_direct_enqueue(vfl, cid, workers):
    """A captured CUDA graph of a window of steps replays exactly what the
    direct enqueue computes, advances the cursor, and refuses the wrong cursor."""
    import synth
    p = synth.preset(cid)
    if workers:
        p = p.with_(workers=workers)
    q, xp, xa, y, params = setup(p, CASES[cid])
    n = q.steps_per_epoch + 2
    tp, ta = schedule(q, 2 * n)
    direct = new_context(vfl, q, xp, xa, y, params)
    direct.train_steps(0, 2 * n, tp, ta)
    g_ctx = new_context(vfl, q, xp, xa, y, params)
    g0 = g_ctx.capture(0, n, tp, ta)
    assert g_ctx.cursor() == 0                      # capture does not run anything
    g_ctx.launch_graph(g0)
    with pytest.raises(vfl.VflError) as ei:
        g_ctx.launch_graph(g0)                      # cursor is now n, the graph starts at 0
    assert ei.value.status == vfl.VFL_E_STATE
    g1 = g_ctx.capture(n, n, tp, ta)
    g_ctx.launch_graph(g1)
    assert g_ctx.cursor() == 2 * n
    np.testing.assert_array_equal(g_ctx.read_losses(0, 2 * n), direct.read_losses(0, 2 * n))
    for key, (W, b) in direct.get_params().items():
        Wg, bg = g_ctx.get_params()[key]
        np.testing.assert_array_equal(W, Wg)
        np.testing.assert_array_equal(b, bg)


def test_direct_enqueue_after_graph_replay(vfl):
    """Direct phase calls continue exactly after a graph replay."""
    import synth
    q, xp, xa, y, params = setup(synth.preset(2), CASES[2])
    n = q.steps_per_epoch
    tp, ta = schedule(q, 3 * n)
    direct = new_context(vfl, q, xp, xa, y, params)
    direct.train_steps(0, 3 * n, tp, ta)
    mixed = new_context(vfl, q, xp, xa, y, params)
    mixed.launch_graph(mixed.capture(0, n, tp, ta))
    mixed.train_steps(n, n, tp, ta)
    mixed.launch_graph(mixed.capture(2 * n, n, tp, ta))
    np.testing.assert_array_equal(mixed.read_losses(0, 3 * n), direct.read_losses(0, 3 * n))
