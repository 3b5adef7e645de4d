"""GPU parity of the intra-party semi-asynchronous parameter server (Sec. 4.1,
Eq. 5): per-worker replicas updated by their own steps and averaged after the
epochs Eq. 5 selects, against the oracle on the same seeded inputs, step by
step (every tap, gradient and the updated replica); then the concurrent
enqueue (all workers' chains in flight at once, directly and from CUDA graphs)
against the sequential one, bit for bit, and checkpoint / restore."""
import numpy as np
import pytest

import oracle
import synth
from _parity import TOL, new_context, rel_err, run_sequential, schedule, setup

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


def ps_preset(cid, workers, dt0, rows, **kw):
    return synth.preset(cid).with_(n_rows=rows, workers=workers, ps_dt0=dt0, staleness=0, schedule="sync", **kw)


def assert_parity(vfl, q, steps):
    worst, failures = run_sequential(vfl, q, q.n_rows, steps=steps)
    assert not failures, f"{q.name}: {failures[:3]}; worst {sorted(worst.items(), key=lambda t: -t[1])[:6]}"
    return worst


def kernels_used(vfl, q, steps):
    q2, xp, xa, y, params = setup(q, q.n_rows)
    ctx = new_context(vfl, q2, xp, xa, y, params)
    tp, ta = schedule(q2, steps)
    ctx.profile(True)
    ctx.train_steps(0, steps, tp, ta)
    ctx.profile(False)
    return {k: v[0] for k, v in ctx.profile_summary().items()}


@pytest.mark.parametrize("workers,dt0,rows", [
    (2, 4, 3 * 256 + 37),     # 4 steps per epoch: averaged after epochs 1, 2 and 4, not 3
    (3, 1, 3 * 256 + 37),     # W does not divide the epoch; averaged after every epoch
    (3, 2, 256 + 37),         # 2 steps per epoch < W: the first average meets an untouched replica
])
@pytest.mark.parametrize("path", ["fused", "generic"])
def test_ps_fp32(vfl, workers, dt0, rows, path, monkeypatch):
    if path == "generic":
        monkeypatch.setenv("VFL_DISABLE_FUSED", "1")
    q = ps_preset(1, workers, dt0, rows)
    nb = -(-rows // q.batch)
    steps = 4 * nb + 1
    used = kernels_used(vfl, q, steps)
    assert ("fused_passive_fwd" in used) == (path == "fused"), used
    n_avg = sum(1 for e in range(steps) if (e + 1) % nb == 0 and oracle.ps_aggregates_after((e + 1) // nb, dt0))
    assert used.get("ps_average", 0) == 2 * n_avg, used      # one launch per party per average
    assert_parity(vfl, q, steps)


def test_ps_bf16(vfl):
    """bf16 (tensor-core kernels), two workers, teacher-forced replicas."""
    q = ps_preset(3, 2, 1, 2 * 4096 + 288)
    assert_parity(vfl, q, steps=7)


def train(vfl, q, steps, mode):
    q2, xp, xa, y, params = setup(q, q.n_rows)
    ctx = new_context(vfl, q2, xp, xa, y, params)
    tp, ta = schedule(q2, steps)
    if mode == "phases":                     # one step at a time, each step's phases in order
        for k in range(steps):
            ctx.passive_forward(k, 0)
            ctx.active_step(k, 0)
            ctx.passive_backward(k)
    elif mode == "train_steps":
        ctx.train_steps(0, steps, tp, ta)
    else:                                    # graphs of one epoch each after a direct step
        ctx.train_steps(0, 1, tp, ta)
        k = 1
        while k < steps:
            m = min(ctx.nb, steps - k)
            ctx.launch_graph(ctx.capture(k, m, tp, ta))
            k += m
    ctx.synchronize()
    return ctx


@pytest.mark.parametrize("cid,workers,dt0", [(1, 4, 2), (2, 3, 4), (3, 2, 1)])
def test_concurrent_workers_equal_sequential(vfl, cid, workers, dt0):
    rows = {1: 5 * 256 + 37, 2: 5 * 1024 + 304, 3: 3 * 4096 + 288}[cid]
    q = ps_preset(cid, workers, dt0, rows)
    steps = 3 * (-(-rows // q.batch)) + 2
    ref = train(vfl, q, steps, "phases")
    want = ref.read_losses(0, steps)
    for mode in ("train_steps", "graphs"):
        ctx = train(vfl, q, steps, mode)
        np.testing.assert_array_equal(ctx.read_losses(0, steps), want, err_msg=mode)
        for w in range(workers):
            for key, (W, b) in ctx.get_replica(w).items():
                W2, b2 = ref.get_replica(w)[key]
                np.testing.assert_array_equal(W, W2, err_msg=f"{mode} replica {w} {key}")
                np.testing.assert_array_equal(b, b2, err_msg=f"{mode} replica {w} {key}")


def test_ps_checkpoint_restore(vfl):
    q = ps_preset(1, 3, 2, 3 * 256 + 37)
    q2, xp, xa, y, params = setup(q, q.n_rows)
    n = 4 * 4 + 1
    tp, ta = schedule(q2, 2 * n)
    a = new_context(vfl, q2, xp, xa, y, params)
    a.train_steps(0, n, tp, ta)
    ck = a.checkpoint()
    assert ck[0] == n and sorted(ck[1]) == [0, 1, 2]
    a.train_steps(n, n, tp, ta)
    b = new_context(vfl, q2, xp, xa, y, params)
    b.restore(ck)
    b.train_steps(n, n, tp, ta)
    np.testing.assert_array_equal(b.read_losses(n, n), a.read_losses(n, n))
    for w in range(3):
        for key, (W, bias) in a.get_replica(w).items():
            np.testing.assert_array_equal(b.get_replica(w)[key][0], W)
            np.testing.assert_array_equal(b.get_replica(w)[key][1], bias)


def test_ps_api_guards(vfl):
    q = ps_preset(1, 2, 2, 3 * 256 + 37)
    q2, xp, xa, y, params = setup(q, q.n_rows)
    ctx = new_context(vfl, q2, xp, xa, y, params)
    with pytest.raises(vfl.VflError):
        ctx.get_version(0)
    ctx.passive_forward(0, 0)
    ctx.passive_forward(1, 0)            # worker 1's replica needs no earlier update
    with pytest.raises(vfl.VflError):
        ctx.passive_forward(2, 0)        # worker 0's replica: step 0's update is not enqueued
    ctx.active_step(0, 0)
    ctx.passive_backward(0)
    ctx.passive_forward(2, 0)
    ctx.synchronize()
    plain = new_context(vfl, *setup(synth.preset(1).with_(n_rows=600), 600))
    with pytest.raises(vfl.VflError):
        plain.get_replica(0)


def test_ps_average_matches_the_replica_mean(vfl):
    """Right after an averaging step every replica equals the mean of the
    oracle's pre-average replicas (the result the oracle's _ps_average pins)."""
    q = ps_preset(1, 3, 1, 2 * 256)
    q2, xp, xa, y, params = setup(q, q.n_rows)
    ctx = new_context(vfl, q2, xp, xa, y, params)
    o = oracle.Oracle(q2, xp, xa, y, params, dp_seed=q2.seed)
    tp, ta = schedule(q2, 4)
    o.run(tp, ta, 4)                     # epochs 1 and 2 end at steps 1 and 3: both averaged
    ctx.train_steps(0, 4, tp, ta)
    r = [ctx.get_replica(w) for w in range(3)]
    for key in r[0]:
        for w in (1, 2):
            np.testing.assert_array_equal(r[w][key][0], r[0][key][0])
            np.testing.assert_array_equal(r[w][key][1], r[0][key][1])
        assert rel_err(r[0][key][0], o.replica_params(0)[key][0]) < TOL["fp32"]
        assert rel_err(r[0][key][1], o.replica_params(0)[key][1]) < TOL["fp32"]


def test_ps_with_embedding_dp(vfl):
    """The parameter server with DP on the published embedding (fused kernels), against the oracle."""
    q = ps_preset(1, 2, 1, 3 * 256 + 37, dp_clip=1.0, dp_sigma=0.5, dp_target="emb")
    assert_parity(vfl, q, steps=9)


def test_ps_host_data_equals_resident(vfl):
    """Replicas trained from pinned host rows equal the device-resident run bit for bit."""
    import torch
    q = ps_preset(2, 3, 2, 4 * 1024 + 304)
    steps = 3 * 5 + 2
    ref = train(vfl, q, steps, "train_steps")
    q2, xp, xa, y, params = setup(q, q.n_rows)
    tp, ta = schedule(q2, steps)
    ctx = vfl.Context(q2, q2.n_rows)
    ctx.set_params(params)
    pins = [torch.from_numpy(a).pin_memory() for a in (xp, xa, y)]
    loss = torch.full((steps,), float("nan"), dtype=torch.float32).pin_memory()
    ctx.bind_host_data(*pins, loss_out=loss)
    ctx.train_steps(0, steps, tp, ta)
    ctx.synchronize()
    np.testing.assert_array_equal(loss.numpy(), ref.read_losses(0, steps))
    for w in range(3):
        for key, (W, b) in ctx.get_replica(w).items():
            np.testing.assert_array_equal(W, ref.get_replica(w)[key][0])
            np.testing.assert_array_equal(b, ref.get_replica(w)[key][1])


def test_ps_at_the_worker_limit(vfl):
    """16 workers (one version slot and one replica each, the library's limit), averaged every epoch."""
    q = ps_preset(1, 16, 1, 20 * 64 + 9, batch=64)
    assert_parity(vfl, q, steps=2 * 21 + 3)
