"""Shared helpers of the GPU parity tests: run the same seeded inputs through
the C ABI and through the oracle and compare."""
import numpy as np

import oracle
import synth

# Tolerances (relative, infinity norm): fp32 path 1e-5 per step and 1e-3 on
# the epoch loss; bf16 path 2e-2 per step.
TOL = {"fp32": 1e-5, "bf16": 2e-2}
EPOCH_LOSS_TOL = 1e-3


def rel_err(got, ref):
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    if ref.size == 0:
        return 0.0
    return float(np.abs(got - ref).max() / max(np.abs(ref).max(), 1e-30))


def schedule(p, n_steps):
    kind = oracle.SCHED_SYNC if p.schedule == "sync" else oracle.SCHED_SEEDED
    return oracle.make_schedule(p.seed, p.staleness, kind, n_steps)


def setup(p, n_rows=None, rows=None):
    """(preset with n_rows, xp, xa, y, params) for the first n_rows rows of the workload."""
    n_rows = n_rows or p.n_rows
    xp, xa, y = synth.make_dataset(p, rows=(0, n_rows)) if rows is None else rows
    q = p.with_(n_rows=n_rows)
    return q, xp, xa, y, synth.init_params(q)


def new_context(vfl, q, xp, xa, y, params):
    ctx = vfl.Context(q, q.n_rows)
    ctx.load_data(xp, xa, y)
    ctx.set_params(params)
    return ctx


def tensor_err(got, ref, dtype):
    """Error of one tensor against the oracle, in the metric of its dtype.

    fp32: relative infinity norm.  bf16: relative Frobenius norm, reported as
    failing outright (1.0) when more than 1 % of the rows hold an element off by
    more than 2e-2 of the tensor's largest magnitude.  Rows that differ are the
    ones where a pre-activation within rounding distance of zero takes the other
    ReLU branch; bf16 rounding upstream makes that happen in a few rows per
    step, and a whole row's downstream gradient then moves."""
    if dtype == "fp32":
        return rel_err(got, ref)
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    if ref.size == 0:
        return 0.0
    fro = float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-30))
    d = np.abs(got - ref) > TOL["bf16"] * max(np.abs(ref).max(), 1e-30)
    rows_off = d.reshape(d.shape[0], -1).any(axis=1).mean() if d.ndim > 1 else d.mean()
    return fro if rows_off <= 0.01 else 1.0


def compare_step(vfl, ctx, rec, tol, check_grads=True):
    """Per-step taps, gradients and updated parameters against an oracle record."""
    k = rec.k
    dt = ctx.p.dtype
    errs = {
        "zp": tensor_err(ctx.tap(k, vfl.TAP_EMB), rec.zp, dt),
        "dzp": tensor_err(ctx.tap(k, vfl.TAP_GRAD), rec.dzp, dt),
        "logits": tensor_err(ctx.tap(k, vfl.TAP_LOGITS), rec.logits, dt),
        "za": tensor_err(ctx.tap(k, vfl.TAP_ZA), rec.za, dt),
        "dza": tensor_err(ctx.tap(k, vfl.TAP_DZA), rec.dza * (rec.za > 0), dt),
    }
    loss = ctx.read_losses(k, 1)[0]
    errs["loss"] = abs(loss - rec.loss) / max(abs(rec.loss), 1e-30)
    if check_grads:
        g = ctx.get_grads(worker=k % ctx.p.workers)
        out_layer = (2, len(ctx.p.top) - 1)
        for key, (dW, db) in g.items():
            errs[f"dW{key}"] = tensor_err(dW, rec.grads[key][0], dt)
            if key == out_layer and dt == "fp32":
                # db of the output layer is the column sum of d(logits), whose signed per-row terms
                # cancel as the model calibrates: its error is taken against the sum of the terms'
                # magnitudes, the scale that bounds the rounding error of a sum
                scale = float(np.abs(rec.ds).sum(axis=0).max())
                ref = np.asarray(rec.grads[key][1], np.float64)
                errs[f"db{key}"] = float(np.abs(np.asarray(db, np.float64) - ref).max() /
                                         max(np.abs(ref).max(), scale, 1e-30))
            else:
                errs[f"db{key}"] = tensor_err(db, rec.grads[key][1], dt)
    # the parameter-server mode: the replica the step updated (the oracle records the same one)
    params = ctx.get_replica(k % ctx.p.workers) if ctx.ps else ctx.get_params()
    for key, (W, b) in params.items():
        errs[f"W{key}"] = tensor_err(W, rec.params[key][0], dt)
        errs[f"b{key}"] = tensor_err(b, rec.params[key][1], dt)
    bad = {name: e for name, e in errs.items() if not e <= tol}
    return errs, bad


def oracle_version(o, v):
    """{(party, layer): (W, b)} of the oracle's stored weight version v."""
    out = {}
    for l, (W, b) in enumerate(o.versions_p[v]):
        out[(0, l)] = (W, b)
    A, T = o.versions_a[v]
    for l, (W, b) in enumerate(A):
        out[(1, l)] = (W, b)
    for l, (W, b) in enumerate(T):
        out[(2, l)] = (W, b)
    return out


def force_gpu_state(ctx, o, S):
    """Put the GPU context into the oracle's state before step o.k: cursor and
    every stored weight version, or every replica in the parameter-server mode
    (oracle -> GPU only)."""
    k = o.k
    ctx.set_cursor(k)
    ctx.set_drops(o.k - o.n_done)
    if ctx.ps:
        for w in range(ctx.p.workers):
            ctx.set_replica(w, o.replica_params(w))
        return
    for v in range(max(0, k - S), k + 1):
        ctx.set_version(v, oracle_version(o, v))


def compare_dropped(ctx, rec, tol):
    """A dropped step: NaN loss, and the parameters (or the step's replica) the oracle kept."""
    errs = {"loss_nan": 0.0 if np.isnan(ctx.read_losses(rec.k, 1)[0]) else 1.0}
    params = ctx.get_replica(rec.k % ctx.p.workers) if ctx.ps else ctx.get_params()
    for key, (W, b) in params.items():
        errs[f"W{key}"] = tensor_err(W, rec.params[key][0], ctx.p.dtype)
        errs[f"b{key}"] = tensor_err(b, rec.params[key][1], ctx.p.dtype)
    return errs, {name: e for name, e in errs.items() if not e <= tol}


def run_sequential(vfl, cid, n_rows, steps=None, teacher_forced=None, workers=None, drops=None, publish_dropped=True):
    """Step-by-step comparison.  bf16 presets are teacher-forced: before each
    step the GPU takes the oracle's weight versions, so one step's error is
    measured without the drift of earlier roundings (a bf16 weight copy that
    rounds the other way moves later ReLU masks).  `drops` marks steps whose
    subscriber gives up (vfl_drop_step); with publish_dropped False their
    publisher never runs."""
    p = synth.preset(cid) if isinstance(cid, int) else cid
    if workers:
        p = p.with_(workers=workers)
    q, xp, xa, y, params = setup(p, n_rows)
    nb = -(-n_rows // q.batch)
    steps = steps or nb + 2                      # one epoch and two steps of the next
    if teacher_forced is None:
        teacher_forced = q.dtype == "bf16"
    tp, ta = schedule(q, steps)
    ctx = new_context(vfl, q, xp, xa, y, params)
    o = oracle.Oracle(q, xp, xa, y, params, dp_seed=q.seed)
    worst = {}
    failures = []
    for k in range(steps):
        if teacher_forced and k > 0:
            force_gpu_state(ctx, o, q.staleness)
        dropped = drops is not None and bool(drops[k])
        rec = o.step(int(tp[k]), int(ta[k]), record=True, drop=dropped)
        if dropped:
            if publish_dropped:
                ctx.passive_forward(k, int(tp[k]))
            ctx.drop_step(k)
            ctx.passive_backward(k)
            errs, bad = compare_dropped(ctx, rec, TOL[q.dtype])
        else:
            ctx.passive_forward(k, int(tp[k]))
            ctx.active_step(k, int(ta[k]))
            ctx.passive_backward(k)
            errs, bad = compare_step(vfl, ctx, rec, TOL[q.dtype])
        for name, e in errs.items():
            worst[name] = max(worst.get(name, 0.0), e)
        if bad:
            failures.append((k, bad))
    return worst, failures
