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


def tensor_err(got, ref, dtype, excused=None):
    """Error of one tensor against the oracle: the relative infinity norm (largest
    elementwise error over the tensor's largest magnitude).  For a bf16 tensor
    whose first axis is the step's rows, rows in `excused` (rows where a ReLU
    unit took the other branch on the GPU, see flipped_rows) are left out of
    the maximum; every other row is held to the same norm."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    if ref.size == 0:
        return 0.0
    scale = max(np.abs(ref).max(), 1e-30)
    d = np.abs(got - ref)
    if dtype == "bf16" and excused is not None and d.ndim >= 1 and d.shape[0] == len(excused):
        d = d[~excused]
        if d.size == 0:
            return 0.0
    return float(d.max() / scale)


# ---------------------------------------------------------------------------
# bf16 branch flips.  The GPU rounds each stored activation to bf16 after an fp32
# accumulation, the oracle after an fp64 one; where the two land on different
# sides of a bf16 rounding boundary, the next layer's pre-activations move by
# about one bf16 unit of that input's term, and a unit whose pre-activation lies
# that close to zero can take the other ReLU branch.  That changes its row (and
# only its row) downstream.  Such rows are found explicitly: the GPU's stored
# activation masks (vfl_tap of every hidden layer) against the oracle's, and
# every flipped unit must lie within one bf16 unit of its terms' magnitude of
# zero in the oracle's pre-activation, else the step fails.
# ---------------------------------------------------------------------------
FLIP_BAND = 2.0 ** -7          # one bf16 unit (relative) of the summed |w_ij h_j|
FLIP_ROWS_MAX = 0.10           # at most 10 % of a step's rows may be excused


def oracle_forward(o, tau_p, tau_a):
    """Pre-activations and stored activations {(party, layer): (pre, mag, h)} of
    every Linear+ReLU layer of the oracle's next step (party 0 passive, 1 active,
    2 the top's hidden layers), computed from the oracle's state before the step
    as its own step computes them; mag = sum_j |w_ij h_j| + |b_i|."""
    c = o.cfg
    k = o.k
    _, r0, r1 = o.batch_rows()
    if o.ps:
        w = k % c.workers
        Pm, Am, Tm = o.replicas[w]
    else:
        Pm = o.versions_p[k - tau_p]
        Am, Tm = o.versions_a[k - tau_a]
    out = {}
    weights = {}

    def chain(party, layers, x, relu_last):
        h = x
        for i, (W, b) in enumerate(o._compute(layers)):
            weights[(party, i)] = (W, h)
            pre = h @ W.T + b
            if i == len(layers) - 1 and not relu_last:
                return pre
            mag = np.abs(h) @ np.abs(W).T + np.abs(b)
            h = oracle.bf16_round(np.maximum(pre, 0.0)) if o.dtype == "bf16" else np.maximum(pre, 0.0)
            out[(party, i)] = (pre, mag, h)
        return h

    zp = chain(0, Pm, o.xp_c[r0:r1], True)
    za = chain(1, Am, o.xa_c[r0:r1], True)
    if c.dp_clip > 0.0 and getattr(c, "dp_target", "grad") == "emb":
        zp = oracle.bf16_round(oracle.dp_embed(zp, k, c.dp_clip, c.dp_sigma, o.dp_seed)[0])
    chain(2, Tm, np.concatenate([za, zp], axis=1), False)
    out["weights"] = weights
    return out


def flip_allowance(fwd, rec, rows):
    """{(party, layer): (EW, Eb)}: for the weight and bias gradients, twice the
    magnitude of the oracle's contributions of the excused rows (sum over those
    rows of |dpre_ri| |h_rj|, and of |dpre_ri|).  A row whose forward took another
    branch on the GPU contributes other terms there; their difference is bounded
    by the two contributions' magnitudes, each taken as the oracle's.  The oracle's
    d(pre-activations) are rebuilt here from its own record by the chain rule."""
    W = fwd["weights"]
    out = {}
    if not rows.any():
        return out

    def back(party, n, g, relu_last):
        for i in reversed(range(n)):
            Wc, hin = W[(party, i)]
            relu = relu_last or i < n - 1
            dpre = g * (fwd[(party, i)][2] > 0) if relu else g
            a = np.abs(dpre[rows])
            out[(party, i)] = (2.0 * a.T @ np.abs(hin[rows]), 2.0 * a.sum(axis=0))
            g = oracle.bf16_round(dpre @ Wc)
        return g

    n_t = sum(1 for key in W if key[0] == 2)
    back(2, n_t, rec.ds, False)
    back(1, sum(1 for key in W if key[0] == 1), rec.dza, True)
    back(0, sum(1 for key in W if key[0] == 0), rec.dzp, True)
    return out


def flipped_rows(vfl, ctx, k, fwd):
    """(excused rows, count of flipped units, worst flip) of GPU step k against the
    oracle's forward `fwd`: rows where any hidden unit's GPU mask differs from the
    oracle's.  A flip further from zero than FLIP_BAND of its terms' magnitude is
    reported in `worst` (> 1 fails the step)."""
    rows = None
    worst = 0.0
    nflip = 0
    for key, val in fwd.items():
        if key == "weights":
            continue
        (party, layer), (pre, mag, h) = key, val
        g = ctx.tap(k, vfl.TAP_ACT(party, layer))
        flip = (g > 0) != (h > 0)
        if rows is None:
            rows = np.zeros(h.shape[0], bool)
        if flip.any():
            nflip += int(flip.sum())
            rows |= flip.any(axis=1)
            worst = max(worst, float((np.abs(pre[flip]) / (FLIP_BAND * mag[flip] + 1e-30)).max()))
    if rows is None:
        rows = np.zeros(0, bool)
    return rows, nflip, worst


def grad_err(got, ref, allow=None):
    """Relative infinity norm of a gradient, each element's error first reduced by
    its allowance for excused rows (flip_allowance)."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    if ref.size == 0:
        return 0.0
    d = np.abs(got - ref)
    if allow is not None:
        d = np.maximum(d - allow, 0.0)
    return float(d.max() / max(np.abs(ref).max(), 1e-30))


def compare_step(vfl, ctx, rec, tol, check_grads=True, excused=None, allowance=None):
    """Per-step taps, gradients and updated parameters against an oracle record,
    in the relative infinity norm; bf16 row tensors leave out the `excused` rows,
    and the gradients (and the parameters they update) take their allowance for
    those rows."""
    k = rec.k
    dt = ctx.p.dtype
    errs = {
        "zp": tensor_err(ctx.tap(k, vfl.TAP_EMB), rec.zp, dt, excused),
        "dzp": tensor_err(ctx.tap(k, vfl.TAP_GRAD), rec.dzp, dt, excused),
        "logits": tensor_err(ctx.tap(k, vfl.TAP_LOGITS), rec.logits, dt, excused),
        "za": tensor_err(ctx.tap(k, vfl.TAP_ZA), rec.za, dt, excused),
        "dza": tensor_err(ctx.tap(k, vfl.TAP_DZA), rec.dza * (rec.za > 0), dt, excused),
    }
    loss = ctx.read_losses(k, 1)[0]
    errs["loss"] = abs(loss - rec.loss) / max(abs(rec.loss), 1e-30)
    if check_grads:
        g = ctx.get_grads(worker=k % ctx.p.workers)
        out_layer = (2, len(ctx.p.top) - 1)
        allowance = allowance or {}
        for key, (dW, db) in g.items():
            aw, ab = allowance.get(key, (None, None))
            errs[f"dW{key}"] = grad_err(dW, rec.grads[key][0], aw)
            if key == out_layer:
                # db of the output layer is the column sum of d(logits), whose signed per-row terms
                # cancel as the model calibrates: its error is taken against the sum of the terms'
                # magnitudes, the scale that bounds the rounding error of a sum
                scale = float(np.abs(rec.ds).sum(axis=0).max())
                ref = np.asarray(rec.grads[key][1], np.float64)
                errs[f"db{key}"] = float(np.abs(np.asarray(db, np.float64) - ref).max() /
                                         max(np.abs(ref).max(), scale, 1e-30))
            else:
                errs[f"db{key}"] = grad_err(db, rec.grads[key][1], ab)
    # the parameter-server mode: the replica the step updated (the oracle records the same one);
    # an updated parameter moves by lr times its gradient's allowance at most
    lr = ctx.p.lr
    allowance = allowance or {}
    params = ctx.get_replica(k % ctx.p.workers) if ctx.ps else ctx.get_params()
    for key, (W, b) in params.items():
        aw, ab = allowance.get(key, (None, None))
        errs[f"W{key}"] = grad_err(W, rec.params[key][0], None if aw is None else lr * aw)
        errs[f"b{key}"] = grad_err(b, rec.params[key][1], None if ab is None else lr * ab)
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
    rounds the other way moves later ReLU masks); their row tensors leave out the
    rows with a flipped ReLU unit (flipped_rows), whose largest count per step and
    total of flipped units are reported in worst["flipped_rows_max"] and
    worst["flipped_units_total"].  `drops` marks steps whose
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
    flips = {}
    for k in range(steps):
        if teacher_forced and k > 0:
            force_gpu_state(ctx, o, q.staleness)
        dropped = drops is not None and bool(drops[k])
        fwd = oracle_forward(o, int(tp[k]), int(ta[k])) if q.dtype == "bf16" and not dropped else None
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
            excused = None
            if fwd is not None:
                excused, nflip, far = flipped_rows(vfl, ctx, k, fwd)
                flips[k] = (int(excused.sum()), nflip)
            allowance = flip_allowance(fwd, rec, excused) if fwd is not None and excused.size else None
            errs, bad = compare_step(vfl, ctx, rec, TOL[q.dtype], excused=excused, allowance=allowance)
            if fwd is not None:
                errs["flip_distance"] = far            # <= 1: every flip lies within its rounding band
                errs["flipped_row_fraction"] = float(excused.mean()) / FLIP_ROWS_MAX if excused.size else 0.0
                if far > 1.0:
                    bad["flip_distance"] = far
                if excused.size and excused.mean() > FLIP_ROWS_MAX:
                    bad["flipped_row_fraction"] = float(excused.mean())
        for name, e in errs.items():
            worst[name] = max(worst.get(name, 0.0), e)
        if bad:
            failures.append((k, bad))
    if flips:
        worst["flipped_rows_max"] = float(max(v[0] for v in flips.values()))
        worst["flipped_units_total"] = float(sum(v[1] for v in flips.values()))
    return worst, failures
