"""Calibrate the system planner (Sec. 4.2-4.3) on this GPU and check its choice.

The paper estimates the pipelined system's delays from a synchronous run:
each phase of a step timed alone, at several batch sizes, fitted to the power
laws of Eq. 7-9, and the memory per worker fitted to Eq. 14.  Here:

* a context with one worker per party and staleness 0 runs steps phase by
  phase, each phase bracketed by CUDA events on its own stream and followed by
  a synchronize (the synchronous baseline); the median over the timed steps,
  divided by the batch size, is the phase's delay per sample at that batch
  size (the paper's fitted exponents, all negative, describe delays per
  sample; minimising Eq. 17 then maximises throughput);
* T_f^(p) = the passive forward, T_b^(p) = the passive backward with its
  update, and the active side's forward, top model, backward and update (one
  fused chain on this path) = the lambda_a term; phi_a and the top terms stay 0;
* the memory per worker is the library's workspace size as a function of the
  batch (exactly affine: chi = 1), against the device's free memory;
* C_a = C_p = 1 (both parties share one GPU); the exchange is a write and a
  read of HBM that the measured phases already contain, so the separate
  communication term is 0 (bytes_per_row = 0).

vfl_plan (Algorithm 2) then picks (w_a, w_p, B).  The validation times the
whole pipelined step (CUDA graphs, every worker count and batch size of the
search space, w_a = w_p since the library runs one worker count per party)
and reports the measured throughput next to the model's prediction.

Run: python -m paper_2510_12494_gb300.calibrate [--config N] [--batches ...] [--workers ...]
"""
from __future__ import annotations

import argparse
import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def _phase_times(vfl, p, steps, warmup):
    """Median delay (ms per step) of each phase of a synchronous run: passive forward, active step,
    passive backward."""
    import torch
    import synth
    q = p.with_(staleness=0, schedule="sync", workers=1, ps_dt0=0)
    xp, xa, y = synth.make_dataset(q)
    ctx = vfl.Context(q, q.n_rows)
    ctx.load_data(xp, xa, y)
    ctx.set_params(synth.init_params(q))
    ps, as_ = ctx.streams
    out = {"pf": [], "act": [], "pb": []}
    for k in range(warmup + steps):
        for name, s, call in (("pf", ps, lambda: ctx.passive_forward(k, 0)), ("act", as_, lambda: ctx.active_step(k, 0)),
                              ("pb", ps, lambda: ctx.passive_backward(k))):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record(s)
            call()
            e1.record(s)
            torch.cuda.synchronize()
            if k >= warmup:
                out[name].append(e0.elapsed_time(e1))
    ctx.close()
    return {k: float(np.median(v)) for k, v in out.items()}


def _pipelined_throughput(vfl, p, epochs):
    """Samples/s of the pipelined training (graphs of one epoch, L2 not flushed: the planner's comparison)."""
    import torch
    import synth
    xp, xa, y = synth.make_dataset(p)
    ctx = vfl.Context(p, p.n_rows)
    ctx.load_data(xp, xa, y)
    ctx.set_params(synth.init_params(p))
    nb = p.steps_per_epoch
    n = nb * (epochs + 1)
    kind = vfl.SCHED_SYNC if p.schedule == "sync" else vfl.SCHED_SEEDED
    tp, ta = vfl.make_schedule(p.seed, p.staleness, kind, n)
    ctx.train_steps(0, nb, tp, ta)                       # warm-up epoch
    ctx.synchronize()
    main = torch.cuda.Stream()
    total_ms = 0.0
    for e in range(epochs):
        g = ctx.capture(nb * (e + 1), nb, tp, ta)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        with torch.cuda.stream(main):
            torch.cuda._sleep(1_000_000)                  # host enqueue stays outside the timed interval
            e0.record(main)
        for s in ctx.streams:
            s.wait_event(e0)
        ctx.launch_graph(g)
        for s in ctx.streams:
            ev = torch.cuda.Event()
            ev.record(s)
            main.wait_event(ev)
        e1.record(main)
        main.synchronize()
        total_ms += e0.elapsed_time(e1)
    ctx.close()
    return epochs * p.n_rows / (total_ms / 1e3)


def calibrate(vfl, p, batches, steps=40, warmup=10):
    """Fitted vfl_plan_model constants (as a dict) and the measured phase delays per batch size."""
    import torch
    meas = {}
    for b in batches:
        meas[b] = _phase_times(vfl, p.with_(batch=b), steps, warmup)
    bs = np.array(batches, np.float64)
    lam_p, gam_p = vfl.fit_power(bs, [meas[b]["pf"] / b for b in batches])
    phi_p, bet_p = vfl.fit_power(bs, [meas[b]["pb"] / b for b in batches])
    lam_a, gam_a = vfl.fit_power(bs, [meas[b]["act"] / b for b in batches])
    # memory per worker: the workspace as a function of the batch, affine (chi = 1)
    ws = np.array([vfl.workspace_bytes(p.with_(batch=b, workers=1, ps_dt0=0, staleness=0), p.n_rows)
                   for b in batches], np.float64)
    rho, m0 = np.polyfit(bs, ws, 1)
    free, _ = torch.cuda.mem_get_info()
    model = dict(lambda_a=lam_a, gamma_a=gam_a, lambda_p=lam_p, gamma_p=gam_p, phi_p=phi_p, beta_p=bet_p,
                 C_a=1.0, C_p=1.0, bytes_per_row=0.0, bandwidth=1.0,
                 M_A0=float(m0), rho_A=float(max(rho, 1e-9)), M_A_max=float(free), M_P0=float(m0),
                 rho_P=float(max(rho, 1e-9)), M_P_max=float(free), chi=1.0)
    return model, meas


def main(argv=None):
    import torch
    import synth
    import paper_2510_12494_gb300 as vfl
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("--config", type=int, default=2)
    ap.add_argument("--batches", type=int, nargs="+", default=[256, 512, 1024, 2048, 4096])
    ap.add_argument("--workers", type=int, nargs=2, default=[1, 4], metavar=("LO", "HI"))
    ap.add_argument("--epochs", type=int, default=3, help="timed epochs per validation point")
    args = ap.parse_args(argv)
    assert torch.cuda.is_available(), "calibration needs a CUDA device"
    p = synth.preset(args.config)
    model, meas = calibrate(vfl, p, args.batches)
    m = vfl.plan_model(**model)
    lo, hi = args.workers
    wa, wp, b, o = vfl.plan(m, (lo, hi), (lo, hi), args.batches)
    grid = {}
    for w in range(lo, hi + 1):
        for bb in args.batches:
            q = p.with_(batch=bb, workers=w)
            grid[f"{w}x{bb}"] = {"measured_samples_per_s": _pipelined_throughput(vfl, q, args.epochs),
                                 "model_ms_per_sample": vfl.plan_delay(m, w, w, float(bb))}
    best = max(grid, key=lambda k: grid[k]["measured_samples_per_s"])
    print(json.dumps({"workload": p.name, "model": model, "phase_ms": {str(k): v for k, v in meas.items()},
                      "b_max": vfl.plan_bmax(m), "plan": {"w_a": wa, "w_p": wp, "batch": b, "ms_per_sample": o},
                      "validation": grid, "measured_best": best}, indent=1))


if __name__ == "__main__":
    main()
