#!/usr/bin/env python
"""Throughput of the split-VFL training step on GB300, through the C ABI.

One "step" is one training mini-batch through the whole path: passive bottom
forward, publish, active bottom forward, top forward, loss, backward, publish
the cut-layer gradient, both bottoms' backward and the SGD updates (Algorithm 1
with the delayed update of App. D).  Default workload: the credit-shaped
preset with the most rows, bytes and FLOPs per epoch: wide-dp (1,000,000 rows,
1000/1000 binary features, 1000-512-256 bottoms, top 512-256-1, BCE, batch
8192, staleness 4 on the seeded schedule, bf16 with fp32 accumulation, DP
clipping + Gaussian noise on the published gradient).  Prints one JSON line.

Timing: the K timed steps run as R >= 5 windows (one epoch each when K allows),
the L2 flushed before each; value and ms_per_step are the median window's.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference] [--config C]

--impl reference times the CPU oracle (the only other implementation of the
method) on the same workload.  With N > 1 (torchrun) every rank runs an
independent replica of the workload on its own GPU (the path has no exchange
between GPUs); value = all ranks' samples / the slowest rank's time.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "split-VFL training samples/sec at 1 GB300; % of roofline per kernel"


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=0, help="timed steps (default: 5 epochs of the workload)")
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", type=int, default=4, help="workload preset 1..5 (default 4, wide-dp)")
    ap.add_argument("--rows", type=int, default=0, help="override the preset's row count")
    ap.add_argument("--workers", type=int, default=0, help="worker streams per party (default: the preset's, or "
                    "BENCH_WORKERS where the workload leaves them open)")
    ap.add_argument("--dp-target", choices=["grad", "emb"], default=None,
                    help="with DP: the published gradient (the preset's) or the published embedding (App. C)")
    ap.add_argument("--dp", type=float, nargs=2, default=None, metavar=("CLIP", "SIGMA"),
                    help="enable DP with this clip norm and noise multiplier")
    ap.add_argument("--ps-dt0", type=int, default=0, metavar="DT0",
                    help="intra-party parameter server (Eq. 5): per-worker replicas averaged per Delta T_0 = DT0 "
                         "(sets the staleness to 0)")
    ap.add_argument("--drop-rate", type=float, default=0.0, metavar="R",
                    help="waiting-deadline drops: each step's subscriber gives up with probability R (seeded draws); "
                         "dropped steps train nothing and count no samples")
    ap.add_argument("--skip-e2e", action="store_true")
    ap.add_argument("--skip-cpu", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--no-graphs", action="store_true", help="enqueue every step directly instead of replaying "
                    "a CUDA graph captured before each timed iteration")
    return ap.parse_args(argv)


# Worker streams per party (the paper's w_a = w_p) where the workload leaves them open: the count measured
# fastest on GB300 (results do not depend on it: every step computes the same thing on any stream).
BENCH_WORKERS = {3: 3, 4: 3}


def workload(args):
    import synth
    p = synth.preset(args.config)
    if args.rows:
        p = p.with_(n_rows=args.rows)
    if args.workers:
        p = p.with_(workers=args.workers)
    elif args.config in BENCH_WORKERS and not args.ps_dt0:
        p = p.with_(workers=BENCH_WORKERS[args.config])
    if args.dp:
        p = p.with_(dp_clip=args.dp[0], dp_sigma=args.dp[1])
    if args.dp_target:
        p = p.with_(dp_target=args.dp_target)
    if args.ps_dt0:
        p = p.with_(ps_dt0=args.ps_dt0, staleness=0, schedule="sync")
    desc = (f"{p.name}: N={p.n_rows}, d_p/d_a={p.d_passive}/{p.d_active}, "
            f"passive {'-'.join(map(str, (p.d_passive,) + p.passive))}, "
            f"active {'-'.join(map(str, (p.d_active,) + p.active))}, "
            f"top {'-'.join(map(str, (p.e_active + p.e_passive,) + p.top))} {p.loss.upper()}, "
            f"B={p.batch}, S={p.staleness} ({p.schedule} schedule), {p.dtype}, "
            f"{p.workers} worker stream(s) per party" +
            (f", DP on the {'embedding' if p.dp_target == 'emb' else 'embedding gradient'} C={p.dp_clip} "
             f"sigma={p.dp_sigma}" if p.dp_clip else "") +
            (f", parameter server per worker (replicas averaged per Eq. 5, Delta T_0={p.ps_dt0})"
             if p.ps_dt0 else "") +
            (f", waiting-deadline drops at rate {args.drop_rate} (batch reassigned to the next step)"
             if getattr(args, "drop_rate", 0.0) else ""))
    return p, desc


def dtype_tag(p):
    return "f32" if p.dtype == "fp32" else "bf16"


def rows_of(p, k):
    j = k % p.steps_per_epoch
    r0 = j * p.batch
    return r0, min(p.n_rows, r0 + p.batch)


def samples(p, k0, n, drops=None):
    """Rows trained by steps [k0, k0+n): a dropped step trains none and hands its batch to the next."""
    if drops is None:
        return sum(rows_of(p, k)[1] - rows_of(p, k)[0] for k in range(k0, k0 + n))
    tot = 0
    for k in range(k0, k0 + n):
        if not drops[k]:
            r0, r1 = rows_of(p, k - int(drops[:k].sum()))
            tot += r1 - r0
    return tot


def sched_kind(p):
    return 0 if p.schedule == "sync" else 2


# --------------------------------------------------------------------------
# clocks during the timed region
# --------------------------------------------------------------------------
class Clocks:
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        self.dev = device_index
        try:
            self.p = subprocess.Popen(["nvidia-smi", "-i", str(device_index), f"--query-gpu={self.Q}",
                                       "--format=csv,noheader,nounits", "-lms", "20"],
                                      stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None

    def stop(self):
        if self.p is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.p.terminate()
        self.p.wait()
        self.f.flush()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.f.name) as fh:
            for line in fh:
                parts = [t.strip() for t in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx.append(float(parts[2]))
                except ValueError:
                    continue
                for name, v in zip(names, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(name)
        os.unlink(self.f.name)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------------------
# CPU oracle timing (subprocess: its own threads, no CUDA)
# --------------------------------------------------------------------------
CPU_SNIPPET = r"""
import sys, time, json, os
sys.path.insert(0, {root!r})
import numpy as np, synth, oracle
p = synth.VflPreset(**{fields!r})      # the workload exactly as the GPU arm runs it
nb = p.steps_per_epoch

def build(n_steps):
    # the rows the first n_steps steps train (step k < nb trains batch k): the sample's steps see
    # exactly the batches, versions and schedule of the full workload
    rows = p.n_rows if n_steps >= nb else n_steps * p.batch
    xp, xa, y = synth.make_dataset(p, rows=(0, rows))
    q = p.with_(n_rows=rows)
    tp, ta = oracle.make_schedule(q.seed, q.staleness, {kind}, n_steps)
    drops = oracle.make_drops(q.seed, {drop_rate}, n_steps)
    return oracle.Oracle(q, xp, xa, y, synth.init_params(q), dp_seed=q.seed), tp, ta, drops

# size the sample from one probe step, so that only the rows it trains are generated
o, tp, ta, drops = build(1)
t0 = time.perf_counter(); o.step(0, 0); t_probe = time.perf_counter() - t0
n_steps = max(1, min({n_steps}, int({budget} / max(t_probe, 1e-6)) + 1))
o, tp, ta, drops = build(n_steps)
t0 = time.perf_counter(); done = 0; nsamp = 0
while done < n_steps:
    r = o.step(int(tp[done]), int(ta[done]), drop=bool(drops[done]))
    nsamp += 0 if r.dropped else r.rows[1] - r.rows[0]
    done += 1
    if time.perf_counter() - t0 > {budget}: break
dt = time.perf_counter() - t0
print(json.dumps(dict(steps=done, samples=nsamp, seconds=dt)))
"""


def cpu_model():
    """The host CPU's model name (lscpu; /proc/cpuinfo as a fallback)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform
    return platform.processor() or platform.machine()


def run_oracle(p, args, n_steps, budget, threads=None):
    """The oracle as it stands, timed in a subprocess (no CUDA) with `threads` BLAS threads (default:
    every host core): at most n_steps steps and about `budget` seconds of the workload's first steps."""
    cores = threads or os.cpu_count() or 1
    env = dict(os.environ)
    for v in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        env[v] = str(cores)
    env["CUDA_VISIBLE_DEVICES"] = ""
    fields = {f: getattr(p, f) for f in p.__dataclass_fields__}
    code = CPU_SNIPPET.format(root=ROOT, fields=fields, n_steps=n_steps, kind=sched_kind(p), budget=budget,
                              drop_rate=float(args.drop_rate))
    r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env)
    if r.returncode != 0:
        raise RuntimeError(f"oracle timing failed: {r.stderr[-2000:]}")
    res = json.loads(r.stdout.strip().splitlines()[-1])
    res["cores"] = cores
    return res


def cpu_baseline(p, args, n_steps):
    """The oracle on the host cores, all of them and one: value = the all-cores figure."""
    model = cpu_model()
    full = run_oracle(p, args, n_steps, args.cpu_seconds)
    one = run_oracle(p, args, n_steps, args.cpu_seconds, threads=1)

    def leg(res):
        return {"value": res["samples"] / res["seconds"], "threads": res["cores"], "steps": res["steps"],
                "samples": res["samples"], "seconds": round(res["seconds"], 3)}
    return {"value": full["samples"] / full["seconds"], "unit": "samples/s", "cores": full["cores"], "kind": "oracle",
            "cpu_model": model, "all_cores": leg(full), "single_thread": leg(one),
            "sample": f"first {full['steps']} training steps ({full['samples']} samples) of the same workload "
                      f"(single thread: {one['steps']} steps), float64 numpy oracle, {full['seconds']:.2f} s with "
                      f"BLAS threads={full['cores']} on {model}"}


# --------------------------------------------------------------------------
# the GPU arm
# --------------------------------------------------------------------------
def peaks():
    """Roofline denominators: HBM copy and bf16 GEMM from MEASURED_PEAKS.json, the FP32 FMA and TF32
    warp-MMA peaks from profiles/peaks.json (python -m paper_2510_12494_gb300.peaks)."""
    out = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "src": "fallback"}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        out = {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
               "bf16_tflops_sustained": d.get("bf16_tflops_sustained", d["bf16_tflops"]), "src": "measured"}
    except (OSError, KeyError, ValueError):
        pass
    try:
        with open(os.path.join(ROOT, "profiles", "peaks.json")) as f:
            d = json.load(f)
        out["ffma_tflops"], out["x3tf32_tflops"] = d["fp32_ffma"]["tflops"], d["fp32_3xtf32_tflops"]
        out["fp32_src"] = "measured"
    except (OSError, KeyError, ValueError):
        # nominal: 152 SMs x 128 FP32 lanes x 2 x 2070 MHz; TF32 at 1.1/2.25 of the bf16 peak, / 3 for 3xTF32
        out["ffma_tflops"], out["x3tf32_tflops"] = 80.5, out["bf16_tflops_sustained"] * 1.1 / 2.25 / 3
        out["fp32_src"] = "nominal"
    return out


# event class -> the kernel function that runs it (the launch list and the ncu captures are per function)
KERNEL_OF_CLASS = {
    "gemm_tc_fwd": "tc_gemm_kernel", "gemm_tc_dx": "tc_gemm_kernel", "gemm_tc_dw": "tc_dw_kernel",
    "gemm_tc_dw_sgd": "tc_dw_kernel", "gemm_tc_chain": "tc_chain_kernel", "gemm_simt_fwd": "gemm_simt_kernel", "gemm_simt_dx": "gemm_simt_kernel",
    "gemm_simt_dw": "gemm_simt_kernel", "head_loss": "head_kernel", "loss": "loss_kernel",
    "dp_clip_noise": "dp_kernel", "relu_mask": "relu_mask_kernel", "sgd": "sgd_kernel",
    "channel_header": "write_header_kernel", "cast": "cast_rows_kernel",
    "fused_passive_fwd": "fused_passive_fwd_kernel", "fused_active_step": "fused_active_kernel",
    "fused_passive_bwd": "fused_passive_bwd_kernel", "fused_update": "fused_update_kernel",
    "ps_average": "ps_average_kernel"}
KERNEL_SOURCE = {"tc_": "kernels_tc.cu", "fused_": "kernels_fused.cu",
                 "stage_rows_bits": "kernels_io.cu"}   # everything else: kernels_simt.cu


def file_digest(src):
    import hashlib
    with open(os.path.join(ROOT, "paper_2510_12494_gb300", "csrc", src), "rb") as f:
        return hashlib.sha256(f.read()).hexdigest()


def source_digest(kernel):
    return file_digest(next((f for pre, f in KERNEL_SOURCE.items() if kernel.startswith(pre)), "kernels_simt.cu"))


def profile_record(name):
    try:
        with open(os.path.join(ROOT, "profiles", name)) as f:
            return json.load(f)
    except (OSError, ValueError):
        return None


def profiled_traffic(kernel, classes, workload_name, launch_units):
    """DRAM bytes (read + write) per launch of `kernel` from the committed ncu captures
    (profiles/kernels.json): the captured launches of the same event classes on the same workload,
    per unit, scaled to `launch_units`; None when nothing matches or the kernel's source has changed
    since the counters were taken."""
    rec = profile_record("kernels.json")
    if not rec:
        return None
    for k in rec["kernels"]:
        if k["kernel"] != kernel or k["workload"] != workload_name or k["source_sha256"] != source_digest(kernel):
            continue
        ls = [x for x in k["launches"] if x.get("class") in classes] or k["launches"]
        dram = [(x["dram_read"] or 0) + (x["dram_write"] or 0) for x in ls]
        per_unit = sum(dram) / len(dram) / k["units_per_launch"]
        return {"bytes_per_launch": per_unit * launch_units, "captured_launches": len(ls),
                "source": "profiles/" + k["file"]}
    return None


def launch_list_check(kernel, workload_name, flops_per_launch, bytes_per_launch, bound, peak):
    """The dominant kernel seen from the committed ncu launch list of the same workload
    (profiles/launches.json: serialised launches, kernel time only): its share of all kernel time,
    whether it is the largest there too, and its roofline fraction on the launch list's warm duration."""
    rec = profile_record("launches.json")
    if not rec or workload_name not in rec.get("workloads", {}):
        return None
    w = rec["workloads"][workload_name]
    mine = next((f for pre, f in KERNEL_SOURCE.items() if kernel.startswith(pre)), "kernels_simt.cu")
    stale = [f for f, h in w.get("sources_sha256", {}).items() if h != file_digest(f) and f == mine]
    ks = w["kernels"]
    top = max(ks, key=lambda n: ks[n]["warm_share"])
    me = ks.get(kernel)
    out = {"largest_warm": top, "agrees": top == kernel, "stale_sources": stale, "command": w["command"]}
    if me:
        sec = me["warm_avg_us"] * 1e-6
        ach = (flops_per_launch / sec / 1e12) if bound in ("tensor", "alu") else (bytes_per_launch / sec / 1e9)
        out.update({"warm_share": me["warm_share"], "cold_share": me["cold_share"],
                    "warm_avg_us": me["warm_avg_us"], "cold_avg_us": me["cold_avg_us"],
                    "achieved": ach, "frac": ach / peak})
    return out


HOST_ENQUEUE_CYCLES = 1_000_000       # ~0.5 ms of GPU spin before each timed iteration (not timed)


def roofline(prof, pk, workload_name, units):
    """The dominant kernel (largest summed event time over its classes) against its bound.  Its
    achieved rate is the algorithmic work per launch over the event-timed launch duration, and again
    over the kernel-only duration of the committed ncu launch list."""
    if not prof:
        return None
    by_kernel = {}
    for cls, (n, ms, flops, nbytes) in prof.items():
        k = KERNEL_OF_CLASS.get(cls, cls)
        a = by_kernel.setdefault(k, [0, 0.0, 0.0, 0.0, []])
        a[0] += n; a[1] += ms; a[2] += flops; a[3] += nbytes; a[4].append(cls)
    # the dominant kernel: the largest share of kernel time in the committed launch list of this workload
    # when that list is current (serialised kernel time, no launch latency or stream overlap in it), else
    # the largest summed event time
    rec = profile_record("launches.json")
    wl = (rec or {}).get("workloads", {}).get(workload_name)
    srcs = {next((f for pre, f in KERNEL_SOURCE.items() if k.startswith(pre)), "kernels_simt.cu") for k in by_kernel}
    fresh = wl is not None and all(wl.get("sources_sha256", {}).get(f) == file_digest(f) for f in srcs)
    if fresh and any(k in wl["kernels"] for k in by_kernel):
        name = max((k for k in by_kernel if k in wl["kernels"]), key=lambda k: wl["kernels"][k]["warm_share"])
        selected_by = "largest warm share of the committed ncu launch list"
    else:
        name = max(by_kernel, key=lambda k: by_kernel[k][1])
        selected_by = "largest summed event time"
    n, ms, flops, nbytes, classes = by_kernel[name]
    sec = ms / 1e3
    if name.startswith("tc_"):
        bound, peak, unit = "tensor", pk["bf16_tflops_sustained"], "TFLOP/s"
        peak_src = f"{pk['src']} sustained bf16 GEMM"
    elif name.startswith("fused_"):
        # fp32 contractions on the TF32 tensor path in 3xTF32 form: three TF32 products per fp32 one
        bound, peak, unit = "tensor", pk["x3tf32_tflops"], "TFLOP/s"
        peak_src = f"{pk['fp32_src']} TF32 warp-MMA peak / 3 (3xTF32)"
    else:
        balance = pk["ffma_tflops"] * 1e12 / (pk["hbm_gbs"] * 1e9)
        if flops > 0 and flops / max(nbytes, 1.0) > balance:
            bound, peak, unit = "alu", pk["ffma_tflops"], "TFLOP/s"
            peak_src = f"{pk['fp32_src']} FFMA peak"
        else:
            bound, peak, unit = "hbm", pk["hbm_gbs"], "GB/s"
            peak_src = f"{pk['src']} HBM copy"
    ach = flops / sec / 1e12 if unit == "TFLOP/s" else nbytes / sec / 1e9
    tr = profiled_traffic(name, classes, workload_name, units)
    ll = launch_list_check(name, workload_name, flops / n, nbytes / n, "tensor" if unit == "TFLOP/s" else "hbm",
                           peak)
    return {"kernel": name, "selected_by": selected_by, "classes": classes, "bound": bound, "achieved": ach, "peak": peak, "unit": unit,
            "frac": ach / peak, "traffic": tr["bytes_per_launch"] if tr else None,
            "traffic_source": tr, "algorithmic_per_launch": {"flops": flops / n, "bytes": nbytes / n},
            "launches": n, "avg_us": ms / n * 1e3, "timing": "CUDA event pair around each launch, on its stream",
            "peak_src": peak_src, "launch_list": ll,
            "all_kernels_ms": {k: round(v[1], 4) for k, v in sorted(by_kernel.items(), key=lambda kv: -kv[1][1])}}


def slowest_rank(x: float) -> float:
    """The maximum of x over the ranks of the default process group (x itself
    without one): a multi-GPU job is as fast as its slowest replica."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return x
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(samples_per_rank: int, world: int, slowest_seconds: float) -> float:
    """Whole-job samples/s: every rank's samples over the slowest rank's time."""
    return samples_per_rank * world / slowest_seconds


def plan(p, args):
    """(W, K, window, n_e2e): warm-up and timed steps, steps per timed window (R >= 5 windows of one
    training run of the workload each when K allows), and the end-to-end leg's steps per method (at
    least one epoch, so that its per-epoch graph updates amortise)."""
    nb = p.steps_per_epoch
    run_len = nb * max(1, p.epochs)
    K = args.steps or 5 * run_len
    window = run_len if K >= 5 * run_len else max(1, -(-K // 5))
    return max(args.warmup, 3), K, window, max(nb, K)


def config_of(desc, world):
    """The `config` object both arms print: the workload and how it is spread over devices."""
    return {"workload": desc, "parallelism": f"replicas x{world} (one per GPU)" if world > 1 else "single device"}


def run_ours(args):
    import numpy as np
    import torch
    import paper_2510_12494_gb300 as vfl
    from paper_2510_12494_gb300 import build
    import synth

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    build.build()

    p, desc = workload(args)
    W, K, window, n_e2e = plan(p, args)
    cpu = None
    if rank == 0 and world == 1 and not args.skip_cpu:
        cpu = cpu_baseline(p, args, W + K)   # before the GPU work: the oracle runs on idle host cores

    xp, xa, y = synth.make_dataset(p)
    params = synth.init_params(p)
    total = W + 2 * K + 2 * n_e2e
    tp, ta = vfl.make_schedule(p.seed, p.staleness, sched_kind(p), total)
    drops = vfl.make_drops(p.seed, args.drop_rate, total) if args.drop_rate > 0 else None
    ctx = vfl.Context(p, p.n_rows)
    ctx.load_data(xp, xa, y)
    ctx.set_params(params)
    main = torch.cuda.Stream()
    flush = torch.empty(256 * 2 ** 20, dtype=torch.uint8, device="cuda")   # > 129 MB L2
    nb = p.steps_per_epoch
    use_graphs = not args.no_graphs

    def timed_block(k0, n, profile=False):
        """Time steps [k0, k0+n) in windows of `window` steps, the L2 flushed before each; with graphs
        each window's graph is captured (untimed) just before it runs.  Returns [(steps, samples, ms)]
        per window and the per-class profile when asked."""
        out = []
        k = k0
        if profile:
            ctx.profile(True)
        while k < k0 + n:
            m = min(window, k0 + n - k)
            graph = ctx.capture(k, m, tp, ta, drops) if use_graphs else None
            with torch.cuda.stream(main):
                flush.zero_()
                # keep the GPU busy while the host enqueues this window, so that the host's launch
                # latency stays outside the device-timed interval that starts at e0
                torch.cuda._sleep(HOST_ENQUEUE_CYCLES)
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record(main)
            for s in ctx.streams:
                s.wait_event(e0)
            if graph is not None:
                ctx.launch_graph(graph)
            else:
                ctx.train_steps(k, m, tp, ta, drops)
            for s in ctx.streams:
                ev = torch.cuda.Event()
                ev.record(s)
                main.wait_event(ev)
            e1.record(main)
            main.synchronize()
            out.append((m, samples(p, k, m, drops), e0.elapsed_time(e1)))
            k += m
        prof = None
        if profile:
            ctx.profile(False)
            prof = ctx.profile_summary()
        return out, prof

    # warm-up
    ctx.train_steps(0, W, tp, ta, drops)
    ctx.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    clocks = Clocks(local)
    l0 = ctx.launches
    x0 = ctx.exchange_bytes()
    wins, _ = timed_block(W, K)
    launches = ctx.launches - l0
    x1 = ctx.exchange_bytes()
    torch.cuda.synchronize()
    clk = clocks.stop()
    # the median window (by samples/s) decides; max over ranks of its per-sample time
    rates = sorted(wins, key=lambda t: t[1] / t[2])
    mid = rates[len(rates) // 2]
    ms_med = slowest_rank(mid[2])
    value = job_throughput(mid[1], world, ms_med / 1e3)
    ms_per_step = ms_med / mid[0]

    # per-kernel timing: the same workload again, every launch bracketed by CUDA events (recorded
    # inside the replayed graphs when graphs are on, so each duration is the kernel as the step runs it)
    _, prof = timed_block(W + K, K, profile=True)
    # units per launch of the dominant kernel: every kernel of the step processes one batch per launch
    roof = roofline(prof, peaks(), p.name, p.batch)

    # end to end through the public API with host buffers: the dataset stays in pinned host memory,
    # every step copies its rows in and its loss out (vfl_bind_host_data) inside the timed region
    e2e = None
    if not args.skip_e2e:
        # the host keeps the features compactly (untimed, once): bit-packed when every feature is 0 or 1
        # (vfl_bind_host_data_bits: 1/16 of bf16's bytes, exact), else in the compute dtype (bf16 presets:
        # rounded exactly as the resident load rounds them); each step's staging kernel reads its rows
        def all_binary(a, rows=65536):
            return all(((c == 0) | (c == 1)).all() for c in (a[i:i + rows] for i in range(0, len(a), rows)))

        binary = all_binary(xp) and all_binary(xa)
        host_bf16 = p.dtype == "bf16" and not binary
        pin_y = torch.from_numpy(y).pin_memory()
        loss_host = torch.full((n_e2e,), float("nan"), dtype=torch.float32).pin_memory()
        if binary:
            pin_xp = torch.from_numpy(vfl.pack_bits(xp)).pin_memory()
            pin_xa = torch.from_numpy(vfl.pack_bits(xa)).pin_memory()
            ctx.bind_host_bits(pin_xp, pin_xa, pin_y, loss_out=loss_host)
        else:
            pin_xp = torch.from_numpy(xp).pin_memory()
            pin_xa = torch.from_numpy(xa).pin_memory()
            if host_bf16:
                pin_xp = pin_xp.to(torch.bfloat16).pin_memory()
                pin_xa = pin_xa.to(torch.bfloat16).pin_memory()
            ctx.bind_host_data(pin_xp, pin_xa, pin_y, loss_out=loss_host)

        def e2e_run(k0, graphs):
            """Wall time of steps [k0, k0+n_e2e): enqueued directly, or in the uniform dependency order as
            one graph per epoch, re-recorded and updated in place by the host while the previous epoch's
            replay runs (a new capture only when the window's shape changes; all of it timed)."""
            loss_host.fill_(float("nan"))
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            if graphs:
                ctx.set_order(True)
                # (window length, first worker) -> graph: a window's shape depends on both
                cache = {}
                k = k0
                while k < k0 + n_e2e:
                    m = min(nb, k0 + n_e2e - k)
                    key = (m, k % p.workers)
                    g = cache.get(key)
                    if g is not None and ctx.update_graph(g, k, m, tp, ta, drops):
                        counts["updated"] += 1
                    else:
                        g = cache[key] = ctx.capture(k, m, tp, ta, drops)
                        counts["captured"] += 1
                    ctx.launch_graph(g)
                    k += m
            else:
                ctx.train_steps(k0, n_e2e, tp, ta, drops)
            ctx.synchronize()
            dt = slowest_rank(time.perf_counter() - t0)
            ctx.set_order(False)
            kept = np.ones(n_e2e, bool)        # the host ring's slot k mod n_e2e holds step k's loss
            if drops is not None:
                steps = np.arange(k0, k0 + n_e2e)
                kept[steps % n_e2e] = drops[steps] == 0
            assert np.isfinite(loss_host.numpy()[kept]).all() and np.isnan(loss_host.numpy()[~kept]).all()
            return job_throughput(samples(p, k0, n_e2e, drops), world, dt)

        counts = {"updated": 0, "captured": 0}
        direct = e2e_run(W + 2 * K, False)
        piped = e2e_run(W + 2 * K + n_e2e, True) if use_graphs else None
        ctx.bind_host_data(None, None, None)
        if binary:
            h2d = p.batch * ((p.d_passive + 31) // 32 + (p.d_active + 31) // 32) * 4 + p.batch * 4
        else:
            h2d = p.batch * (p.d_passive + p.d_active) * (2 if host_bf16 else 4) + p.batch * 4
        e2e = {"value": max(direct, piped or 0.0), "unit": "samples/s", "h2d_bytes_per_step": h2d,
               "host_features": "bit-packed (every feature 0 or 1)" if binary else ("bf16" if host_bf16 else "fp32"),
               "d2h_bytes_per_step": 4, "steps": n_e2e, "direct_enqueue": direct,
               "uniform_order_graph_updates": piped, "graph_windows": counts,
               "method": "uniform-order graphs updated in flight" if piped and piped > direct else "direct enqueue"}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "samples/s", "n_gpus": world, "steps": K, "warmup": W,
            "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": dtype_tag(p), "data": "synthetic (seeded stand-in for the paper's tabular data)",
            "config": config_of(desc, world),
            "timing": {"windows": len(wins), "steps_per_window": window,
                       "window_ms": [round(t[2], 4) for t in wins],
                       "window_samples_per_s": [t[1] / t[2] * 1e3 for t in wins],
                       "statistic": "median window (value, ms_per_step); max over ranks",
                       "l2": "flushed (256 MiB write) before each window; inputs larger than L2",
                       "launch": "CUDA graph per window, captured before it runs (untimed)" if use_graphs
                       else "direct enqueue",
                       "streams": f"{p.workers} worker stream(s) per party"},
            "clocks": clk, "e2e": e2e, "gpu_launches": launches, "roofline": roof, "cpu_baseline": cpu,
            # Sec. 5's communication cost: payload bytes through the two channels per timed step
            "exchange_bytes_per_step": {"embedding": (x1[0] - x0[0]) / K, "gradient": (x1[1] - x0[1]) / K},
        }
        print(json.dumps(line))
    ctx.close()
    if world > 1:
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()


def run_reference(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    p, desc = workload(args)
    W, K, _, _ = plan(p, args)
    budget = 60.0
    t0 = time.perf_counter()
    # warm-up steps, then the timed steps, each a bounded sample of the workload
    run_oracle(p, args, max(W, 1), 20.0)
    res = run_oracle(p, args, K, budget)
    value = res["samples"] / res["seconds"]
    model = cpu_model()
    cpu = {"value": value, "unit": "samples/s", "cores": res["cores"], "kind": "oracle", "cpu_model": model,
           "sample": f"first {res['steps']} of {K} training steps ({res['samples']} samples), "
                     f"float64 numpy oracle, {res['seconds']:.2f} s with BLAS threads={res['cores']} on {model}"}
    line = {"metric": METRIC, "value": value, "unit": "samples/s", "n_gpus": world, "steps": res["steps"],
            "warmup": W, "ms_per_step": res["seconds"] / max(res["steps"], 1) * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded stand-in for the paper's tabular data)", "impl": "reference",
            "config": config_of(desc, world),
            "cpu_baseline": cpu, "e2e": {"value": value, "unit": "samples/s", "h2d_bytes_per_step": 0,
                                         "d2h_bytes_per_step": 0},
            "wall_s": time.perf_counter() - t0}
    print(json.dumps(line))


if __name__ == "__main__":
    a = parse()
    if a.impl == "reference":
        run_reference(a)
    else:
        run_ours(a)
