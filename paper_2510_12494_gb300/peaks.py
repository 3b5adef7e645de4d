"""Measure the fp32 roofline denominators of this GPU and write profiles/peaks.json.

  python -m paper_2510_12494_gb300.peaks

FP32 FMA (SIMT) and TF32 warp-MMA throughput from vfl_measure_peak, the best of
five timed launches each, with the SM clock sampled by nvidia-smi (read-only)
during the runs.  The 3xTF32 figure (three TF32 products per fp32 product, the
form the fused fp32 kernels use) is the TF32 one divided by three.  Clocks are
never set: a run whose samples show a slowdown reason is reported as such.
"""
from __future__ import annotations

import json
import os
import statistics
import subprocess
import tempfile
import time

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _clock_sampler():
    f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
    q = "clocks.sm,clocks.max.sm,clocks_event_reasons.hw_slowdown,clocks_event_reasons.sw_thermal_slowdown"
    try:
        p = subprocess.Popen(["nvidia-smi", "-i", "0", f"--query-gpu={q}", "--format=csv,noheader,nounits",
                              "-lms", "20"], stdout=f, stderr=subprocess.DEVNULL)
    except OSError:
        p = None
    return f, p


def _clock_stop(f, p):
    if p is None:
        return {"sm_mhz": None, "sm_max_mhz": None, "slowdown": None}
    p.terminate()
    p.wait()
    f.flush()
    sm, mx, slow = [], [], False
    with open(f.name) as fh:
        for line in fh:
            parts = [t.strip() for t in line.split(",")]
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except (ValueError, IndexError):
                continue
            slow = slow or any(v.lower() == "active" for v in parts[2:4])
    os.unlink(f.name)
    return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
            "slowdown": slow, "samples": len(sm)}


def measure(reps: int = 5):
    import torch
    import paper_2510_12494_gb300 as vfl
    from paper_2510_12494_gb300 import build
    build.build()
    torch.cuda.set_device(0)
    out = {"command": "python -m paper_2510_12494_gb300.peaks", "gpu": torch.cuda.get_device_name(0),
           "how": "vfl_measure_peak: 8 blocks x 256 threads per SM, 8 independent FMA chains per thread (FFMA) or "
                  "8 independent m16n8k8 TF32 accumulators per warp (MMA); best of %d timed launches, CUDA events; "
                  "SM clock sampled by nvidia-smi during the runs, never set" % reps,
           "when": time.strftime("%Y-%m-%dT%H:%M:%SZ", time.gmtime())}
    for name, kind, iters in (("fp32_ffma", vfl.PEAK_FFMA, 1 << 16), ("tf32_mma", vfl.PEAK_TF32_MMA, 1 << 14)):
        f, p = _clock_sampler()
        best = 0.0
        for _ in range(reps):
            flop, ms = vfl.measure_peak(kind, iters)
            best = max(best, flop / (ms * 1e-3) / 1e12)
        clk = _clock_stop(f, p)
        out[name] = {"tflops": best, "clocks": clk}
    out["fp32_3xtf32_tflops"] = out["tf32_mma"]["tflops"] / 3.0
    return out


def main():
    res = measure()
    path = os.path.join(ROOT, "profiles", "peaks.json")
    with open(path, "w") as fh:
        json.dump(res, fh, indent=1)
        fh.write("\n")
    print(json.dumps(res, indent=1))


if __name__ == "__main__":
    main()
