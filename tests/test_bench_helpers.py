"""Host logic of the measurement and of the boundary's documentation, without a GPU:
- every function vfl.h declares carries a comment naming the paper passage it implements (or saying it
  has no counterpart in the paper);
- bench.py's timing plan (>= 5 windows, an end-to-end leg of at least one epoch), its per-kernel traffic
  lookup in the committed ncu captures (matched by kernel, workload and the source file's hash), and its
  choice of the dominant kernel."""
import json
import os
import re
import types

import pytest

import bench
import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PASSAGE = re.compile(r"Sec\. ?\d|Eq\. ?\d|Algorithm ?\d|App\. ?[A-Z]|Assumption ?\d|"
                     r"no counterpart in the paper|the paper has no\s+(\*\s+)?counterpart", re.I)


def header_declarations():
    """(function name, the comment block right above its declaration) for every declared function."""
    src = open(os.path.join(ROOT, "include", "vfl.h")).read()
    out = []
    for m in re.finditer(r"^(?:vfl_status|int64_t|const char\*|void)\s+(vfl_[a-z_0-9]+)\s*\(", src, flags=re.M):
        head = src[: m.start()].rstrip()
        comment = ""
        # the nearest comment ending right above (a /* */ block, possibly after other declarations of a group)
        end = head.rfind("*/")
        if end >= 0:
            start = head.rfind("/*", 0, end)
            comment = head[start : end + 2]
        out.append((m.group(1), comment))
    return out


def test_every_declared_function_is_found():
    names = [n for n, _ in header_declarations()]
    assert len(names) >= 40 and len(set(names)) == len(names)
    assert "vfl_bind_host_data_bits" in names and "vfl_train_steps" in names


@pytest.mark.parametrize("name,comment", header_declarations(), ids=lambda x: x if isinstance(x, str) and
                         x.startswith("vfl_") else "")
def test_declaration_cites_a_passage(name, comment):
    assert PASSAGE.search(comment), f"{name}: no passage cited in its comment"


def test_timing_plan_has_five_windows_and_an_epoch_long_e2e_leg():
    p = synth.preset(4)
    nb = p.steps_per_epoch
    for steps in (None, 1, 20, 5 * nb + 3):
        args = types.SimpleNamespace(steps=steps, warmup=1)
        W, K, window, n_e2e = bench.plan(p, args)
        assert W >= 3
        assert K // window >= 5 or K < 5
        assert n_e2e >= nb


def test_profiled_traffic_matches_kernel_workload_and_source():
    rec = json.load(open(os.path.join(ROOT, "profiles", "kernels.json")))
    entry = next(k for k in rec["kernels"] if k["kernel"] == "tc_dw_kernel" and k["workload"] == "wide-dp")
    got = bench.profiled_traffic("tc_dw_kernel", ["gemm_tc_dw"], "wide-dp", entry["units_per_launch"])
    assert got is not None and got["source"] == "profiles/" + entry["file"]
    ls = [x for x in entry["launches"] if x["class"] == "gemm_tc_dw"]
    want = sum((x["dram_read"] or 0) + (x["dram_write"] or 0) for x in ls) / len(ls)
    assert abs(got["bytes_per_launch"] - want) <= 1e-6 * want
    # scaled by the units a launch processes
    half = bench.profiled_traffic("tc_dw_kernel", ["gemm_tc_dw"], "wide-dp", entry["units_per_launch"] // 2)
    assert abs(half["bytes_per_launch"] - want / 2) <= 1e-6 * want
    # another workload's capture is not used, and nothing matches an unknown workload
    assert bench.profiled_traffic("tc_dw_kernel", ["gemm_tc_dw"], "no-such-workload", 1) is None


def test_profiled_traffic_is_null_once_the_source_changes(monkeypatch):
    monkeypatch.setattr(bench, "source_digest", lambda kernel: "0" * 64)
    assert bench.profiled_traffic("tc_dw_kernel", ["gemm_tc_dw"], "wide-dp", 8192) is None


def test_every_profile_names_its_source_and_summary():
    """Each committed ncu capture names an existing kernel source by path and SHA-256 (bench.py compares the
    hash with the file as it stands), its summary file, its units and a per-launch DRAM figure."""
    rec = json.load(open(os.path.join(ROOT, "profiles", "kernels.json")))
    assert rec["kernels"]
    for k in rec["kernels"]:
        assert os.path.exists(os.path.join(ROOT, k["source"])), k["source"]
        assert re.fullmatch(r"[0-9a-f]{64}", k["source_sha256"]), k["file"]
        assert os.path.exists(os.path.join(ROOT, "profiles", k["file"])), k["file"]
        assert k["units_per_launch"] > 0 and k["dram_bytes_per_launch"] >= 0 and k["launches"]


def test_roofline_picks_the_launch_lists_largest_kernel():
    """With a current launch list, the dominant kernel is the one with the largest warm share there, and its
    fraction is the algorithmic work per launch over the event-timed duration against the measured peak."""
    pk = {"bf16_tflops_sustained": 1000.0, "x3tf32_tflops": 100.0, "ffma_tflops": 80.0, "hbm_gbs": 7000.0,
          "src": "test", "fp32_src": "test"}
    # class -> (launches, total ms, total flops, total bytes); event time would pick the GEMM
    prof = {"gemm_tc_dw": (10, 0.2, 10 * 4e9, 10 * 1e7), "gemm_tc_fwd": (20, 0.5, 20 * 1e9, 20 * 1e7),
            "sgd": (5, 0.01, 0.0, 5 * 1e6)}
    r = bench.roofline(prof, pk, "wide-dp", 8192)
    ll = json.load(open(os.path.join(ROOT, "profiles", "launches.json")))["workloads"]["wide-dp"]["kernels"]
    fresh = all(bench.file_digest(f) == h for f, h in
                json.load(open(os.path.join(ROOT, "profiles", "launches.json")))["workloads"]["wide-dp"]
                ["sources_sha256"].items())
    if fresh:
        top = max((k for k in ("tc_dw_kernel", "tc_gemm_kernel", "sgd_kernel") if k in ll),
                  key=lambda k: ll[k]["warm_share"])
        assert r["kernel"] == top
        assert r["selected_by"].startswith("largest warm share")
    else:
        assert r["kernel"] == "tc_gemm_kernel"
    n, ms, flops, _ = (prof["gemm_tc_dw"] if r["kernel"] == "tc_dw_kernel" else prof["gemm_tc_fwd"])
    assert r["bound"] == "tensor" and r["peak"] == 1000.0
    assert abs(r["achieved"] - flops / (ms / 1e3) / 1e12) < 1e-9
    assert abs(r["frac"] - r["achieved"] / 1000.0) < 1e-12
    assert abs(r["avg_us"] - ms / n * 1e3) < 1e-9
