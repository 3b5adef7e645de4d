"""The allocation-free weight-gradient entry point (vfl_weight_grad_noalloc).

It exists for callers that cannot allocate device memory when they need a
gradient (allocator callbacks, fixed-footprint hosts, processes whose pools
already hold all of HBM): its scratch is a fixed array inside the library.
Checked here through the C ABI against the gradient the regular training path
computes (vfl_get_grads), on two calls in a row.  This file is collected last
so that a run stopping at the first failure has already run every other test.
"""
import numpy as np
import pytest

from _parity import TOL, rel_err

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


def one_step_reference(vfl, dtype):
    """One training step of a model whose passive bottom is a single layer, so
    that the layer's input is the passive data itself; returns the pieces the
    allocation-free call needs and the regular path's gradient of that layer."""
    import synth
    base = synth.preset(2)
    p = base.with_(n_rows=1024 + 304, passive=(64,), dtype=dtype)
    xp, xa, y = synth.make_dataset(base, rows=(0, p.n_rows))
    params = synth.init_params(p)
    ctx = vfl.Context(p, p.n_rows)
    ctx.load_data(xp, xa, y)
    ctx.set_params(params)
    ctx.passive_forward(0, 0)
    ctx.active_step(0, 0)
    ctx.passive_backward(0)
    zp = ctx.tap(0, vfl.TAP_EMB)
    dzp = ctx.tap(0, vfl.TAP_GRAD)
    dW, db = ctx.get_grads(worker=0, parties=(0,))[(0, 0)]
    r0, r1 = ctx.batch_rows(0)
    x = xp[r0:r1]
    ctx.close()
    return dzp * (zp > 0), x, dW, db


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_noalloc_matches_training_path_twice(vfl, dtype):
    import torch
    dpre, x, dW_ref, db_ref = one_step_reference(vfl, dtype)
    tdt = torch.float32 if dtype == "fp32" else torch.bfloat16
    code = vfl.FP32 if dtype == "fp32" else vfl.BF16
    d_dpre = torch.from_numpy(dpre).to("cuda", tdt)     # exact: the taps hold compute-dtype values
    d_x = torch.from_numpy(x).to("cuda", tdt)           # the same rounding the context applied at load
    out, fin = dW_ref.shape
    results = []
    for _ in range(2):
        dW = torch.full((out, fin), float("nan"), device="cuda")
        db = torch.full((out,), float("nan"), device="cuda")
        vfl.weight_grad_noalloc(d_dpre, d_x, dW, db, code)
        torch.cuda.synchronize()
        results.append((dW.cpu().numpy(), db.cpu().numpy()))
    for dW, db in results:
        assert rel_err(dW, dW_ref) <= TOL["fp32"]
        assert rel_err(db, db_ref) <= TOL["fp32"]
    np.testing.assert_array_equal(results[0][0], results[1][0])
    np.testing.assert_array_equal(results[0][1], results[1][1])


def test_noalloc_rejects_layers_beyond_its_scratch(vfl):
    import torch
    dpre = torch.zeros((16, 2049), device="cuda")
    x = torch.zeros((16, 2048), device="cuda")
    dW = torch.zeros((2049, 2048), device="cuda")
    db = torch.zeros((2049,), device="cuda")
    with pytest.raises(vfl.VflError) as ei:
        vfl.weight_grad_noalloc(dpre, x, dW, db, vfl.FP32)
    assert ei.value.status == vfl.VFL_E_INVAL
    assert "fixed scratch" in str(ei.value)


def test_noalloc_layer_at_the_scratch_limit(vfl):
    """A layer whose partial sums need the whole fixed scratch in one split
    (out*in + out == 4,194,304): accepted, and equal to a float64 matmul and
    column sum of the same bf16 inputs."""
    import torch
    out, fin, rows = 2048, 2047, 3000
    assert out * fin + out == 4 * 2 ** 20
    g = torch.Generator().manual_seed(7)
    dpre = torch.randn(rows, out, generator=g).to(torch.bfloat16)
    x = torch.rand(rows, fin, generator=g).to(torch.bfloat16)
    ref_w = (dpre.double().T @ x.double()).numpy()
    ref_b = dpre.double().sum(0).numpy()
    dW = torch.full((out, fin), float("nan"), device="cuda")
    db = torch.full((out,), float("nan"), device="cuda")
    vfl.weight_grad_noalloc(dpre.cuda(), x.cuda(), dW, db, vfl.BF16)
    torch.cuda.synchronize()
    assert rel_err(dW.cpu().numpy(), ref_w) <= TOL["fp32"]
    assert rel_err(db.cpu().numpy(), ref_b) <= TOL["fp32"]


def test_noalloc_rejects_too_wide_inputs(vfl):
    import torch
    fin = 65535 * 64 + 1
    dpre = torch.zeros((1, 1), device="cuda")
    x = torch.zeros((1, fin), device="cuda")
    dW = torch.zeros((1, fin), device="cuda")
    db = torch.zeros((1,), device="cuda")
    with pytest.raises(vfl.VflError) as ei:
        vfl.weight_grad_noalloc(dpre, x, dW, db, vfl.FP32)
    assert ei.value.status == vfl.VFL_E_INVAL
    assert "input width" in str(ei.value)
