"""GPU parity of the DP mechanism on the published embedding (App. C): the
clipped and noised embedding the active party consumes, the straight-through
passive backward, every gradient and updated parameter, against the oracle on
the same seeded inputs (tolerances as in test_gpu_parity)."""
import numpy as np
import pytest

import synth
from _parity import new_context, run_sequential, schedule, setup

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


def assert_parity(vfl, q, steps=None):
    worst, failures = run_sequential(vfl, q, q.n_rows, steps=steps)
    assert not failures, f"{q.name}: {failures[:3]}; worst {sorted(worst.items(), key=lambda t: -t[1])[:6]}"
    return worst


def kernels_used(vfl, q, steps=2):
    q2, xp, xa, y, params = setup(q, q.n_rows)
    ctx = new_context(vfl, q2, xp, xa, y, params)
    tp, ta = schedule(q2, steps)
    ctx.profile(True)
    ctx.train_steps(0, steps, tp, ta)
    ctx.profile(False)
    return {k: v[0] for k, v in ctx.profile_summary().items()}


@pytest.mark.parametrize("path", ["fused", "generic"])
@pytest.mark.parametrize("clip,sigma", [(1.0, 1.0), (0.3, 0.0), (1e30, 0.0)])
def test_embedding_dp_fp32(vfl, clip, sigma, path, monkeypatch):
    """fp32, S = 2 seeded, a ragged last batch: clipping with noise, clipping
    alone (every row scaled) and neither (the mechanism's identity case), on the
    fused row kernels (the mechanism in the passive forward's epilogue) and on
    the per-layer kernels."""
    if path == "generic":
        monkeypatch.setenv("VFL_DISABLE_FUSED", "1")
    q = synth.preset(1).with_(n_rows=2 * 256 + 37, staleness=2, schedule="seeded", dp_clip=clip, dp_sigma=sigma,
                              dp_target="emb")
    used = kernels_used(vfl, q)
    assert ("fused_passive_fwd" in used) == (path == "fused"), used
    assert_parity(vfl, q)


def test_embedding_dp_bf16_wide(vfl):
    """The wide-dp workload with the embedding as the DP target (bf16, S = 4)."""
    q = synth.preset(4).with_(n_rows=8192 + 576, dp_target="emb")
    assert_parity(vfl, q)


def test_embedding_dp_is_not_the_gradient_mechanism(vfl):
    """Same seed and constants, the two targets: the published embeddings differ
    (noised only under the embedding target) and so do the losses."""
    base = synth.preset(1).with_(n_rows=1024, staleness=2, schedule="seeded", dp_clip=1.0, dp_sigma=1.0)
    out = {}
    for target in ("grad", "emb"):
        q, xp, xa, y, params = setup(base.with_(dp_target=target), 1024)
        ctx = new_context(vfl, q, xp, xa, y, params)
        tp, ta = schedule(q, 4)
        ctx.train_steps(0, 4, tp, ta)
        out[target] = (ctx.tap(3, vfl.TAP_EMB), ctx.read_losses(0, 4))
    assert not np.allclose(out["grad"][0], out["emb"][0])
    assert not np.allclose(out["grad"][1][1:], out["emb"][1][1:])
