"""The layer-chain forward (a bf16 bottom model's layers in one launch, its
activations kept in shared memory between layers) against the per-layer
tensor-core GEMMs it replaces: bit for bit on multiclass-shaped models
(27-256-256-128 bottoms) over an epoch with a ragged last batch, directly and
from a graph; and the chain is what runs (fewer launches a step)."""
import os

import numpy as np
import pytest

import synth
from _parity import new_context, schedule, setup

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


def run(vfl, q, xp, xa, y, params, n, tp, ta, chain, graph):
    if chain:
        os.environ.pop("VFL_DISABLE_CHAIN", None)
    else:
        os.environ["VFL_DISABLE_CHAIN"] = "1"
    try:
        ctx = new_context(vfl, q, xp, xa, y, params)
    finally:
        os.environ.pop("VFL_DISABLE_CHAIN", None)
    l0 = ctx.launches
    if graph:
        ctx.train_steps(0, 2, tp, ta)
        ctx.launch_graph(ctx.capture(2, n - 2, tp, ta))
    else:
        ctx.train_steps(0, n, tp, ta)
    ctx.synchronize()
    out = ctx.read_losses(0, n), ctx.get_params(), ctx.launches - l0
    ctx.close()
    return out


@pytest.mark.parametrize("workers,graph", [(1, False), (3, True)])
def test_chain_equals_per_layer(vfl, workers, graph):
    p = synth.preset(3).with_(workers=workers)
    q, xp, xa, y, params = setup(p, 2 * 4096 + 288)
    n = q.steps_per_epoch + 1
    tp, ta = schedule(q, n)
    la, pa, na = run(vfl, q, xp, xa, y, params, n, tp, ta, True, graph)
    lb, pb, nb = run(vfl, q, xp, xa, y, params, n, tp, ta, False, graph)
    np.testing.assert_array_equal(la, lb)
    for key, (W, b) in pa.items():
        np.testing.assert_array_equal(W, pb[key][0])
        np.testing.assert_array_equal(b, pb[key][1])
    if not graph:
        assert na == nb - 4 * n     # two 3-layer bottoms: 6 launches a step become 2
