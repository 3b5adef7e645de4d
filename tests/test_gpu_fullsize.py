"""The wide-dp workload at its full size (1,000,000 rows, 2000 binary features,
batch 8192, bf16, staleness 4, DP on the published gradient) in the launch
configuration bench.py times: a few steps enqueued directly, then a window of
steps captured as one CUDA graph and replayed.  The oracle runs the same first
steps on just the rows they train (step k < ceil(n / B) trains batch k in both),
so the per-step losses and the final weights can be compared with it."""
import numpy as np
import pytest

import oracle
import synth
from _parity import TOL, new_context, rel_err, schedule

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


def test_wide_dp_full_size_bench_configuration(vfl):
    p = synth.preset(4)
    assert p.n_rows == 1_000_000 and p.batch == 8192
    warm, window = 3, 5
    n = warm + window
    xp, xa, y = synth.make_dataset(p)
    params = synth.init_params(p)
    tp, ta = schedule(p, n)
    ctx = new_context(vfl, p, xp, xa, y, params)
    ctx.train_steps(0, warm, tp, ta)                     # the bench's warm-up: direct enqueue
    ctx.launch_graph(ctx.capture(warm, window, tp, ta))  # a timed window: one captured graph
    ctx.synchronize()
    got = ctx.read_losses(0, n)
    gp = ctx.get_params()
    ctx.close()

    rows = n * p.batch
    q = p.with_(n_rows=rows)
    o = oracle.Oracle(q, xp[:rows], xa[:rows], y[:rows], params, dp_seed=q.seed)
    ref, _ = o.run(tp, ta, n)
    assert np.isfinite(got).all()
    assert np.abs(got - ref).max() <= TOL["bf16"] * np.abs(ref).max(), (got, ref)
    out_layer = (2, len(p.top) - 1)
    for key, (W, b) in gp.items():
        assert rel_err(W, o.current_params()[key][0]) < TOL["bf16"], key
        if key != out_layer:   # the output bias: a column sum of d(logits) whose terms cancel
            assert rel_err(b, o.current_params()[key][1]) < TOL["bf16"], key
