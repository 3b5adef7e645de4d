"""GPU parity on the edge cases of the step: ragged tails of 1 and 17 rows,
batches of a single row, the largest staleness bound, models at and just past
the limits of the fused kernels and of the folded output layer, and one-layer
towers.  Each case runs the CUDA path through the C ABI step by step against
the oracle on the same seeded inputs (tolerances as in test_gpu_parity), and
checks which kernels carried it."""
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


def kernels_used(vfl, q, steps=2):
    """Kernel classes (name -> launches) of the first `steps` steps of q."""
    q2, xp, xa, y, params = setup(q, q.n_rows)
    ctx = new_context(vfl, q2, xp, xa, y, params)
    tp, ta = schedule(q2, steps)
    ctx.profile(True)
    ctx.train_steps(0, steps, tp, ta)
    ctx.profile(False)
    return {k: v[0] for k, v in ctx.profile_summary().items()}


def assert_parity(vfl, q, steps=None):
    worst, failures = run_sequential(vfl, q, q.n_rows, steps=steps)
    assert not failures, f"{q.name}: {failures[:3]}; worst {sorted(worst.items(), key=lambda t: -t[1])[:6]}"


# a small bf16 model of the multiclass shape
SMALL_BF16 = synth.preset(3).with_(cid=0, name="small-bf16", n_rows=2 * 256 + 40, passive=(64, 32), active=(64, 32),
                                   top=(64, 7), batch=256)


@pytest.mark.parametrize("cid,tail", [(1, 1), (1, 17), (2, 1), (2, 15), (3, 1), (3, 17)])
def test_ragged_tail(vfl, cid, tail):
    """An epoch whose last batch holds `tail` rows: one partial 16-row tile,
    one row past a full tile, a tensor-core row block of one row."""
    p = synth.preset(cid)
    q = p.with_(n_rows=2 * p.batch + tail)
    assert_parity(vfl, q, steps=4)


@pytest.mark.parametrize("base", ["tiny", "bf16"])
def test_single_row_batches(vfl, base):
    q = (synth.preset(1) if base == "tiny" else SMALL_BF16).with_(batch=1, n_rows=5)
    assert_parity(vfl, q, steps=7)


def test_largest_staleness_bound(vfl):
    """S = 15, the largest the context takes: sixteen weight versions and
    channel slots in flight, with three worker streams per party."""
    q = synth.preset(1).with_(staleness=15, schedule="seeded", workers=3)
    assert_parity(vfl, q, steps=40)


# fp32, 256-wide inputs; the active step stages f_a and g: with f_a = 256-32-64 its
# shared memory is 212 KB, within the 227 KB a block may use; with f_a = 256-64-64 it is
# 253 KB and the model runs on the per-layer kernels
WIDE = synth.preset(1).with_(cid=0, name="wide-fp32", n_rows=2 * 512 + 100, d_passive=256, d_active=256, passive=(64, 64),
                             active=(32, 64), top=(64, 1), batch=512, staleness=2, schedule="seeded")


def test_fused_at_width_limit(vfl):
    used = kernels_used(vfl, WIDE)
    assert used.get("fused_active_step", 0) == 2, used
    assert_parity(vfl, WIDE)


def test_past_fused_shared_memory_falls_back(vfl):
    q = WIDE.with_(active=(64, 64))
    used = kernels_used(vfl, q)
    assert "fused_active_step" not in used and "fused_passive_fwd" not in used, used
    assert_parity(vfl, q)


def test_past_fused_width_falls_back(vfl):
    q = WIDE.with_(d_passive=264, active=(32, 64))
    used = kernels_used(vfl, q)
    assert "fused_active_step" not in used, used
    assert_parity(vfl, q)


@pytest.mark.parametrize("n_out", [2, 16, 17])
def test_fused_softmax_widths(vfl, n_out):
    """Softmax cross-entropy on the fused path: the output layer folded into
    the hidden layer's epilogue up to 16 outputs, a row-tile layer past that."""
    q = synth.preset(1).with_(cid=0, top=(32, n_out), loss="ce")
    used = kernels_used(vfl, q)
    assert used.get("fused_active_step", 0) == 2, used
    assert_parity(vfl, q)


def test_generic_softmax_two_classes(vfl, monkeypatch):
    """Two-class softmax on the per-layer kernels: the output bias gradient is
    a sum of per-row terms that nearly cancel."""
    monkeypatch.setenv("VFL_DISABLE_FUSED", "1")
    q = synth.preset(1).with_(cid=0, top=(32, 2), loss="ce")
    assert "fused_active_step" not in kernels_used(vfl, q)
    assert_parity(vfl, q)


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_one_layer_towers(vfl, dtype):
    """Bottoms of one layer and a top of one (output) layer."""
    base = synth.preset(1) if dtype == "fp32" else SMALL_BF16
    q = base.with_(passive=(16,), active=(16,), top=(base.top[-1],))
    assert_parity(vfl, q, steps=6)


@pytest.mark.parametrize("n_out,head", [(12, True), (13, False)])
def test_bf16_head_limit(vfl, n_out, head):
    """The bf16 output layer and loss run as one kernel up to 12 outputs, as
    separate GEMM and loss kernels past that."""
    q = SMALL_BF16.with_(top=(64, n_out))
    used = kernels_used(vfl, q)
    assert ("head_loss" in used) == head and ("loss" in used) != head, used
    assert_parity(vfl, q, steps=4)


@pytest.mark.parametrize("dtype", ["fp32", "bf16"])
def test_unit_dimensions(vfl, dtype):
    """Every GEMM dimension at 1 somewhere: one feature per party, width-1 layers and cut layers, one logit
    (M = 1 is the single-row batch case above)."""
    base = synth.preset(1) if dtype == "fp32" else SMALL_BF16.with_(loss="bce")
    q = base.with_(cid=0, name=f"unit-{dtype}", d_passive=1, d_active=1, passive=(1,), active=(3, 1), top=(1, 1),
                   loss="bce", n_rows=300, batch=128)
    assert_parity(vfl, q, steps=5)
