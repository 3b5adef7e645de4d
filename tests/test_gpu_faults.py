"""Failure detection without a GPU fault: ordering violations are refused on
the host, a bounded device-side wait on a channel nobody publishes gives up
with VFL_E_TIMEOUT, a stale channel header is reported as VFL_E_VERSION, and
the context keeps working (and stays exact) afterwards."""
import numpy as np
import pytest

import oracle
from _parity import new_context, rel_err, schedule, setup

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


@pytest.fixture
def ctx(vfl):
    import synth
    q, xp, xa, y, params = setup(synth.preset(2), 3 * 1024 + 304)
    c = new_context(vfl, q, xp, xa, y, params)
    c._data = (q, xp, xa, y, params)
    yield c
    c.close()


def test_out_of_order_calls_are_refused(vfl, ctx):
    E = vfl.VFL_E_STATE
    for call in (lambda: ctx.active_step(0, 0),            # no embedding published yet
                 lambda: ctx.passive_backward(0),          # no gradient published yet
                 lambda: ctx.passive_forward(1, 0),        # steps publish in order
                 lambda: ctx.passive_forward(0, 1)):       # tau_p > k
        with pytest.raises(vfl.VflError) as ei:
            call()
        assert ei.value.status == E
    ctx.passive_forward(0, 0)
    with pytest.raises(vfl.VflError) as ei:
        ctx.set_cursor(0)                                  # a step is in flight
    assert ei.value.status == E
    ctx.active_step(0, 0)
    ctx.passive_backward(0)
    ctx.passive_forward(1, 1)
    ctx.active_step(1, 0)
    ctx.passive_backward(1)
    with pytest.raises(vfl.VflError) as ei:
        ctx.passive_forward(2, 3)                          # beyond the staleness bound S = 2
    assert ei.value.status == E


def test_bounded_wait_times_out_and_context_survives(vfl, ctx):
    q, xp, xa, y, params = ctx._data
    # nothing ever publishes step 7: the device-side wait gives up instead of hanging
    with pytest.raises(vfl.VflError) as ei:
        ctx.wait_channel(0, 7, 20000)
    assert ei.value.status == vfl.VFL_E_TIMEOUT
    with pytest.raises(vfl.VflError) as ei:
        ctx.wait_channel(1, 7, 20000)
    assert ei.value.status == vfl.VFL_E_TIMEOUT
    # the context still trains, exactly
    tp, ta = schedule(q, 3)
    ctx.train_steps(0, 3, tp, ta)
    ctx.wait_channel(0, 2, 20000)                          # published: returns at once
    o = oracle.Oracle(q, xp, xa, y, params)
    ref, _ = o.run(tp, ta, 3)
    assert rel_err(ctx.read_losses(0, 3), ref) < 1e-5


def test_stale_header_is_reported(vfl, ctx):
    q, *_ = ctx._data
    tp, ta = schedule(q, 4)
    ctx.train_steps(0, 4, tp, ta)
    ctx.check_channel(0, 3)
    ctx.check_channel(1, 3)
    # slot 0 (S + 1 = 3 slots) now carries step 3; a subscriber of step 0 must notice
    with pytest.raises(vfl.VflError) as ei:
        ctx.check_channel(0, 0)
    assert ei.value.status == vfl.VFL_E_VERSION
    with pytest.raises(vfl.VflError) as ei:
        ctx.check_channel(1, 0)
    assert ei.value.status == vfl.VFL_E_VERSION
    ctx.check_channel(0, 3)                                # the status word was cleared


def test_invalid_arguments(vfl, ctx):
    for call in (lambda: ctx.wait_channel(2, 0, 10), lambda: ctx.wait_channel(0, 0, 0),
                 lambda: ctx.check_channel(0, -1), lambda: ctx.read_losses(0, 5)):
        with pytest.raises(vfl.VflError) as ei:
            call()
        assert ei.value.status == vfl.VFL_E_INVAL
