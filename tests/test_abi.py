"""The C-ABI library without a GPU: it loads, exports every function the header
declares, validates its arguments, and its host-side schedule matches the
oracle bit for bit."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def vfl():
    from paper_2510_12494_gb300 import build
    build.build()
    import paper_2510_12494_gb300 as v
    return v


def declared_functions():
    src = open(os.path.join(ROOT, "include", "vfl.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(vfl_[a-z_0-9]+)\s*\(", src)))


def test_library_exports_every_declared_function(vfl):
    names = declared_functions()
    assert len(names) >= 20
    L = ctypes.CDLL(vfl.LIB_PATH)
    missing = [n for n in names if not hasattr(L, n)]
    assert not missing, missing
    assert set(names) == set(vfl.EXPORTS), set(names) ^ set(vfl.EXPORTS)


def test_config_struct_layout_matches_header(vfl):
    # 5 + 3*8 int32, then loss, dtype, batch, lr, staleness, workers, clip, sigma (4 bytes each), then u64,
    # then the int32 dp_target and ps_dt0
    assert ctypes.sizeof(vfl.VflConfig) == (5 + 24 + 8) * 4 + 4 + 8 + 8
    assert vfl.VflConfig.dp_seed.offset % 8 == 0
    assert vfl.VflConfig.dp_target.offset == vfl.VflConfig.dp_seed.offset + 8
    assert vfl.VflConfig.ps_dt0.offset == vfl.VflConfig.dp_target.offset + 4


@pytest.mark.parametrize("S", [0, 1, 2, 4, 7])
@pytest.mark.parametrize("seed", [0, 1, 0xDEADBEEF12345])
@pytest.mark.parametrize("kind", [0, 1, 2])
def test_schedule_matches_oracle_bit_exactly(vfl, S, seed, kind):
    n = 700
    tp, ta = vfl.make_schedule(seed, S, kind, n)
    op, oa = oracle.make_schedule(seed, S, kind, n)
    np.testing.assert_array_equal(tp, op)
    np.testing.assert_array_equal(ta, oa)


def test_schedule_rejects_bad_arguments(vfl):
    with pytest.raises(vfl.VflError):
        vfl.make_schedule(0, -1, 0, 5)
    with pytest.raises(vfl.VflError):
        vfl.make_schedule(0, 1, 9, 5)


@pytest.mark.parametrize("cid", [1, 2, 3, 4, 5])
def test_workspace_sizes(vfl, cid):
    p = synth.preset(cid)
    b = vfl.workspace_bytes(p, p.n_rows)
    es = 4 if p.dtype == "fp32" else 2
    assert b >= p.n_rows * (p.d_passive + p.d_active) * es
    assert b < 64 * 2 ** 30


def test_gdp_sigma_matches_the_oracle(vfl):
    import oracle
    for args in ((1.0, 1024, 30000, 150), (0.25, 256, 4096, 16), (3.0, 8192, 1000000, 123)):
        assert vfl.gdp_sigma(*args) == pytest.approx(oracle.gdp_sigma(*args), rel=1e-15)
    with pytest.raises(vfl.VflError):
        vfl.gdp_sigma(0.0, 1024, 30000, 150)


def test_invalid_configs_are_rejected(vfl):
    p = synth.preset(1)
    for bad in (dict(batch=0), dict(staleness=-1), dict(staleness=40), dict(workers=0), dict(workers=17),
                dict(top=(32, 2)), dict(loss="ce", top=(32, 1)), dict(lr=-1.0)):
        with pytest.raises(vfl.VflError):
            vfl.workspace_bytes(p.with_(**bad), 100)
    with pytest.raises(vfl.VflError):
        vfl.workspace_bytes(p, 0)
    for bad in (dict(ps_dt0=-1), dict(ps_dt0=4, staleness=1, workers=2)):
        with pytest.raises(vfl.VflError):
            vfl.workspace_bytes(p.with_(**bad), 100)
    cfg = vfl.make_config(p.with_(dp_clip=1.0, dp_target="emb"))
    assert cfg.dp_target == vfl.DP_EMB
    cfg.dp_target = 7
    out = ctypes.c_uint64()
    assert vfl.lib().vfl_workspace_bytes(ctypes.byref(cfg), 100, ctypes.byref(out)) == vfl.VFL_E_INVAL


@pytest.mark.parametrize("dt0", [1, 2, 3, 4, 5, 8, 13, 40])
def test_ps_interval_matches_the_oracle(vfl, dt0):
    for t in range(1, 6 * dt0 + 3):
        assert vfl.ps_interval(t, dt0) == oracle.ps_interval(t, dt0), (t, dt0)
    with pytest.raises(vfl.VflError):
        vfl.ps_interval(0, dt0)
    with pytest.raises(vfl.VflError):
        vfl.ps_interval(1, 0)


def test_ps_workspace_holds_a_master_per_replica(vfl):
    p = synth.preset(2).with_(workers=4, staleness=0)
    base = vfl.workspace_bytes(p, p.n_rows)
    with_ps = vfl.workspace_bytes(p.with_(ps_dt0=4), p.n_rows)
    n_params = 0
    for widths, d_in in ((p.passive, p.d_passive), (p.active, p.d_active), (p.top, p.e_active + p.e_passive)):
        for o in widths:
            n_params += o * d_in + o
            d_in = o
    # three more fp32 masters (and the version ring grows from one slot to one per worker)
    assert with_ps - base >= 3 * n_params * 4


@pytest.mark.parametrize("rate", [0.0, 0.01, 0.3, 0.999, 1.0])
@pytest.mark.parametrize("seed", [0, 7, 0xDEADBEEF12345])
def test_drop_draws_match_oracle_bit_exactly(vfl, rate, seed):
    np.testing.assert_array_equal(vfl.make_drops(seed, rate, 3000), oracle.make_drops(seed, rate, 3000))


def test_drop_draws_reject_bad_rates(vfl):
    for rate in (-0.1, 1.5, float("nan")):
        with pytest.raises(vfl.VflError):
            vfl.make_drops(0, rate, 5)
