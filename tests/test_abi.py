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


def _rand_plan_model(vfl, rng):
    kw = {f: float(rng.uniform(0.01, 2.0)) for f in ("lambda_a", "phi_a", "lambda_top", "phi_top", "lambda_p", "phi_p")}
    kw.update({f: float(rng.uniform(-1.2, 0.4)) for f in ("gamma_a", "beta_a", "gamma_top", "beta_top", "gamma_p",
                                                           "beta_p")})
    kw.update(C_a=float(rng.uniform(1, 64)), C_p=float(rng.uniform(1, 64)), bytes_per_row=float(rng.uniform(0, 2e-3)),
              bandwidth=float(rng.uniform(1, 10)), M_A0=1.0, rho_A=float(rng.uniform(1e-4, 1e-2)),
              M_A_max=float(rng.uniform(5, 50)), M_P0=2.0, rho_P=float(rng.uniform(1e-4, 1e-2)),
              M_P_max=float(rng.uniform(5, 50)), chi=float(rng.uniform(0.8, 1.5)))
    return kw


@pytest.mark.parametrize("seed", range(8))
def test_planner_matches_oracle(vfl, seed):
    from types import SimpleNamespace
    rng = np.random.default_rng(100 + seed)
    kw = _rand_plan_model(vfl, rng)
    m, om = vfl.plan_model(**kw), SimpleNamespace(**kw)
    assert vfl.plan_bmax(m) == pytest.approx(oracle.plan_bmax(om), rel=1e-13)
    for wa, wp, b in ((1, 1, 16.0), (3, 7, 333.0), (50, 2, 1024.0)):
        assert vfl.plan_delay(m, wa, wp, b) == pytest.approx(oracle.plan_delay(om, wa, wp, b), rel=1e-13)
    batches = [16, 32, 64, 128, 256, 512, 1024, 2048, 4096]
    try:
        want = oracle.plan(om, (1, 6), (2, 5), batches)
    except ValueError:
        with pytest.raises(vfl.VflError):
            vfl.plan(m, (1, 6), (2, 5), batches)
        return
    got = vfl.plan(m, (1, 6), (2, 5), batches)
    assert got[:3] == want[:3]
    assert got[3] == pytest.approx(want[3], rel=1e-13)
    x = np.array([16, 64, 256, 1024, 4096], np.float64)
    t = 0.5 * x ** 0.8 * np.exp(rng.normal(0, 0.05, x.size))
    c1, e1 = vfl.fit_power(x, t)
    c2, e2 = oracle.fit_power(x, t)
    assert c1 == pytest.approx(c2, rel=1e-10) and e1 == pytest.approx(e2, rel=1e-10)


def test_planner_rejects_bad_arguments(vfl):
    m = vfl.plan_model(lambda_a=1.0)
    for args in (((2, 1), (1, 1), [16]), ((0, 1), (1, 1), [16]), ((1, 1), (1, 1), [])):
        with pytest.raises(vfl.VflError):
            vfl.plan(m, *args)
    with pytest.raises(vfl.VflError):
        vfl.plan(vfl.plan_model(lambda_a=1.0, C_a=0.0), (1, 1), (1, 1), [16])
    with pytest.raises(vfl.VflError):
        vfl.plan_bmax(vfl.plan_model(M_A0=5.0, rho_A=1.0, M_A_max=1.0))
    with pytest.raises(vfl.VflError):
        vfl.fit_power([4.0, 4.0], [1.0, 2.0])
    with pytest.raises(vfl.VflError):
        vfl.fit_power([1.0, 2.0], [1.0, -2.0])
