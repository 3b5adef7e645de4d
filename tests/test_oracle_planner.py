"""Pins of the oracle's system planner (Sec. 4.2-4.3, Eq. 7-17, Algorithm 2):
optima worked out by hand (the crossing of a falling and a rising delay, the
memory bound of Eq. 15, the communication term), the monotonicity the model
implies in the worker counts, and the power-law fit recovering known
constants (the paper's Table 8 values as ground truth)."""
import math
from types import SimpleNamespace

import numpy as np
import pytest

import oracle


def model(**kw):
    base = {f: 0.0 for f in oracle.PLAN_FIELDS}
    base.update(C_a=1.0, C_p=1.0, bandwidth=1.0, chi=1.0)
    base.update(kw)
    return SimpleNamespace(**base)


def test_crossing_of_falling_and_rising_delays():
    # T_A = 100 / B falls, T_P = B rises; they cross at B = 10.  Over {4, 8, 16, 32} the max is
    # 25, 12.5, 16, 32: B = 8 wins with O = 12.5.
    m = model(lambda_a=100.0, gamma_a=-1.0, lambda_p=1.0, gamma_p=1.0)
    assert oracle.plan(m, (1, 1), (1, 1), [4, 8, 16, 32]) == (1, 1, 8, 12.5)
    # order of the candidates does not matter for a strict minimum
    assert oracle.plan(m, (1, 1), (1, 1), [32, 16, 8, 4])[2] == 8


def test_memory_bound_of_eq15():
    # active: ((10 - 2) / 0.5)^(1/2) = 4; passive: ((50 - 1) / 1)^(1/2) = 7 -> B_max = 4
    m = model(lambda_a=100.0, gamma_a=-1.0, M_A0=2.0, rho_A=0.5, M_A_max=10.0, M_P0=1.0, rho_P=1.0,
              M_P_max=50.0, chi=2.0)
    assert oracle.plan_bmax(m) == pytest.approx(4.0, rel=1e-15)
    # T_A = 100 / B alone would take the largest batch; 8 is over the bound, so 4
    assert oracle.plan(m, (1, 1), (1, 1), [2, 4, 8])[2] == 4
    with pytest.raises(ValueError):
        oracle.plan(m, (1, 1), (1, 1), [8, 16])
    # no memory model: no bound
    assert oracle.plan_bmax(model()) == math.inf


def test_communication_term():
    # equal compute at every batch (exponent 0); (E + G) / B_b = 2 B * 3 / 6 = B decides: the smallest batch
    m = model(lambda_a=5.0, lambda_p=5.0, bytes_per_row=3.0, bandwidth=6.0)
    assert oracle.plan_delay(m, 1, 1, 16.0) == pytest.approx(5.0 + 16.0)
    assert oracle.plan(m, (1, 1), (1, 1), [64, 16, 32])[2:] == (16, pytest.approx(21.0))


def test_passive_backward_uses_its_own_constant():
    # the passive party's time is lambda_p B^gamma_p + phi_p B^beta_p (Eq. 8), not phi_a
    m = model(phi_a=1000.0, lambda_p=1.0, gamma_p=1.0, phi_p=2.0, beta_p=1.0, C_a=1e9)
    assert oracle.plan_delay(m, 1, 1, 4.0) == pytest.approx(12.0)


@pytest.mark.parametrize("seed", range(5))
def test_smallest_worker_counts_win_under_the_printed_model(seed):
    # every term scales with w / C, so O never decreases with either worker count: the scan's first
    # strict minimum is at the lower ends of both ranges
    rng = np.random.default_rng(seed)
    kw = {f: float(rng.uniform(0.01, 2.0)) for f in ("lambda_a", "phi_a", "lambda_top", "phi_top", "lambda_p", "phi_p")}
    kw.update({f: float(rng.uniform(-1.2, 1.2)) for f in ("gamma_a", "beta_a", "gamma_top", "beta_top", "gamma_p", "beta_p")})
    m = model(C_a=32.0, C_p=32.0, bytes_per_row=float(rng.uniform(0, 1)), bandwidth=100.0, **kw)
    wa, wp, b, o = oracle.plan(m, (2, 9), (3, 7), [16, 32, 64, 128, 256, 512, 1024])
    assert (wa, wp) == (2, 3)
    assert o == min(oracle.plan_delay(m, 2, 3, float(bb)) for bb in (16, 32, 64, 128, 256, 512, 1024))


def test_paper_constants_take_the_largest_batch():
    # Table 8's exponents are all negative: every compute delay falls with B; without a communication
    # cost or a memory bound the largest candidate wins, on C_a + C_p = 64 cores split evenly
    t8 = dict(lambda_a=0.018, gamma_a=-0.8015, lambda_p=0.010, gamma_p=-1.0071, lambda_top=0.011,
              gamma_top=-0.7514, phi_a=0.066, beta_a=-0.6069, phi_p=0.038, beta_p=-1.0546, beta_top=-0.7834,
              phi_top=0.072)
    m = model(C_a=32.0, C_p=32.0, **t8)
    assert oracle.plan(m, (2, 50), (2, 50), [16, 32, 64, 128, 256, 512, 1024])[:3] == (2, 2, 1024)


def test_fit_recovers_power_laws():
    b = np.array([16, 32, 64, 128, 256, 512, 1024], np.float64)
    for coef, expo in ((0.018, -0.8015), (0.066, -0.6069), (0.038, -1.0546), (3.5, 1.0)):
        c, e = oracle.fit_power(b, coef * b ** expo)
        assert c == pytest.approx(coef, rel=1e-9) and e == pytest.approx(expo, abs=1e-9)
    # multiplicative noise of a few per cent moves the exponent by little
    rng = np.random.default_rng(3)
    c, e = oracle.fit_power(b, 2.0 * b ** 0.7 * np.exp(rng.normal(0, 0.02, b.size)))
    assert abs(e - 0.7) < 0.02 and abs(c / 2.0 - 1) < 0.1
