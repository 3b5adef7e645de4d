"""System planning of PubSub-VFL (Sec. 4.2-4.3) -- TEST INFRASTRUCTURE ONLY.

The delay model of one iteration (Eq. 7-9): every term is coef * B^exp * w / C,
  T_A = (lambda_a B^gamma_a + phi_a B^beta_a + lambda_top B^gamma_top + phi_top B^beta_top) w_a / C_a,
  T_P = (lambda_p B^gamma_p + phi_p B^beta_p) w_p / C_p;
the communication delay (Eq. 10) (E + G) / B_b with E = G = B * bytes_per_row;
the memory bound (Eq. 14-15) B_max = min over the parties of ((M_max - M0) / rho)^(1/chi);
the objective (Eq. 17) O = max(T_A, T_P) + (E + G) / B_b; and Algorithm 2, the
exhaustive scan over the candidate batches (as given), then w_a, then w_p, that
keeps the first strict minimum.

Readings: the state cost printed after Eq. 17 writes phi_a in the passive term
and swaps the names of the worker ranges, and drops the communication term;
this follows Eq. 8 (phi_p), the ranges as Algorithm 2 loops them (w_a over
[P, Q], w_p over [M, N]) and Eq. 17's objective with the communication term,
which Algorithm 2 also adds.  The model's `w / C` form is kept as printed.
The fit of the constants is a least-squares line in log-log space.
"""
from __future__ import annotations

import math

import numpy as np

FIELDS = ("lambda_a", "gamma_a", "phi_a", "beta_a", "lambda_top", "gamma_top", "phi_top", "beta_top",
          "lambda_p", "gamma_p", "phi_p", "beta_p", "C_a", "C_p", "bytes_per_row", "bandwidth",
          "M_A0", "rho_A", "M_A_max", "M_P0", "rho_P", "M_P_max", "chi")


def _term(coef, b, expo):
    return 0.0 if coef == 0.0 else coef * b ** expo


def plan_bmax(m) -> float:
    """B_max of Eq. 15 (a party with rho <= 0 sets no bound)."""
    out = math.inf
    for m0, rho, mmax in ((m.M_A0, m.rho_A, m.M_A_max), (m.M_P0, m.rho_P, m.M_P_max)):
        if rho > 0.0:
            room = (mmax - m0) / rho
            if room < 0.0:
                raise ValueError("memory budget below the base consumption")
            out = min(out, room ** (1.0 / m.chi))
    return out


def plan_delay(m, w_a: int, w_p: int, b: float) -> float:
    """O(w_a, w_p, B) of Eq. 17."""
    t_a = (_term(m.lambda_a, b, m.gamma_a) + _term(m.phi_a, b, m.beta_a) +
           _term(m.lambda_top, b, m.gamma_top) + _term(m.phi_top, b, m.beta_top)) * w_a / m.C_a
    t_p = (_term(m.lambda_p, b, m.gamma_p) + _term(m.phi_p, b, m.beta_p)) * w_p / m.C_p
    return max(t_a, t_p) + 2.0 * b * m.bytes_per_row / m.bandwidth


def plan(m, wa_range, wp_range, batches):
    """Algorithm 2: (w_a, w_p, B, O) minimising Eq. 17 over the feasible candidates."""
    bmax = plan_bmax(m)
    best = None
    for b in batches:
        if not (1 <= b <= bmax):
            continue
        for wa in range(wa_range[0], wa_range[1] + 1):
            for wp in range(wp_range[0], wp_range[1] + 1):
                o = plan_delay(m, wa, wp, float(b))
                if best is None or o < best[3]:
                    best = (wa, wp, int(b), o)
    if best is None:
        raise ValueError("no feasible candidate")
    return best


def fit_power(x, t):
    """(coef, expo) of t = coef * x^expo, least squares on (log x, log t)."""
    expo, logc = np.polyfit(np.log(np.asarray(x, np.float64)), np.log(np.asarray(t, np.float64)), 1)
    return math.exp(logc), float(expo)
