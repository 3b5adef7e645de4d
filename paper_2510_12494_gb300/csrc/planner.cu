// System planning of PubSub-VFL (Sec. 4.2-4.3): the delay model of Eq. 7-12, the memory bound of
// Eq. 14-15, the objective of Eq. 17 and the exhaustive search of Algorithm 2, plus the power-law
// fit that turns measured delays into the model's constants.  Host code only.
#include <algorithm>
#include <cmath>
#include <limits>

#include "vfl.h"

namespace {

// coef * B^expo, the form of every term of Eq. 7-9
double term(double coef, double batch, double expo) { return coef == 0.0 ? 0.0 : coef * std::pow(batch, expo); }

// ((M_max - M0) / rho)^(1/chi) of one party (+inf when rho <= 0), or NaN when the budget is below M0
double party_bmax(double m0, double rho, double mmax, double chi) {
    if (!(rho > 0.0)) return std::numeric_limits<double>::infinity();
    const double room = (mmax - m0) / rho;
    if (room < 0.0) return std::numeric_limits<double>::quiet_NaN();
    return std::pow(room, 1.0 / chi);
}

bool model_ok(const vfl_plan_model* m) {
    return m && m->C_a > 0.0 && m->C_p > 0.0 && m->bandwidth > 0.0 && m->chi > 0.0 && m->bytes_per_row >= 0.0;
}

double delay(const vfl_plan_model* m, int wa, int wp, double b) {
    const double ta = (term(m->lambda_a, b, m->gamma_a) + term(m->phi_a, b, m->beta_a) +
                       term(m->lambda_top, b, m->gamma_top) + term(m->phi_top, b, m->beta_top)) * wa / m->C_a;
    const double tp = (term(m->lambda_p, b, m->gamma_p) + term(m->phi_p, b, m->beta_p)) * wp / m->C_p;
    const double comm = 2.0 * b * m->bytes_per_row / m->bandwidth;   // (E + G) / B_b
    return std::max(ta, tp) + comm;
}

}  // namespace

extern "C" {

vfl_status vfl_plan_bmax(const vfl_plan_model* m, double* bmax) {
    if (!model_ok(m) || !bmax) return VFL_E_INVAL;
    const double a = party_bmax(m->M_A0, m->rho_A, m->M_A_max, m->chi);
    const double p = party_bmax(m->M_P0, m->rho_P, m->M_P_max, m->chi);
    if (std::isnan(a) || std::isnan(p)) return VFL_E_INVAL;
    *bmax = std::min(a, p);
    return VFL_OK;
}

vfl_status vfl_plan_delay(const vfl_plan_model* m, int32_t w_a, int32_t w_p, double batch, double* out) {
    if (!model_ok(m) || !out || w_a < 1 || w_p < 1 || !(batch > 0.0)) return VFL_E_INVAL;
    *out = delay(m, w_a, w_p, batch);
    return VFL_OK;
}

vfl_status vfl_plan(const vfl_plan_model* m, int32_t wa_lo, int32_t wa_hi, int32_t wp_lo, int32_t wp_hi,
                    const int32_t* batches, int32_t n_batches, int32_t* w_a, int32_t* w_p, int32_t* batch,
                    double* out) {
    if (!model_ok(m) || !batches || n_batches < 1 || !w_a || !w_p || !batch || !out) return VFL_E_INVAL;
    if (wa_lo < 1 || wp_lo < 1 || wa_hi < wa_lo || wp_hi < wp_lo) return VFL_E_INVAL;
    double bmax = 0.0;
    if (vfl_plan_bmax(m, &bmax) != VFL_OK) return VFL_E_INVAL;
    double best = std::numeric_limits<double>::infinity();
    bool found = false;
    for (int r = 0; r < n_batches; ++r) {
        const double b = batches[r];
        if (!(b >= 1.0) || b > bmax) continue;
        for (int wa = wa_lo; wa <= wa_hi; ++wa)
            for (int wp = wp_lo; wp <= wp_hi; ++wp) {
                const double o = delay(m, wa, wp, b);
                if (o < best) {
                    best = o;
                    *w_a = wa;
                    *w_p = wp;
                    *batch = batches[r];
                    found = true;
                }
            }
    }
    if (!found) return VFL_E_INVAL;
    *out = best;
    return VFL_OK;
}

vfl_status vfl_fit_power(const double* x, const double* t, int32_t n, double* coef, double* expo) {
    if (!x || !t || !coef || !expo || n < 2) return VFL_E_INVAL;
    double mx = 0.0, my = 0.0;
    for (int i = 0; i < n; ++i) {
        if (!(x[i] > 0.0) || !(t[i] > 0.0)) return VFL_E_INVAL;
        mx += std::log(x[i]);
        my += std::log(t[i]);
    }
    mx /= n;
    my /= n;
    double sxx = 0.0, sxy = 0.0;
    for (int i = 0; i < n; ++i) {
        const double dx = std::log(x[i]) - mx;
        sxx += dx * dx;
        sxy += dx * (std::log(t[i]) - my);
    }
    if (!(sxx > 0.0)) return VFL_E_INVAL;
    *expo = sxy / sxx;
    *coef = std::exp(my - *expo * mx);
    return VFL_OK;
}

}  // extern "C"
