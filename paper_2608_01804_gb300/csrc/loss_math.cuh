// Per-token clipped-surrogate arithmetic shared by the loss kernels (Eq. 3,
// KL skipped): log-prob from a row's (max, scaled sum), ratio, clipped term,
// gradient coefficient, and the per-row outputs.
#pragma once

#include "leap_internal.h"

namespace leap {

struct TokenLoss {
    float logp, lse, ell, rho, g;
    bool active;
};

// Clipped surrogate for one token given its row max m (raw logits), the
// scaled sum s = sum_v 2^((z_v - m) inv_temp log2 e) and the target logit zy.
__device__ __forceinline__ TokenLoss token_loss(const RowArgs& a, float m, float s, float zy, float old,
                                                float A, float wk) {
    TokenLoss r;
    const float lnS = logf(s);
    r.lse = fmaf(m, a.inv_temp, lnS);
    r.logp = a.inv_temp * (zy - m) - lnS;
    r.rho = expf(r.logp - old);
    const float lo = 1.f - a.eps_low, hi = 1.f + a.eps_high;
    const float clipped = fminf(fmaxf(r.rho, lo), hi);
    r.ell = -fminf(r.rho * A, clipped * A);
    r.active = (A >= 0.f) ? (r.rho <= hi) : (r.rho >= lo);
    r.g = r.active ? -wk * A * r.rho : 0.f;
    if (isnan(r.rho)) {  // fminf / fmaxf would drop a NaN: keep it in the loss and the gradient
        r.ell = r.rho;
        r.g = r.rho;
        r.active = false;
    }
    return r;
}

__device__ __forceinline__ void write_row_outputs(const RowArgs& a, int64_t row, const TokenLoss& r, float wk) {
    if (a.logp) a.logp[row] = r.logp;
    if (a.lse) a.lse[row] = r.lse;
    if (a.ell) a.ell[row] = r.ell;
    if (a.ws_contrib) {
        a.ws_contrib[row] = (double)wk * (double)r.ell;
        a.ws_rho[row] = r.rho;
        a.ws_flag[row] = (uint8_t)(1u | (r.active ? 0u : 2u));
    }
}

__device__ __forceinline__ void write_masked_outputs(const RowArgs& a, int64_t row) {
    if (a.logp) a.logp[row] = 0.f;
    if (a.lse) a.lse[row] = 0.f;
    if (a.ell) a.ell[row] = 0.f;
    if (a.ws_contrib) {
        a.ws_contrib[row] = 0.0;
        a.ws_rho[row] = 0.f;
        a.ws_flag[row] = 0;
    }
}

}  // namespace leap
