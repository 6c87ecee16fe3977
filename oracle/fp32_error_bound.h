/*
 * First-order forward error bounds of an fp32 evaluation of a
 * proxy-denominator residual chain (reading R11 of resispec_oracle.c).
 * TEST INFRASTRUCTURE ONLY: the parity tests widen their tolerance by these
 * bounds on rows whose test denominator is the proxy; they are not part of
 * the verification rule the oracle computes.
 */
#ifndef FP32_ERROR_BOUND_H_
#define FP32_ERROR_BOUND_H_

/* Bounds e[i] of the rounding of fp32 tempered softmax values v[i]. */
void fp32err_init(const double* v, int V, double* e);

/* Carries the bounds (eR, eD) of R and D through one ResiSpec rejection of
 * x0 (R, D before; r, K after; budget Z, level, fill fraction mu) and leaves
 * the bounds of R' = r / sum r and D' = K in (eR, eD). */
void fp32err_reject(const double* R, const double* D, const double* r, const double* K, int V,
                    int x0, double Z, double level, double mu, double* eR, double* eD);

#endif
