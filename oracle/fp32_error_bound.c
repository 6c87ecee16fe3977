/*
 * First-order forward error bounds of an fp32 evaluation of a
 * proxy-denominator residual chain (reading R11 of resispec_oracle.c).
 *
 * TEST INFRASTRUCTURE ONLY, and not the paper's rule: resispec_oracle.c
 * computes the verification walk; this file computes how far a correct
 * single-precision evaluation of the same walk may land from it on rows
 * whose test denominator is each rejection's proxy (the paper's EAGLE
 * integration, App. C).  There the proxy K = R - r is a difference that
 * cancels on tokens just below the level, and a later rejection may divide
 * it by a small budget, so the fp32 result can differ from the fp64 one by
 * far more than one rounding on a few tokens.  The parity tests add these
 * per-token bounds to their tolerance on such rows only.
 *
 * Model.  Every quantity x of the chain carries an absolute error bound e_x,
 * propagated to first order (products of errors dropped) through the steps
 * of one rejection in the order GetProxy takes them:
 *   m = min(level D, R)   t = R - m   r = m + mu t   K = R - r off x0
 *   Z = D(x0) - R(x0)     mu = (Z - sum m) / sum t   R' = r / sum r
 * plus one unit roundoff EPS of each rounded result.  A min whose operands
 * are within their error bounds of each other may take either side.
 * Pinned by tests/test_oracle_walk.py (an fp32 emulation of the chain stays
 * inside the bound on every token) and tests/test_oracle_pins.py (a
 * two-rejection example worked by hand, tests/golden/fp32_error_bound_v3.json).
 */
#include <math.h>

#include "fp32_error_bound.h"

static const double ERR_EPS = 5.9604644775390625e-08; /* 2^-24, fp32's unit roundoff */

/* Rounding of an fp32 tempered softmax value 2^a / S, a = log2(v / max v):
 * the exponent's argument is rounded relative to |a|, plus a few roundings
 * of the exponential and the normaliser. */
void fp32err_init(const double* v, int V, double* e) {
  double mx = 0.0;
  for (int i = 0; i < V; ++i)
    if (v[i] > mx) mx = v[i];
  for (int i = 0; i < V; ++i)
    e[i] = v[i] > 0.0 ? v[i] * ERR_EPS * (4.0 + 0.7 * fabs(log2(v[i] / mx))) : 0.0;
}

/* Bounds of m = min(level D, R) and t = R - m at one token (R > 0, not x0). */
static void err_min(double R, double D, double eR, double eD, double level, double* m,
                    double* em, double* t, double* et) {
  const double lD = level == INFINITY ? (D > 0.0 ? INFINITY : 0.0) : level * D;
  const double le = level == INFINITY ? 0.0 : level * eD;
  *m = fmin(lD, R);
  if (fabs(R - lD) <= eR + le + ERR_EPS * R)
    *em = fmax(eR, le) + ERR_EPS * R; /* either side of the min */
  else
    *em = (lD < R) ? le + ERR_EPS * *m : eR;
  *t = R - *m;
  *et = eR + *em + ERR_EPS * *t;
}

void fp32err_reject(const double* R, const double* D, const double* r, const double* K, int V,
                    int x0, double Z, double level, double mu, double* eR, double* eD) {
  double S = 0.0, slope = 0.0, sum_t = 0.0, sum_em = 0.0, sum_et = 0.0;
  for (int i = 0; i < V; ++i) {
    S += r[i];
    if (i == x0 || R[i] == 0.0) continue;
    double m, em, t, et;
    err_min(R[i], D[i], eR[i], eD[i], level, &m, &em, &t, &et);
    sum_t += t;
    sum_em += em;
    sum_et += et;
    if (level != INFINITY && level * D[i] < R[i]) slope += D[i];
  }
  if (!(S > 0.0)) return;
  const double eZ = eD[x0] + eR[x0] + ERR_EPS * Z;
  /* mu = (Z - sum m) / sum t: its numerator may cancel */
  const double emu = mu > 0.0 && sum_t > 0.0
                         ? (eZ + sum_em + ERR_EPS * Z) / sum_t + mu * sum_et / sum_t
                         : 0.0;
  double er_sum = 0.0;
  for (int i = 0; i < V; ++i) {
    double er, eK;
    if (i == x0 || R[i] == 0.0) {
      er = 0.0; /* taken out exactly; a rejected token stays at 0 */
      eK = (i == x0) ? eD[i] : 0.0;
    } else {
      double m, em, t, et;
      err_min(R[i], D[i], eR[i], eD[i], level, &m, &em, &t, &et);
      er = em + mu * et + emu * t + ERR_EPS * r[i];
      eK = (1.0 - mu) * et + emu * t + ERR_EPS * K[i];
    }
    eR[i] = er; /* bound of r for now */
    eD[i] = eK;
    er_sum += er;
  }
  /* the level's response to an error in Z moves the tokens below it
     together: relative dZ / (mass below the level) on them, dZ / Z on all */
  const double below = (level == INFINITY) ? 0.0 : level * slope;
  for (int i = 0; i < V; ++i) {
    const double Rn = r[i] / S;
    double e = eR[i] / S + Rn * (er_sum / S + eZ / Z);
    if (i != x0 && R[i] > 0.0 && below > 0.0 && level != INFINITY && level * D[i] < R[i])
      e += Rn * eZ / below;
    eR[i] = e;
  }
}

/* Entry points for the pins (ctypes). */
void oracle_fp32err_init(const double* v, int V, double* e) { fp32err_init(v, V, e); }

void oracle_fp32err_reject(const double* R, const double* D, const double* r, const double* K,
                           int V, int x0, double Z, double level, double mu, double* eR,
                           double* eD) {
  fp32err_reject(R, D, r, K, V, x0, Z, level, mu, eR, eD);
}
