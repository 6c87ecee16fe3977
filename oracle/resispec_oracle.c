/*
 * ResiSpec verification oracle: plain, slow, fp64 CPU reference.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may link or call
 * this file; only the tests, the smoke check and the benchmark's CPU-baseline
 * leg do.  It shares no code, header, table or constant generator with the
 * CUDA library.
 *
 * What it computes (paper: "ResiSpec: Enhancing Multi-Candidate Speculative
 * Sampling via Residual Distribution Shaping"):
 *
 *   - tempered distributions p = softmax(z_target / T), q = softmax(z_draft / T)
 *     (Sec. 6.1 / Appendix C "Decoding configurations": temperature, no top-p);
 *   - the multi-candidate verification walk over a draft token tree
 *     (Sec. 3 "Multi-candidate Tree-structured Verification"): at each visited
 *     node the children are tested in ascending node order; acceptance
 *     descends into the accepted child, rejection of all children ends the
 *     walk with a sample from the residual;
 *   - the accept test  u < R(x) / D(x)  (Algorithm 1);
 *   - on rejection, mode RESISPEC: K = GetProxy(R, Q, x0) and
 *     R <- norm(max(R - K, 0))  (Algorithm 1, function GetProxy; budget from
 *     Sec. 5.3, Eq. for s(x0));
 *     mode SPECINFER: R <- norm(max(R - q, 0))  (Eq. 2, Sec. 3);
 *   - the final sample x ~ R by inverse CDF over ascending token ids
 *     (Algorithm 1, last step), or, when an accepted node has no children,
 *     the bonus token from that node's own target distribution (speculative
 *     decoding convention; the paper does not spell it out);
 *   - counter-based randomness: Philox4x64-10 (Salmon, Moraes, Dror, Shaw,
 *     "Parallel random numbers: as easy as 1, 2, 3", SC 2011), key
 *     (seed, 0), counter (row, seq, 0, 0); output word `draw` gives
 *     u = (word >> 40) * 2^-24.  Word 0 of the block of row c+1 is the
 *     accept-test uniform of candidate node c; word 1 of the block of row r
 *     is the residual/bonus uniform of the node whose logits are row r.
 *
 * Readings of points the paper leaves open:
 *   R1  budget Z = q(x0) - R(x0) with R the current residual (Algorithm 1
 *       calls GetProxy(R, Q, x_i)); positive on every rejection.
 *   R2  the deficit is water-filled in proportion to the remaining capacity
 *       R - r over tokens other than x0:  r += Delta * cap / sum(cap).
 *       parity unpinned beyond the hand-worked example and the L1 closed form
 *       of Theorem 2: the paper does not fix how the deficit is split.
 *   R3  slack s is zero off x0, so K = R - r everywhere and then K(x0) = q(x0)
 *       (GetProxy prose, step 3).
 *   R4  the test denominator D stays the node's draft distribution q for all
 *       siblings (Algorithm 1 never updates D).
 *   R5  degenerate rejection (Z <= 0, or an all-zero residual from rounding):
 *       R is left unchanged and the event is counted.
 *   R7  budget variant Z_applied (Sec. 5.3 heuristic, flag): Z =
 *       max(Z*, |q(x0) - R(x0)|) with Z* = min over q > 0 of R/q, the
 *       capacity bound of Prop. "Capacity Bound of Ideal Shaping" taken on
 *       the current residual, clamped to Z <= 1 - R(x0) so that the
 *       water-fill of step 3 stays feasible (r <= R off x0 sums to Z).
 *   R8  proxy-as-denominator variant (flag; App. C, the EAGLE integration
 *       "updates the current target distribution p and draft/proxy
 *       distribution q ... before verifying the next sibling"): after a
 *       ResiSpec rejection the test denominator D becomes the proxy K of
 *       that rejection (K = R - r off x0, K(x0) = D(x0): a distribution),
 *       and the next GetProxy takes D in place of q.  D starts as q at each
 *       node.
 *   R9  drafting (flag; Algorithm 1's "x_1..x_k ~ Q i.i.d."): the children of
 *       each visited node are drawn from that node's tempered draft
 *       distribution q by inverse CDF over ascending token ids, child c
 *       with u = word 2 of the Philox block of row c + 1, in child order
 *       before the node's accept tests; the drawn tokens replace cand.
 *   R10 lambda-level fill (flag; another reading of step 3, which only asks
 *       that the deficit go to tokens still below their capacity p): the
 *       filled mass is the draft raised to a common level, r = min(lam q, p)
 *       off x0 with lam chosen so that sum r = Z.  sum_{i != x0} min(lam q_i,
 *       p_i) is continuous, nondecreasing and linear between the ratios
 *       p_i / q_i, so lam is found exactly on the sorted ratios.  If even
 *       r = p on the support of q leaves a deficit, the tokens with q = 0
 *       (other than x0) take it in proportion to p, the rule of R2.
 *   R11 tolerance of the proxy-denominator chain (R8): the proxy K = R - r
 *       is a difference that cancels on tokens just below the level, and a
 *       later rejection may divide it by a small budget, so an fp32
 *       evaluation of the chain can be far from the fp64 one on a few
 *       tokens.  For such rows the oracle also returns a first-order forward
 *       error bound per token of the final distribution (out_dist_err): the
 *       absolute errors of R and D are carried through every rejection
 *       (min, R - m, r = m + mu t, K, the budget Z = D(x0) - R(x0), the
 *       level's response to Z and the normaliser), starting from the
 *       rounding of fp32 tempered softmax values; it is test infrastructure
 *       that widens the parity tolerance only where the arithmetic does.
 *   R6  the accept decision is the paper's test u < R(x) / D(x) in fp64
 *       (decide_fp64 = 1, what the Python wrapper passes by default);
 *       decide_fp64 = 0 takes it as u * D(x) < R(x) on operands rounded to
 *       fp32, a diagnostic only.  The margin |u - R/D| is reported in fp64
 *       for near-tie accounting.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#include "fp32_error_bound.h"

#define OR_MODE_RESISPEC 0
#define OR_MODE_SPECINFER 1

#define OR_F32 0
#define OR_BF16 1

/* Per-sequence status bits.  Same meaning as the library's device word. */
#define OR_ERR_TREE 1       /* parent index not in [-1, child) */
#define OR_ERR_TOKEN 2      /* candidate token outside [0, V) */
#define OR_ERR_NONFINITE 4  /* NaN or +inf logit in a visited row */
#define OR_ERR_EMPTY_ROW 8  /* every logit of a visited row is -inf */
#define OR_ERR_DEPTH 16     /* more accepted tokens than max_depth */
#define OR_INFO_DEGENERATE 256 /* a rejection left R unchanged (R5) */

/* ------------------------------------------------------------------ */
/* Philox4x64-10, from the round function and key schedule published in
 * Salmon et al., SC 2011 (Sec. 4.2 of that paper): two 64x64->128
 * multiplications per round, a permutation of the four words, and a Weyl
 * sequence on the key. */
static const uint64_t PHILOX_M0 = 0xD2E7470EE14C6C93ULL;
static const uint64_t PHILOX_M1 = 0xCA5A826395121157ULL;
static const uint64_t PHILOX_W0 = 0x9E3779B97F4A7C15ULL; /* golden ratio */
static const uint64_t PHILOX_W1 = 0xBB67AE8584CAA73BULL; /* sqrt(3) - 1 */

void oracle_philox4x64_10(const uint64_t ctr[4], const uint64_t key[2],
                          uint64_t out[4]) {
  uint64_t x0 = ctr[0], x1 = ctr[1], x2 = ctr[2], x3 = ctr[3];
  uint64_t k0 = key[0], k1 = key[1];
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += PHILOX_W0;
      k1 += PHILOX_W1;
    }
    unsigned __int128 a = (unsigned __int128)PHILOX_M0 * x0;
    unsigned __int128 b = (unsigned __int128)PHILOX_M1 * x2;
    uint64_t hi0 = (uint64_t)(a >> 64), lo0 = (uint64_t)a;
    uint64_t hi1 = (uint64_t)(b >> 64), lo1 = (uint64_t)b;
    uint64_t y0 = hi1 ^ x1 ^ k0;
    uint64_t y1 = lo1;
    uint64_t y2 = hi0 ^ x3 ^ k1;
    uint64_t y3 = lo0;
    x0 = y0;
    x1 = y1;
    x2 = y2;
    x3 = y3;
  }
  out[0] = x0;
  out[1] = x1;
  out[2] = x2;
  out[3] = x3;
}

/* U(seed, seq, row, draw) in [0, 1), a multiple of 2^-24. */
double oracle_uniform(uint64_t seed, int64_t seq, int64_t row, int draw) {
  uint64_t ctr[4] = {(uint64_t)row, (uint64_t)seq, 0, 0};
  uint64_t key[2] = {seed, 0};
  uint64_t w[4];
  oracle_philox4x64_10(ctr, key, w);
  return (double)(w[draw & 3] >> 40) * (1.0 / 16777216.0);
}

/* ------------------------------------------------------------------ */
static double bf16_to_double(uint16_t bits) {
  uint32_t u = (uint32_t)bits << 16;
  float f;
  memcpy(&f, &u, sizeof f);
  return (double)f;
}

static void load_row(const void* base, int dtype, size_t offset, int V,
                     double* z) {
  if (dtype == OR_BF16) {
    const uint16_t* s = (const uint16_t*)base + offset;
    for (int i = 0; i < V; ++i) z[i] = bf16_to_double(s[i]);
  } else {
    const float* s = (const float*)base + offset;
    for (int i = 0; i < V; ++i) z[i] = (double)s[i];
  }
}

/* Tempered softmax: a = z / T, m = max a, p = exp(a - m) / sum exp(a - m).
 * Returns 0, OR_ERR_NONFINITE or OR_ERR_EMPTY_ROW. */
int oracle_softmax(const double* z, int V, double T, double* p) {
  double m = -INFINITY;
  for (int i = 0; i < V; ++i) {
    double a = z[i] / T;
    if (isnan(a) || a == INFINITY) return OR_ERR_NONFINITE;
    p[i] = a;
    if (a > m) m = a;
  }
  if (m == -INFINITY) return OR_ERR_EMPTY_ROW;
  double s = 0.0;
  for (int i = 0; i < V; ++i) {
    p[i] = exp(p[i] - m);
    s += p[i];
  }
  for (int i = 0; i < V; ++i) p[i] /= s;
  return 0;
}

/* GetProxy(p, q, x0) of Algorithm 1, with p the current residual R.
 *   step 1  Z = q(x0) - p(x0)                         (budget, Sec. 5.3)
 *   step 2  r_i = min(Z q_i, p_i) for i != x0, r_x0 = 0 (projection)
 *   step 3  Delta = Z - sum r; fill Delta into the capacity p - r (R2), or
 *           raise the draft to a common level (fill 1, R10)
 *   step 4  k = p - r + s, then k(x0) = q(x0)          (s = 0 off x0, R3)
 * Writes k and r (either may be NULL) and returns Z.  The caller must only
 * use k when Z > 0 (R5). */
double oracle_get_proxy_z(const double* p, const double* q, int V, int x0, double Z, int fill,
                          double* k, double* r);

double oracle_get_proxy(const double* p, const double* q, int V, int x0,
                        double* k, double* r) {
  return oracle_get_proxy_z(p, q, V, x0, q[x0] - p[x0], 0, k, r);
}

/* The budget of a rejection of x0: rule 0 = Algorithm 1 (R1), rule 1 =
 * Z_applied (R7). */
double oracle_budget(const double* R, const double* q, int V, int x0, int rule) {
  const double gap = q[x0] - R[x0];
  if (rule == 0) return gap;
  double zstar = INFINITY;
  for (int i = 0; i < V; ++i)
    if (q[i] > 0.0 && R[i] / q[i] < zstar) zstar = R[i] / q[i];
  double Z = fmax(zstar, fabs(gap));
  return fmin(Z, 1.0 - R[x0]);
}

typedef struct {
  double ratio;
  int i;
} ratio_item;

static int by_ratio(const void* a, const void* b) {
  const double x = ((const ratio_item*)a)->ratio, y = ((const ratio_item*)b)->ratio;
  return x < y ? -1 : (x > y ? 1 : 0);
}

/* The level of R10: the lam >= 0 with sum_{i != x0, q_i > 0} min(lam q_i,
 * p_i) = Z, or INFINITY when even lam = inf leaves the sum below Z.  The
 * ratios p_i / q_i are visited in ascending order; before ratio j the tokens
 * below it are saturated (they give p_i) and the rest give lam q_i, so the
 * crossing piece is solved in closed form. */
static double lambda_level(const double* p, const double* q, int V, int x0, double Z) {
  int n = 0;
  ratio_item* it = (ratio_item*)malloc(sizeof(ratio_item) * (size_t)(V > 0 ? V : 1));
  double* suf_q = (double*)malloc(sizeof(double) * (size_t)(V + 1));
  for (int i = 0; i < V; ++i)
    if (i != x0 && q[i] > 0.0) {
      it[n].ratio = p[i] / q[i];
      it[n].i = i;
      ++n;
    }
  qsort(it, (size_t)n, sizeof(ratio_item), by_ratio);
  suf_q[n] = 0.0;
  for (int j = n - 1; j >= 0; --j) suf_q[j] = suf_q[j + 1] + q[it[j].i];
  double lam = INFINITY, pre_p = 0.0;
  for (int j = 0; j < n; ++j) {
    const double at = pre_p + it[j].ratio * suf_q[j]; /* S(ratio_j) */
    if (at >= Z) {
      lam = (Z - pre_p) / suf_q[j];
      break;
    }
    pre_p += p[it[j].i];
  }
  free(it);
  free(suf_q);
  return lam;
}

/* GetProxy with the budget Z and the fill rule given (steps 2-4 below);
 * *level_out / *mu_out (optional) receive the level of step 2 (INFINITY: the
 * support of q saturated) and the fraction of the capacity filled in step 3. */
static double get_proxy_full(const double* p, const double* q, int V, int x0, double Z, int fill,
                             double* k, double* r, double* level_out, double* mu_out) {
  double* rr = r ? r : (double*)malloc(sizeof(double) * (size_t)V);
  const double level = fill == 1 ? lambda_level(p, q, V, x0, Z) : Z;
  double mu = 0.0;
  double sum_r = 0.0;
  for (int i = 0; i < V; ++i) {
    /* step 2 at the level Z (R2), or at the level that meets Z (R10); with
       lam = inf the support of q is saturated */
    const double lq = (level == INFINITY) ? (q[i] > 0.0 ? INFINITY : 0.0) : level * q[i];
    rr[i] = (i == x0) ? 0.0 : fmin(lq, p[i]);
    sum_r += rr[i];
  }
  double delta = Z - sum_r;
  double sum_cap = 0.0;
  for (int i = 0; i < V; ++i)
    if (i != x0) sum_cap += p[i] - rr[i];
  /* the capacity fill (R2; for R10 only the deficit that the level cannot
     meet, which leaves capacity on q = 0 tokens alone) */
  if (sum_cap > 0.0 && (fill != 1 || level == INFINITY)) {
    mu = delta / sum_cap;
    for (int i = 0; i < V; ++i)
      if (i != x0) rr[i] += delta * (p[i] - rr[i]) / sum_cap;
  }
  if (k) {
    for (int i = 0; i < V; ++i) k[i] = p[i] - rr[i];
    k[x0] = q[x0];
  }
  if (!r) free(rr);
  if (level_out) *level_out = level;
  if (mu_out) *mu_out = mu;
  return Z;
}

double oracle_get_proxy_z(const double* p, const double* q, int V, int x0, double Z, int fill,
                          double* k, double* r) {
  return get_proxy_full(p, q, V, x0, Z, fill, k, r, NULL, NULL);
}

/* R <- norm(max(R - K, 0)).  Returns the normaliser (0: R left unchanged). */
static double residual_from(double* R, const double* K, int V, double* tmp) {
  double s = 0.0;
  for (int i = 0; i < V; ++i) {
    tmp[i] = fmax(R[i] - K[i], 0.0);
    s += tmp[i];
  }
  if (!(s > 0.0)) return 0.0;
  for (int i = 0; i < V; ++i) R[i] = tmp[i] / s;
  return s;
}

int oracle_reject_ex(int mode, double* R, const double* q, int V, int x0,
                     double* K, double* r, double* tmp, double* inv_err,
                     double* norm_out);
int oracle_reject_z(int mode, int z_rule, int fill, double* R, const double* q, int V, int x0,
                    double* K, double* r, double* tmp, double* inv_err, double* norm_out);

/* One rejection of token x0 applied to the residual R (length V).
 * mode SPECINFER: R <- norm(max(R - q, 0))              (Eq. 2, Sec. 3)
 * mode RESISPEC:  K = GetProxy(R, q, x0); R <- norm(max(R - K, 0)) (Alg. 1)
 * Returns 1 if R changed, 0 on a degenerate rejection (R5).  When inv_err is
 * non-NULL the GetProxy invariants of Sec. 5.1 / Algorithm 1 are measured and
 * the largest violation is max-ed into *inv_err. */
int oracle_reject(int mode, double* R, const double* q, int V, int x0,
                  double* K, double* r, double* tmp, double* inv_err) {
  return oracle_reject_ex(mode, R, q, V, x0, K, r, tmp, inv_err, NULL);
}

/* As oracle_reject; *norm_out receives the SpecInfer normaliser
 * sum (R - q)_+ of this rejection (1 in ResiSpec mode). */
int oracle_reject_ex(int mode, double* R, const double* q, int V, int x0,
                     double* K, double* r, double* tmp, double* inv_err,
                     double* norm_out) {
  return oracle_reject_z(mode, 0, 0, R, q, V, x0, K, r, tmp, inv_err, norm_out);
}

static int reject_full(int mode, int z_rule, int fill, double* R, const double* q, int V, int x0,
                       double* K, double* r, double* tmp, double* inv_err, double* norm_out,
                       double* Z_out, double* level_out, double* mu_out);

/* As oracle_reject_ex with the ResiSpec budget chosen by z_rule (R1 / R7)
 * and the fill of step 3 by fill (0: R2, 1: R10). */
int oracle_reject_z(int mode, int z_rule, int fill, double* R, const double* q, int V, int x0,
                    double* K, double* r, double* tmp, double* inv_err, double* norm_out) {
  return reject_full(mode, z_rule, fill, R, q, V, x0, K, r, tmp, inv_err, norm_out, NULL, NULL,
                     NULL);
}

static int reject_full(int mode, int z_rule, int fill, double* R, const double* q, int V, int x0,
                       double* K, double* r, double* tmp, double* inv_err, double* norm_out,
                       double* Z_out, double* level_out, double* mu_out) {
  if (norm_out) *norm_out = 1.0;
  if (mode == OR_MODE_SPECINFER) {
    double changed = residual_from(R, q, V, tmp);
    if (norm_out && changed > 0.0) *norm_out = changed;
    if (inv_err && changed > 0.0) {
      double s = 0.0, e = 0.0;
      for (int i = 0; i < V; ++i) {
        s += R[i];
        if (-R[i] > e) e = -R[i];
      }
      if (fabs(s - 1.0) > e) e = fabs(s - 1.0);
      if (e > *inv_err) *inv_err = e;
    }
    return changed > 0.0;
  }
  const double Z = oracle_budget(R, q, V, x0, z_rule);
  if (Z_out) *Z_out = Z;
  if (!(Z > 0.0)) return 0;
  get_proxy_full(R, q, V, x0, Z, fill, K, r, level_out, mu_out);
  double e = 0.0;
  if (inv_err) {
    double sr = 0.0, sk = 0.0;
    for (int i = 0; i < V; ++i) {
      sr += r[i];
      sk += K[i];
      if (-r[i] > e) e = -r[i];
      if (r[i] - R[i] > e) e = r[i] - R[i];
      if (-K[i] > e) e = -K[i];
    }
    if (fabs(sr - Z) > e) e = fabs(sr - Z);
    if (fabs(r[x0]) > e) e = fabs(r[x0]);
    /* sum K = 1 with K(x0) = q(x0) holds for the budget of Algorithm 1 only;
       under Z_applied the slack that would restore it is unspecified (it
       never reaches R' = r / Z), so only r is checked there. */
    if (z_rule == 0) {
      if (fabs(sk - 1.0) > e) e = fabs(sk - 1.0);
      if (fabs(K[x0] - q[x0]) > e) e = fabs(K[x0] - q[x0]);
    }
  }
  double norm = residual_from(R, K, V, tmp);
  if (!(norm > 0.0)) return 0;
  if (inv_err) {
    double s = 0.0;
    for (int i = 0; i < V; ++i) {
      s += R[i];
      if (-R[i] > e) e = -R[i];
      /* R' = r / Z, compared on the unnormalised scale: R - K = r is formed
         by a cancellation whose rounding is relative to R, not to r. */
      double d = fabs(R[i] * Z - r[i]);
      if (d > e) e = d;
    }
    if (fabs(s - 1.0) > e) e = fabs(s - 1.0);
    if (e > *inv_err) *inv_err = e;
  }
  return 1;
}

/* Inverse-CDF draw: the smallest token x with C(x) > u * C(V-1), C the
 * inclusive prefix sum over ascending token ids.  *margin receives
 * min(|u C(V-1) - C(x-1)|, |C(x) - u C(V-1)|) / C(V-1). */
int oracle_sample(const double* R, int V, double u, double* margin) {
  double total = 0.0;
  for (int i = 0; i < V; ++i) total += R[i];
  double tau = u * total;
  double c = 0.0;
  int last_pos = -1;
  for (int i = 0; i < V; ++i) {
    double prev = c;
    c += R[i];
    if (R[i] > 0.0) last_pos = i;
    if (c > tau) {
      if (margin) {
        double a = tau - prev, b = c - tau;
        *margin = (a < b ? a : b) / total;
      }
      return i;
    }
  }
  if (margin) *margin = 0.0;
  return last_pos < 0 ? 0 : last_pos;
}

/* ------------------------------------------------------------------ */
typedef struct {
  int32_t B, N, V, D;
  int32_t dtype;
  int32_t mode;
  int32_t decide_fp64; /* 1: the fp64 test u < R/D (R6); 0: fp32 diagnostic */
  int32_t check_invariants;
  int32_t nthreads;
  int32_t pad_;
  int64_t seq_stride; /* elements between sequences; 0 = shared rows */
  const void* target;
  const void* draft;
  const int32_t* parents;  /* [N], or [B, N] with parents_stride = N */
  const int32_t* cand;     /* [B, N] */
  const int32_t* seq_ids;  /* [B] global sequence index for the RNG, or NULL */
  double temperature;
  uint64_t seed;
  /* outputs, each optional (NULL) */
  int32_t* out_tokens;     /* [B, D+1], -1 padded */
  int32_t* out_len;        /* [B], -1 on a data error */
  int32_t* out_nodes;      /* [B, D], -1 padded */
  double* out_dist;        /* [B, V] distribution of the final draw */
  double* out_accept_margin; /* [B] min |u - R/q| over the tests */
  double* out_sample_margin; /* [B] relative margin of the final draw */
  int32_t* out_status;     /* [B] */
  int32_t* out_rejects;    /* [B] rejections along the walk */
  int32_t* out_rows;       /* [B] logit rows read (target + draft) */
  double* out_inv_err;     /* [B] largest invariant violation */
  double* out_cond;        /* [B] 1 / prod of the SpecInfer normalisers at the
                              final node (1 without SpecInfer rejections) */
  int64_t parents_stride;  /* elements between sequences' parent arrays:
                              0 = one tree for all, N = parents is [B, N]
                              (per-sequence, dynamic trees) */
  int32_t z_rule;          /* ResiSpec budget: 0 Algorithm 1 (R1), 1 Z_applied (R7) */
  int32_t denom_update;    /* 1: the test denominator becomes the proxy after
                              each ResiSpec rejection (R8) */
  int32_t* draft_out;      /* non-NULL: draft the children of visited nodes
                              (R9) into [B, N] (-1 elsewhere) instead of
                              reading cand */
  double* out_draft_margin; /* [B] smallest relative CDF margin of those draws */
  int32_t fill;            /* ResiSpec fill of step 3: 0 capacity (R2), 1 level (R10) */
  int32_t pad2_;
  double* out_dist_err;    /* [B, V] forward error bound of out_dist for rows with
                              the proxy denominator (R11); 0 elsewhere */
} oracle_args;

typedef struct {
  const oracle_args* a;
  int tid, nthreads;
  int tree_bad;
} worker_ctx;

/* A tree is valid when every node's parent precedes it (-1: the root). */
static int tree_is_bad(const int32_t* parents, int N) {
  for (int c = 0; c < N; ++c)
    if (parents[c] < -1 || parents[c] >= c) return 1;
  return 0;
}

static void verify_sequence(const oracle_args* a, int lb, int tree_bad,
                            double* z, double* p, double* q, double* R,
                            double* K, double* r, double* tmp, double* Dbuf,
                            double* eR, double* eD, double* Rb, int32_t* kids) {
  const int V = a->V, N = a->N, D = a->D;
  const int32_t* parents = a->parents + (size_t)(a->parents_stride * lb);
  if (a->parents_stride) tree_bad = tree_is_bad(parents, N);
  const int64_t gb = a->seq_ids ? a->seq_ids[lb] : lb;
  const double T = a->temperature;
  int32_t* toks = a->out_tokens ? a->out_tokens + (size_t)lb * (D + 1) : NULL;
  int32_t* drafted = a->draft_out ? a->draft_out + (size_t)lb * N : NULL;
  double dmargin = INFINITY;
  if (drafted)
    for (int c = 0; c < N; ++c) drafted[c] = -1;
  int32_t* nodes = a->out_nodes ? a->out_nodes + (size_t)lb * D : NULL;
  if (toks)
    for (int i = 0; i <= D; ++i) toks[i] = -1;
  if (nodes)
    for (int i = 0; i < D; ++i) nodes[i] = -1;
  int status = 0, depth = 0, rejects = 0, rows = 0;
  double amargin = INFINITY, smargin = INFINITY, inv = 0.0, cond = 1.0;
  double* inv_ptr = a->check_invariants ? &inv : NULL;
  const size_t seq_off = (size_t)(a->seq_stride * lb);

  if (tree_bad) {
    status = OR_ERR_TREE;
    goto done;
  }
  int node = -1, row = 0;
  for (;;) {
    int nk = 0;
    for (int c = 0; c < N; ++c)
      if (parents[c] == node) kids[nk++] = c;

    load_row(a->target, a->dtype, seq_off + (size_t)row * V, V, z);
    rows += 1;
    int st = oracle_softmax(z, V, T, p);
    if (st) {
      status |= st;
      goto done;
    }
    if (nk == 0) {
      /* bonus token: the accepted node has no children (or N == 0) */
      cond = 1.0;
      double u = oracle_uniform(a->seed, gb, row, 1);
      int y = oracle_sample(p, V, u, &smargin);
      if (toks) toks[depth] = y;
      if (a->out_dist) memcpy(a->out_dist + (size_t)lb * V, p, sizeof(double) * V);
      if (a->out_dist_err) memset(a->out_dist_err + (size_t)lb * V, 0, sizeof(double) * V);
      break;
    }
    load_row(a->draft, a->dtype, seq_off + (size_t)row * V, V, z);
    rows += 1;
    st = oracle_softmax(z, V, T, q);
    if (st) {
      status |= st;
      goto done;
    }
    if (drafted) /* x_1..x_k ~ Q i.i.d. (R9) */
      for (int j = 0; j < nk; ++j) {
        double m = INFINITY;
        drafted[kids[j]] = oracle_sample(q, V, oracle_uniform(a->seed, gb, kids[j] + 1, 2), &m);
        if (m < dmargin) dmargin = m;
      }
    memcpy(R, p, sizeof(double) * V); /* R <- P, D <- Q (Algorithm 1) */
    double* Dn = q;                   /* the test denominator */
    if (a->denom_update && a->mode == OR_MODE_RESISPEC) {
      memcpy(Dbuf, q, sizeof(double) * V);
      Dn = Dbuf;                      /* becomes each rejection's proxy (R8) */
    }
    const int track = a->out_dist_err != NULL && Dn == Dbuf; /* R11 */
    if (track) {
      fp32err_init(p, V, eR);
      fp32err_init(q, V, eD);
    }
    cond = 1.0;
    int accepted = -1;
    for (int j = 0; j < nk; ++j) {
      int c = kids[j];
      int x = drafted ? drafted[c] : a->cand[(size_t)lb * N + c];
      if (x < 0 || x >= V) {
        status |= OR_ERR_TOKEN;
        goto done;
      }
      double u = oracle_uniform(a->seed, gb, c + 1, 0);
      if (Dn[x] > 0.0) {
        double m = fabs(u - R[x] / Dn[x]);
        if (m < amargin) amargin = m;
      }
      int accept;
      if (a->decide_fp64) {
        accept = (Dn[x] > 0.0) ? (u < R[x] / Dn[x]) : (R[x] > 0.0);
      } else {
        float uf = (float)u, qf = (float)Dn[x], Rf = (float)R[x];
        float lhs = uf * qf;
        accept = lhs < Rf;
      }
      if (accept) {
        accepted = c;
        break;
      }
      rejects += 1;
      double norm = 1.0, Zj = 0.0, level = 0.0, mu = 0.0;
      if (track) memcpy(Rb, R, sizeof(double) * V);
      if (!reject_full(a->mode, a->z_rule, a->fill, R, Dn, V, x, K, r, tmp, inv_ptr, &norm, &Zj,
                       &level, &mu)) {
        status |= OR_INFO_DEGENERATE;
      } else if (Dn == Dbuf) {
        if (track) fp32err_reject(Rb, Dbuf, r, K, V, x, Zj, level, mu, eR, eD);
        memcpy(Dbuf, K, sizeof(double) * V);
      }
      cond /= norm;
    }
    if (accepted < 0) {
      double u = oracle_uniform(a->seed, gb, row, 1);
      int y = oracle_sample(R, V, u, &smargin);
      if (toks) toks[depth] = y;
      if (a->out_dist) memcpy(a->out_dist + (size_t)lb * V, R, sizeof(double) * V);
      if (a->out_dist_err) {
        if (track)
          memcpy(a->out_dist_err + (size_t)lb * V, eR, sizeof(double) * V);
        else
          memset(a->out_dist_err + (size_t)lb * V, 0, sizeof(double) * V);
      }
      break;
    }
    if (depth >= D) {
      status |= OR_ERR_DEPTH;
      goto done;
    }
    if (toks) toks[depth] = drafted ? drafted[accepted] : a->cand[(size_t)lb * N + accepted];
    if (nodes) nodes[depth] = accepted;
    depth += 1;
    node = accepted;
    row = accepted + 1;
  }
done:
  if (status & ~OR_INFO_DEGENERATE) {
    if (toks)
      for (int i = 0; i <= D; ++i) toks[i] = -1;
    if (nodes)
      for (int i = 0; i < D; ++i) nodes[i] = -1;
    depth = -1;
  }
  if (a->out_len) a->out_len[lb] = depth;
  if (a->out_status) a->out_status[lb] = status;
  if (a->out_accept_margin) a->out_accept_margin[lb] = amargin;
  if (a->out_sample_margin) a->out_sample_margin[lb] = smargin;
  if (a->out_draft_margin) a->out_draft_margin[lb] = dmargin;
  if (a->out_rejects) a->out_rejects[lb] = rejects;
  if (a->out_rows) a->out_rows[lb] = rows;
  if (a->out_inv_err) a->out_inv_err[lb] = inv;
  if (a->out_cond) a->out_cond[lb] = cond;
}

static void* worker(void* arg) {
  worker_ctx* w = (worker_ctx*)arg;
  const oracle_args* a = w->a;
  size_t V = (size_t)(a->V > 0 ? a->V : 1);
  double* buf = (double*)malloc(sizeof(double) * V * 11);
  int32_t* kids = (int32_t*)malloc(sizeof(int32_t) * (size_t)(a->N > 0 ? a->N : 1));
  for (int lb = w->tid; lb < a->B; lb += w->nthreads)
    verify_sequence(a, lb, w->tree_bad, buf, buf + V, buf + 2 * V, buf + 3 * V,
                    buf + 4 * V, buf + 5 * V, buf + 6 * V, buf + 7 * V, buf + 8 * V,
                    buf + 9 * V, buf + 10 * V, kids);
  free(kids);
  free(buf);
  return NULL;
}

/* Runs the walk for every sequence of the batch.  Returns 0, or -1 on bad
 * sizes.  Per-sequence data errors are reported through out_status and
 * out_len = -1. */
int oracle_verify(const oracle_args* a) {
  if (a->B < 0 || a->N < 0 || a->V < 1 || a->D < 0 || !(a->temperature > 0.0))
    return -1;
  if (a->parents_stride < 0) return -1;
  const int tree_bad = a->parents_stride ? 0 : tree_is_bad(a->parents, a->N);
  int nt = a->nthreads > 0 ? a->nthreads : 1;
  if (nt > a->B) nt = a->B > 0 ? a->B : 1;
  worker_ctx* ctx = (worker_ctx*)calloc((size_t)nt, sizeof(worker_ctx));
  pthread_t* th = (pthread_t*)calloc((size_t)nt, sizeof(pthread_t));
  for (int t = 0; t < nt; ++t) {
    ctx[t].a = a;
    ctx[t].tid = t;
    ctx[t].nthreads = nt;
    ctx[t].tree_bad = tree_bad;
  }
  for (int t = 1; t < nt; ++t) pthread_create(&th[t], NULL, worker, &ctx[t]);
  worker(&ctx[0]);
  for (int t = 1; t < nt; ++t) pthread_join(th[t], NULL);
  free(th);
  free(ctx);
  return 0;
}

int oracle_abi_version(void) { return 1; }
int oracle_args_size(void) { return (int)sizeof(oracle_args); }
