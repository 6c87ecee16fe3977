// Element arithmetic of the SpecInfer residual in the streaming kernel.
//
// The residual after n rejections at a node is (Eq. 2, Sec. 3)
//   R_n = (R_{n-1} - q)_+ / S_n = (p - C_n q)_+ / N_n
// for one scalar C_n: subtracting multiples of q and clipping at zero
// compose.  In the kernel's unnormalised units (p~ = 2^(z_t c - M_t),
// q~ = 2^(z_d c - M_d), c = log2(e) / T) this is r~ = (p~ - K_n q~)_+ with
//   K_1 = S_t / S_d,   K_{n+1} = K_n + T_n / S_d,   T_n = sum r~ (after K_n),
// S_t, S_d the sums of p~ and q~.  The residual is T_n^-1 r~.
//
// Conditioning.  Where p(x) is close to C_n q(x) the residual is a small
// difference of two large terms, and the normalised residual moves by about
// p(x) / N_n times the relative error of K_n or of p~(x), q~(x).  After a
// few rejections N_n (the product of the rejected masses) can be 1e-2 or
// less, so single-precision sums and the ~2^-22 relative error of ex2.approx
// would put errors of 1e-6 and more on such tokens.  Hence:
//   - K_n, S_t, S_d and T_n are double-float (dfloat.cuh);
//   - the exponent z c - M uses c = c_hi + c_lo (log2(e) / T to 48 bits);
//   - tokens with p~ (or, in S_d, q~) at least 2^-kDomBits of the row's
//     maximum ("dominant") get 2^x as a double-float (a 64-entry table of
//     2^(j/64) and a short series), their residual p~ - K q~ in
//     double-float, and a compensated addition each;
//   - the other tokens keep the fp32 path: their values are below
//     2^-kDomBits of the maximum and their absolute error below 2^-21 of
//     that (2^-33 of the maximum: below 1e-6 of the normalised residual
//     while T_n > 1.2e-4, T_n in units of the maximum).  A thread sums its
//     at most 8 such values of a chunk in fp32 (rounding relative 2^-24 per
//     addition, unbiased) and adds that sum to the double-float once.
// A thread first marks the dominant elements of its chunk in a bit mask and
// then takes them one at a time, so a warp runs the double-float path as
// often as its lane with the most dominant elements, not once per element
// position that any lane needs.
#pragma once
#include "dfloat.cuh"
#include "ptx.cuh"

namespace rs {

constexpr int kDomBits = 12;
constexpr float kDomArg = -(float)kDomBits;  // exponent threshold of the double-float path
constexpr int kExp2Tab = 64;                 // 2^(j / 64), j = -32 .. 31, as double-floats

// ln 2 split into an fp32 head and the fp32 rounding of the rest.
constexpr double kLn2d = 0.69314718055994530941723212145818;
constexpr float kLn2Hi = (float)kLn2d;
constexpr float kLn2Lo = (float)(kLn2d - (double)kLn2Hi);

// Exact power of two 2^n for n in [-126, 127].
__device__ __forceinline__ float pow2i(int n) { return __int_as_float((n + 127) << 23); }

// 2^(a_hi + a_lo) as a double-float (relative error about 1e-11) for a_hi in
// [-126, 125] and |a_lo| well below 1: a_hi = n + j / 64 + g exactly with
// integers n, j (-32 <= j < 32; j = 32 is taken as n + 1, j = -32) and
// |g| <= 1/128; 2^(j/64) comes from the table and 2^(g + a_lo) = e^u,
// u = (g + a_lo) ln 2 (|u| < 0.0055), from u + u^2 (1/2 + u (1/6 + u / 24)),
// whose omitted terms are below 2^-43.
__device__ __forceinline__ DF exp2_df(float a_hi, float a_lo, const float (*tab)[2]) {
  const float n = rintf(a_hi);
  const float f = __fsub_rn(a_hi, n);                    // exact, |f| <= 1/2
  const float jf = rintf(__fmul_rn(f, 64.f));            // -32 .. 32
  const float g = __fsub_rn(f, __fmul_rn(jf, 0.015625f)); // exact, |g| <= 1/128
  DF u = two_prod(g, kLn2Hi);
  u = fast_two_sum(u.hi, __fmaf_rn(g, kLn2Lo, __fmaf_rn(a_lo, kLn2Hi, u.lo)));
  const float uh = u.hi;
  const float poly =
      __fmul_rn(__fmul_rn(uh, uh), __fmaf_rn(uh, __fmaf_rn(uh, 1.f / 24.f, 1.f / 6.f), 0.5f));
  const DF em1 = fast_two_sum(uh, __fadd_rn(u.lo, poly));  // e^u - 1
  const int wrap = jf == 32.f;
  const int j = (int)jf + 32 - 64 * wrap;
  const DF t = DF{tab[j][0], tab[j][1]};
  const DF r = df_add(t, df_mul(t, em1));
  const float s = pow2i((int)n + wrap);
  return DF{__fmul_rn(r.hi, s), __fmul_rn(r.lo, s)};
}

// The exponent z (c_hi + c_lo) - M as a double-float (exact up to the
// rounding of c_lo z and of the final fast sum).
__device__ __forceinline__ DF exponent_df(float z, float c_hi, float c_lo, float M) {
  const DF pz = two_prod(z, c_hi);
  const DF a = two_sum(pz.hi, -M);
  return fast_two_sum(a.hi, __fadd_rn(a.lo, __fmaf_rn(z, c_lo, pz.lo)));
}

// The fp32 exponent z (c_hi + c_lo) - M of the fast path (-inf for z = -inf,
// whatever the sign of c_lo).
__device__ __forceinline__ float exponent_f(float z, float c_hi, float c_lo, float M) {
  const float a = __fmaf_rn(z, c_hi, -M);
  return a == -INFINITY ? a : __fmaf_rn(z, c_lo, a);
}

// p~ (or q~) of a dominant element as a double-float.
__device__ __forceinline__ DF unnorm_dom(float z, float c_hi, float c_lo, float M,
                                         const float (*tab)[2]) {
  const DF e = exponent_df(z, c_hi, c_lo, M);
  return exp2_df(e.hi, e.lo, tab);
}

// p~ (or q~) of one element as a double-float: the table path above the
// threshold, ex2.approx below it.  -inf logits give 0.
__device__ __forceinline__ DF unnorm_df(float z, float c_hi, float c_lo, float M,
                                        const float (*tab)[2]) {
  const float a = exponent_f(z, c_hi, c_lo, M);
  if (!(a > kDomArg)) return df(ex2(a));
  return unnorm_dom(z, c_hi, c_lo, M, tab);
}

// Per-visit constants of the SpecInfer residual.
struct SpecConst {
  float c_hi, c_lo;  // log2(e) / T
  float Mt, Md;      // the row references
  DF K;              // the current threshold K_n (0 before the node's first rejection)
};

// r~ of an element whose p~ is below the threshold, from its target
// exponent a_t: fp32 (value and error below 2^-kDomBits and
// 2^-(kDomBits+21) of the row's maximum).
__device__ __forceinline__ float residual_f(float at, float zd, const SpecConst& S) {
  const float p = ex2(at);
  const float q = ex2(exponent_f(zd, S.c_hi, S.c_lo, S.Md));
  return fmaxf(__fmaf_rn(-S.K.hi, q, p), 0.f);
}

// r~ = (p~ - K q~)_+ of an element whose p~ is dominant, in double-float.
__device__ __forceinline__ DF residual_dom(float zt, float zd, const SpecConst& S,
                                           const float (*tab)[2]) {
  const DF p = unnorm_dom(zt, S.c_hi, S.c_lo, S.Mt, tab);
  const DF q = unnorm_df(zd, S.c_hi, S.c_lo, S.Md, tab);
  const DF r = df_add(p, df_neg(df_mul(S.K, q)));
  return r.hi > 0.f ? r : df(0.f);
}

// r~ = (p~ - K q~)_+ of one element, as a double-float.
__device__ __forceinline__ DF spec_residual(float zt, float zd, const SpecConst& S,
                                            const float (*tab)[2]) {
  const float at = exponent_f(zt, S.c_hi, S.c_lo, S.Mt);
  if (!(at > kDomArg)) return df(residual_f(at, zd, S));
  return residual_dom(zt, zd, S, tab);
}

// acc += sum of p~ (or q~) over the NE elements of a thread's chunk: the
// fp32 sum of the elements below the threshold, then the dominant ones.
// z(j) gives element j for a compile-time j (from registers); zr(j) gives it
// for a run-time j (from shared memory), so the values need not stay in
// registers across the second loop.
template <int NE, class Elem, class ElemR>
__device__ __forceinline__ void unnorm_sum(const Elem& z, const ElemR& zr, float c_hi, float c_lo,
                                           float M, const float (*tab)[2], DF& acc) {
  float fs = 0.f;
  unsigned dom = 0;
#pragma unroll
  for (int j = 0; j < NE; ++j) {
    const float a = exponent_f(z(j), c_hi, c_lo, M);
    const bool d = a > kDomArg;
    dom |= (unsigned)d << j;
    fs = __fadd_rn(fs, d ? 0.f : ex2(a));
  }
  acc = df_add(acc, fs);
  while (dom) {
    const int j = __ffs(dom) - 1;
    dom &= dom - 1;
    acc = df_add(acc, unnorm_dom(zr(j), c_hi, c_lo, M, tab));
  }
}

// acc += sum of r~ over the NE elements of a thread's chunk (target zt,
// draft zd, fetched as in unnorm_sum); returns the same sum in fp32 (for the
// chunk records).
template <int NE, class Elem, class ElemR>
__device__ __forceinline__ float residual_sum(const Elem& zt, const Elem& zd, const ElemR& ztr,
                                              const ElemR& zdr, const SpecConst& S,
                                              const float (*tab)[2], DF& acc) {
  float fs = 0.f;
  unsigned dom = 0;
#pragma unroll
  for (int j = 0; j < NE; ++j) {
    const float a = exponent_f(zt(j), S.c_hi, S.c_lo, S.Mt);
    const bool d = a > kDomArg;
    dom |= (unsigned)d << j;
    fs = __fadd_rn(fs, d ? 0.f : residual_f(a, zd(j), S));
  }
  float cr = fs;
  acc = df_add(acc, fs);
  while (dom) {
    const int j = __ffs(dom) - 1;
    dom &= dom - 1;
    const DF r = residual_dom(ztr(j), zdr(j), S, tab);
    acc = df_add(acc, r);
    cr = __fadd_rn(cr, r.hi);
  }
  return cr;
}

}  // namespace rs
