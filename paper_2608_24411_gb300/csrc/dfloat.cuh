// Double-float arithmetic: a value is the unevaluated sum hi + lo of two
// fp32 numbers (|lo| <= ulp(hi) / 2 after normalisation), which carries
// about 48 significant bits through additions and products.  The error-free
// transformations are the classical ones: Knuth's TwoSum (TAOCP vol. 2,
// 4.2.2), Dekker's Fast2Sum and the exact product with a fused multiply-add
// (Dekker 1971, "A floating-point technique for extending the available
// precision").  Every operation is written with explicitly rounded
// intrinsics so that the compiler cannot contract or reorder it.
//
// Used by the SpecInfer instance of the streaming kernel, whose residual
// (p - K q)_+ / N amplifies any relative error of the normalisers and of K
// by p / N (see verify_stream.cuh).
#pragma once

namespace rs {

struct DF {
  float hi, lo;
};

__device__ __forceinline__ DF df(float a) { return DF{a, 0.f}; }

// s + e = a + b exactly (any magnitudes).
__device__ __forceinline__ DF two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  const float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
  return DF{s, e};
}

// s + e = a + b exactly when |a| >= |b| (or a = 0).
__device__ __forceinline__ DF fast_two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  return DF{s, __fsub_rn(b, __fsub_rn(s, a))};
}

// p + e = a * b exactly (no underflow).
__device__ __forceinline__ DF two_prod(float a, float b) {
  const float p = __fmul_rn(a, b);
  return DF{p, __fmaf_rn(a, b, -p)};
}

__device__ __forceinline__ DF df_add(DF a, DF b) {
  const DF s = two_sum(a.hi, b.hi);
  return fast_two_sum(s.hi, __fadd_rn(s.lo, __fadd_rn(a.lo, b.lo)));
}

__device__ __forceinline__ DF df_add(DF a, float b) {
  const DF s = two_sum(a.hi, b);
  return fast_two_sum(s.hi, __fadd_rn(s.lo, a.lo));
}

__device__ __forceinline__ DF df_neg(DF a) { return DF{-a.hi, -a.lo}; }

__device__ __forceinline__ DF df_mul(DF a, DF b) {
  const DF p = two_prod(a.hi, b.hi);
  return fast_two_sum(p.hi, __fmaf_rn(a.hi, b.lo, __fmaf_rn(a.lo, b.hi, p.lo)));
}

__device__ __forceinline__ DF df_mul(DF a, float b) {
  const DF p = two_prod(a.hi, b);
  return fast_two_sum(p.hi, __fmaf_rn(a.lo, b, p.lo));
}

// a / b: one quotient digit, its remainder, a second digit (long division).
__device__ __forceinline__ DF df_div(DF a, DF b) {
  const float q1 = __fdiv_rn(a.hi, b.hi);
  const DF r = df_add(a, df_neg(df_mul(b, q1)));
  const float q2 = __fdiv_rn(r.hi, b.hi);
  return fast_two_sum(q1, q2);
}

__device__ __forceinline__ float df_value(DF a) { return __fadd_rn(a.hi, a.lo); }

// Butterfly sum of a double-float over groups of 2^LEVELS lanes (every lane
// of a group gets the same bits).
template <int LEVELS>
__device__ __forceinline__ DF df_group_sum(DF v) {
#pragma unroll
  for (int o = 1 << (LEVELS - 1); o; o >>= 1) {
    DF w;
    w.hi = __shfl_xor_sync(0xffffffffu, v.hi, o);
    w.lo = __shfl_xor_sync(0xffffffffu, v.lo, o);
    // the same operand order on both lanes of a pair: lower lane first
    v = (threadIdx.x & o) ? df_add(w, v) : df_add(v, w);
  }
  return v;
}

}  // namespace rs
