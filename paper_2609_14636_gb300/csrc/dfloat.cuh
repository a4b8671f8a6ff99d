// dfloat.cuh -- double-float (unevaluated sum hi + lo of two floats)
// arithmetic for the tiled scan (sm_103a).
//
// GB300 runs FP64 at 1/64 of its FP32 rate, and the tiled scan's sums are a
// chain of dependent additions over every row of a tile (the block scan, the
// prefix combine, the per-trajectory scan).  A pair of floats carries about
// 48 significant bits, far more than the 1e-5 relative bound on sums and the
// 1e-3 band around lambda need, and its addition is a handful of FP32
// operations.  The error-free transformations are the published ones:
// Knuth's TwoSum (exact sum and rounding error of two floats), Dekker's
// Fast2Sum (the same when |a| >= |b|), and the FMA product split (exact
// product and error); the double-float sum follows the accurate addition of
// Bailey's double-double arithmetic, renormalised twice.  The intrinsics
// (__fadd_rn and friends) keep the compiler from contracting or
// reassociating any step.
#pragma once

#include <cuda_runtime.h>

namespace stride {

struct dfloat {
  float hi, lo;  // value hi + lo, |lo| <= ulp(hi) / 2 once normalised
};

__device__ __forceinline__ dfloat df_two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  const float bb = __fsub_rn(s, a);
  const float e = __fadd_rn(__fsub_rn(a, __fsub_rn(s, bb)), __fsub_rn(b, bb));
  return dfloat{s, e};
}

// requires |a| >= |b| (or a == 0)
__device__ __forceinline__ dfloat df_fast_two_sum(float a, float b) {
  const float s = __fadd_rn(a, b);
  return dfloat{s, __fsub_rn(b, __fsub_rn(s, a))};
}

__device__ __forceinline__ dfloat df_from(float x) { return dfloat{x, 0.f}; }

__device__ __forceinline__ dfloat df_from_double(double d) {
  const float hi = __double2float_rn(d);
  return dfloat{hi, __double2float_rn(d - (double)hi)};
}

__device__ __forceinline__ double df_to_double(dfloat a) { return (double)a.hi + (double)a.lo; }

__device__ __forceinline__ dfloat df_add(dfloat a, dfloat b) {
  dfloat s = df_two_sum(a.hi, b.hi);
  const dfloat t = df_two_sum(a.lo, b.lo);
  s.lo = __fadd_rn(s.lo, t.hi);
  s = df_fast_two_sum(s.hi, s.lo);
  s.lo = __fadd_rn(s.lo, t.lo);
  return df_fast_two_sum(s.hi, s.lo);
}

__device__ __forceinline__ dfloat df_neg(dfloat a) { return dfloat{-a.hi, -a.lo}; }

// exact product of two floats
__device__ __forceinline__ dfloat df_mul_ff(float a, float b) {
  const float p = __fmul_rn(a, b);
  return dfloat{p, __fmaf_rn(a, b, -p)};
}

// a / n for a count n (exact in float: n < 2^24): the quotient's leading
// float, the exact remainder by FMA, and its quotient as the trailing part.
__device__ __forceinline__ dfloat df_div_count(dfloat a, float n) {
  const float q1 = __fdiv_rn(a.hi, n);
  const float r = __fadd_rn(__fmaf_rn(-q1, n, a.hi), a.lo);
  return df_fast_two_sum(q1, __fdiv_rn(r, n));
}

// Comparisons with a float threshold; false for NaN, as for the double
// comparisons they replace.
__device__ __forceinline__ bool df_lt(dfloat a, float x) { return a.hi < x || (a.hi == x && a.lo < 0.f); }
__device__ __forceinline__ bool df_ge(dfloat a, float x) { return a.hi > x || (a.hi == x && a.lo >= 0.f); }

__device__ __forceinline__ dfloat df_shfl_up(dfloat v, int d) {
  return dfloat{__shfl_up_sync(0xffffffffu, v.hi, d), __shfl_up_sync(0xffffffffu, v.lo, d)};
}

}  // namespace stride
