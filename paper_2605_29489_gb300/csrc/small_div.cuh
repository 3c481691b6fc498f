// Division by a small positive integer count with a precomputed reciprocal.
//
// q = RN(a * y) with y = RN(1/c), then one correction step with the residual
// r = RN(a - q * c) (one fma): q' = RN(q + r * y).  This is Markstein's correction
// (P. W. Markstein, "Computation of elementary functions on the IBM RISC System/6000
// processor", IBM J. Res. Dev. 34(1), 1990): with y within half an ulp of 1/c and q within
// an ulp of a/c it yields the correctly rounded quotient while the quotient and the
// residual stay in the normal range.  Numerators 0 < |a| < 2^-100 (quotients that may be
// subnormal after dividing by c <= 32) take the IEEE division instead.  For every finite
// a other than -0 (the correction turns -0 / c into +0; the merge never divides -0) and
// every c in 1..32 the result equals a / c rounded to nearest-even; an exhaustive GPU
// test checks exactly that against the CUDA division.
#pragma once

namespace mp {

// the correction step alone: a / c rounded to nearest-even unless div_small_needs_ieee(a)
__device__ __forceinline__ float div_small_fast(float a, float c, float y) {
  const float q = __fmul_rn(a, y);
  const float r = __fmaf_rn(-q, c, a);
  return __fmaf_rn(r, y, q);
}

// true for the numerators 0 < |a| < 2^-100, which take the IEEE division
__device__ __forceinline__ bool div_small_needs_ieee(float a) {
  return (__float_as_uint(a) & 0x7FFFFFFFu) - 1u < 0x0D7FFFFFu;  // bits of 2^-100 are 0x0D800000
}

// a / c for a small integer c given as the float c and its reciprocal y = RN(1/c)
__device__ __forceinline__ float div_small(float a, float c, float y) {
  return div_small_needs_ieee(a) ? __fdiv_rn(a, c) : div_small_fast(a, c, y);
}

}  // namespace mp
