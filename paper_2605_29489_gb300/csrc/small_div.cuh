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

// a / c for a small integer c given as the float c and its reciprocal y = RN(1/c)
__device__ __forceinline__ float div_small(float a, float c, float y) {
  const float q = __fmul_rn(a, y);
  const float r = __fmaf_rn(-q, c, a);
  float out = __fmaf_rn(r, y, q);
  const float aa = fabsf(a);
  if (aa < 0x1p-100f && aa > 0.0f) out = __fdiv_rn(a, c);
  return out;
}

}  // namespace mp
