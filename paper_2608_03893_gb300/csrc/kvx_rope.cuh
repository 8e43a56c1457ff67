// Device-side RoPE angle: cos / sin of t * omega_i in fp32 with a float-float angle.
//
// Sec. 3.3 rotates pair i of a key at absolute position t by t * omega_i, omega_i =
// theta^(-2i/d).  A plain fp32 product t * omega loses up to t * 2^-24 rad (2e-3 rad
// at t = 32767), which would show in the output after the target re-rotation.  Here
// the product is kept as a float-float pair (the exact rounding error of t * omega_hi
// recovered with one FMA, plus t * omega_lo), reduced by 2*pi with the Cody-Waite
// two-constant split (W. J. Cody and W. Waite, "Software Manual for the Elementary
// Functions", 1980) using FMAs, and only then passed to the __sincosf intrinsic, whose
// documented absolute error on [-pi, pi] is 2^-21.41.  Reduction error (below 5e-7
// rad for every t < 2^24) plus that bound keeps cos and sin within 1e-6 of the
// exact values.
#pragma once

#include <cuda_runtime.h>

namespace kvx {

__device__ __forceinline__ void rope_sincos(int t, float w_hi, float w_lo, float two_pi_hi,
                                            float two_pi_lo, float inv_two_pi, float* s,
                                            float* c) {
  const float tf = static_cast<float>(t);                  // exact for t < 2^24
  const float a_hi = __fmul_rn(tf, w_hi);
  const float a_err = __fmaf_rn(tf, w_hi, -a_hi);          // exact: t*w_hi - a_hi
  const float a_lo = __fmaf_rn(tf, w_lo, a_err);
  const float q = rintf(__fmul_rn(a_hi, inv_two_pi));
  float r = __fmaf_rn(-q, two_pi_hi, a_hi);
  r = __fmaf_rn(-q, two_pi_lo, r);
  r = __fadd_rn(r, a_lo);
  __sincosf(r, s, c);
}

}  // namespace kvx
