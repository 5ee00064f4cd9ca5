// Activation functions shared by the GEMM epilogues and the one-launch
// forward, so that both compute bit-identical values.
#pragma once
#include "ptx.cuh"

namespace elasto {

// GELU, phi in Eq. 5 (the exact x * Phi(x) of the base ViT), in the logistic
// form of the Hendrycks & Gimpel (2016) tanh approximation with one more odd
// term: GELU(x) ~= x / (1 + 2^v), v = -2 log2(e) u(x),
//   u(x) = x (a0 + a1 s + a2 s^2),  s = min(x^2, 36),
// a0..a2 refitted by minimax on [0, 8] (paper_2609_10018_gb300/gelu_fit.py).
// |error| <= 2.52e-5 for every x (the error is even in x, and the clamp keeps
// u increasing past |x| = 6, where the logistic has saturated), against the
// 2^-9 relative rounding of the bf16 output. Two MUFU operations (ex2, rcp)
// and six FMA-pipe operations: the FC1 epilogue is issue-bound, and an
// Abramowitz & Stegun 7.1.26 erf costs about twice as many.
__device__ __forceinline__ float gelu(float x) {
  constexpr float kB0 = -2.3011213394560093f;  // -2 log2(e) a0
  constexpr float kB1 = -0.10677572400312792f;  // -2 log2(e) a1
  constexpr float kB2 = 0.0010142630552981257f;  // -2 log2(e) a2
  const float s = fminf(x * x, 36.0f);
  const float v = x * fmaf(fmaf(kB2, s, kB1), s, kB0);
  return __fdividef(x, 1.0f + ex2_approx(v));
}

}  // namespace elasto
