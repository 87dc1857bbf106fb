// The GELU forms of the translator MLPs (App. C.2: phi = GELU), one definition
// each, shared by the kernels that evaluate them and by the device probe that
// measures them against the exact erf form.
//
//   gelu_gate_pair   tensor-core MLP epilogues (split, pair, routed and on-chip
//                    schedules): the fp32 accumulator pair rounded to fp16, plus
//                    the fp16 bias, then GELU(u) * gtilde in packed fp16x2 with
//                    the tanh form on the hardware tanh unit; fp16 result.
//   gelu_tanh        backbone translators: the tanh form in fp32 on the
//                    hardware tanh unit.
//   gelu_erf         SIMT path: the exact form with erff.
//
// The tanh form is 0.5 u (1 + tanh(sqrt(2/pi) (u + 0.044715 u^3))) (Hendrycks
// and Gimpel); it is at most 4.7e-4 from the erf form (at |u| = 2.7).
#pragma once

#include <cuda_fp16.h>

#include "ptx.cuh"

namespace mot {

// GELU(u) * g with half_g = g / 2 (the tanh form) on two fp16 lanes at once
// (HFMA2 + tanh.approx.f16x2).
__device__ __forceinline__ __half2 gelu_times_h2(__half2 u, __half2 half_g) {
  const __half2 k0 = __float2half2_rn(0.7978845608028654f);
  const __half2 k1 = __float2half2_rn(0.7978845608028654f * 0.044715f);
  const __half2 arg = __hmul2(u, __hfma2(__hmul2(u, u), k1, k0));
  const uint32_t tb = tanh_approx_f16x2(*reinterpret_cast<const uint32_t*>(&arg));
  const __half2 t = *reinterpret_cast<const __half2*>(&tb);
  const __half2 hu = __hmul2(u, half_g);
  return __hfma2(hu, t, hu);
}

// Epilogue of the first translator layer on two accumulator columns (fp32
// bits a, b) with their fp16 biases (packed in bias2): fp16x2 GELU(u) * gtilde.
__device__ __forceinline__ uint32_t gelu_gate_pair(uint32_t a, uint32_t b, uint32_t bias2,
                                                   __half2 half_g) {
  __half2 u = __float22half2_rn(make_float2(__uint_as_float(a), __uint_as_float(b)));
  u = __hadd2(u, *reinterpret_cast<const __half2*>(&bias2));
  const __half2 o = gelu_times_h2(u, half_g);
  return *reinterpret_cast<const uint32_t*>(&o);
}

// GELU(u) in fp32, the tanh form on the hardware tanh unit.
__device__ __forceinline__ float gelu_tanh(float u) {
  const float k0 = 0.7978845608028654f, k1 = 0.7978845608028654f * 0.044715f;
  const float t = tanh_approx(u * fmaf(k1, u * u, k0));
  const float hu = 0.5f * u;
  return fmaf(hu, t, hu);
}

// GELU(u) in fp32, the exact form.
__device__ __forceinline__ float gelu_erf(float u) {
  return 0.5f * u * (1.f + erff(u * 0.70710678118654752f));
}

}  // namespace mot
