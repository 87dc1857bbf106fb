// Helpers shared by the replay attention kernels (App. C.4): replay.cu (selection,
// SIMT attention, V transpose), replay_fmha.cu (full causal attention on the tensor
// cores) and replay_gattn.cu (source-guided attention on the tensor cores).
#pragma once

#include <cuda_bf16.h>

#include "replay_internal.h"
#include "ptx.cuh"

namespace mot {

// GQA group sizes with an instantiated attention kernel
__host__ __device__ constexpr bool group_ok(int g) {
  return (g >= 1 && g <= 8) || g == 12 || g == 16;
}

namespace {

__device__ __forceinline__ float bf16f(uint16_t b) { return __uint_as_float(uint32_t(b) << 16); }

// 2^x on the special-function unit (PTX ex2.approx.ftz: relative error about 2^-22, results
// below the normal range flushed to 0), for the softmax probabilities that are then rounded
// to bf16.
__device__ __forceinline__ float ex2_fast(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Order-preserving map of bf16 bits to unsigned 16-bit: larger value -> larger key.
__device__ __forceinline__ uint32_t ord16(uint16_t b) {
  return (b & 0x8000u) ? (~uint32_t(b) & 0xFFFFu) : (uint32_t(b) | 0x8000u);
}

__device__ __forceinline__ int seq_len_of(const ReplayArgs& a, int b) {
  if (b >= a.batch) return 0;
  const int L = a.seq_lens[b];
  return L < 0 ? 0 : (L > a.d.N ? a.d.N : L);
}

}  // namespace
}  // namespace mot
