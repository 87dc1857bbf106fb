// Storage-type conversions used when the weights are loaded.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "mot_internal.h"

namespace mot {
namespace {

// bf16 -> fp16 in place (same element size), round to nearest even. The
// values here are translator weights, far inside fp16's normal range.
__global__ void bf16_to_f16_kernel(uint16_t* buf, size_t n) {
  for (size_t i = blockIdx.x * size_t(blockDim.x) + threadIdx.x; i < n;
       i += size_t(gridDim.x) * blockDim.x) {
    const float f = __bfloat162float(__ushort_as_bfloat16(buf[i]));
    buf[i] = __half_as_ushort(__float2half_rn(f));
  }
}

__global__ void f32_to_f16_kernel(const float* src, uint16_t* dst, size_t n) {
  for (size_t i = blockIdx.x * size_t(blockDim.x) + threadIdx.x; i < n;
       i += size_t(gridDim.x) * blockDim.x)
    dst[i] = __half_as_ushort(__float2half_rn(src[i]));
}

// b2t[g][c][m] = fp16(b2[g][m][c]) for m < E, 0 for E <= m < 64.
__global__ void build_b2t_kernel(const float* b2, uint16_t* b2t, int G, int E, int Dt) {
  const size_t n = size_t(G) * Dt * 64;
  for (size_t i = blockIdx.x * size_t(blockDim.x) + threadIdx.x; i < n;
       i += size_t(gridDim.x) * blockDim.x) {
    const int m = static_cast<int>(i % 64);
    const size_t gc = i / 64;
    const int c = static_cast<int>(gc % Dt), g = static_cast<int>(gc / Dt);
    const float v = m < E ? b2[(size_t(g) * E + m) * Dt + c] : 0.f;
    b2t[i] = __half_as_ushort(__float2half_rn(v));
  }
}

// wg16[g][n][c] = wg[g][n][c] for n < E, 0 for E <= n < 16 (bf16 bits).
__global__ void build_wg16_kernel(const uint16_t* wg, uint16_t* wg16, int G, int E, int Ds) {
  const size_t n = size_t(G) * 16 * Ds;
  for (size_t i = blockIdx.x * size_t(blockDim.x) + threadIdx.x; i < n;
       i += size_t(gridDim.x) * blockDim.x) {
    const int c = static_cast<int>(i % Ds);
    const size_t gn = i / Ds;
    const int r = static_cast<int>(gn % 16), g = static_cast<int>(gn / 16);
    wg16[i] = r < E ? wg[(size_t(g) * E + r) * Ds + c] : uint16_t(0);
  }
}

}  // namespace

cudaError_t launch_build_wg16(const void* wg, void* wg16, int G, int E, int Ds, cudaStream_t st) {
  if (G == 0) return cudaSuccess;
  build_wg16_kernel<<<1024, 256, 0, st>>>(static_cast<const uint16_t*>(wg),
                                          static_cast<uint16_t*>(wg16), G, E, Ds);
  return cudaGetLastError();
}

cudaError_t launch_build_b2t(const float* b2, void* b2t, int G, int E, int Dt, cudaStream_t st) {
  if (G == 0) return cudaSuccess;
  build_b2t_kernel<<<1024, 256, 0, st>>>(b2, static_cast<uint16_t*>(b2t), G, E, Dt);
  return cudaGetLastError();
}

cudaError_t launch_bf16_to_f16_inplace(void* buf, size_t n, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  bf16_to_f16_kernel<<<1024, 256, 0, st>>>(static_cast<uint16_t*>(buf), n);
  return cudaGetLastError();
}

cudaError_t launch_f32_to_f16(const float* src, void* dst, size_t n, cudaStream_t st) {
  if (n == 0) return cudaSuccess;
  f32_to_f16_kernel<<<1024, 256, 0, st>>>(src, static_cast<uint16_t*>(dst), n);
  return cudaGetLastError();
}

}  // namespace mot
