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

}  // namespace

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
