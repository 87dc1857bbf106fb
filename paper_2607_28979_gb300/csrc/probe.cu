// mot_debug_gelu: the device GELU forms the translation kernels use, evaluated
// on caller-given points, so a test can measure each against the exact erf
// form of GELU (App. C.2: phi = GELU) on the GPU itself.
#include <cuda_fp16.h>
#include <stdint.h>

#include "gelu.cuh"
#include "mot_internal.h"

namespace mot {
namespace {

__global__ void __launch_bounds__(256) gelu_probe_kernel(int form, const float* __restrict__ u,
                                                         const float* __restrict__ g, int64_t n,
                                                         float* __restrict__ out) {
  for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < n;
       i += int64_t(gridDim.x) * blockDim.x) {
    const float x = u[i], gg = g[i];
    float y;
    if (form == 0) {   // the tensor-core MLP epilogue, zero bias: low lane of the fp16 pair
      const uint32_t p = gelu_gate_pair(__float_as_uint(x), __float_as_uint(x), 0u,
                                        __float2half2_rn(0.5f * gg));
      y = __half2float(__ushort_as_half(static_cast<unsigned short>(p & 0xFFFFu)));
    } else if (form == 1) {   // backbone epilogues: gtilde * GELU(u)
      y = gg * gelu_tanh(x);
    } else {                  // SIMT path: GELU(u) * gtilde
      y = gelu_erf(x) * gg;
    }
    out[i] = y;
  }
}

}  // namespace
}  // namespace mot

extern "C" mot_status mot_debug_gelu(int32_t form, const float* u, const float* gate, int64_t n,
                                     float* out, mot_stream_t stream) {
  if (form < 0 || form > 2 || n < 0) return MOT_ERR_INVALID_ARG;
  if (n == 0) return MOT_OK;
  if (!u || !gate || !out) return MOT_ERR_INVALID_ARG;
  const int64_t blocks = (n + 255) / 256;
  const unsigned grid = static_cast<unsigned>(blocks < 152 * 8 ? blocks : 152 * 8);
  mot::gelu_probe_kernel<<<grid, 256, 0, reinterpret_cast<cudaStream_t>(stream)>>>(form, u, gate,
                                                                                    n, out);
  return cudaGetLastError() == cudaSuccess ? MOT_OK : MOT_ERR_CUDA;
}
