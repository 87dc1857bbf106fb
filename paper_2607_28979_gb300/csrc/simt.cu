// SIMT translation path: plain fp32 FFMA GEMMs (no TF32, no tensor cores).
// Used for fp32 caches, where the accuracy target needs true fp32 products,
// and for bf16 shapes that the tcgen05 tiling does not cover.
//
//   GEMM1:  a2[row][j] = GELU(z_row . W1cat[j] + b1[j]) * gate[row][j / H]
//   GEMM2:  y[row][c]  = a2[row] . W2cat[c] + sum_m gate[row][m] * b2[m][c]
//           stored into the target cache at (layer, b, c / d_t, s, c % d_t).
// GELU is the exact erf form; a2 is kept in fp32.
#include <cuda_bf16.h>

#include "gelu.cuh"
#include "mot_internal.h"

namespace mot {
namespace {

constexpr int BM = 64, BN = 64, BK = 32;

__device__ __forceinline__ float ld_f(const float* p) { return *p; }
__device__ __forceinline__ float ld_f(const __nv_bfloat16* p) { return __bfloat162float(*p); }
__device__ __forceinline__ void st_v(float* p, float v) { *p = v; }
__device__ __forceinline__ void st_v(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }

// Grid (2*tiles_max, ceil(EH/64), gp), 256 threads, 4x4 outputs per thread.
template <typename T>
__global__ void __launch_bounds__(256) simt_gemm1_kernel(PathArgs a) {
  const Dims& d = a.d;
  const int m = blockIdx.x >> 1, half = blockIdx.x & 1;
  if (m >= *a.n_tiles) return;
  const TileInfo ti = a.tiles[m];
  const int row0 = half * BM;   // row offset inside the 128-row tile
  if (row0 >= ti.rows) return;
  const int gl = blockIdx.z, grp = a.g0 + gl;
  const GroupInfo gi = a.groups[grp];
  const int n0 = blockIdx.y * BN;
  const T* __restrict__ src = static_cast<const T*>(a.src[gi.x]);
  const T* __restrict__ w1 = static_cast<const T*>(a.w1) + static_cast<size_t>(grp) * d.EH * d.Ds;

  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};

  for (int k0 = 0; k0 < d.Ds; k0 += BK) {
    for (int e = threadIdx.x; e < BM * BK; e += 256) {
      const int r = e / BK, kk = e % BK, c = k0 + kk;
      float v = 0.f;
      if (row0 + r < ti.rows && c < d.Ds) {
        const int h = c / d.d_s, i = c - h * d.d_s;
        v = ld_f(src + ((((static_cast<size_t>(gi.src_layer) * d.B + ti.b) * d.H_s + h) * d.S +
                         (ti.s0 + row0 + r)) * d.d_s + i));
      }
      As[kk][r] = v;
    }
    for (int e = threadIdx.x; e < BN * BK; e += 256) {
      const int j = e / BK, kk = e % BK, c = k0 + kk;
      Bs[kk][j] = (n0 + j < d.EH && c < d.Ds) ? ld_f(w1 + static_cast<size_t>(n0 + j) * d.Ds + c) : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < BK; ++kk) {
      float av[4], bv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) av[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) bv[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
    }
    __syncthreads();
  }
  float* __restrict__ a2 = static_cast<float*>(a.a2);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = row0 + ty * 4 + i;   // row inside the tile
    if (r >= ti.rows) continue;
    const size_t grow = static_cast<size_t>(m) * kTileM + r;
    const float* g = a.gate + (static_cast<size_t>(grp) * d.tpad + grow) * d.E;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int col = n0 + tx * 4 + j;
      if (col >= d.EH) continue;
      const float u = acc[i][j] + a.b1[static_cast<size_t>(grp) * d.EH + col];
      a2[(static_cast<size_t>(gl) * d.tpad + grow) * d.EH + col] = gelu_erf(u) * g[col / d.H];
    }
  }
}

// Grid (2*tiles_max, ceil(Dt/64), gp), 256 threads, 4x4 outputs per thread.
template <typename T>
__global__ void __launch_bounds__(256) simt_gemm2_kernel(PathArgs a) {
  const Dims& d = a.d;
  const int m = blockIdx.x >> 1, half = blockIdx.x & 1;
  if (m >= *a.n_tiles) return;
  const TileInfo ti = a.tiles[m];
  const int row0 = half * BM;
  if (row0 >= ti.rows) return;
  const int gl = blockIdx.z, grp = a.g0 + gl;
  const GroupInfo gi = a.groups[grp];
  const int n0 = blockIdx.y * BN;
  const float* __restrict__ a2 = static_cast<const float*>(a.a2);
  const T* __restrict__ w2 = static_cast<const T*>(a.w2) + static_cast<size_t>(grp) * d.Dt * d.EH;

  __shared__ float As[BK][BM + 4];
  __shared__ float Bs[BK][BN + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  float acc[4][4] = {};

  for (int k0 = 0; k0 < d.EH; k0 += BK) {
    for (int e = threadIdx.x; e < BM * BK; e += 256) {
      const int r = e / BK, kk = e % BK, j = k0 + kk;
      float v = 0.f;
      if (row0 + r < ti.rows && j < d.EH)
        v = a2[(static_cast<size_t>(gl) * d.tpad + static_cast<size_t>(m) * kTileM + row0 + r) * d.EH + j];
      As[kk][r] = v;
    }
    for (int e = threadIdx.x; e < BN * BK; e += 256) {
      const int c = e / BK, kk = e % BK, j = k0 + kk;
      Bs[kk][c] = (n0 + c < d.Dt && j < d.EH) ? ld_f(w2 + static_cast<size_t>(n0 + c) * d.EH + j) : 0.f;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < BK; ++kk) {
      float av[4], bv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) av[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) bv[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
    }
    __syncthreads();
  }
  T* __restrict__ dst = static_cast<T*>(a.dst[gi.x]);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = row0 + ty * 4 + i;
    if (r >= ti.rows) continue;
    const int s = ti.s0 + r;
    const float* g = a.gate + (static_cast<size_t>(grp) * d.tpad + static_cast<size_t>(m) * kTileM + r) * d.E;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int c = n0 + tx * 4 + j;
      if (c >= d.Dt) continue;
      float y = acc[i][j];
      for (int e = 0; e < d.E; ++e)
        y = fmaf(g[e], a.b2[(static_cast<size_t>(grp) * d.E + e) * d.Dt + c], y);
      const int h = c / d.d_t, ii = c - h * d.d_t;
      st_v(dst + ((((static_cast<size_t>(gi.tgt_layer) * d.B + ti.b) * d.H_t + h) * d.S + s) * d.d_t + ii), y);
    }
  }
}

}  // namespace

cudaError_t launch_simt_gemm1(const PathArgs& a, cudaStream_t st) {
  const Dims& d = a.d;
  dim3 grid(2 * d.tiles_max, (d.EH + BN - 1) / BN, a.gp);
  if (d.dtype == 0)
    simt_gemm1_kernel<__nv_bfloat16><<<grid, 256, 0, st>>>(a);
  else
    simt_gemm1_kernel<float><<<grid, 256, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_simt_gemm2(const PathArgs& a, cudaStream_t st) {
  const Dims& d = a.d;
  dim3 grid(2 * d.tiles_max, (d.Dt + BN - 1) / BN, a.gp);
  if (d.dtype == 0)
    simt_gemm2_kernel<__nv_bfloat16><<<grid, 256, 0, st>>>(a);
  else
    simt_gemm2_kernel<float><<<grid, 256, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace mot
