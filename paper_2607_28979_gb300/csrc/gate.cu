// Ragged token-tile list and the per-token gate (Def. 3.1).
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "mot_internal.h"

namespace mot {

// ---------------------------------------------------------------- tile list

// One block. Clamps every length into [0, S] (flagging kStatusSeqLen), then
// lays the 128-token tiles of all batch entries out contiguously: tile i
// covers rows [i*128, i*128+128) of the gate / A2 workspaces.
__global__ void prep_tiles_kernel(const int32_t* __restrict__ seq_lens, int32_t batch, int32_t S,
                                  TileInfo* __restrict__ tiles, int32_t* __restrict__ n_tiles,
                                  int32_t* __restrict__ status) {
  __shared__ int32_t s_len[4096];
  __shared__ int32_t s_off[4096];
  for (int b = threadIdx.x; b < batch; b += blockDim.x) {
    int32_t L = seq_lens[b];
    if (L < 0 || L > S) {
      atomicOr(status, kStatusSeqLen);
      L = L < 0 ? 0 : S;
    }
    s_len[b] = L;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int32_t acc = 0;
    for (int b = 0; b < batch; ++b) {
      s_off[b] = acc;
      acc += (s_len[b] + kTileM - 1) / kTileM;
    }
    *n_tiles = acc;
  }
  __syncthreads();
  for (int b = threadIdx.x; b < batch; b += blockDim.x) {
    const int32_t L = s_len[b];
    const int32_t nt = (L + kTileM - 1) / kTileM;
    for (int t = 0; t < nt; ++t) {
      TileInfo ti;
      ti.b = b;
      ti.s0 = t * kTileM;
      ti.rows = min(kTileM, L - t * kTileM);
      ti.pad = 0;
      tiles[s_off[b] + t] = ti;
    }
  }
}

cudaError_t launch_prep(const int32_t* seq_lens, int32_t batch, const Dims& d, TileInfo* tiles,
                        int32_t* n_tiles, int32_t* status, cudaStream_t st) {
  prep_tiles_kernel<<<1, 256, 0, st>>>(seq_lens, batch, d.S, tiles, n_tiles, status);
  return cudaGetLastError();
}

// ---------------------------------------------------------------- gate

template <typename T>
struct Vec;
template <>
struct Vec<__nv_bfloat16> {
  static constexpr int N = 8;   // 16-byte loads
  __device__ static void load(const __nv_bfloat16* p, float (&v)[8]) {
    const uint4 u = *reinterpret_cast<const uint4*>(p);
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&u);
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 f = __bfloat1622float2(h[k]);
      v[2 * k] = f.x;
      v[2 * k + 1] = f.y;
    }
  }
};
template <>
struct Vec<float> {
  static constexpr int N = 4;
  __device__ static void load(const float* p, float (&v)[4]) {
    const float4 u = *reinterpret_cast<const float4*>(p);
    v[0] = u.x; v[1] = u.y; v[2] = u.z; v[3] = u.w;
  }
};

// The fp16 gate row of the tensor-core path: gtilde in columns [0, E), zeros up
// to 64 (one K block of GEMM2's bias step). `g` may be null (all zeros).
__device__ __forceinline__ void write_gate16(const PathArgs& a, int grp, size_t row, const float* g,
                                             int E) {
  if (!a.gate16) return;
  uint4* out = reinterpret_cast<uint4*>(static_cast<uint16_t*>(a.gate16) +
                                        (static_cast<size_t>(grp) * a.d.tpad + row) * 64);
#pragma unroll
  for (int v = 0; v < 8; ++v) {
    uint32_t w[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int e0 = v * 8 + 2 * k;
      const float lo = (g && e0 < E) ? g[e0] : 0.f, hi = (g && e0 + 1 < E) ? g[e0 + 1] : 0.f;
      const __half2 h = __floats2half2_rn(lo, hi);
      w[k] = *reinterpret_cast<const uint32_t*>(&h);
    }
    out[v] = make_uint4(w[0], w[1], w[2], w[3]);
  }
}

__device__ __forceinline__ float to_f(float x) { return x; }
__device__ __forceinline__ float to_f(__nv_bfloat16 x) { return __bfloat162float(x); }

// Grid (tiles_max, gp), 256 threads: each warp produces the gate of 16 token
// rows of one tile for one (layer, K/V) group. Lanes split the D_s channels
// (VEC-wide vectors when the head dim allows it), reduce the E logits with
// warp shuffles, and lane 0 applies the max-subtracted softmax and the Top-K
// renormalisation. Rows past the tile's length get a zero gate.
template <typename T, bool VEC>
__global__ void __launch_bounds__(256) gate_kernel(PathArgs a) {
  const Dims& d = a.d;
  const int m = blockIdx.x;
  const int grp = a.g0 + blockIdx.y;
  if (m >= *a.n_tiles) return;
  const TileInfo ti = a.tiles[m];
  const GroupInfo gi = a.groups[grp];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int E = d.E;
  const T* __restrict__ src = static_cast<const T*>(a.src[gi.x]);
  const T* __restrict__ wg = static_cast<const T*>(a.wg) + static_cast<size_t>(grp) * E * d.Ds;
  const float* __restrict__ bg = a.bg + static_cast<size_t>(grp) * E;
  constexpr int NV = VEC ? Vec<T>::N : 1;

  for (int r = warp; r < kTileM; r += 8) {
    float* __restrict__ gout = a.gate + (static_cast<size_t>(grp) * d.tpad + static_cast<size_t>(m) * kTileM + r) * E;
    if (r >= ti.rows) {
      if (lane < E) gout[lane] = 0.f;
      if (lane == 0) write_gate16(a, grp, static_cast<size_t>(m) * kTileM + r, nullptr, E);
      continue;
    }
    const int s = ti.s0 + r;
    float acc[kMaxE];
#pragma unroll
    for (int e = 0; e < kMaxE; ++e) acc[e] = 0.f;
    for (int c = lane * NV; c < d.Ds; c += 32 * NV) {
      const int h = c / d.d_s, i = c - h * d.d_s;
      const T* zp = src + ((((static_cast<size_t>(gi.src_layer) * d.B + ti.b) * d.H_s + h) * d.S + s) * d.d_s + i);
      float z[NV];
      if constexpr (VEC) {
        Vec<T>::load(zp, z);
      } else {
        z[0] = to_f(*zp);
      }
#pragma unroll
      for (int e = 0; e < kMaxE; ++e) {
        if (e < E) {
          float w[NV];
          if constexpr (VEC) {
            Vec<T>::load(wg + static_cast<size_t>(e) * d.Ds + c, w);
          } else {
            w[0] = to_f(wg[static_cast<size_t>(e) * d.Ds + c]);
          }
#pragma unroll
          for (int k = 0; k < NV; ++k) acc[e] = fmaf(w[k], z[k], acc[e]);
        }
      }
    }
#pragma unroll
    for (int e = 0; e < kMaxE; ++e) {
      if (e < E) {
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], off);
      }
    }
    if (lane == 0) {
      float g[kMaxE];
      float mx = -INFINITY;
#pragma unroll
      for (int e = 0; e < kMaxE; ++e)
        if (e < E) {
          g[e] = acc[e] + bg[e];
          mx = fmaxf(mx, g[e]);
        }
      float sum = 0.f;
#pragma unroll
      for (int e = 0; e < kMaxE; ++e)
        if (e < E) {
          g[e] = expf(g[e] - mx);
          sum += g[e];
        }
      const float inv = 1.f / sum;
#pragma unroll
      for (int e = 0; e < kMaxE; ++e)
        if (e < E) g[e] *= inv;
      if (d.top_k > 0 && d.top_k < E) {
        // keep the top_k largest scores (equal scores: lower index first)
        uint32_t keep = 0;
        for (int k = 0; k < d.top_k; ++k) {
          int best = -1;
          float bv = 0.f;
#pragma unroll
          for (int e = 0; e < kMaxE; ++e)
            if (e < E && !((keep >> e) & 1u) && (best < 0 || g[e] > bv)) {
              best = e;
              bv = g[e];
            }
          keep |= 1u << best;
        }
        float ks = 0.f;
#pragma unroll
        for (int e = 0; e < kMaxE; ++e)
          if (e < E && ((keep >> e) & 1u)) ks += g[e];
        const float kinv = 1.f / ks;
#pragma unroll
        for (int e = 0; e < kMaxE; ++e)
          if (e < E) g[e] = ((keep >> e) & 1u) ? g[e] * kinv : 0.f;
      }
#pragma unroll
      for (int e = 0; e < kMaxE; ++e)
        if (e < E) gout[e] = g[e];
      write_gate16(a, grp, static_cast<size_t>(m) * kTileM + r, g, E);
    }
  }
}

// Tile-wide variant for head dims that split into CPR 16-byte chunks with CPR
// dividing 256: block (tile m, group) of 256 threads; thread t owns channel
// chunk t % CPR of every head and rows t / CPR + p * (256 / CPR), p < P. A
// warp's loads of one head then cover 512 contiguous bytes of the cache (the
// tile's rows of one head are contiguous), every load is independent, and the
// CPR partial dot products of a row are summed with shuffles inside a warp.
template <typename T, int CPR, int P, int EMAX>
__global__ void __launch_bounds__(256) gate_tile_kernel(PathArgs a) {
  const Dims& d = a.d;
  const int m = blockIdx.x;
  const int grp = a.g0 + blockIdx.y;
  if (m >= *a.n_tiles) return;
  const TileInfo ti = a.tiles[m];
  const GroupInfo gi = a.groups[grp];
  constexpr int NV = Vec<T>::N;
  constexpr int RPP = 256 / CPR;   // rows per pass
  const int E = d.E;
  const int cp = (threadIdx.x % CPR) * NV;   // channel offset inside a head
  const int r0 = threadIdx.x / CPR;
  const T* __restrict__ src = static_cast<const T*>(a.src[gi.x]);
  const T* __restrict__ wg = static_cast<const T*>(a.wg) + static_cast<size_t>(grp) * E * d.Ds;
  float acc[P][EMAX];
#pragma unroll
  for (int p = 0; p < P; ++p)
#pragma unroll
    for (int e = 0; e < EMAX; ++e) acc[p][e] = 0.f;
  // Software pipeline over heads: the raw 16-byte loads of head h + 1 are in
  // flight while head h is multiplied, so each thread keeps 2 * P loads
  // outstanding instead of P.
  const size_t head_stride = static_cast<size_t>(d.S) * d.d_s;
  const T* base0 = src + ((static_cast<size_t>(gi.src_layer) * d.B + ti.b) * d.H_s * d.S + ti.s0) * d.d_s + cp;
  uint4 raw_cur[P], raw_nxt[P];
#pragma unroll
  for (int p = 0; p < P; ++p) {
    const int r = r0 + p * RPP;
    raw_cur[p] = r < ti.rows ? *reinterpret_cast<const uint4*>(base0 + static_cast<size_t>(r) * d.d_s)
                             : make_uint4(0, 0, 0, 0);
  }
  for (int h = 0; h < d.H_s; ++h) {
    if (h + 1 < d.H_s) {
      const T* bn = base0 + (h + 1) * head_stride;
#pragma unroll
      for (int p = 0; p < P; ++p) {
        const int r = r0 + p * RPP;
        raw_nxt[p] = r < ti.rows ? *reinterpret_cast<const uint4*>(bn + static_cast<size_t>(r) * d.d_s)
                                 : make_uint4(0, 0, 0, 0);
      }
    }
    float w[EMAX][NV];
#pragma unroll
    for (int e = 0; e < EMAX; ++e) {
      if (e < E) {
        Vec<T>::load(wg + static_cast<size_t>(e) * d.Ds + h * d.d_s + cp, w[e]);
      } else {
#pragma unroll
        for (int k = 0; k < NV; ++k) w[e][k] = 0.f;
      }
    }
#pragma unroll
    for (int p = 0; p < P; ++p) {
      float z[NV];
      Vec<T>::load(reinterpret_cast<const T*>(&raw_cur[p]), z);
#pragma unroll
      for (int e = 0; e < EMAX; ++e)
#pragma unroll
        for (int k = 0; k < NV; ++k) acc[p][e] = fmaf(w[e][k], z[k], acc[p][e]);
    }
#pragma unroll
    for (int p = 0; p < P; ++p) raw_cur[p] = raw_nxt[p];
  }
#pragma unroll
  for (int p = 0; p < P; ++p)
#pragma unroll
    for (int e = 0; e < EMAX; ++e)
#pragma unroll
      for (int off = CPR / 2; off > 0; off >>= 1)
        acc[p][e] += __shfl_xor_sync(0xffffffffu, acc[p][e], off);
  // Every thread of a row's CPR group now holds the row's logits: each one
  // evaluates the softmax (cheap, E values) and writes its slice of the fp16
  // gate row; the group's first thread also writes the fp32 gate.
  const int j = threadIdx.x % CPR;
  constexpr int kSlice = 64 / CPR;   // fp16 gate16 elements per thread (8 or 4)
  const float* __restrict__ bg = a.bg + static_cast<size_t>(grp) * E;
#pragma unroll
  for (int p = 0; p < P; ++p) {
    const int r = r0 + p * RPP;
    const size_t row = static_cast<size_t>(m) * kTileM + r;
    float* __restrict__ gout = a.gate + (static_cast<size_t>(grp) * d.tpad + row) * E;
    float g[EMAX];
    if (r >= ti.rows) {
#pragma unroll
      for (int e = 0; e < EMAX; ++e) g[e] = 0.f;
    } else {
      float mx = -INFINITY;
#pragma unroll
      for (int e = 0; e < EMAX; ++e)
        if (e < E) {
          g[e] = acc[p][e] + bg[e];
          mx = fmaxf(mx, g[e]);
        }
      float sum = 0.f;
#pragma unroll
      for (int e = 0; e < EMAX; ++e)
        if (e < E) {
          g[e] = expf(g[e] - mx);
          sum += g[e];
        }
      const float inv = 1.f / sum;
#pragma unroll
      for (int e = 0; e < EMAX; ++e) g[e] = e < E ? g[e] * inv : 0.f;
      if (d.top_k > 0 && d.top_k < E) {
        uint32_t keep = 0;
        for (int k = 0; k < d.top_k; ++k) {
          int best = -1;
          float bv = 0.f;
#pragma unroll
          for (int e = 0; e < EMAX; ++e)
            if (e < E && !((keep >> e) & 1u) && (best < 0 || g[e] > bv)) {
              best = e;
              bv = g[e];
            }
          keep |= 1u << best;
        }
        float ks = 0.f;
#pragma unroll
        for (int e = 0; e < EMAX; ++e)
          if (e < E && ((keep >> e) & 1u)) ks += g[e];
        const float kinv = 1.f / ks;
#pragma unroll
        for (int e = 0; e < EMAX; ++e) g[e] = (e < E && ((keep >> e) & 1u)) ? g[e] * kinv : 0.f;
      }
    }
    if (j == 0) {
#pragma unroll
      for (int e = 0; e < EMAX; ++e)
        if (e < E) gout[e] = g[e];
    }
    if (a.gate16) {
      uint16_t* out = static_cast<uint16_t*>(a.gate16) +
                      (static_cast<size_t>(grp) * d.tpad + row) * 64 + j * kSlice;
      uint32_t w[kSlice / 2];
#pragma unroll
      for (int k = 0; k < kSlice / 2; ++k) {
        const int e0 = j * kSlice + 2 * k;   // this thread's columns e0, e0 + 1
        float lo = 0.f, hi = 0.f;
#pragma unroll
        for (int e = 0; e < EMAX; ++e) {   // register selects, no indexed access
          lo = e == e0 ? g[e] : lo;
          hi = e == e0 + 1 ? g[e] : hi;
        }
        const __half2 hv = __floats2half2_rn(lo, hi);
        w[k] = *reinterpret_cast<const uint32_t*>(&hv);
      }
      if constexpr (kSlice == 8)
        *reinterpret_cast<uint4*>(out) = make_uint4(w[0], w[1], w[2], w[3]);
      else
        *reinterpret_cast<uint2*>(out) = make_uint2(w[0], w[1]);
    }
  }
}

// Gate of groups [a.g0, a.g0 + a.gp).
// Test hook: the gate rows of every tile taken from a caller buffer
// fg[G][B][S][E] (fp32) instead of the gate's linear map and softmax, written
// in the layouts the translators read (fp32 rows and the fp16 bias-block rows).
// Grid (tiles_max, gp), one thread per tile row.
__global__ void __launch_bounds__(kTileM) fixed_gate_kernel(PathArgs a, const float* __restrict__ fg) {
  const Dims& d = a.d;
  const int m = blockIdx.x;
  const int grp = a.g0 + blockIdx.y;
  if (m >= *a.n_tiles) return;
  const TileInfo ti = a.tiles[m];
  const int r = threadIdx.x;
  const bool real = r < ti.rows;
  float g[kMaxE];
#pragma unroll
  for (int e = 0; e < kMaxE; ++e)
    g[e] = (real && e < d.E)
               ? fg[((static_cast<size_t>(grp) * d.B + ti.b) * d.S + ti.s0 + r) * d.E + e]
               : 0.f;
  float* gout = a.gate + (static_cast<size_t>(grp) * d.tpad + static_cast<size_t>(m) * kTileM + r) * d.E;
#pragma unroll
  for (int e = 0; e < kMaxE; ++e)
    if (e < d.E) gout[e] = g[e];
  write_gate16(a, grp, static_cast<size_t>(m) * kTileM + r, real ? g : nullptr, d.E);
}

cudaError_t launch_fixed_gate(const PathArgs& a, const float* fg, cudaStream_t st) {
  if (a.gp <= 0) return cudaSuccess;
  fixed_gate_kernel<<<dim3(a.d.tiles_max, a.gp), kTileM, 0, st>>>(a, fg);
  return cudaGetLastError();
}

cudaError_t launch_gate(const PathArgs& a, cudaStream_t st) {
  const Dims& d = a.d;
  if (a.gp <= 0) return cudaSuccess;
  dim3 grid(d.tiles_max, a.gp);
  // tile-wide kernel: 16-byte chunks per head row (CPR) of 8 or 16, E <= 8
  if (d.dtype == 0 && d.E <= 4 && d.d_s == 64) {
    gate_tile_kernel<__nv_bfloat16, 8, 4, 4><<<grid, 256, 0, st>>>(a);
  } else if (d.dtype == 0 && d.E <= 8 && d.d_s == 64) {
    gate_tile_kernel<__nv_bfloat16, 8, 4, 8><<<grid, 256, 0, st>>>(a);
  } else if (d.dtype == 0 && d.E <= 4 && d.d_s == 128) {
    gate_tile_kernel<__nv_bfloat16, 16, 8, 4><<<grid, 256, 0, st>>>(a);
  } else if (d.dtype == 0 && d.E <= 8 && d.d_s == 128) {
    gate_tile_kernel<__nv_bfloat16, 16, 8, 8><<<grid, 256, 0, st>>>(a);
  } else if (d.dtype == 0) {
    if (d.d_s % 8 == 0)
      gate_kernel<__nv_bfloat16, true><<<grid, 256, 0, st>>>(a);
    else
      gate_kernel<__nv_bfloat16, false><<<grid, 256, 0, st>>>(a);
  } else {
    if (d.d_s % 4 == 0)
      gate_kernel<float, true><<<grid, 256, 0, st>>>(a);
    else
      gate_kernel<float, false><<<grid, 256, 0, st>>>(a);
  }
  return cudaGetLastError();
}

}  // namespace mot
