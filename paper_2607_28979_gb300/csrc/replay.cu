// Replay attention of the post-translation phase (App. C.4) on sm_103a:
// Top-S source-guided sparse attention, and full causal attention for the
// L_Full bottom layers.
//
//   replay_select_kernel  one CTA per context row (b, u): the S positions j <= u
//                         with the largest guidance score A[b][u][j] (ties to the
//                         lower position), written in ascending order. Each
//                         candidate gets the unique 32-bit key
//                         (order-preserving bits of A) << 16 | (0xFFFF - j), so the
//                         selection is exact integer work: an MSB-first radix
//                         select (four 8-bit digits, 256-bin shared histograms)
//                         finds the S-th largest key, and a block scan compacts
//                         the keys at or above it. Rows with u + 1 <= S take every
//                         position.
//   replay_attn_kernel    one CTA per (b, key/value head, u): the query heads of
//                         the GQA group attend to the selected rows (sparse) or to
//                         positions 0..u in 128-key chunks with an online softmax
//                         (full). Thread t scores key t of the chunk against every
//                         query of the group (its key row read as 16-byte vectors),
//                         the softmax is fp32, and thread i accumulates output
//                         dimension i over the chunk's value rows (coalesced
//                         across the warp).
#include <cuda_bf16.h>

#include "mot_internal.h"

namespace mot {
namespace {

constexpr int kSelThreads = 256;
constexpr int kAttnThreads = 128;   // = the key chunk
constexpr int kMaxGroup = 16;       // query heads per key/value head

__device__ __forceinline__ float bf16f(uint16_t b) { return __uint_as_float(uint32_t(b) << 16); }

// Order-preserving map of bf16 bits to unsigned 16-bit: larger value -> larger key.
__device__ __forceinline__ uint32_t ord16(uint16_t b) {
  return (b & 0x8000u) ? (~uint32_t(b) & 0xFFFFu) : (uint32_t(b) | 0x8000u);
}

__device__ __forceinline__ int seq_len_of(const ReplayArgs& a, int b) {
  if (b >= a.batch) return 0;
  const int L = a.seq_lens[b];
  return L < 0 ? 0 : (L > a.d.N ? a.d.N : L);
}

// Exclusive scan of one value per thread over the block (kSelThreads threads).
__device__ __forceinline__ int block_excl_scan(int v, int* warp_sums, int& total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < kSelThreads / 32 ? warp_sums[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < kSelThreads / 32) warp_sums[lane] = w;   // inclusive warp prefix
  }
  __syncthreads();
  const int before = warp > 0 ? warp_sums[warp - 1] : 0;
  total = warp_sums[kSelThreads / 32 - 1];
  __syncthreads();
  return before + x - v;
}

__global__ void __launch_bounds__(kSelThreads) replay_select_kernel(const ReplayArgs a) {
  __shared__ int hist[256];
  __shared__ int warp_sums[kSelThreads / 32];
  __shared__ uint32_t s_prefix;
  __shared__ int s_k;
  const ReplayDims& d = a.d;
  const int row = blockIdx.x;
  const int b = row / d.N, u = row - b * d.N;
  if (u >= seq_len_of(a, b)) return;
  int32_t* out = a.sel + int64_t(row) * d.S;
  const int n = u + 1;
  if (n <= d.S) {
    for (int j = threadIdx.x; j < d.S; j += kSelThreads) out[j] = j < n ? j : -1;
    return;
  }
  const uint16_t* A = static_cast<const uint16_t*>(a.guide) + int64_t(row) * d.N;
  // this thread's contiguous chunk of candidates (ascending positions across threads)
  const int C = (n + kSelThreads - 1) / kSelThreads;
  const int j0 = min(n, int(threadIdx.x) * C), j1 = min(n, j0 + C);
  if (threadIdx.x == 0) {
    s_prefix = 0;
    s_k = d.S;
  }
  // MSB-first radix select of the S-th largest key (digits of 8 bits)
  for (int shift = 24; shift >= 0; shift -= 8) {
    for (int i = threadIdx.x; i < 256; i += kSelThreads) hist[i] = 0;
    __syncthreads();
    const uint32_t prefix = s_prefix;
    const uint32_t hi_mask = shift == 24 ? 0u : (0xFFFFFFFFu << (shift + 8));
    for (int j = j0; j < j1; ++j) {
      const uint32_t key = (ord16(A[j]) << 16) | (0xFFFFu - uint32_t(j));
      if ((key & hi_mask) == prefix) atomicAdd(&hist[(key >> shift) & 0xFFu], 1);
    }
    __syncthreads();
    if (threadIdx.x == 0) {   // from the top bin down: the bin holding the k-th largest
      int k = s_k, bin = 255;
      for (; bin > 0; --bin) {
        if (hist[bin] >= k) break;
        k -= hist[bin];
      }
      s_k = k;
      s_prefix = prefix | (uint32_t(bin) << shift);
    }
    __syncthreads();
  }
  const uint32_t thr = s_prefix;   // the S-th largest key: exactly S keys are >= thr
  int cnt = 0;
  for (int j = j0; j < j1; ++j)
    cnt += ((ord16(A[j]) << 16) | (0xFFFFu - uint32_t(j))) >= thr;
  int total;
  int pos = block_excl_scan(cnt, warp_sums, total);
  for (int j = j0; j < j1; ++j)
    if (((ord16(A[j]) << 16) | (0xFFFFu - uint32_t(j))) >= thr) out[pos++] = j;
}

template <int D>
__global__ void __launch_bounds__(kAttnThreads) replay_attn_kernel(const ReplayArgs a) {
  __shared__ float qs[kMaxGroup][D];
  __shared__ float ps[kMaxGroup][kAttnThreads];
  __shared__ int32_t idx[kAttnThreads];
  __shared__ float red[kMaxGroup][kAttnThreads / 32];
  const ReplayDims& d = a.d;
  const int G = d.Hq / d.Hkv;
  const int u = blockIdx.x;
  const int hk = blockIdx.y % d.Hkv, b = blockIdx.y / d.Hkv;
  if (u >= seq_len_of(a, b)) return;
  const int t = threadIdx.x, lane = t & 31, warp = t >> 5;
  const float scale = rsqrtf(float(D));
  // the group's queries, pre-scaled
  for (int i = t; i < G * D; i += kAttnThreads) {
    const int g = i / D, c = i - g * D;
    const int h = hk * G + g;
    qs[g][c] = bf16f(static_cast<const uint16_t*>(a.q)[((int64_t(b) * d.Hq + h) * d.N + u) * D + c]) *
               scale;
  }
  const bool full = a.full != 0;
  const int n_keys = full ? u + 1 : min(d.S, u + 1);
  const int32_t* sel = a.sel + (int64_t(b) * d.N + u) * d.S;
  const uint16_t* kb = static_cast<const uint16_t*>(a.k) + (int64_t(b) * d.Hkv + hk) * d.N * D;
  const uint16_t* vb = static_cast<const uint16_t*>(a.v) + (int64_t(b) * d.Hkv + hk) * d.N * D;
  float m[kMaxGroup], l[kMaxGroup], acc[kMaxGroup];
  for (int g = 0; g < G; ++g) {
    m[g] = -INFINITY;
    l[g] = 0.f;
    acc[g] = 0.f;
  }
  __syncthreads();
  for (int c0 = 0; c0 < n_keys; c0 += kAttnThreads) {
    const int nc = min(kAttnThreads, n_keys - c0);
    const int j = t < nc ? (full ? c0 + t : sel[c0 + t]) : -1;
    idx[t] = j;
    // scores of key t against every query of the group
    float s[kMaxGroup];
    for (int g = 0; g < G; ++g) s[g] = -INFINITY;
    if (j >= 0) {
      const uint4* k4 = reinterpret_cast<const uint4*>(kb + int64_t(j) * D);
      for (int g = 0; g < G; ++g) s[g] = 0.f;
#pragma unroll 4
      for (int c = 0; c < D / 8; ++c) {
        const uint4 w = __ldg(k4 + c);
        const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const float k0 = __uint_as_float(ww[e] << 16), k1 = __uint_as_float(ww[e] & 0xFFFF0000u);
          for (int g = 0; g < G; ++g)
            s[g] = fmaf(qs[g][8 * c + 2 * e + 1], k1, fmaf(qs[g][8 * c + 2 * e], k0, s[g]));
        }
      }
    }
    // chunk maxima per query
    for (int g = 0; g < G; ++g) {
      float x = s[g];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) x = fmaxf(x, __shfl_xor_sync(0xffffffffu, x, o));
      if (lane == 0) red[g][warp] = x;
    }
    __syncthreads();
    float mnew[kMaxGroup], corr[kMaxGroup];
    for (int g = 0; g < G; ++g) {
      float x = red[g][0];
      for (int w = 1; w < kAttnThreads / 32; ++w) x = fmaxf(x, red[g][w]);
      mnew[g] = fmaxf(m[g], x);
      corr[g] = m[g] == -INFINITY ? 0.f : expf(m[g] - mnew[g]);
      ps[g][t] = j >= 0 ? expf(s[g] - mnew[g]) : 0.f;
    }
    __syncthreads();
    // sums and the weighted value rows (thread t owns output dimension t)
    for (int g = 0; g < G; ++g) {
      float x = ps[g][t];
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
      if (lane == 0) red[g][warp] = x;
    }
    __syncthreads();
    for (int g = 0; g < G; ++g) {
      float x = 0.f;
      for (int w = 0; w < kAttnThreads / 32; ++w) x += red[g][w];
      l[g] = l[g] * corr[g] + x;
      acc[g] *= corr[g];
      m[g] = mnew[g];
    }
    if (t < D) {
      for (int jj = 0; jj < nc; ++jj) {
        const float vv = bf16f(vb[int64_t(idx[jj]) * D + t]);
        for (int g = 0; g < G; ++g) acc[g] = fmaf(ps[g][jj], vv, acc[g]);
      }
    }
    __syncthreads();
  }
  if (t < D) {
    uint16_t* o = static_cast<uint16_t*>(a.out);
    for (int g = 0; g < G; ++g) {
      const int h = hk * G + g;
      __nv_bfloat16 r = __float2bfloat16_rn(acc[g] / l[g]);
      o[((int64_t(b) * d.Hq + h) * d.N + u) * D + t] = *reinterpret_cast<uint16_t*>(&r);
    }
  }
}

}  // namespace

bool replay_supported(const ReplayDims& d) {
  return d.Hkv > 0 && d.Hq % d.Hkv == 0 && d.Hq / d.Hkv <= kMaxGroup &&
         (d.d == 64 || d.d == 128) && d.S >= 1 && d.S <= 4096 && d.N >= 1 && d.N <= 65536;
}

cudaError_t launch_replay_select(const ReplayArgs& a, cudaStream_t st) {
  const int rows = a.d.B * a.d.N;
  if (rows <= 0) return cudaSuccess;
  replay_select_kernel<<<rows, kSelThreads, 0, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_replay_attn(const ReplayArgs& a, cudaStream_t st) {
  dim3 grid(a.d.N, a.d.B * a.d.Hkv);
  if (a.d.d == 128)
    replay_attn_kernel<128><<<grid, kAttnThreads, 0, st>>>(a);
  else
    replay_attn_kernel<64><<<grid, kAttnThreads, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace mot
