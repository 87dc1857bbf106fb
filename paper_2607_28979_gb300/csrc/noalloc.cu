// mot_translate_static: the translation without any device allocation.
//
// Some callers cannot call cudaMalloc: a process whose device memory is
// carved up up front by its own pool allocator and forbids further
// allocations, code that runs where the CUDA allocator must not be entered,
// or a host that loads this library only to run a translation now and then
// and must not grow its footprint per call. For them this entry point needs no
// handle: the caller passes the configuration, the packed weight blob already
// in its own device memory, and the caches. The per-call intermediates (the
// renormalised gate of every token and the gate-weighted hidden activations)
// live in one file-scope __device__ array of kStaticScratchBytes that every
// GPU loading the library holds until the process exits.
//
// One SIMT kernel computes the translation in three phases per translated
// (target layer, K/V) group, each a launch: the gate (softmax over a linear
// map, Top-K renormalisation), the first translator layer with the exact-erf
// GELU times the gate, and the second layer plus the gate-weighted biases,
// stored into the target cache. All arithmetic is fp32 FFMA.
#include <cuda_bf16.h>
#include <stdint.h>

#include <mutex>

#include "mot_internal.h"

namespace mot {
namespace {

constexpr size_t kStaticScratchBytes = size_t(64) << 20;   // 64 MiB per device
static __device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

constexpr int kMaxDevices = 64;
constexpr int kRows = 64, kCols = 64, kK = 32;   // block tile: 64 tokens x 64 columns

struct StaticArgs {
  int32_t L_s, H_s, d_s, H_t, d_t, E, top_k, H, B, S;
  int32_t Ds, Dt, EH, s_pad;
  int32_t src_layer, tgt_layer;
  const void* src;
  void* dst;
  const void* w;               // this group's block of the weight blob
  const int32_t* seq_lens;     // device [batch]
  float* gate;                 // scratch [batch][s_pad][E]
  float* a2;                   // scratch [batch][s_pad][E*H]
};

__device__ __forceinline__ float ldv(const float* p, size_t i) { return p[i]; }
__device__ __forceinline__ float ldv(const __nv_bfloat16* p, size_t i) {
  return __bfloat162float(p[i]);
}
__device__ __forceinline__ void stv(float* p, size_t i, float v) { p[i] = v; }
__device__ __forceinline__ void stv(__nv_bfloat16* p, size_t i, float v) {
  p[i] = __float2bfloat16_rn(v);
}

// Blob offsets inside one group's block (elements).
struct BlobOff {
  size_t bg, exp0, per_exp, b1, w2, b2;   // b1 / w2 / b2 relative to an expert's start
  __device__ BlobOff(const StaticArgs& a) {
    const size_t E = a.E, Ds = a.Ds, Dt = a.Dt, H = a.H;
    bg = E * Ds;
    exp0 = E * Ds + E;
    per_exp = H * Ds + H + Dt * H + Dt;
    b1 = H * Ds;
    w2 = H * Ds + H;
    b2 = H * Ds + H + Dt * H;
  }
};

// Grid (batch * s_pad / 64, column tiles). Phase 0: gate; 1: first layer; 2: second layer.
template <typename T>
__global__ void __launch_bounds__(256) static_translate_kernel(StaticArgs a, int phase) {
  const int nblk = a.s_pad / kRows;
  const int b = blockIdx.x / nblk, s0 = (blockIdx.x % nblk) * kRows;
  int len = a.seq_lens[b];
  len = len < 0 ? 0 : (len > a.S ? a.S : len);
  if (s0 >= len) return;
  const int rows = min(kRows, len - s0);
  const T* __restrict__ src = static_cast<const T*>(a.src);
  const T* __restrict__ w = static_cast<const T*>(a.w);
  const BlobOff o(a);
  const size_t row_base = static_cast<size_t>(b) * a.s_pad + s0;   // scratch row of s0

  if (phase == 0) {
    // one warp per token row: E dot products over D_s, softmax, Top-K
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int r = warp; r < rows; r += 8) {
      const int s = s0 + r;
      float acc[kMaxE];
      for (int e = 0; e < kMaxE; ++e) acc[e] = 0.f;
      for (int c = lane; c < a.Ds; c += 32) {
        const int h = c / a.d_s, i = c - h * a.d_s;
        const float z = ldv(src, (((static_cast<size_t>(a.src_layer) * a.B + b) * a.H_s + h) * a.S + s) * a.d_s + i);
        for (int e = 0; e < a.E; ++e) acc[e] = fmaf(ldv(w, static_cast<size_t>(e) * a.Ds + c), z, acc[e]);
      }
      for (int e = 0; e < a.E; ++e)
        for (int off = 16; off > 0; off >>= 1) acc[e] += __shfl_xor_sync(0xffffffffu, acc[e], off);
      if (lane == 0) {
        float g[kMaxE], mx = -INFINITY, sum = 0.f;
        for (int e = 0; e < a.E; ++e) {
          g[e] = acc[e] + ldv(w, o.bg + e);
          mx = fmaxf(mx, g[e]);
        }
        for (int e = 0; e < a.E; ++e) {
          g[e] = expf(g[e] - mx);
          sum += g[e];
        }
        for (int e = 0; e < a.E; ++e) g[e] /= sum;
        if (a.top_k > 0 && a.top_k < a.E) {
          uint32_t keep = 0;
          for (int k = 0; k < a.top_k; ++k) {
            int best = -1;
            for (int e = 0; e < a.E; ++e)
              if (!((keep >> e) & 1u) && (best < 0 || g[e] > g[best])) best = e;
            keep |= 1u << best;
          }
          float ks = 0.f;
          for (int e = 0; e < a.E; ++e)
            if ((keep >> e) & 1u) ks += g[e];
          for (int e = 0; e < a.E; ++e) g[e] = ((keep >> e) & 1u) ? g[e] / ks : 0.f;
        }
        for (int e = 0; e < a.E; ++e) a.gate[(row_base + r) * a.E + e] = g[e];
      }
    }
    return;
  }

  // phases 1 and 2: a 64 x 64 output tile, 4 x 4 per thread, K staged in shared memory
  __shared__ float As[kK][kRows + 4];
  __shared__ float Bs[kK][kCols + 4];
  const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
  const int n0 = blockIdx.y * kCols;
  const int K = phase == 1 ? a.Ds : a.EH;
  const int N = phase == 1 ? a.EH : a.Dt;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += kK) {
    for (int e = threadIdx.x; e < kRows * kK; e += 256) {
      const int r = e / kK, kk = e % kK, k = k0 + kk;
      float v = 0.f;
      if (r < rows && k < K) {
        if (phase == 1) {
          const int h = k / a.d_s, i = k - h * a.d_s;
          v = ldv(src, (((static_cast<size_t>(a.src_layer) * a.B + b) * a.H_s + h) * a.S + s0 + r) * a.d_s + i);
        } else {
          v = a.a2[(row_base + r) * a.EH + k];
        }
      }
      As[kk][r] = v;
    }
    for (int e = threadIdx.x; e < kCols * kK; e += 256) {
      const int j = e / kK, kk = e % kK, k = k0 + kk, col = n0 + j;
      float v = 0.f;
      if (col < N && k < K) {
        if (phase == 1) {   // W1 of expert col / H, row col % H
          const int m = col / a.H, jj = col - m * a.H;
          v = ldv(w, o.exp0 + m * o.per_exp + static_cast<size_t>(jj) * a.Ds + k);
        } else {            // W2 of expert k / H, row col, column k % H
          const int m = k / a.H, jj = k - m * a.H;
          v = ldv(w, o.exp0 + m * o.per_exp + o.w2 + static_cast<size_t>(col) * a.H + jj);
        }
      }
      Bs[kk][j] = v;
    }
    __syncthreads();
#pragma unroll 8
    for (int kk = 0; kk < kK; ++kk) {
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
  T* __restrict__ dst = static_cast<T*>(a.dst);
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    const int r = ty * 4 + i;
    if (r >= rows) continue;
    const float* g = a.gate + (row_base + r) * a.E;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int col = n0 + tx * 4 + j;
      if (col >= N) continue;
      if (phase == 1) {
        const int m = col / a.H, jj = col - m * a.H;
        const float u = acc[i][j] + ldv(w, o.exp0 + m * o.per_exp + o.b1 + jj);
        a.a2[(row_base + r) * a.EH + col] = 0.5f * u * (1.f + erff(u * 0.70710678118654752f)) * g[m];
      } else {
        float y = acc[i][j];
        for (int m = 0; m < a.E; ++m) y = fmaf(g[m], ldv(w, o.exp0 + m * o.per_exp + o.b2 + col), y);
        const int h = col / a.d_t, ii = col - h * a.d_t;
        stv(dst, (((static_cast<size_t>(a.tgt_layer) * a.B + b) * a.H_t + h) * a.S + s0 + r) * a.d_t + ii, y);
      }
    }
  }
}

// Device address of the scratch array, resolved once per device.
std::mutex g_setup_mutex;
void* g_scratch_ptr[kMaxDevices] = {};

// a * b, saturating at SIZE_MAX (buffer sizes from int32 dimensions).
size_t mul_sat(size_t a, size_t b) {
  if (a != 0 && b > SIZE_MAX / a) return SIZE_MAX;
  return a * b;
}

bool ranges_overlap(const void* a, size_t na, const void* b, size_t nb) {
  const uintptr_t x = reinterpret_cast<uintptr_t>(a), y = reinterpret_cast<uintptr_t>(b);
  const uintptr_t xe = na > UINTPTR_MAX - x ? UINTPTR_MAX : x + na;
  const uintptr_t ye = nb > UINTPTR_MAX - y ? UINTPTR_MAX : y + nb;
  return x < ye && y < xe;
}

}  // namespace
}  // namespace mot

using namespace mot;

extern "C" mot_status mot_translate_static(const mot_config* cfg, const void* weights,
                                           const void* src_k, const void* src_v,
                                           const int32_t* seq_lens, int32_t batch, void* dst_k,
                                           void* dst_v, mot_stream_t stream) {
  if (!cfg || !weights || !src_k || !src_v || !dst_k || !dst_v) return MOT_ERR_INVALID_ARG;
  const mot_config& c = *cfg;
  if (c.n_layers_src <= 0 || c.src_kv_heads <= 0 || c.src_head_dim <= 0 || c.n_layers_tgt <= 0 ||
      c.tgt_kv_heads <= 0 || c.tgt_head_dim <= 0 || c.n_translators <= 0 || c.hidden <= 0 ||
      c.max_batch <= 0 || c.max_seq <= 0 || c.top_k < 0 || c.top_k > c.n_translators ||
      (c.dtype != MOT_BF16 && c.dtype != MOT_FP32))
    return MOT_ERR_INVALID_ARG;
  if (c.layer_map)
    for (int l = 0; l < c.n_layers_tgt; ++l)
      if (c.layer_map[l] < -1 || c.layer_map[l] >= c.n_layers_src) return MOT_ERR_INVALID_ARG;
  if (c.n_translators > kMaxE || c.max_batch > 4096) return MOT_ERR_UNSUPPORTED;
  // S_pad (max_seq rounded up to 64) must stay an int32
  if (c.max_seq > INT32_MAX - (kRows - 1)) return MOT_ERR_UNSUPPORTED;
  if (batch < 0 || batch > c.max_batch || (batch > 0 && !seq_lens)) return MOT_ERR_INVALID_ARG;
  const uintptr_t al = reinterpret_cast<uintptr_t>(weights) | reinterpret_cast<uintptr_t>(src_k) |
                       reinterpret_cast<uintptr_t>(src_v) | reinterpret_cast<uintptr_t>(dst_k) |
                       reinterpret_cast<uintptr_t>(dst_v);
  if (al & 15u) return MOT_ERR_INVALID_ARG;

  // The outputs may overlap neither each other, nor the caches they read, nor
  // the weights: target layer l would overwrite a source layer that a later
  // target layer still reads (the depth-ratio map reuses source layers).
  const size_t es = c.dtype == MOT_BF16 ? 2 : 4;
  int n_translated = 0;
  for (int l = 0; l < c.n_layers_tgt; ++l)
    if (!c.layer_map || c.layer_map[l] >= 0) ++n_translated;
  const size_t src_b = mul_sat(mul_sat(mul_sat(mul_sat(mul_sat(c.n_layers_src, c.max_batch),
                                                       c.src_kv_heads), c.max_seq),
                                       c.src_head_dim), es);
  const size_t dst_b = mul_sat(mul_sat(mul_sat(mul_sat(mul_sat(c.n_layers_tgt, c.max_batch),
                                                       c.tgt_kv_heads), c.max_seq),
                                       c.tgt_head_dim), es);
  const size_t Ds_ = mul_sat(c.src_kv_heads, c.src_head_dim);
  const size_t Dt_ = mul_sat(c.tgt_kv_heads, c.tgt_head_dim);
  size_t per_exp = mul_sat(c.hidden, Ds_);
  per_exp = per_exp + c.hidden;
  per_exp = per_exp + mul_sat(Dt_, c.hidden) + Dt_;
  const size_t group_elems = mul_sat(c.n_translators, Ds_) + c.n_translators +
                             mul_sat(c.n_translators, per_exp);
  const size_t w_b = mul_sat(mul_sat(2 * size_t(n_translated), group_elems), es);
  // the kernels index with int32 widths
  if (Ds_ > INT32_MAX || Dt_ > INT32_MAX ||
      mul_sat(c.n_translators, c.hidden) > size_t(INT32_MAX))
    return MOT_ERR_UNSUPPORTED;

  StaticArgs a{};
  a.L_s = c.n_layers_src; a.H_s = c.src_kv_heads; a.d_s = c.src_head_dim;
  a.H_t = c.tgt_kv_heads; a.d_t = c.tgt_head_dim;
  a.E = c.n_translators; a.top_k = c.top_k; a.H = c.hidden;
  a.B = c.max_batch; a.S = c.max_seq;
  a.Ds = a.H_s * a.d_s; a.Dt = a.H_t * a.d_t; a.EH = a.E * a.H;
  a.s_pad = (a.S + kRows - 1) / kRows * kRows;
  // scratch: gate rows then hidden rows, both fp32, for every (batch entry, position)
  const size_t rows = size_t(batch) * size_t(a.s_pad);
  const size_t gate_bytes = (rows * a.E * 4 + 255) / 256 * 256;
  const size_t need = gate_bytes + mul_sat(mul_sat(rows, size_t(a.EH)), 4);
  if (need > kStaticScratchBytes) return MOT_ERR_UNSUPPORTED;   // scratch too small
  if (ranges_overlap(dst_k, dst_b, dst_v, dst_b) || ranges_overlap(dst_k, dst_b, src_k, src_b) ||
      ranges_overlap(dst_k, dst_b, src_v, src_b) || ranges_overlap(dst_v, dst_b, src_k, src_b) ||
      ranges_overlap(dst_v, dst_b, src_v, src_b) || ranges_overlap(dst_k, dst_b, weights, w_b) ||
      ranges_overlap(dst_v, dst_b, weights, w_b))
    return MOT_ERR_INVALID_ARG;

  if (batch == 0) return MOT_OK;

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) {
    cudaGetLastError();
    return MOT_ERR_CUDA;
  }
  if (dev < 0 || dev >= kMaxDevices) return MOT_ERR_UNSUPPORTED;
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    if (!g_scratch_ptr[dev]) {
      void* p = nullptr;
      if (cudaGetSymbolAddress(&p, g_static_scratch) != cudaSuccess || !p) {
        cudaGetLastError();
        return MOT_ERR_CUDA;
      }
      g_scratch_ptr[dev] = p;
    }
    scratch = g_scratch_ptr[dev];
  }
  a.gate = static_cast<float*>(scratch);
  a.a2 = reinterpret_cast<float*>(static_cast<unsigned char*>(scratch) + gate_bytes);
  a.seq_lens = seq_lens;

  const size_t gsz = size_t(a.E) * a.Ds + a.E +
                     size_t(a.E) * (size_t(a.H) * a.Ds + a.H + size_t(a.Dt) * a.H + a.Dt);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const dim3 block(256);
  const unsigned gx = static_cast<unsigned>(batch) * (a.s_pad / kRows);
  int r = 0;   // translated layers so far (blob order)
  for (int l = 0; l < c.n_layers_tgt; ++l) {
    int sl;
    if (c.layer_map) {
      sl = c.layer_map[l];
    } else if (c.n_layers_tgt == 1) {
      sl = 0;
    } else {   // depth-ratio map (App. C.3): round(l*(L_s-1)/(L_t-1)), halves up
      const long long num = (long long)l * (c.n_layers_src - 1), den = c.n_layers_tgt - 1;
      sl = static_cast<int>((2 * num + den) / (2 * den));
    }
    if (sl < 0) continue;
    for (int x = 0; x < 2; ++x) {
      a.src_layer = sl;
      a.tgt_layer = l;
      a.src = x ? src_v : src_k;
      a.dst = x ? dst_v : dst_k;
      a.w = static_cast<const char*>(weights) + (size_t(2 * r + x) * gsz) * es;
      const dim3 g0(gx, 1), g1(gx, (a.EH + kCols - 1) / kCols), g2(gx, (a.Dt + kCols - 1) / kCols);
      if (c.dtype == MOT_BF16) {
        static_translate_kernel<__nv_bfloat16><<<g0, block, 0, st>>>(a, 0);
        static_translate_kernel<__nv_bfloat16><<<g1, block, 0, st>>>(a, 1);
        static_translate_kernel<__nv_bfloat16><<<g2, block, 0, st>>>(a, 2);
      } else {
        static_translate_kernel<float><<<g0, block, 0, st>>>(a, 0);
        static_translate_kernel<float><<<g1, block, 0, st>>>(a, 1);
        static_translate_kernel<float><<<g2, block, 0, st>>>(a, 2);
      }
      if (cudaGetLastError() != cudaSuccess) return MOT_ERR_CUDA;
    }
    ++r;
  }
  return MOT_OK;
}
