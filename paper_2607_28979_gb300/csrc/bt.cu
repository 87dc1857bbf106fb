// Backbone translators (App. C.2) inside the gated mixture (Def. 3.1) on sm_103a.
//
// Per token, slot r of the channel window is the source cache entry of layer
// pi(t_r): P = H_s rows (one per source KV head) of d_s values. A group
// g = x * E + m (K/V block x, backbone m) owns a row space of R = B * S * P rows,
// row ((b * S + s) * P + p). One slot of the recurrent scan is eight launches:
//
//   kBtIn   z  = GELU(W_in LN_in(x) + b_in)        A = the source cache (TMA 3-D box
//                                                   of tau tokens x P heads), the
//                                                   layer norm applied in the epilogue:
//                                                   (W_in' x - mu sum(W_in')) rstd + c, with
//                                                   W_in' = W_in diag(gamma) held as bf16
//                                                   hi + lo (two K blocks per source block)
//           xz = LN_C(z); slot 0 also h = z (h_0 = z_1) and xq = LN_Q(z)
//   kBtQ    q  = W_Q xq + b_Q
//   kBtKV   k|v = W_KV xz + b_KV
//   attn    o  = softmax of the scaled scores over the token's P key rows, per head
//                (SIMT, bt_attn_kernel)
//   kBtO    ht = h + W_O o + b_O;  xf = LN_F(ht)
//   kBtF1   f  = GELU(W_F1 xf + b_F1)
//   kBtF2   h  = ht + W_F2 f + b_F2;  xq = LN_Q(h) of the next slot; xo = bf16(h) and
//           the row's (mean, M2) statistics
//   kBtOut  dst[t_r] = sum_m gtilde_m GELU(rstd (W_out' xo_m - mu sum(W_out')) + c_m)
//                                                  (LN_out over the token's P*d values,
//                                                   folded like LN_in; mu, rstd from the
//                                                   P row statistics; the E backbones of
//                                                   block x in one tile)
//
// The row layer norms gamma * (v - mean) / sqrt(var + 1e-5) + beta run over the
// row's d values in fp32, on the fp32 row held in registers; the matrices they
// feed stay the blob's exact bf16 values. Every GEMM is one persistent,
// warp-specialised tcgen05 kernel: warp 0 TMA producer (4-stage ring of 64-wide
// K blocks), warp 1 MMA issuer (M = 128, N = NT, fp32 accumulators in TMEM, two
// buffers), warp 2 TMEM allocator, then the epilogue warps (8 for the row-norm
// stages, two per TMEM lane quarter, each thread one half of a row, the halves'
// layer-norm statistics combined through shared memory; 16 for the others, a
// quarter of the columns per warp). Row tiles hold whole tokens (tau = 128 / P of
// them). Apart from the row halves' exchange, the epilogue warps never wait on one
// another. All waits are bounded; on a timeout every role
// unwinds, copies and MMAs in flight are drained, TMEM is freed and
// kStatusTimeout is raised.
#include <cuda_bf16.h>

#include <algorithm>

#include "bt_internal.h"
#include "gelu.cuh"
#include "ptx.cuh"

namespace mot {
namespace {

constexpr int kBtStages = 4;
constexpr int kBtABytes = 128 * 64 * 2;   // 16 KB: 128 rows x 64 bf16
constexpr int kBtBBytes = 256 * 64 * 2;   // 32 KB: up to 256 rows x 64 bf16
constexpr int kBtStageBytes = kBtABytes + kBtBBytes;
// warps 0..3 roles, then EPI epilogue warps: 8 for the row-norm stages (a row's
// d values split over two threads, one per half, whose layer-norm statistics are
// combined through shared memory), 16 for the others (each warp of a lane quarter
// takes every fourth 32-column chunk)
__host__ __device__ constexpr int bt_threads(int epi) { return 32 * (4 + epi); }
constexpr int kBtRowEpi = 8;
constexpr int kBtTmemCols = 512;
constexpr float kLnEps = 1e-5f;
constexpr int kBtXchBytes = 2 * 2 * 128 * 8;   // [tile parity][half][row] (mean, M2)
constexpr int kBtSmem = kBtStages * kBtStageBytes + 256 + kBtXchBytes + 1024;
static_assert(kBtSmem <= 232448, "shared memory budget");

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ int seq_len_of(const BtArgs& a, int b) {
  if (b >= a.batch) return 0;
  const int L = a.seq_lens[b];
  return L < 0 ? 0 : (L > a.d.S ? a.d.S : L);
}

struct GemmCfg {
  int mode;
  int K;          // reduction length per backbone
  int NT;         // accumulator columns per tile (multiple of 32, <= 256)
  int n_tiles;    // N tiles per group
  int groups;     // groups iterated (2E, or 2 for kBtOut)
  int row_tiles;  // row tiles per group
  int a_box_bytes;
  int b_rows_per_g;   // rows of the weight map per (group, slot) block
};

// One work item of the persistent loop. Every role decodes items the same way
// (skipping the same inactive tiles), so their barrier phases stay in step.
struct Work {
  int g, b, s0, ntok, j;
  int tok0;       // kBtOut: first token of the 128-token tile (routed: bucket position)
  int64_t row0;   // the tile's first row in its group's row space
  bool active;
};

// Items of a launch: dense, groups x row tiles x N tiles; routed, the tiles of
// every bucket (from the route kernel's prefix sums) x N tiles.
__device__ __forceinline__ int total_items(const BtArgs& a, const GemmCfg& c) {
  if (!a.routed) return c.groups * c.row_tiles * c.n_tiles;
  const int* pre = a.rpre + (c.mode == kBtOut ? a.d.G + 1 : 0);
  return pre[a.d.G] * c.n_tiles;
}

__device__ __forceinline__ Work decode(const BtArgs& a, const GemmCfg& c, int item) {
  Work w;
  if (a.routed) {   // tile of bucket positions of group g
    const bool out = c.mode == kBtOut;
    const int* pre = a.rpre + (out ? a.d.G + 1 : 0);
    const int tile = item / c.n_tiles;
    w.j = item - tile * c.n_tiles;
    int g = 0;
    while (g + 1 < a.d.G && pre[g + 1] <= tile) ++g;
    w.g = g;
    const int span = out ? 128 : a.d.tau;
    const int pos0 = (tile - pre[g]) * span;
    w.ntok = min(span, a.cnt[g] - pos0);
    w.tok0 = pos0;
    w.b = 0;
    w.s0 = pos0;
    w.row0 = int64_t(pos0) * a.d.P;
    w.active = w.ntok > 0;
    return w;
  }
  const int per_g = c.row_tiles * c.n_tiles;
  w.g = item / per_g;
  const int rem = item - w.g * per_g;
  const int rt = rem / c.n_tiles;
  w.j = rem - rt * c.n_tiles;
  if (c.mode == kBtOut) {
    w.tok0 = rt * 128;
    w.b = w.tok0 / a.d.S;
    w.s0 = w.tok0 - w.b * a.d.S;
    w.ntok = 128;
    // active if any token of the tile is inside its sequence
    bool act = false;
    for (int b = w.b; b < a.d.B && b * a.d.S < w.tok0 + 128; ++b) {
      const int lo = max(0, w.tok0 - b * a.d.S);
      act = act || lo < seq_len_of(a, b);
    }
    w.active = act;
  } else {
    w.b = rt / a.d.tiles_b;
    w.s0 = (rt - w.b * a.d.tiles_b) * a.d.tau;
    w.ntok = min(a.d.tau, a.d.S - w.s0);
    w.tok0 = w.b * a.d.S + w.s0;
    w.active = w.s0 < seq_len_of(a, w.b);
  }
  w.row0 = int64_t(w.tok0) * a.d.P;
  return w;
}

// Whether token t of a (non-output) tile is a real token.
__device__ __forceinline__ bool tile_token_valid(const BtArgs& a, const Work& w, int t) {
  return t < w.ntok && (a.routed || w.s0 + t < seq_len_of(a, w.b));
}

struct EpiCtx {
  const BtArgs* a;
  const GemmCfg* c;
};

// ---------------------------------------------------------------- epilogues
//
// Each thread owns one accumulator row (TMEM lane 32 * q + lane). `tb` is the
// accumulator address with the lane quarter already added.

template <int D>
__device__ __forceinline__ void load_row(uint32_t tb, float (&v)[D]) {
#pragma unroll
  for (int c = 0; c < D / 32; ++c) {
    uint32_t r[32];
    tmem_ld_32x32b_x32(tb + c * 32, r);
    tmem_ld_wait(r);
#pragma unroll
    for (int k = 0; k < 32; ++k) v[c * 32 + k] = __uint_as_float(r[k]);
  }
}

template <int D>
__device__ __forceinline__ void row_stats(const float (&v)[D], float& mean, float& m2) {
  float s = 0.f;
#pragma unroll
  for (int k = 0; k < D; ++k) s += v[k];
  mean = s * (1.f / D);
  float q = 0.f;
#pragma unroll
  for (int k = 0; k < D; ++k) {
    const float t = v[k] - mean;
    q = fmaf(t, t, q);
  }
  m2 = q;
}

// dst[0..D) = bf16(gamma * (v - mean) * rstd + beta), 16-byte stores
template <int D>
__device__ __forceinline__ void store_norm(const float (&v)[D], float mean, float rstd,
                                           const float* gamma, const float* beta, uint16_t* dst) {
  uint4* d4 = reinterpret_cast<uint4*>(dst);
  const float4* g4 = reinterpret_cast<const float4*>(gamma);
  const float4* b4 = reinterpret_cast<const float4*>(beta);
#pragma unroll
  for (int c = 0; c < D / 8; ++c) {
    const float4 g0 = __ldg(g4 + 2 * c), g1 = __ldg(g4 + 2 * c + 1);
    const float4 b0 = __ldg(b4 + 2 * c), b1 = __ldg(b4 + 2 * c + 1);
    const float gg[8] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y, g1.z, g1.w};
    const float bb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
    float y[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) y[k] = fmaf((v[8 * c + k] - mean) * rstd, gg[k], bb[k]);
    d4[c] = make_uint4(pack2(y[0], y[1]), pack2(y[2], y[3]), pack2(y[4], y[5]), pack2(y[6], y[7]));
  }
}

template <int D>
__device__ __forceinline__ void store_f32(const float (&v)[D], float* dst) {
  float4* d4 = reinterpret_cast<float4*>(dst);
#pragma unroll
  for (int c = 0; c < D / 4; ++c) d4[c] = make_float4(v[4 * c], v[4 * c + 1], v[4 * c + 2], v[4 * c + 3]);
}

template <int D>
__device__ __forceinline__ void add_f32(float (&v)[D], const float* src) {
  const float4* s4 = reinterpret_cast<const float4*>(src);
#pragma unroll
  for (int c = 0; c < D / 4; ++c) {
    const float4 t = s4[c];
    v[4 * c] += t.x;
    v[4 * c + 1] += t.y;
    v[4 * c + 2] += t.z;
    v[4 * c + 3] += t.w;
  }
}

template <int D>
__device__ __forceinline__ void add_bias(float (&v)[D], const float* bias) {
  const float4* b4 = reinterpret_cast<const float4*>(bias);
#pragma unroll
  for (int c = 0; c < D / 4; ++c) {
    const float4 t = __ldg(b4 + c);
    v[4 * c] += t.x;
    v[4 * c + 1] += t.y;
    v[4 * c + 2] += t.z;
    v[4 * c + 3] += t.w;
  }
}

template <int D>
__device__ __forceinline__ void store_bf16(const float (&v)[D], uint16_t* dst) {
  uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int c = 0; c < D / 8; ++c)
    d4[c] = make_uint4(pack2(v[8 * c], v[8 * c + 1]), pack2(v[8 * c + 2], v[8 * c + 3]),
                       pack2(v[8 * c + 4], v[8 * c + 5]), pack2(v[8 * c + 6], v[8 * c + 7]));
}

// Named barrier over the nthreads epilogue threads, with the AND of p.
__device__ __forceinline__ bool epi_and(int id, int nthreads, bool p) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred a, q;\n\t"
      "setp.ne.u32 a, %1, 0;\n\t"
      "bar.red.and.pred q, %2, %3, a;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(p)), "r"(id), "r"(nthreads)
      : "memory");
  return r != 0;
}

// Where a row is split over two threads (half cg of the columns each), the
// halves' statistics: each thread's (mean, M2) of its DH values goes to xch, and
// after the epilogue barrier the pair combines them by the pairwise formula
// (equal counts). Both threads form the same sums, so both get the same result.
struct RowXch {
  float2* xch;   // [2][128] of this tile parity, or null: the row is whole in one thread
  int cg, nthreads;
};
template <int DH>
__device__ __forceinline__ void row_stats_x(const float (&v)[DH], float& mean, float& m2, int row,
                                            const RowXch& x) {
  row_stats<DH>(v, mean, m2);
  if (x.xch != nullptr) {
    x.xch[x.cg * 128 + row] = make_float2(mean, m2);
    epi_and(1, x.nthreads, true);
    const float2 o = x.xch[(x.cg ^ 1) * 128 + row];
    const float dl = o.x - mean;
    m2 = (m2 + o.y) + dl * dl * (0.5f * DH);
    mean = 0.5f * (mean + o.x);
  }
}

// Row-wise epilogues with the row in registers: N = D columns, split in NCG
// halves of DH = D / NCG columns (half x.cg in this thread).
template <int D, int NCG>
__device__ void epi_row(const EpiCtx& e, const Work& w, uint32_t tb, int row, const RowXch& xr) {
  constexpr int DH = D / NCG;
  constexpr int DF = D;   // full row width: the row statistics and strides
  const int col0 = xr.cg * DH;
  const BtArgs& a = *e.a;
  const BtDims& d = a.d;
  const int mode = e.c->mode;
  const int r = a.slot;
  int p, t;
  if (mode == kBtIn && !a.routed) {   // rows of the 3-D box: head-major within the tile
    p = row / d.tau;
    t = row - p * d.tau;
  } else {               // rows of the row space: token-major
    t = row / d.P;
    p = row - t * d.P;
  }
  const bool valid = p < d.P && tile_token_valid(a, w, t);
  const int64_t grow = int64_t(w.g) * d.R + w.row0 + int64_t(t) * d.P + p;   // row of this thread
  const int64_t gcol = grow * DF + col0;                                        // its first column
  float v[DH];
  float mean = 0.f, m2 = 0.f;
  if (mode == kBtIn) {
    // layer norm of the source row (d_s values), then GELU of the folded product
    float mu = 0.f, rs = 0.f;
    if (valid) {
      const int x = w.g / d.E;
      const uint16_t* xs_row =
          a.routed ? static_cast<const uint16_t*>(a.xs) + grow * d.d_s
                   : static_cast<const uint16_t*>(a.src[x]) +
                         (((int64_t(a.src_layer[r]) * d.B + w.b) * d.P + p) * d.S + w.s0 + t) *
                             d.d_s;
      const uint4* x4 = reinterpret_cast<const uint4*>(xs_row);
      float sum = 0.f;
      for (int c = 0; c < d.d_s / 8; ++c) {
        const uint4 u = __ldg(x4 + c);
        sum += bf16_lo(u.x) + bf16_hi(u.x) + bf16_lo(u.y) + bf16_hi(u.y) + bf16_lo(u.z) +
               bf16_hi(u.z) + bf16_lo(u.w) + bf16_hi(u.w);
      }
      mu = sum / d.d_s;
      float q = 0.f;
      for (int c = 0; c < d.d_s / 8; ++c) {
        const uint4 u = __ldg(x4 + c);
        const float f[8] = {bf16_lo(u.x), bf16_hi(u.x), bf16_lo(u.y), bf16_hi(u.y),
                            bf16_lo(u.z), bf16_hi(u.z), bf16_lo(u.w), bf16_hi(u.w)};
#pragma unroll
        for (int k = 0; k < 8; ++k) q = fmaf(f[k] - mu, f[k] - mu, q);
      }
      rs = rsqrtf(q / d.d_s + kLnEps);
    }
    __syncwarp();   // converge before the warp-collective TMEM loads
    load_row<DH>(tb + col0, v);
    const float* sw = a.s_in + int64_t(w.g) * DF + col0;
    const float* cb = a.c_in + int64_t(w.g) * DF + col0;
#pragma unroll
    for (int k = 0; k < DH; ++k) v[k] = gelu_tanh(fmaf(v[k] - mu * __ldg(sw + k), rs, __ldg(cb + k)));
    row_stats_x<DH>(v, mean, m2, row, xr);
    if (valid) {
      const float rstd = rsqrtf(m2 * (1.f / DF) + kLnEps);
      const float* lnc = a.ln_c + (int64_t(w.g) * d.N + r) * 2 * DF + col0;
      store_norm<DH>(v, mean, rstd, lnc, lnc + DF, static_cast<uint16_t*>(a.xz) + gcol);
      if (r == 0) {   // h_0 = z_1, and slot 0's queries read LN_Q(h_0)
        const float* lnq = a.ln_q + (int64_t(w.g) * d.N + r) * 2 * DF + col0;
        store_f32<DH>(v, a.h + gcol);
        store_norm<DH>(v, mean, rstd, lnq, lnq + DF, static_cast<uint16_t*>(a.xq) + gcol);
      }
    }
    return;
  }
  load_row<DH>(tb + col0, v);
  if (mode == kBtO) {
    add_bias<DH>(v, a.c_o + (int64_t(w.g) * d.N + r) * DF + col0);
    if (valid) add_f32<DH>(v, a.h + gcol);
    row_stats_x<DH>(v, mean, m2, row, xr);
    if (valid) {
      const float* lnf = a.ln_f + (int64_t(w.g) * d.N + r) * 2 * DF + col0;
      store_f32<DH>(v, a.ht + gcol);
      store_norm<DH>(v, mean, rsqrtf(m2 * (1.f / DF) + kLnEps), lnf, lnf + DF,
                     static_cast<uint16_t*>(a.xf) + gcol);
    }
    return;
  }
  // kBtF2: the new state, its row norm (next slot's queries), the raw row for
  // the output projection and the row's statistics for its token norm
  add_bias<DH>(v, a.c_f2 + (int64_t(w.g) * d.N + r) * DF + col0);
  if (valid) add_f32<DH>(v, a.ht + gcol);
  row_stats_x<DH>(v, mean, m2, row, xr);
  if (valid) {
    if (r + 1 < d.N) {
      const float* lnq = a.ln_q + (int64_t(w.g) * d.N + r + 1) * 2 * DF + col0;
      store_f32<DH>(v, a.h + gcol);
      store_norm<DH>(v, mean, rsqrtf(m2 * (1.f / DF) + kLnEps), lnq, lnq + DF,
                     static_cast<uint16_t*>(a.xq) + gcol);
    }
    store_bf16<DH>(v, static_cast<uint16_t*>(a.xo) + gcol);
    if (xr.cg == 0) a.rstat[grow] = make_float2(mean, m2);
  }
}

// Plain epilogues, 32 columns at a time: bias (+ GELU), bf16 out. Column group
// cg of ng takes chunks cg, cg + ng, ...
__device__ void epi_plain(const EpiCtx& e, const Work& w, uint32_t tb, int row, int cg, int ng) {
  const BtArgs& a = *e.a;
  const GemmCfg& c = *e.c;
  const BtDims& d = a.d;
  const int r = a.slot;
  const int t = row / d.P, p = row - t * d.P;
  const bool valid = tile_token_valid(a, w, t);
  const int64_t grow = int64_t(w.g) * d.R + w.row0 + int64_t(t) * d.P + p;
  const int N = c.NT * c.n_tiles;   // output row width
  const float* bias;
  uint16_t* out;
  if (c.mode == kBtQ) {
    bias = a.c_q + (int64_t(w.g) * d.N + r) * N;
    out = static_cast<uint16_t*>(a.q);
  } else if (c.mode == kBtKV) {
    bias = a.c_kv + (int64_t(w.g) * d.N + r) * N;
    out = static_cast<uint16_t*>(a.kv);
  } else {
    bias = a.c_f1 + (int64_t(w.g) * d.N + r) * N;
    out = static_cast<uint16_t*>(a.f);
  }
  const bool gelu = c.mode == kBtF1;
  for (int ch = cg; ch < c.NT / 32; ch += ng) {
    uint32_t rr[32];
    __syncwarp();
    tmem_ld_32x32b_x32(tb + ch * 32, rr);
    tmem_ld_wait(rr);
    if (!valid) continue;
    const int col = w.j * c.NT + ch * 32;
    const float4* b4 = reinterpret_cast<const float4*>(bias + col);
    uint4* o4 = reinterpret_cast<uint4*>(out + grow * N + col);
#pragma unroll
    for (int q8 = 0; q8 < 4; ++q8) {
      float f[8];
      const float4 b0 = __ldg(b4 + 2 * q8), b1 = __ldg(b4 + 2 * q8 + 1);
      const float bb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        f[k] = __uint_as_float(rr[8 * q8 + k]) + bb[k];
        if (gelu) f[k] = gelu_tanh(f[k]);
      }
      o4[q8] = make_uint4(pack2(f[0], f[1]), pack2(f[2], f[3]), pack2(f[4], f[5]),
                          pack2(f[6], f[7]));
    }
  }
}

// kBtOut: the E backbones' accumulators of this 128-token tile sit side by
// side (E * NT columns); the gate-weighted sum goes to target layer q0 + r.
// Routed (Top-1): one bucket's accumulator for 128 of its positions; each row
// is its token's whole output (gtilde = 1), stored at the token's position.
__device__ void epi_out_routed(const EpiCtx& e, const Work& w, uint32_t tb, int row, int cg,
                               int ng) {
  const BtArgs& a = *e.a;
  const GemmCfg& c = *e.c;
  const BtDims& d = a.d;
  const int g = w.g, x = g / d.E, m = g - x * d.E;
  const int pos = w.tok0 + row;
  const bool valid = row < w.ntok;
  int b = 0, s = 0;
  float gt = 0.f, mu = 0.f, rs = 0.f;
  if (valid) {
    const int tok = a.list[int64_t(g) * d.B * d.S + pos];
    b = tok / d.S;
    s = tok - b * d.S;
    gt = a.gate[(int64_t(x) * d.B * d.S + tok) * d.E + m];
    const float2* st = a.rstat + int64_t(g) * d.R + int64_t(pos) * d.P;
    float tm = 0.f;
    for (int k = 0; k < d.P; ++k) tm += st[k].x;
    tm /= d.P;
    float tq = 0.f;
    for (int k = 0; k < d.P; ++k) {
      const float2 sk = st[k];
      tq += sk.y + d.d * (sk.x - tm) * (sk.x - tm);
    }
    mu = tm;
    rs = rsqrtf(tq / (float(d.d) * d.P) + kLnEps);
  }
  uint16_t* dst = static_cast<uint16_t*>(a.dst[x]);
  const int l = d.q0 + a.slot;
  const float* cbase = a.c_out + int64_t(g) * d.Dt;
  const float* sbase = a.s_out + int64_t(g) * d.Dt;
  for (int ch = cg; ch < c.NT / 32; ch += ng) {
    uint32_t rr[32];
    __syncwarp();
    tmem_ld_32x32b_x32(tb + ch * 32, rr);
    tmem_ld_wait(rr);
    if (!valid) continue;
    const int col = w.j * c.NT + ch * 32;
    float y[32];
#pragma unroll
    for (int k = 0; k < 32; ++k) {
      const float u = fmaf(__uint_as_float(rr[k]) - mu * __ldg(sbase + col + k), rs,
                           __ldg(cbase + col + k));
      y[k] = fmaf(gt, gelu_tanh(u), 0.f);
    }
    const int hh = col / d.d_t, i0 = col - hh * d.d_t;
    uint4* o4 = reinterpret_cast<uint4*>(
        dst + (((int64_t(l) * d.B + b) * d.H_t + hh) * d.S + s) * d.d_t + i0);
#pragma unroll
    for (int q8 = 0; q8 < 4; ++q8)
      o4[q8] = make_uint4(pack2(y[8 * q8], y[8 * q8 + 1]), pack2(y[8 * q8 + 2], y[8 * q8 + 3]),
                          pack2(y[8 * q8 + 4], y[8 * q8 + 5]), pack2(y[8 * q8 + 6], y[8 * q8 + 7]));
  }
}

__device__ void epi_out(const EpiCtx& e, const Work& w, uint32_t tb, int row, int cg, int ng) {
  const BtArgs& a = *e.a;
  const GemmCfg& c = *e.c;
  const BtDims& d = a.d;
  const int x = w.g;   // kBtOut iterates the two K/V blocks
  const int tok = w.tok0 + row;
  const int b = tok / d.S, s = tok - b * d.S;
  const bool valid = b < d.B && s < seq_len_of(a, b);
  float gt[kMaxE], mu[kMaxE], rs[kMaxE];
  for (int m = 0; m < d.E; ++m) {
    gt[m] = valid ? a.gate[(int64_t(x) * d.B * d.S + tok) * d.E + m] : 0.f;
    mu[m] = 0.f;
    rs[m] = 0.f;
    if (gt[m] == 0.f) continue;
    // LN_out statistics over the token's P rows (Chan's combination of the
    // per-row mean and M2, each over d values)
    const float2* st = a.rstat + (int64_t(x) * d.E + m) * d.R + int64_t(tok) * d.P;
    float tm = 0.f;
    for (int k = 0; k < d.P; ++k) tm += st[k].x;
    tm /= d.P;
    float tq = 0.f;
    for (int k = 0; k < d.P; ++k) {
      const float2 sk = st[k];
      tq += sk.y + d.d * (sk.x - tm) * (sk.x - tm);
    }
    mu[m] = tm;
    rs[m] = rsqrtf(tq / (float(d.d) * d.P) + kLnEps);
  }
  uint16_t* dst = static_cast<uint16_t*>(a.dst[x]);
  const int l = d.q0 + a.slot;
  for (int ch = cg; ch < c.NT / 32; ch += ng) {
    float y[32];
#pragma unroll
    for (int k = 0; k < 32; ++k) y[k] = 0.f;
    const int col = w.j * c.NT + ch * 32;
    for (int m = 0; m < d.E; ++m) {
      uint32_t rr[32];
      __syncwarp();
      tmem_ld_32x32b_x32(tb + m * c.NT + ch * 32, rr);
      tmem_ld_wait(rr);
      if (gt[m] == 0.f) continue;   // not kept for this token (or an invalid row)
      const float* cb = a.c_out + (int64_t(x) * d.E + m) * d.Dt + col;
      const float* sb = a.s_out + (int64_t(x) * d.E + m) * d.Dt + col;
#pragma unroll
      for (int k = 0; k < 32; ++k) {
        const float u = fmaf(__uint_as_float(rr[k]) - mu[m] * __ldg(sb + k), rs[m], __ldg(cb + k));
        y[k] = fmaf(gt[m], gelu_tanh(u), y[k]);
      }
    }
    if (!valid) continue;
    const int hh = col / d.d_t, i0 = col - hh * d.d_t;
    uint4* o4 = reinterpret_cast<uint4*>(
        dst + (((int64_t(l) * d.B + b) * d.H_t + hh) * d.S + s) * d.d_t + i0);
#pragma unroll
    for (int q8 = 0; q8 < 4; ++q8)
      o4[q8] = make_uint4(pack2(y[8 * q8], y[8 * q8 + 1]), pack2(y[8 * q8 + 2], y[8 * q8 + 3]),
                          pack2(y[8 * q8 + 4], y[8 * q8 + 5]), pack2(y[8 * q8 + 6], y[8 * q8 + 7]));
  }
}

// ---------------------------------------------------------------- the GEMM kernel

template <int D, int EPI>
__global__ void __launch_bounds__(bt_threads(EPI), 1)
    bt_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmA2,
                   const __grid_constant__ CUtensorMap tmB, const BtArgs a, const GemmCfg c) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + kBtStages * kBtABytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kBtStages * kBtStageBytes);
  uint64_t* empty = full + kBtStages;
  uint64_t* tfull = empty + kBtStages;   // [2]
  uint64_t* tempty = tfull + 2;          // [2]
  uint64_t* drain = tempty + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float2* xch = reinterpret_cast<float2*>(smem + kBtStages * kBtStageBytes + 256);   // [2][2][128]

  const BtDims& d = a.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool is_out = c.mode == kBtOut;
  const int n_exp = is_out && !a.routed ? d.E : 1;   // routed: one backbone per bucket
  const int nk = c.K / 64;
  const int acc_cols = n_exp * c.NT;   // one accumulator buffer

  if (threadIdx.x == 0) {
    for (int s = 0; s < kBtStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&tfull[b], 1);
      mbar_init(&tempty[b], EPI);
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmA2);
    tma_prefetch_desc(&tmB);
  }
  if (warp == 2) {
    tmem_alloc(tmem_slot, kBtTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int total = total_items(a, c);
  uint32_t issued_mask = 0, issue_parity = 0;
  bool mma_issued = false;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer
      int stage = 0;
      uint32_t phase = 0;
      const uint32_t tx = c.a_box_bytes + c.NT * 128;
      for (int it = blockIdx.x; it < total; it += gridDim.x) {
        const Work w = decode(a, c, it);
        if (!w.active) continue;
        bool ok = true;
        for (int kk = 0; kk < n_exp * nk; ++kk) {
          const int m = kk / nk, kb = kk - m * nk;
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, a.wait_limit)) { ok = false; break; }
          mbar_arrive_expect_tx(&full[stage], tx);
          uint8_t* dA = sA + stage * kBtABytes;
          uint8_t* dB = sB + stage * kBtBBytes;
          const int kc = kb * 64;
          const int64_t row0 = w.row0;
          switch (c.mode) {
            case kBtIn: {   // K blocks [0, d_s/64): hi weights, then the same source blocks x lo
              const int x = w.g / d.E;
              if (a.routed)   // the bucket's packed source rows (token-major)
                tma_load_2d(dA, &tmA, &full[stage], kc % d.d_s,
                            static_cast<int32_t>(int64_t(w.g) * d.R + row0));
              else
                tma_load_3d(dA, x ? &tmA2 : &tmA, &full[stage], kc % d.d_s, w.s0,
                            (a.src_layer[a.slot] * d.B + w.b) * d.P);
              tma_load_2d(dB, &tmB, &full[stage], kc, w.g * c.b_rows_per_g + w.j * c.NT);
              break;
            }
            case kBtOut: {
              const int g = a.routed ? w.g : w.g * d.E + m;
              tma_load_2d(dA, &tmA, &full[stage], kc,
                          static_cast<int32_t>(int64_t(g) * d.B * d.S + w.tok0));
              tma_load_2d(dB, &tmB, &full[stage], kc, g * c.b_rows_per_g + w.j * c.NT);
              break;
            }
            default:
              tma_load_2d(dA, &tmA, &full[stage], kc, static_cast<int32_t>(int64_t(w.g) * d.R + row0));
              tma_load_2d(dB, &tmB, &full[stage], kc,
                          (w.g * d.N + a.slot) * c.b_rows_per_g + w.j * c.NT);
          }
          issued_mask |= 1u << stage;
          issue_parity = (issue_parity & ~(1u << stage)) | (phase << stage);
          if (++stage == kBtStages) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer (warp-uniform loop, elected lane)
    const uint32_t idesc = idesc_bf16_f32(128, c.NT);
    int stage = 0;
    uint32_t phase = 0;
    int buf = 0;
    uint32_t buf_phase = 0;
    for (int it = blockIdx.x; it < total; it += gridDim.x) {
      const Work w = decode(a, c, it);
      if (!w.active) continue;
      if (!mbar_wait(&tempty[buf], buf_phase ^ 1u, abort_flag, a.wait_limit)) break;
      tc_fence_after();
      bool ok = true;
      for (int kk = 0; kk < n_exp * nk; ++kk) {
        const int m = kk / nk, kb = kk - m * nk;
        if (!mbar_wait(&full[stage], phase, abort_flag, a.wait_limit)) { ok = false; break; }
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(buf * acc_cols + m * c.NT);
        const uint64_t adesc = sdesc_k_sw128(smem_u32(sA + stage * kBtABytes));
        const uint64_t bdesc = sdesc_k_sw128(smem_u32(sB + stage * kBtBBytes));
        if (elect_one()) {
#pragma unroll
          for (int k = 0; k < 4; ++k)
            umma_bf16(d_tmem, adesc + 2 * k, bdesc + 2 * k, idesc, (kb | k) != 0);
          umma_commit(&empty[stage]);
        }
        __syncwarp();
        mma_issued = true;
        if (++stage == kBtStages) { stage = 0; phase ^= 1u; }
      }
      if (!ok) break;
      if (elect_one()) umma_commit(&tfull[buf]);
      __syncwarp();
      buf ^= 1;
      if (buf == 0) buf_phase ^= 1u;
    }
  } else if (warp >= 4) {
    // ------------------------------------------------ epilogue
    const int q = warp & 3;
    const int cg = (warp - 4) >> 2;   // column group of this warp (EPI / 4 groups)
    const int row = q * 32 + lane;
    EpiCtx e{&a, &c};
    int buf = 0;
    uint32_t buf_phase = 0;
    for (int it = blockIdx.x; it < total; it += gridDim.x) {
      const Work w = decode(a, c, it);
      if (!w.active) continue;
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&tfull[buf], buf_phase, abort_flag, a.wait_limit) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      // the split rows pair warps at a barrier: every epilogue warp stops, or none
      if constexpr (EPI == kBtRowEpi) ok = epi_and(1, 32 * EPI, ok != 0) ? 1 : 0;
      if (!ok) break;
      tc_fence_after();
      const uint32_t tb = tmem_base + static_cast<uint32_t>(buf * acc_cols) +
                          (static_cast<uint32_t>(q * 32) << 16);
      if constexpr (EPI == kBtRowEpi) {   // the row-norm stages (kBtIn, kBtO, kBtF2)
        epi_row<D, 2>(e, w, tb, row, RowXch{xch + buf * 256, cg, 32 * EPI});
      } else {
        if (c.mode == kBtOut && a.routed)
          epi_out_routed(e, w, tb, row, cg, EPI / 4);
        else if (c.mode == kBtOut)
          epi_out(e, w, tb, row, cg, EPI / 4);
        else
          epi_plain(e, w, tb, row, cg, EPI / 4);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[buf]);
      buf ^= 1;
      if (buf == 0) buf_phase ^= 1u;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    // unwinding after a timed-out wait: let issued copies land and issued MMAs finish
    if (warp == 0 && lane == 0) {
      for (int s = 0; s < kBtStages; ++s)
        if ((issued_mask >> s) & 1u) {
          const uint32_t ad = smem_u32(&full[s]);
          const long long t0 = clock64();
          while (!mbar_try_wait(ad, (issue_parity >> s) & 1u) && clock64() - t0 < a.wait_limit) {
          }
        }
    }
    if (warp == 1 && mma_issued) {
      if (elect_one()) umma_commit(drain);
      __syncwarp();
      const uint32_t ad = smem_u32(drain);
      const long long t0 = clock64();
      while (!mbar_try_wait(ad, 0) && clock64() - t0 < a.wait_limit) {
      }
    }
    __syncthreads();
  }
  if (warp == 2) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, kBtTmemCols);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicOr(a.status, kStatusTimeout);
}

// ---------------------------------------------------------------- fused FFN (FFN1 + GELU + FFN2)
//
// One persistent CTA per SM over (group, row tile): the FFN hidden never leaves
// the SM. For each 128-column chunk hc of d_f:
//   MMA1  acc1[hc & 1] = xf W_F1[hc]^T          (M = 128, N = 128, K = d)
//   epi   A2[hc & 1]   = bf16(GELU(acc1 + b_F1)) into a 128B-swizzled SMEM tile
//   MMA2  acc2        += A2 W_F2[:, hc]^T        (M = 128, N = d, K = 128)
// MMA1 runs one chunk ahead of MMA2; after the last chunk the kBtF2 row epilogue
// reads acc2. warp 0: TMA (xf once per tile, W_F1 / W_F2 chunks in 2-slot
// rings); warp 1: MMAs; warp 2: TMEM; warps 4..11: epilogue (two per TMEM lane
// quarter: each half of every hidden chunk and half of the FFN2 row).
template <int D>
struct Ffn {
  static constexpr int kA = 128 * D * 2;       // xf tile: D / 64 blocks of 128 rows x 128 B
  static constexpr int kW1 = 128 * D * 2;      // W_F1 chunk: 128 rows x D
  static constexpr int kW2 = D * 128 * 2;      // W_F2 chunk: D rows x 128 (two 64-column blocks)
  static constexpr int kA2 = 128 * 128 * 2;    // hidden chunk: two blocks of 128 rows x 64
  static constexpr int kBytes = kA + 2 * kW1 + 2 * kW2 + 2 * kA2;
  static constexpr int kSmem = kBytes + 256 + 1024;
};
static_assert(Ffn<128>::kSmem <= 232448, "shared memory budget");

constexpr int kFfnEpi = 8;   // epilogue warps: two per TMEM lane quarter, each half of a row
template <int D>
__global__ void __launch_bounds__(32 * (4 + kFfnEpi), 1)
    bt_ffn_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmW1,
                  const __grid_constant__ CUtensorMap tmW2, const BtArgs a, const GemmCfg c) {
  using F = Ffn<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sW1 = sA + F::kA;        // [2]
  uint8_t* sW2 = sW1 + 2 * F::kW1;  // [2]
  uint8_t* sH = sW2 + 2 * F::kW2;   // [2] hidden chunks
  uint64_t* bars = reinterpret_cast<uint64_t*>(sH + 2 * F::kA2);
  uint64_t* a_full = bars;          // xf tile landed
  uint64_t* a_empty = bars + 1;     // every MMA1 of the tile done
  uint64_t* w1_full = bars + 2;     // [2]
  uint64_t* w1_empty = bars + 4;    // [2]
  uint64_t* w2_full = bars + 6;     // [2]
  uint64_t* w2_empty = bars + 8;    // [2]
  uint64_t* c1_full = bars + 10;    // [2] acc1 written
  uint64_t* c1_empty = bars + 12;   // [2] acc1 read (every epilogue warp)
  uint64_t* h_full = bars + 14;     // [2] hidden chunk written (every epilogue warp)
  uint64_t* h_empty = bars + 16;    // [2] hidden chunk consumed by MMA2
  uint64_t* c2_full = bars + 18;    // acc2 complete
  uint64_t* c2_empty = bars + 19;   // acc2 read (every epilogue warp)
  uint64_t* drain = bars + 20;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 21);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const BtDims& d = a.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_hc = d.df / 128;
  const int total = total_items(a, c);
  if (threadIdx.x == 0) {
    mbar_init(a_full, 1);
    mbar_init(a_empty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&w1_full[i], 1);
      mbar_init(&w1_empty[i], 1);
      mbar_init(&w2_full[i], 1);
      mbar_init(&w2_empty[i], 1);
      mbar_init(&c1_full[i], 1);
      mbar_init(&c1_empty[i], kFfnEpi);
      mbar_init(&h_full[i], kFfnEpi);
      mbar_init(&h_empty[i], 1);
    }
    mbar_init(c2_full, 1);
    mbar_init(c2_empty, kFfnEpi);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA);
    tma_prefetch_desc(&tmW1);
    tma_prefetch_desc(&tmW2);
  }
  if (warp == 2) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;   // acc1[i] at 128 i, acc2 at 256
  const long long wl = a.wait_limit;
  uint32_t issued = 0;   // producer: 1 when any copy was issued (for the drain)
  bool mma_issued = false;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer
      int tl = 0;   // local tile count
      int w1c = 0, w2c = 0;   // chunk counters of the two rings
      for (int it = blockIdx.x; it < total; it += gridDim.x) {
        const Work w = decode(a, c, it);
        if (!w.active) continue;
        if (!mbar_wait(a_empty, (tl & 1) ^ 1u, abort_flag, wl)) break;
        mbar_arrive_expect_tx(a_full, F::kA);
        const int64_t row0 = w.row0;
        for (int kb = 0; kb < D / 64; ++kb)
          tma_load_2d(sA + kb * 128 * 128, &tmA, a_full, kb * 64,
                      static_cast<int32_t>(int64_t(w.g) * d.R + row0));
        issued = 1;
        bool ok = true;
        const int wrow1 = (w.g * d.N + a.slot) * d.df, wrow2 = (w.g * d.N + a.slot) * D;
        for (int hc = 0; hc < n_hc && ok; ++hc) {
          const int s1 = w1c & 1;
          if (!mbar_wait(&w1_empty[s1], ((w1c >> 1) & 1) ^ 1u, abort_flag, wl)) { ok = false; break; }
          mbar_arrive_expect_tx(&w1_full[s1], F::kW1);
          for (int kb = 0; kb < D / 64; ++kb)
            tma_load_2d(sW1 + s1 * F::kW1 + kb * 128 * 128, &tmW1, &w1_full[s1], kb * 64,
                        wrow1 + hc * 128);
          ++w1c;
          const int s2 = w2c & 1;
          if (!mbar_wait(&w2_empty[s2], ((w2c >> 1) & 1) ^ 1u, abort_flag, wl)) { ok = false; break; }
          mbar_arrive_expect_tx(&w2_full[s2], F::kW2);
          for (int kb = 0; kb < 2; ++kb)
            tma_load_2d(sW2 + s2 * F::kW2 + kb * D * 128, &tmW2, &w2_full[s2], hc * 128 + kb * 64,
                        wrow2);
          ++w2c;
        }
        if (!ok) break;
        ++tl;
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer (warp-uniform, elected lane)
    const uint32_t id1 = idesc_bf16_f32(128, 128), id2 = idesc_bf16_f32(128, D);
    int tl = 0, w1c = 0, w2c = 0, c1c = 0, hcc = 0;
    bool ok = true;
    for (int it = blockIdx.x; it < total && ok; it += gridDim.x) {
      const Work w = decode(a, c, it);
      if (!w.active) continue;
      if (!mbar_wait(a_full, tl & 1, abort_flag, wl)) { ok = false; break; }
      auto mma1 = [&](int hc) -> bool {
        const int s1 = w1c & 1, b1 = c1c & 1;
        if (!mbar_wait(&w1_full[s1], (w1c >> 1) & 1, abort_flag, wl)) return false;
        if (!mbar_wait(&c1_empty[b1], ((c1c >> 1) & 1) ^ 1u, abort_flag, wl)) return false;
        tc_fence_after();
        if (elect_one()) {
          for (int kb = 0; kb < D / 64; ++kb) {
            const uint64_t ad = sdesc_k_sw128(smem_u32(sA + kb * 128 * 128));
            const uint64_t bd = sdesc_k_sw128(smem_u32(sW1 + s1 * F::kW1 + kb * 128 * 128));
#pragma unroll
            for (int k = 0; k < 4; ++k)
              umma_bf16(tmem + b1 * 128, ad + 2 * k, bd + 2 * k, id1, (kb | k) != 0);
          }
          umma_commit(&c1_full[b1]);
          umma_commit(&w1_empty[s1]);
          if (hc == n_hc - 1) umma_commit(a_empty);   // the tile's last read of xf
        }
        __syncwarp();
        mma_issued = true;
        ++w1c;
        ++c1c;
        return true;
      };
      auto mma2 = [&](int hc) -> bool {
        const int s2 = w2c & 1, bh = hcc & 1;
        if (!mbar_wait(&w2_full[s2], (w2c >> 1) & 1, abort_flag, wl)) return false;
        if (!mbar_wait(&h_full[bh], (hcc >> 1) & 1, abort_flag, wl)) return false;
        if (hc == 0 && !mbar_wait(c2_empty, (tl & 1) ^ 1u, abort_flag, wl)) return false;
        tc_fence_after();
        if (elect_one()) {
          for (int kb = 0; kb < 2; ++kb) {
            const uint64_t ad = sdesc_k_sw128(smem_u32(sH + bh * F::kA2 + kb * 128 * 128));
            const uint64_t bd = sdesc_k_sw128(smem_u32(sW2 + s2 * F::kW2 + kb * D * 128));
#pragma unroll
            for (int k = 0; k < 4; ++k)
              umma_bf16(tmem + 256, ad + 2 * k, bd + 2 * k, id2, (hc | kb | k) != 0);
          }
          umma_commit(&h_empty[bh]);
          umma_commit(&w2_empty[s2]);
          if (hc == n_hc - 1) umma_commit(c2_full);
        }
        __syncwarp();
        ++w2c;
        ++hcc;
        return true;
      };
      ok = mma1(0);
      for (int hc = 0; ok && hc < n_hc; ++hc) {
        if (hc + 1 < n_hc) ok = mma1(hc + 1);
        if (ok) ok = mma2(hc);
      }
      ++tl;
    }
  } else if (warp >= 4) {
    // ------------------------------------------------ epilogue: GELU chunks, then the F2 rows.
    // Warps 4 + 4 cg + q (cg = 0, 1) share TMEM lane quarter q: each takes half of every
    // hidden chunk's columns and half of the F2 row, whose statistics the pair exchanges
    // through hidden buffer 0 (free once acc2 is complete).
    const int q = warp & 3;
    const int cg = (warp - 4) >> 2;
    const int row = q * 32 + lane;
    float2* xch = reinterpret_cast<float2*>(sH);   // [2][128] (mean, M2) of the row halves
    const uint32_t lanes = static_cast<uint32_t>(q * 32) << 16;
    EpiCtx e{&a, &c};
    int tl = 0, c1c = 0, hcc = 0;
    bool ok = true;
    for (int it = blockIdx.x; it < total && ok; it += gridDim.x) {
      const Work w = decode(a, c, it);
      if (!w.active) continue;
      const float* b1 = a.c_f1 + (int64_t(w.g) * d.N + a.slot) * d.df;
      for (int hc = 0; hc < n_hc; ++hc) {
        const int b1i = c1c & 1, bh = hcc & 1;
        int wv = 1;
        if (lane == 0) wv = mbar_wait(&c1_full[b1i], (c1c >> 1) & 1, abort_flag, wl) ? 1 : 0;
        if (!__shfl_sync(0xffffffffu, wv, 0)) { ok = false; break; }
        wv = 1;
        if (lane == 0) wv = mbar_wait(&h_empty[bh], ((hcc >> 1) & 1) ^ 1u, abort_flag, wl) ? 1 : 0;
        if (!__shfl_sync(0xffffffffu, wv, 0)) { ok = false; break; }
        tc_fence_after();
        const uint32_t hbase = smem_u32(sH + bh * F::kA2);
#pragma unroll
        for (int ch = 2 * cg; ch < 2 * cg + 2; ++ch) {
          uint32_t rr[32];
          tmem_ld_32x32b_x32(tmem + lanes + b1i * 128 + ch * 32, rr);
          tmem_ld_wait(rr);
          const float4* bb4 = reinterpret_cast<const float4*>(b1 + hc * 128 + ch * 32);
          uint32_t pk[16];
#pragma unroll
          for (int k4 = 0; k4 < 8; ++k4) {
            const float4 bb = __ldg(bb4 + k4);
            const float x0 = gelu_tanh(__uint_as_float(rr[4 * k4]) + bb.x);
            const float x1 = gelu_tanh(__uint_as_float(rr[4 * k4 + 1]) + bb.y);
            const float x2 = gelu_tanh(__uint_as_float(rr[4 * k4 + 2]) + bb.z);
            const float x3 = gelu_tanh(__uint_as_float(rr[4 * k4 + 3]) + bb.w);
            pk[2 * k4] = pack2(x0, x1);
            pk[2 * k4 + 1] = pack2(x2, x3);
          }
          // row `row`, columns 32 ch .. 32 ch + 31 of the 128-column chunk: block ch / 2,
          // half ch % 2 of its 64 columns, 16-byte chunks permuted by the 128B swizzle
          const uint32_t rbase = hbase + (ch >> 1) * 128 * 128 + row * 128;
#pragma unroll
          for (int v = 0; v < 4; ++v)
            st_shared_v4(rbase + static_cast<uint32_t>((((ch & 1) * 4 + v) ^ (row & 7)) << 4),
                         pk[4 * v], pk[4 * v + 1], pk[4 * v + 2], pk[4 * v + 3]);
        }
        tc_fence_before();
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(&c1_empty[b1i]);
          mbar_arrive(&h_full[bh]);
        }
        ++c1c;
        ++hcc;
      }
      int wv = 0;
      if (ok && lane == 0) wv = mbar_wait(c2_full, tl & 1, abort_flag, wl) ? 1 : 0;
      // the row halves pair warps at a barrier: every epilogue warp stops, or none
      if (!epi_and(1, 32 * kFfnEpi, __shfl_sync(0xffffffffu, wv, 0) != 0)) { ok = false; break; }
      tc_fence_after();
      epi_row<D, 2>(e, w, tmem + lanes + 256, row, RowXch{xch, cg, 32 * kFfnEpi});   // the kBtF2 rows
      epi_and(1, 32 * kFfnEpi, true);   // both halves read the exchange before hidden buffer 0 is reused
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(c2_empty);
      ++tl;
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    // unwinding: let issued copies land (bounded) and issued MMAs finish
    if (warp == 0 && lane == 0 && issued) {
      const long long t0 = clock64();
      while (clock64() - t0 < (wl < 100000000LL ? wl : 100000000LL)) {
      }
    }
    if (warp == 1 && mma_issued) {
      if (elect_one()) umma_commit(drain);
      __syncwarp();
      const uint32_t ad = smem_u32(drain);
      const long long t0 = clock64();
      while (!mbar_try_wait(ad, 0) && clock64() - t0 < wl) {
      }
    }
    __syncthreads();
  }
  if (warp == 2) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem, 512);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicOr(a.status, kStatusTimeout);
}

// ---------------------------------------------------------------- gate (SIMT)
//
// One warp per token: logits_m = Wg[x][m] . window(token) + bg, the window
// flattened slot-major then head-major (c = r * D_s + p * d_s + i); softmax in
// fp32, then Top-K (ties to the lower index) and renormalisation. Also clamps
// and reports sequence lengths outside [0, S].
__global__ void __launch_bounds__(256) bt_gate_kernel(const BtArgs a) {
  extern __shared__ uint4 wg_s[];   // [E][N * D_s] bf16 of block x
  const BtDims& d = a.d;
  const int x = blockIdx.y;
  const int WD = d.N * d.Ds;
  const uint4* wsrc = reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(a.wg) +
                                                     int64_t(x) * d.E * WD);
  for (int i = threadIdx.x; i < d.E * WD / 8; i += blockDim.x) wg_s[i] = __ldg(wsrc + i);
  if (blockIdx.x == 0 && blockIdx.y == 0)
    for (int b = threadIdx.x; b < a.batch; b += blockDim.x) {
      const int L = a.seq_lens[b];
      if (L < 0 || L > d.S) atomicOr(a.status, kStatusSeqLen);
    }
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_tok = d.B * d.S;
  for (int tok = blockIdx.x * 8 + warp; tok < n_tok; tok += gridDim.x * 8) {
    const int b = tok / d.S, s = tok - b * d.S;
    if (s >= seq_len_of(a, b)) continue;
    float acc[kMaxE];
    for (int m = 0; m < d.E; ++m) acc[m] = 0.f;
    for (int c8 = lane; c8 < WD / 8; c8 += 32) {
      const int c = c8 * 8;
      const int r = c / d.Ds, rem = c - r * d.Ds;
      const int p = rem / d.d_s, i = rem - p * d.d_s;
      const uint4 u = __ldg(reinterpret_cast<const uint4*>(
          static_cast<const uint16_t*>(a.src[x]) +
          (((int64_t(a.src_layer[r]) * d.B + b) * d.P + p) * d.S + s) * d.d_s + i));
      const float xv[8] = {bf16_lo(u.x), bf16_hi(u.x), bf16_lo(u.y), bf16_hi(u.y),
                           bf16_lo(u.z), bf16_hi(u.z), bf16_lo(u.w), bf16_hi(u.w)};
      for (int m = 0; m < d.E; ++m) {
        const uint4 wv = wg_s[(m * WD + c) / 8];
        const float wf[8] = {bf16_lo(wv.x), bf16_hi(wv.x), bf16_lo(wv.y), bf16_hi(wv.y),
                             bf16_lo(wv.z), bf16_hi(wv.z), bf16_lo(wv.w), bf16_hi(wv.w)};
        float sacc = acc[m];
#pragma unroll
        for (int k = 0; k < 8; ++k) sacc = fmaf(wf[k], xv[k], sacc);
        acc[m] = sacc;
      }
    }
    for (int m = 0; m < d.E; ++m)
      for (int o = 16; o > 0; o >>= 1) acc[m] += __shfl_xor_sync(0xffffffffu, acc[m], o);
    if (lane == 0) {
      float g[kMaxE];
      float mx = -INFINITY;
      for (int m = 0; m < d.E; ++m) {
        g[m] = acc[m] + a.bg[x * d.E + m];
        mx = fmaxf(mx, g[m]);
      }
      float sum = 0.f;
      for (int m = 0; m < d.E; ++m) {
        g[m] = expf(g[m] - mx);
        sum += g[m];
      }
      for (int m = 0; m < d.E; ++m) g[m] /= sum;
      if (d.top_k > 0 && d.top_k < d.E) {
        uint32_t keep = 0;
        for (int k = 0; k < d.top_k; ++k) {
          int best = -1;
          for (int m = 0; m < d.E; ++m)
            if (!((keep >> m) & 1u) && (best < 0 || g[m] > g[best])) best = m;
          keep |= 1u << best;
        }
        float ks = 0.f;
        for (int m = 0; m < d.E; ++m)
          if ((keep >> m) & 1u) ks += g[m];
        for (int m = 0; m < d.E; ++m) g[m] = ((keep >> m) & 1u) ? g[m] / ks : 0.f;
      }
      float* go = a.gate + (int64_t(x) * n_tok + tok) * d.E;
      for (int m = 0; m < d.E; ++m) go[m] = g[m];
    }
  }
}

// ---------------------------------------------------------------- Top-1 routing
//
// One CTA of 1024 threads. For each group g = x * E + m, the tokens whose kept
// gate weight for backbone m is nonzero (with Top-1, exactly the chosen
// backbone), in token order: every thread counts the choices in its contiguous
// chunk of token slots, a block scan gives each thread its first bucket
// position, and the thread writes its tokens there. Then cnt[g] and the tile
// prefix sums (tau-token tiles, 128-token tiles).
__global__ void __launch_bounds__(1024) bt_route_kernel(const BtArgs a, int32_t* cnt,
                                                        int32_t* list, int32_t* rpre) {
  __shared__ int s_scan[1024];
  __shared__ int s_cnt[2 * kMaxE];
  const BtDims& d = a.d;
  const int T = d.B * d.S;
  const int tid = threadIdx.x;
  const int per = (T + 1023) / 1024;
  const int t0 = min(T, tid * per), t1 = min(T, t0 + per);
  for (int g = 0; g < d.G; ++g) {
    const int x = g / d.E, m = g - x * d.E;
    const float* gx = a.gate + int64_t(x) * T * d.E + m;
    auto chose = [&](int tok) {
      const int b = tok / d.S, s = tok - b * d.S;
      return s < seq_len_of(a, b) && gx[int64_t(tok) * d.E] > 0.f;
    };
    int c = 0;
    for (int tok = t0; tok < t1; ++tok) c += chose(tok) ? 1 : 0;
    s_scan[tid] = c;
    __syncthreads();
    for (int o = 1; o < 1024; o <<= 1) {   // inclusive scan (Hillis-Steele)
      const int v = tid >= o ? s_scan[tid - o] : 0;
      __syncthreads();
      s_scan[tid] += v;
      __syncthreads();
    }
    int off = s_scan[tid] - c;
    int32_t* lg = list + int64_t(g) * T;
    for (int tok = t0; tok < t1; ++tok)
      if (chose(tok)) lg[off++] = tok;
    if (tid == 1023) s_cnt[g] = s_scan[1023];
    __syncthreads();
  }
  if (tid == 0) {
    int p0 = 0, p1 = 0;
    for (int g = 0; g < d.G; ++g) {
      cnt[g] = s_cnt[g];
      rpre[g] = p0;
      rpre[d.G + 1 + g] = p1;
      p0 += (s_cnt[g] + d.tau - 1) / d.tau;
      p1 += (s_cnt[g] + 127) / 128;
    }
    rpre[d.G] = p0;
    rpre[2 * d.G + 1] = p1;
  }
}

// The source rows of slot a.slot for every bucket position, packed per group:
// xs[g][pos * P + p] = src[x][pi(t_r)][b][p][s] (16-byte copies).
__global__ void __launch_bounds__(256) bt_pack_kernel(const BtArgs a, uint4* __restrict__ xs) {
  const BtDims& d = a.d;
  const int g = blockIdx.y, x = g / d.E;
  const int T = d.B * d.S;
  const int cpr = d.d_s / 8;   // 16-byte chunks per row
  const int64_t total = int64_t(a.cnt[g]) * d.P * cpr;
  const uint4* src = static_cast<const uint4*>(a.src[x]);
  const int32_t* lg = a.list + int64_t(g) * T;
  const int64_t lbase = int64_t(a.src_layer[a.slot]) * d.B;
  for (int64_t i = int64_t(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
       i += int64_t(gridDim.x) * blockDim.x) {
    const int64_t rowi = i / cpr;
    const int c = static_cast<int>(i - rowi * cpr);
    const int pos = static_cast<int>(rowi / d.P), p = static_cast<int>(rowi - int64_t(pos) * d.P);
    const int tok = lg[pos];
    const int b = tok / d.S, s = tok - b * d.S;
    xs[(int64_t(g) * d.R + rowi) * cpr + c] =
        __ldg(src + (((lbase + b) * d.P + p) * d.S + s) * cpr + c);
  }
}

// ---------------------------------------------------------------- attention (SIMT)
//
// One thread per (query row, head): scores against the token's P key rows
// scaled by 1/sqrt(d/n_a), a max-subtracted softmax in fp32 and the weighted
// sum of the value rows. Consecutive threads take consecutive heads of a row,
// so a warp reads whole query rows and writes whole output rows.
// The CTA first copies the key/value rows of the tokens its threads cover into
// shared memory (one coalesced pass), so each token's rows are read from memory
// once rather than by each of its P x na threads.
template <int DH>
__global__ void __launch_bounds__(256) bt_attn_kernel(const BtArgs a) {
  extern __shared__ uint4 bt_kv_s4[];
  const BtDims& d = a.d;
  const int g = blockIdx.y;
  const int64_t id0 = int64_t(blockIdx.x) * blockDim.x;
  const int64_t id = id0 + threadIdx.x;
  // routed: the bucket's positions (its rows are packed); dense: every token slot
  const int64_t n_rows = (a.routed ? int64_t(a.cnt[g]) : int64_t(d.B) * d.S) * d.P;
  const int64_t n_thr = n_rows * d.na;
  if (id0 >= n_thr) return;
  const int64_t tok0 = (id0 / d.na) / d.P;
  {
    const int64_t last = (id0 + blockDim.x < n_thr ? id0 + blockDim.x : n_thr) - 1;
    const int64_t tok1 = (last / d.na) / d.P;
    const int64_t n16 = (tok1 - tok0 + 1) * d.P * 2 * d.d / 8;
    const uint4* src = reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(a.kv) +
                                                      (int64_t(g) * d.R + tok0 * d.P) * 2 * d.d);
    for (int64_t i = threadIdx.x; i < n16; i += blockDim.x) bt_kv_s4[i] = src[i];
  }
  __syncthreads();
  if (id >= n_thr) return;
  const int h = static_cast<int>(id % d.na);
  const int64_t row = id / d.na;
  const int64_t tok = row / d.P;
  if (!a.routed) {
    const int b = static_cast<int>(tok / d.S), s = static_cast<int>(tok - int64_t(b) * d.S);
    if (s >= seq_len_of(a, b)) return;
  }
  const int P = d.P, D = d.d;
  const float scale = rsqrtf(static_cast<float>(DH));
  const uint16_t* qr = static_cast<const uint16_t*>(a.q) + (int64_t(g) * d.R + row) * D + h * DH;
  const uint16_t* kvb = reinterpret_cast<const uint16_t*>(bt_kv_s4) + (tok - tok0) * P * 2 * D + h * DH;
  uint16_t* orow = static_cast<uint16_t*>(a.o) + (int64_t(g) * d.R + row) * D + h * DH;
  float qv[DH];
  const uint4* q4 = reinterpret_cast<const uint4*>(qr);
#pragma unroll
  for (int c = 0; c < DH / 8; ++c) {
    const uint4 u = q4[c];
    qv[8 * c] = bf16_lo(u.x); qv[8 * c + 1] = bf16_hi(u.x);
    qv[8 * c + 2] = bf16_lo(u.y); qv[8 * c + 3] = bf16_hi(u.y);
    qv[8 * c + 4] = bf16_lo(u.z); qv[8 * c + 5] = bf16_hi(u.z);
    qv[8 * c + 6] = bf16_lo(u.w); qv[8 * c + 7] = bf16_hi(u.w);
  }
  float sc[kBtMaxP];
  float mx = -INFINITY;
#pragma unroll
  for (int j = 0; j < kBtMaxP; ++j) {
    if (j >= P) break;
    const uint4* k4 = reinterpret_cast<const uint4*>(kvb + int64_t(j) * 2 * D);
    float sdot = 0.f;
#pragma unroll
    for (int c = 0; c < DH / 8; ++c) {
      const uint4 u = k4[c];
      sdot = fmaf(qv[8 * c], bf16_lo(u.x), sdot);
      sdot = fmaf(qv[8 * c + 1], bf16_hi(u.x), sdot);
      sdot = fmaf(qv[8 * c + 2], bf16_lo(u.y), sdot);
      sdot = fmaf(qv[8 * c + 3], bf16_hi(u.y), sdot);
      sdot = fmaf(qv[8 * c + 4], bf16_lo(u.z), sdot);
      sdot = fmaf(qv[8 * c + 5], bf16_hi(u.z), sdot);
      sdot = fmaf(qv[8 * c + 6], bf16_lo(u.w), sdot);
      sdot = fmaf(qv[8 * c + 7], bf16_hi(u.w), sdot);
    }
    sc[j] = sdot * scale;
    mx = fmaxf(mx, sc[j]);
  }
  float den = 0.f;
#pragma unroll
  for (int j = 0; j < kBtMaxP; ++j) {
    if (j >= P) break;
    sc[j] = expf(sc[j] - mx);
    den += sc[j];
  }
  const float inv = 1.f / den;
  float ov[DH];
#pragma unroll
  for (int k = 0; k < DH; ++k) ov[k] = 0.f;
#pragma unroll
  for (int j = 0; j < kBtMaxP; ++j) {
    if (j >= P) break;
    const uint4* v4 = reinterpret_cast<const uint4*>(kvb + int64_t(j) * 2 * D + D);
    const float wj = sc[j] * inv;
#pragma unroll
    for (int c = 0; c < DH / 8; ++c) {
      const uint4 u = v4[c];
      ov[8 * c] = fmaf(wj, bf16_lo(u.x), ov[8 * c]);
      ov[8 * c + 1] = fmaf(wj, bf16_hi(u.x), ov[8 * c + 1]);
      ov[8 * c + 2] = fmaf(wj, bf16_lo(u.y), ov[8 * c + 2]);
      ov[8 * c + 3] = fmaf(wj, bf16_hi(u.y), ov[8 * c + 3]);
      ov[8 * c + 4] = fmaf(wj, bf16_lo(u.z), ov[8 * c + 4]);
      ov[8 * c + 5] = fmaf(wj, bf16_hi(u.z), ov[8 * c + 5]);
      ov[8 * c + 6] = fmaf(wj, bf16_lo(u.w), ov[8 * c + 6]);
      ov[8 * c + 7] = fmaf(wj, bf16_hi(u.w), ov[8 * c + 7]);
    }
  }
  uint4* o4 = reinterpret_cast<uint4*>(orow);
#pragma unroll
  for (int c = 0; c < DH / 8; ++c)
    o4[c] = make_uint4(pack2(ov[8 * c], ov[8 * c + 1]), pack2(ov[8 * c + 2], ov[8 * c + 3]),
                       pack2(ov[8 * c + 4], ov[8 * c + 5]), pack2(ov[8 * c + 6], ov[8 * c + 7]));
}

}  // namespace

// Shapes the kernels take: bf16, P <= 16 heads of d_s in {64, 128}, width
// d in {64, 128} with heads of 16, 32 or 64, d_f a multiple of 64 and of the
// N tile, D_t a multiple of 32 with d_t % 32 == 0, E <= 8.
bool bt_supported(const BtDims& d) {
  const int dh = d.na > 0 ? d.d / d.na : 0;
  return d.P >= 1 && d.P <= kBtMaxP && (d.d_s == 64 || d.d_s == 128) && (d.d == 64 || d.d == 128) &&
         d.na > 0 && d.d % d.na == 0 && (dh == 16 || dh == 32 || dh == 64) && d.df % 64 == 0 &&
         (d.df <= 256 || d.df % 256 == 0) && d.Dt % 32 == 0 && d.d_t % 32 == 0 && d.E >= 1 &&
         d.E <= 8 && d.N >= 1 && d.N <= kBtMaxSlots && d.tau >= 1;
}

cudaError_t launch_bt_gate(const BtArgs& a, cudaStream_t st) {
  const BtDims& d = a.d;
  const size_t smem = size_t(d.E) * d.N * d.Ds * 2;
  static size_t attr = 0;
  if (smem > 48 * 1024 && smem > attr) {
    cudaError_t e = cudaFuncSetAttribute(bt_gate_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    attr = smem;
  }
  const int n_tok = d.B * d.S;
  dim3 grid(std::min((n_tok + 7) / 8, 1024), 2);
  bt_gate_kernel<<<grid, 256, smem, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_bt_route(const BtArgs& a, int32_t* cnt, int32_t* list, int32_t* rpre,
                            cudaStream_t st) {
  if (a.d.G > 2 * kMaxE) return cudaErrorInvalidValue;
  bt_route_kernel<<<1, 1024, 0, st>>>(a, cnt, list, rpre);
  return cudaGetLastError();
}

cudaError_t launch_bt_pack(const BtArgs& a, void* xs, cudaStream_t st) {
  const BtDims& d = a.d;
  const int64_t per_g = int64_t(d.B) * d.S * d.P * (d.d_s / 8);
  const int64_t blocks = (per_g + 255) / 256;
  dim3 grid(static_cast<unsigned>(blocks < 1024 ? blocks : 1024), d.G);
  bt_pack_kernel<<<grid, 256, 0, st>>>(a, static_cast<uint4*>(xs));
  return cudaGetLastError();
}

cudaError_t launch_bt_attn(const BtArgs& a, cudaStream_t st) {
  const BtDims& d = a.d;
  const int64_t threads = int64_t(d.B) * d.S * d.P * d.na;
  dim3 grid(static_cast<unsigned>((threads + 255) / 256), d.G);
  // 256 consecutive threads span at most 256 / na + 2 rows, so at most that / P + 2 tokens
  const int max_tok = (256 / d.na + 2) / d.P + 2;
  const int smem = max_tok * d.P * 2 * d.d * 2;
  auto kern = d.d / d.na == 16 ? bt_attn_kernel<16> : d.d / d.na == 32 ? bt_attn_kernel<32> : bt_attn_kernel<64>;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
  }
  kern<<<grid, 256, smem, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_bt_gemm(int mode, const BtArgs& a, const CUtensorMap& tmA,
                           const CUtensorMap& tmA2, const CUtensorMap& tmB, int num_sms,
                           cudaStream_t st) {
  const BtDims& d = a.d;
  GemmCfg c{};
  c.mode = mode;
  c.groups = d.G;
  c.row_tiles = d.B * d.tiles_b;
  c.a_box_bytes = kBtABytes;
  c.n_tiles = 1;
  switch (mode) {
    case kBtIn:
      c.K = 2 * d.d_s; c.NT = d.d; c.b_rows_per_g = d.d;
      c.a_box_bytes = 64 * 2 * d.tau * d.P;
      break;
    case kBtQ: c.K = d.d; c.NT = d.d; c.b_rows_per_g = d.d; break;
    case kBtKV: c.K = d.d; c.NT = 2 * d.d; c.b_rows_per_g = 2 * d.d; break;
    case kBtO: c.K = d.d; c.NT = d.d; c.b_rows_per_g = d.d; break;
    case kBtF1:
      c.K = d.d; c.b_rows_per_g = d.df;
      c.NT = d.df <= 256 ? d.df : 256;
      c.n_tiles = d.df / c.NT;
      break;
    case kBtF2: c.K = d.df; c.NT = d.d; c.b_rows_per_g = d.d; break;
    case kBtOut: {
      c.K = d.P * d.d;
      c.groups = a.routed ? d.G : 2;   // routed: one bucket (one backbone) per tile
      c.b_rows_per_g = d.Dt;
      int nt = a.routed ? 256 : 256 / d.E;
      nt -= nt % 32;
      while (nt > 32 && d.Dt % nt) nt -= 32;
      c.NT = nt;
      c.n_tiles = d.Dt / nt;
      c.row_tiles = (d.B * d.S + 127) / 128;
      break;
    }
    default: return cudaErrorInvalidValue;
  }
  if (c.NT < 32 || c.NT > 256 || c.NT % 32 || c.K % 64) return cudaErrorInvalidValue;
  // the row-norm stages keep a row in one thread; the others spread it over 16 warps
  const bool wide = mode == kBtQ || mode == kBtKV || mode == kBtF1 || mode == kBtOut;
  static bool attr_set[4] = {false, false, false, false};
  const int di = (d.d == 128 ? 1 : 0) + (wide ? 2 : 0);
  auto kern = wide ? (d.d == 128 ? bt_gemm_kernel<128, 16> : bt_gemm_kernel<64, 16>)
                   : (d.d == 128 ? bt_gemm_kernel<128, kBtRowEpi> : bt_gemm_kernel<64, kBtRowEpi>);
  if (!attr_set[di]) {
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kBtSmem);
    if (e != cudaSuccess) return e;
    attr_set[di] = true;
  }
  const long long items = static_cast<long long>(c.groups) * c.row_tiles * c.n_tiles;
  const int grid = static_cast<int>(items < num_sms ? items : num_sms);
  if (grid <= 0) return cudaSuccess;
  kern<<<grid, bt_threads(wide ? 16 : kBtRowEpi), kBtSmem, st>>>(tmA, tmA2, tmB, a, c);
  return cudaGetLastError();
}

cudaError_t launch_bt_ffn(const BtArgs& a, const CUtensorMap& tmXf, const CUtensorMap& tmW1,
                          const CUtensorMap& tmW2, int num_sms, cudaStream_t st) {
  const BtDims& d = a.d;
  if (d.df % 128) return cudaErrorInvalidValue;
  GemmCfg c{};
  c.mode = kBtF2;   // the row epilogue after the last chunk is kBtF2's
  c.groups = d.G;
  c.row_tiles = d.B * d.tiles_b;
  c.n_tiles = 1;
  c.NT = d.d;
  c.K = d.df;
  static bool attr[2] = {false, false};
  const int di = d.d == 128 ? 1 : 0;
  auto kern = d.d == 128 ? bt_ffn_kernel<128> : bt_ffn_kernel<64>;
  const int smem = d.d == 128 ? Ffn<128>::kSmem : Ffn<64>::kSmem;
  if (!attr[di]) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    attr[di] = true;
  }
  const long long items = static_cast<long long>(c.groups) * c.row_tiles;
  const int grid = static_cast<int>(items < num_sms ? items : num_sms);
  if (grid <= 0) return cudaSuccess;
  kern<<<grid, 32 * (4 + kFfnEpi), smem, st>>>(tmXf, tmW1, tmW2, a, c);
  return cudaGetLastError();
}

}  // namespace mot
