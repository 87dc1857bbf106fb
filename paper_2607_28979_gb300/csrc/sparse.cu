// Top-K routing with per-expert token buckets (Def. 3.1 with top_k < E).
//
// With a Top-K gate, translator m contributes only to the tokens whose top_k
// choices include m, so its MLP needs to run on those tokens only: the
// combine sum_m gtilde_m Tr_m(z) has top_k nonzero terms per token. For a
// pass of groups:
//   route    count the tokens of every (group, expert) bucket, lay the buckets
//            out in a packed row space (each padded to whole 256-row pair
//            tiles, in bucket order), list the pair tiles, then write each
//            bucket's token rows in ascending token order with their slot
//            (the expert's rank among the token's choices) and gtilde;
//   pack     gather the source rows of the packed tokens (all heads) into zp;
//   GEMMs    umma2.cu's pair kernels over the pair-tile list;
//   combine  y = sum of the token's top_k slot rows (slot order) -> target.
// Every step is deterministic: no atomics on data, fixed summation order.
#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include <algorithm>

#include "mot_internal.h"

namespace mot {
namespace {

constexpr int kRouteThreads = 1024;

__device__ __forceinline__ int n_rows_of(const PathArgs& a) {
  return min(*a.n_tiles, a.d.tiles_max) * kTileM;
}

// Block-wide sum (1024 threads); s_warp holds at least 33 ints.
__device__ __forceinline__ int block_sum(int v, int* s_warp) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  if (lane == 0) s_warp[warp] = v;
  __syncthreads();
  if (warp == 0) {
    int t = s_warp[lane];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
    if (lane == 0) s_warp[32] = t;
  }
  __syncthreads();
  const int total = s_warp[32];
  __syncthreads();   // s_warp is reused by the next call
  return total;
}

// Block-wide exclusive scan of one flag per thread (1024 threads): returns the
// thread's prefix and writes the block total to *total.
__device__ __forceinline__ int block_scan_flag(int f, int* s_warp, int* total) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t bal = __ballot_sync(0xffffffffu, f);
  const int within = __popc(bal & ((1u << lane) - 1u));
  if (lane == 0) s_warp[warp] = __popc(bal);
  __syncthreads();
  if (warp == 0) {
    const int v = s_warp[lane];
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int n = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += n;
    }
    s_warp[32 + lane] = incl - v;   // exclusive prefix of warp totals
    if (lane == 31) *total = incl;
  }
  __syncthreads();
  const int pre = s_warp[32 + warp] + within;
  __syncthreads();   // s_warp is reused by the next call
  return pre;
}

// grid (gp, E): tokens of bucket (local group, expert).
__global__ void __launch_bounds__(kRouteThreads) route_count_kernel(PathArgs a, SparseArgs s) {
  const int g = blockIdx.x, m = blockIdx.y, grp = a.g0 + g, E = a.d.E;
  const int n_rows = n_rows_of(a);
  const uint32_t* __restrict__ sel = a.sel + static_cast<size_t>(grp) * a.d.tpad;
  int cnt = 0;
  for (int r = threadIdx.x; r < n_rows; r += kRouteThreads) cnt += (sel[r] >> m) & 1u;
  __shared__ int s_part[32];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) cnt += __shfl_xor_sync(0xffffffffu, cnt, o);
  if ((threadIdx.x & 31) == 0) s_part[threadIdx.x >> 5] = cnt;
  __syncthreads();
  if (threadIdx.x < 32) {
    int v = s_part[threadIdx.x];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    if (threadIdx.x == 0) {
      s.counts[g * E + m] = v;
      s.counts_all[grp * E + m] = v;
    }
  }
}

// One block: packed-row layout of the buckets and the pair-tile list.
__global__ void __launch_bounds__(kRouteThreads) route_plan_kernel(PathArgs a, SparseArgs s) {
  const int nb = a.gp * a.d.E;
  __shared__ int s_rows[kRouteThreads], s_pairs[kRouteThreads];
  // each thread owns a contiguous range of buckets
  const int per = (nb + kRouteThreads - 1) / kRouteThreads;
  const int b0 = min(nb, threadIdx.x * per), b1 = min(nb, b0 + per);
  int rows = 0, pairs = 0;
  for (int b = b0; b < b1; ++b) {
    const int np = (s.counts[b] + 2 * kTileM - 1) / (2 * kTileM);
    pairs += np;
    rows += np * 2 * kTileM;
  }
  s_rows[threadIdx.x] = rows;
  s_pairs[threadIdx.x] = pairs;
  __syncthreads();
  if (threadIdx.x == 0) {   // exclusive scan over the 1024 partial sums
    int r = 0, q = 0;
    for (int i = 0; i < kRouteThreads; ++i) {
      const int vr = s_rows[i], vq = s_pairs[i];
      s_rows[i] = r;
      s_pairs[i] = q;
      r += vr;
      q += vq;
    }
    // the capacity covers the worst case (every token in top_k buckets, each
    // bucket padded by under 256 rows); the check only keeps writes in bounds
    const bool fits = r <= s.R && q <= s.max_pairs;
    s.plan[0] = fits ? q : 0;
    s.plan[1] = fits ? r : 0;
  }
  __syncthreads();
  if (s.plan[0] == 0 && s.plan[1] == 0) return;
  int row = s_rows[threadIdx.x], pair = s_pairs[threadIdx.x];
  for (int b = b0; b < b1; ++b) {
    const int c = s.counts[b];
    const int np = (c + 2 * kTileM - 1) / (2 * kTileM);
    s.row0[b] = row;
    for (int q = 0; q < np; ++q) {
      SparsePair sp;
      sp.vg = b;
      sp.p0 = row + q * 2 * kTileM;
      sp.rows0 = max(0, min(kTileM, c - q * 2 * kTileM));
      sp.rows1 = max(0, min(kTileM, c - q * 2 * kTileM - kTileM));
      s.pairs[pair + q] = sp;
    }
    row += np * 2 * kTileM;
    pair += np;
  }
}

// Bucket lists: block (g, m, c) writes the packed rows of bucket (g, m) for the
// tokens of row chunk c, in token order: it first counts the bucket's tokens in the
// rows before its chunk, then scans its chunk 1024 rows at a time. Chunk 0 also
// writes the padding rows of the bucket's last pair tile. Chunks are at least
// kFillChunk rows and at most kFillChunks per bucket, so the counting stays linear
// in the rows times a small factor.
constexpr int kFillChunk = 4096;
constexpr int kFillChunks = 32;

// Rows per chunk for `rows_max` rows (a multiple of kRouteThreads), the same on
// the host (grid) and in the kernel.
__host__ __device__ __forceinline__ int fill_chunk_rows(int rows_max) {
  const int per = (rows_max + kFillChunks - 1) / kFillChunks;
  const int c = per > kFillChunk ? per : kFillChunk;
  return (c + kRouteThreads - 1) / kRouteThreads * kRouteThreads;
}

__global__ void __launch_bounds__(kRouteThreads) route_fill_kernel(PathArgs a, SparseArgs s) {
  const int g = blockIdx.x, m = blockIdx.y, grp = a.g0 + g, E = a.d.E, b = g * E + m;
  if (s.plan[1] == 0) return;
  const int n_rows = n_rows_of(a);
  const int chunk = fill_chunk_rows(a.d.tiles_max * kTileM);
  const int r_lo = blockIdx.z * chunk;
  const int base = s.row0[b], count = s.counts[b];
  uint16_t* g16 = static_cast<uint16_t*>(s.gate16p);
  if (blockIdx.z == 0) {   // padding rows of the bucket's last pair tile
    const int padded = ((count + 2 * kTileM - 1) / (2 * kTileM)) * 2 * kTileM;
    for (int p = base + count + threadIdx.x; p < base + padded; p += kRouteThreads) {
      s.ltok[p] = -1;
      s.lslot[p] = 0;
      s.gatep[p] = 0.f;
      uint4* row16 = reinterpret_cast<uint4*>(g16 + static_cast<size_t>(p) * 64);
#pragma unroll
      for (int v = 0; v < 8; ++v) row16[v] = make_uint4(0u, 0u, 0u, 0u);
    }
  }
  if (r_lo >= n_rows) return;   // uniform over the block
  const uint32_t* __restrict__ sel = a.sel + static_cast<size_t>(grp) * a.d.tpad;
  const float* __restrict__ gate = a.gate + static_cast<size_t>(grp) * a.d.tpad * E;
  __shared__ int s_warp[64];
  __shared__ int s_total;
  // the bucket's tokens before this chunk
  int before = 0;
  for (int r = threadIdx.x; r < r_lo; r += kRouteThreads) before += (sel[r] >> m) & 1u;
  before = block_sum(before, s_warp);
  const int r_hi = min(n_rows, r_lo + chunk);
  int done = 0;
  for (int r0 = r_lo; r0 < r_hi; r0 += kRouteThreads) {
    const int r = r0 + threadIdx.x;
    const uint32_t sv = r < r_hi ? sel[r] : 0u;
    const int f = (sv >> m) & 1u;
    const int pre = block_scan_flag(f, s_warp, &s_total);
    if (f) {
      const int p = base + before + done + pre;
      const float gv = gate[static_cast<size_t>(r) * E + m];
      s.ltok[p] = r;
      s.lslot[p] = __popc(sv & ((1u << m) - 1u));
      s.gatep[p] = gv;
      uint4* row16 = reinterpret_cast<uint4*>(g16 + static_cast<size_t>(p) * 64);
      const uint16_t hv = __half_as_ushort(__float2half_rn(gv));
#pragma unroll
      for (int v = 0; v < 8; ++v) {
        uint32_t w[4] = {0u, 0u, 0u, 0u};
        if (m / 8 == v) w[(m % 8) / 2] = (m & 1) ? (uint32_t(hv) << 16) : uint32_t(hv);
        row16[v] = make_uint4(w[0], w[1], w[2], w[3]);
      }
    }
    done += s_total;
  }
}

// Packed source rows: zp[h][p] = head row h of the token of packed row p (the
// bucket's rows in token order), 16-byte vectors; packed rows without a token (the
// tail of a bucket's last pair tile) are zeros. grid (x, H_s): block (x, h) takes
// rows p = x * rpb + t / vpr, stepping by gridDim.x * rpb, thread t the row's
// vector t % vpr; all index arithmetic per row is a shift or one small division.
__global__ void __launch_bounds__(256) pack_kernel(PathArgs a, SparseArgs s) {
  const Dims& d = a.d;
  const int rows = s.plan[1];
  const int vpr = d.d_s / 8;     // 16-byte vectors per head row (<= 256, checked at launch)
  const int rpb = 256 / vpr;     // rows per block per step
  const int t = threadIdx.x;
  if (t >= rpb * vpr) return;
  const int v = t % vpr, h = blockIdx.y;
  uint4* zp = static_cast<uint4*>(s.zp) + static_cast<size_t>(h) * s.R * vpr + v;
  const int step = gridDim.x * rpb;
  // eight rows per thread per pass: their chains of dependent loads (token, pair, group
  // and tile, source vector) are in flight together
  constexpr int kRows = 8;
  for (int p0 = blockIdx.x * rpb + t / vpr; p0 < rows; p0 += kRows * step) {
    int tok[kRows];
#pragma unroll
    for (int j = 0; j < kRows; ++j) tok[j] = p0 + j * step < rows ? s.ltok[p0 + j * step] : -1;
    uint4 val[kRows];
#pragma unroll
    for (int j = 0; j < kRows; ++j) {
      val[j] = make_uint4(0u, 0u, 0u, 0u);
      if (tok[j] >= 0) {
        const int vg = s.pairs[(p0 + j * step) / (2 * kTileM)].vg;
        const GroupInfo gi = a.groups[a.g0 + vg / d.E];
        const TileInfo ti = a.tiles[tok[j] / kTileM];
        const size_t pos = static_cast<size_t>(ti.s0) + tok[j] % kTileM;
        const uint4* src = static_cast<const uint4*>(a.src[gi.x]);
        val[j] = src[(((static_cast<size_t>(gi.src_layer) * d.B + ti.b) * d.H_s + h) * d.S + pos) * vpr + v];
      }
    }
#pragma unroll
    for (int j = 0; j < kRows; ++j)
      if (p0 + j * step < rows) zp[static_cast<size_t>(p0 + j * step) * vpr] = val[j];
  }
}

// y = sum over the top_k slots (in slot order) -> bf16 target rows.
// grid (ceil(tpad * D_t / 8 / 256), gp): one thread per 8 channels of a row.
__global__ void combine_kernel(PathArgs a, SparseArgs s) {
  const Dims& d = a.d;
  const int g = blockIdx.y, grp = a.g0 + g, K = d.top_k;
  const int vpr = d.Dt / 8;
  const size_t i = blockIdx.x * size_t(blockDim.x) + threadIdx.x;
  const int n_rows = n_rows_of(a);
  if (i >= static_cast<size_t>(n_rows) * vpr) return;
  const int r = static_cast<int>(i / vpr), v = static_cast<int>(i % vpr);
  const TileInfo ti = a.tiles[r / kTileM];
  if (r % kTileM >= ti.rows) return;
  const GroupInfo gi = a.groups[grp];
  const float4* y = reinterpret_cast<const float4*>(
      s.ybuf + (static_cast<size_t>(g) * d.tpad + r) * K * d.Dt + v * 8);
  float acc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
  for (int k = 0; k < K; ++k) {
    const float4 lo = y[(k * d.Dt) / 4], hi = y[(k * d.Dt) / 4 + 1];
    acc[0] += lo.x; acc[1] += lo.y; acc[2] += lo.z; acc[3] += lo.w;
    acc[4] += hi.x; acc[5] += hi.y; acc[6] += hi.z; acc[7] += hi.w;
  }
  uint32_t w[4];
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    const __nv_bfloat162 b2 = __floats2bfloat162_rn(acc[2 * j], acc[2 * j + 1]);
    w[j] = *reinterpret_cast<const uint32_t*>(&b2);
  }
  const int c = v * 8, h = c / d.d_t, i0 = c - h * d.d_t;
  __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(a.dst[gi.x]);
  const size_t pos = static_cast<size_t>(ti.s0) + r % kTileM;
  *reinterpret_cast<uint4*>(
      dst + ((((static_cast<size_t>(gi.tgt_layer) * d.B + ti.b) * d.H_t + h) * d.S + pos) * d.d_t +
             i0)) = make_uint4(w[0], w[1], w[2], w[3]);
}

}  // namespace

cudaError_t launch_route(const PathArgs& a, const SparseArgs& s, int step, cudaStream_t st) {
  if (a.gp <= 0) return cudaSuccess;
  const dim3 grid(a.gp, a.d.E);
  if (step == 0) {
    route_count_kernel<<<grid, kRouteThreads, 0, st>>>(a, s);
  } else if (step == 1) {
    route_plan_kernel<<<1, kRouteThreads, 0, st>>>(a, s);
  } else {
    const int rows_max = a.d.tiles_max * kTileM, chunk = fill_chunk_rows(rows_max);
    route_fill_kernel<<<dim3(a.gp, a.d.E, (rows_max + chunk - 1) / chunk), kRouteThreads, 0, st>>>(a, s);
  }
  return cudaGetLastError();
}

cudaError_t launch_pack(const PathArgs& a, const SparseArgs& s, cudaStream_t st) {
  if (a.gp <= 0) return cudaSuccess;
  if (a.d.d_s % 8 || a.d.d_s / 8 > 256 || a.d.H_s <= 0) return cudaErrorInvalidValue;
  const dim3 grid(static_cast<unsigned>(std::max(1, 8 * 152 / a.d.H_s)), a.d.H_s);
  pack_kernel<<<grid, 256, 0, st>>>(a, s);
  return cudaGetLastError();
}

cudaError_t launch_combine(const PathArgs& a, const SparseArgs& s, cudaStream_t st) {
  if (a.gp <= 0) return cudaSuccess;
  const size_t per = static_cast<size_t>(a.d.tpad) * (a.d.Dt / 8);
  const dim3 grid(static_cast<unsigned>((per + 255) / 256), a.gp);
  combine_kernel<<<grid, 256, 0, st>>>(a, s);
  return cudaGetLastError();
}

}  // namespace mot
