// Tile geometry and the two fused epilogues shared by the tcgen05 kernels.
//
//   GEMM1 epilogue:  A2[row, n0 + c] = fp16( GELU(acc[row, c] + b1[n0 + c]) * gtilde_m(row) )
//                    (one expert m per 256-column tile since H % 256 == 0), computed in
//                    packed fp16x2 arithmetic and written as 32x32 tiles through
//                    64B-swizzled, double-buffered shared memory + TMA store.
//   GEMM2 epilogue:  y[row, c] = acc[row, c] (the gate-weighted biases
//                    sum_m gtilde_m(row) * b2_m[c] are GEMM2's last K block), rounded to
//                    bf16 and stored as 16-byte vectors into the target cache row
//                    dst[l][b][c / d_t][s][c % d_t] when s < seq_len[b].
#pragma once

#include <cuda_bf16.h>
#include <cuda_fp16.h>

#include "mot_internal.h"
#include "gelu.cuh"
#include "ptx.cuh"

namespace mot {

constexpr int UM = kTileM;   // 128 rows (tokens) per accumulator tile
constexpr int UN = kUmmaN;   // 256 columns per accumulator tile
constexpr int UK = kUmmaK;   // 64 K elements per pipeline stage
constexpr int kStages = 4;
constexpr int kABytes = UM * UK * 2;   // 16 KB
constexpr int kBBytes = UN * UK * 2;   // 32 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kTmemCols = 2 * UN;      // two fp32 accumulators of 256 columns
constexpr int kStoreTileBytes = 2 * 32 * 64;   // one warp's two 32 x 32 fp16 store tiles

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// GEMM1 epilogue of one warp: rows 32*q + lane of the tile, columns
// [col_begin, col_begin + 64 * n_chunks). `tbase` is the accumulator's TMEM
// address including the warp's lane quarter; `tile` this warp's 4 KB of
// shared memory (two 2 KB store tiles). The columns are processed in 32-wide
// sub-chunks: the TMEM load of sub-chunk i+1 is in flight while sub-chunk i is
// evaluated, and each 32x32 fp16 result goes out by TMA store from one of the
// two tiles while the other is refilled.
__device__ __forceinline__ void gemm1_sub(const uint32_t (&r)[32], const uint4* b4, __half2 half_g,
                                          uint32_t (&pk)[16]) {
#pragma unroll
  for (int v = 0; v < 4; ++v) {
    const uint4 bb = __ldg(b4 + v);
    const uint32_t bw[4] = {bb.x, bb.y, bb.z, bb.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int j = v * 8 + 2 * k;
      pk[4 * v + k] = gelu_gate_pair(r[j], r[j + 1], bw[k], half_g);
    }
  }
}

// Gate value of this thread's row for GEMM1 tile (grp, m, n0), and an L1
// prefetch of the warp's bias columns: issued one tile ahead by the caller so
// that neither round trip sits at the start of the tile's epilogue.
__device__ __forceinline__ float gemm1_prefetch(const PathArgs& p, int q, int lane, int grp, int m,
                                                int n0, int col_begin) {
  const Dims& d = p.d;
  const size_t grow = static_cast<size_t>(m) * UM + q * 32 + lane;
  const float g = p.gate[(static_cast<size_t>(grp) * d.tpad + grow) * d.E + n0 / d.H];
  if (lane < 2) {
    const __half* b = static_cast<const __half*>(p.b1h) + static_cast<size_t>(grp) * d.EH + n0 +
                      col_begin + lane * 64;
    asm volatile("prefetch.global.L1 [%0];" ::"l"(b));
  }
  return g;
}

// `bias_col` is the tile's first column in the group's E*H biases; the store
// map's coordinates of the tile are (st_x, st_y, st_z) = (first column, first
// row, group slot) of the A2 layout in use.
__device__ __forceinline__ void epilogue_gemm1(const PathArgs& p, const CUtensorMap* tmS,
                                               uint32_t tbase, uint8_t* tile, int q, int lane,
                                               int grp, int bias_col, int st_x, int st_y,
                                               int st_z, int col_begin, int n_chunks,
                                               float gate) {
  const Dims& d = p.d;
  const __half2 half_g = __float2half2_rn(0.5f * gate);
  const __half* __restrict__ bias =
      static_cast<const __half*>(p.b1h) + static_cast<size_t>(grp) * d.EH + bias_col;
  const uint32_t tile_addr = smem_u32(tile);
  const int n_sub = 2 * n_chunks;
  uint32_t ra[32], rb[32];
  tmem_ld_32x32b_x32(tbase + col_begin, ra);
#pragma unroll 1
  for (int sc = 0; sc < n_sub; sc += 2) {
    // ---- sub-chunk sc (in ra); load sc + 1 into rb meanwhile
    tmem_ld_wait(ra);
    tmem_ld_32x32b_x32(tbase + col_begin + (sc + 1) * 32, rb);
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int s = sc + half;
      const int col0 = col_begin + s * 32;
      uint32_t pk[16];   // columns col0 + 2k, +1 of this row as fp16x2
      if (half == 0) {
        gemm1_sub(ra, reinterpret_cast<const uint4*>(bias + col0), half_g, pk);
      } else {
        tmem_ld_wait(rb);
        if (s + 1 < n_sub) tmem_ld_32x32b_x32(tbase + col_begin + (s + 1) * 32, ra);
        gemm1_sub(rb, reinterpret_cast<const uint4*>(bias + col0), half_g, pk);
      }
      // the store that last used this half's tile must have finished reading it
      if (lane == 0) bulk_wait_group_read<1>();
      __syncwarp();
      // row `lane` of the 32x32 tile (64 bytes); 16-byte chunk cc sits at chunk
      // position cc ^ ((row / 2) % 4), the 64-byte swizzle of the store map
      const uint32_t t_addr = tile_addr + half * 2048;
#pragma unroll
      for (int cc = 0; cc < 4; ++cc)
        st_shared_v4(t_addr + lane * 64 + ((cc ^ ((lane >> 1) & 3)) << 4), pk[4 * cc],
                     pk[4 * cc + 1], pk[4 * cc + 2], pk[4 * cc + 3]);
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) {
        tma_store_3d(tmS, tile + half * 2048, st_x + col0, st_y + q * 32, st_z);
        bulk_commit_group();
      }
    }
  }
}

// GEMM2 epilogue of one warp: row 32*q + lane of the tile, columns
// [col_begin, col_begin + 32 * n_chunks) of output tile n0. The gate-weighted
// biases are already in the accumulator (GEMM2's last K block).
__device__ __forceinline__ void epilogue_gemm2(const PathArgs& p, uint32_t tbase, int q, int lane,
                                               int grp, int m, int n0, int col_begin,
                                               int n_chunks) {
  const Dims& d = p.d;
  const int row = q * 32 + lane;
  const GroupInfo gi = p.groups[grp];
  const TileInfo ti = p.tiles[m];
  const bool valid = row < ti.rows;
  __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(p.dst[gi.x]);
  const size_t s = static_cast<size_t>(ti.s0) + row;
#pragma unroll 1
  for (int ch = 0; ch < n_chunks; ++ch) {
    const int cl = col_begin + ch * 32;
    uint32_t r[32];
    tmem_ld_32x32b_x32(tbase + cl, r);
    tmem_ld_wait(r);
    const int c = n0 + cl;
    if (valid) {
      const int h = c / d.d_t, i0 = c - h * d.d_t;
      uint4* o4 = reinterpret_cast<uint4*>(
          dst + ((((static_cast<size_t>(gi.tgt_layer) * d.B + ti.b) * d.H_t + h) * d.S + s) * d.d_t +
                 i0));
#pragma unroll
      for (int v = 0; v < 4; ++v)
        o4[v] = make_uint4(pack_bf16x2(__uint_as_float(r[8 * v + 0]), __uint_as_float(r[8 * v + 1])),
                           pack_bf16x2(__uint_as_float(r[8 * v + 2]), __uint_as_float(r[8 * v + 3])),
                           pack_bf16x2(__uint_as_float(r[8 * v + 4]), __uint_as_float(r[8 * v + 5])),
                           pack_bf16x2(__uint_as_float(r[8 * v + 6]), __uint_as_float(r[8 * v + 7])));
    }
  }
}

}  // namespace mot
