// Work-item order of the fused persistent translation kernel.
//
// A pass covers F = gp * n_m token tiles ("flat tiles" f = gl * n_m + m). Each
// flat tile has n1 GEMM1 items (one per 256 hidden columns of E*H) and n2
// GEMM2 items (one per 256 output columns of D_t); a GEMM2 item of tile f may
// start only once all n1 GEMM1 items of f are done (it reads their A2 rows).
//
// Flat tiles are grouped into blocks of MB tiles (the last block may be
// short), and items are issued in segments that skew GEMM2 one block behind
// GEMM1:
//   segment 0            GEMM1 items of block 0
//   segment k (1..nb-1)  GEMM1 items of block k, then GEMM2 items of block k-1
//   segment nb           GEMM2 items of block nb-1
// so a GEMM2 item is issued about one block of GEMM1 items after the last
// item it depends on, and its A2 rows are still in L2 when it reads them.
// Inside a block, items run tile by tile with the column index fastest.
#pragma once

#include <stdint.h>

#ifdef __CUDACC__
#define MOT_HD __host__ __device__ __forceinline__
#else
#define MOT_HD inline
#endif

namespace mot {

struct Item {
  int32_t type;   // 1 = GEMM1 (hidden columns), 2 = GEMM2 (output columns)
  int32_t f;      // flat tile
  int32_t n;      // column tile
};

struct Schedule {
  int32_t F;      // flat tiles in the pass
  int32_t n1, n2; // column tiles of GEMM1 / GEMM2
  int32_t MB;     // flat tiles per block

  MOT_HD int32_t blocks() const { return (F + MB - 1) / MB; }
  MOT_HD int32_t total() const { return F * (n1 + n2); }
};

// Item at position i of the issue order, 0 <= i < s.total().
MOT_HD Item schedule_item(const Schedule& s, int32_t i) {
  const int32_t nb = s.blocks();
  const int32_t cl = s.F - (nb - 1) * s.MB;   // tiles in the last block
  int32_t blk, idx, type;
  if (nb == 1) {
    if (i < cl * s.n1) { type = 1; blk = 0; idx = i; }
    else { type = 2; blk = 0; idx = i - cl * s.n1; }
  } else {
    const int32_t g1 = s.MB * s.n1, g2 = s.MB * s.n2, full = g1 + g2;
    if (i < g1) {
      type = 1; blk = 0; idx = i;
    } else {
      const int32_t j = i - g1;
      if (j < (nb - 2) * full) {   // segments 1 .. nb-2
        const int32_t k = 1 + j / full, off = j - (k - 1) * full;
        if (off < g1) { type = 1; blk = k; idx = off; }
        else { type = 2; blk = k - 1; idx = off - g1; }
      } else {
        const int32_t r = j - (nb - 2) * full;   // segments nb-1 and nb
        if (r < cl * s.n1) { type = 1; blk = nb - 1; idx = r; }
        else if (r < cl * s.n1 + g2) { type = 2; blk = nb - 2; idx = r - cl * s.n1; }
        else { type = 2; blk = nb - 1; idx = r - cl * s.n1 - g2; }
      }
    }
  }
  const int32_t nn = type == 1 ? s.n1 : s.n2;
  Item it;
  it.type = type;
  it.f = blk * s.MB + idx / nn;
  it.n = idx % nn;
  return it;
}

}  // namespace mot
