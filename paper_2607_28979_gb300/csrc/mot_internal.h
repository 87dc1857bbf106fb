// Internal declarations shared by the C-ABI layer and the kernel files.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "mot.h"

#include <nvtx3/nvToolsExt.h>

namespace mot {

// NVTX range over a scope (host code): the entry points and every kernel
// launch are named for nsys / ncu NVTX filtering. Without a tool attached the
// push and pop are a null-pointer check each.
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

constexpr int kTileM = 128;   // tokens per token tile (rows of one MMA tile)
constexpr int kMaxE = 16;     // translators per (layer, K/V) group

// Sticky device status bits, OR-ed into the handle's status word.
enum : int32_t { kStatusSeqLen = 1, kStatusTimeout = 2 };

// One 128-token tile of the ragged batch: batch entry b, positions
// [s0, s0 + rows).
struct TileInfo {
  int32_t b, s0, rows, pad;
};

// One translated (target layer, K/V) group.
struct GroupInfo {
  int32_t tgt_layer, src_layer, x, pad;
};

struct Dims {
  int32_t L_s, H_s, d_s, L_t, H_t, d_t, E, top_k, H, B, S;
  int32_t Ds, Dt, EH;
  int32_t G;          // translated groups = 2 * translated target layers
  int32_t tiles_max;  // B * ceil(S / 128): token tiles at full capacity
  int32_t tpad;       // tiles_max * 128: rows of the gate / A2 workspaces
  int32_t dtype;      // 0 = bf16, 1 = fp32
};

// Everything one translation pass needs on the device. Weights are in the
// library's repacked layout:
//   wg [G][E][Ds] (dtype), bg [G][E] (fp32),
//   w1 [G][E*H][Ds] (dtype; the E experts' W1 stacked along rows),
//   b1 [G][E*H] (fp32),
//   w2 [G][Dt][E*H] (dtype; the E experts' W2 side by side along K),
//   b2 [G][E][Dt] (fp32).
// On the tensor-core path w2 holds fp16 (converted from the bf16 blob at
// load) and b1h an fp16 copy of b1, so that GEMM2 runs fp16 x fp16 -> fp32.
// The gate-weighted bias sum_m gtilde_m b2_m is one more K block of GEMM2:
// A = gate16 (the token's gtilde in its first E columns), B = b2t.
// Workspace: gate [G][tpad][E] fp32 (renormalised gate weights per token
// row), a2 [gp][tpad][E*H] (GELU(hidden) * gate: fp16 on the tensor-core path,
// fp32 on the SIMT path).
struct PathArgs {
  Dims d;
  const void* src[2];
  void* dst[2];
  const TileInfo* tiles;
  const int32_t* n_tiles;
  const GroupInfo* groups;
  const void* wg;
  const float* bg;
  const void* w1;
  const float* b1;
  const void* b1h;   // fp16 [G][E*H] (tensor-core path)
  const void* w2;
  const float* b2;
  float* gate;
  void* gate16;      // fp16 [G][tpad][64]: gtilde padded with zeros (tensor-core path, else null)
  const void* b2t;   // fp16 [G][D_t][64]: b2 transposed, zero-padded (tensor-core path)
  void* a2;
  int32_t* status;
  uint32_t* sel;          // [G][tpad] Top-K selection bits per row (sparse routing), else null
  const int32_t* proj_layer;   // MoT-h projection: the target layer of each group
  int32_t g0, gp;         // groups [g0, g0 + gp) of this pass
  long long wait_limit;   // bound of every pipeline wait, in SM cycles
  int32_t stall_test;     // test hook (single-SM GEMM1): CTA 0 withholds its first stage
};

// Top-K routing (0 < top_k < E) on the tensor-core path (sparse.cu): for each
// (group, expert) bucket of a pass the tokens that selected the expert are
// gathered into a packed row space, each bucket padded to whole pairs of
// 128-row tiles, and the translators run on their own tokens only. GEMM2
// writes each (token, slot) row in fp32; the combine sums a token's top_k
// slots in slot order (slot = rank of the expert among the token's choices).
struct SparsePair {       // one 256-row pair tile of one bucket
  int32_t vg;             // bucket: local group * E + expert
  int32_t p0;             // packed row of its first 128-row tile
  int32_t rows0, rows1;   // valid rows of its two tiles
};
struct SparseArgs {
  int32_t* counts;        // [gp * E] tokens per bucket (this pass)
  int32_t* counts_all;    // [G * E] tokens per bucket of the last translation
  int32_t* row0;          // [gp * E] first packed row of each bucket
  int32_t* plan;          // [2]: number of pairs, packed rows in use
  SparsePair* pairs;      // [max_pairs]
  int32_t* ltok;          // [R] token row (index into the tpad rows), -1 for padding
  int32_t* lslot;         // [R] slot of the row's expert among the token's choices
  float* gatep;           // [R] gtilde of the row's expert
  void* gate16p;          // [R][64] fp16: gtilde in the bucket's expert column, else 0
  void* zp;               // [H_s][R][d_s] packed source rows (dtype)
  void* a2p;              // [R][H] fp16 hidden activations
  float* ybuf;            // [gp][tpad][top_k][D_t] per-slot outputs (top_k > 1; top_k = 1
                          // stores the target rows from GEMM2)
  int32_t R;              // packed-row capacity of a pass
  int32_t max_pairs;
};

// Kernel launchers (each returns the launch's cudaError_t).
cudaError_t launch_bf16_to_f16_inplace(void* buf, size_t n, cudaStream_t st);
cudaError_t launch_build_b2t(const float* b2, void* b2t, int G, int E, int Dt, cudaStream_t st);
cudaError_t launch_build_wg16(const void* wg, void* wg16, int G, int E, int Ds, cudaStream_t st);
cudaError_t launch_f32_to_f16(const float* src, void* dst, size_t n, cudaStream_t st);
cudaError_t launch_prep(const int32_t* seq_lens, int32_t batch, const Dims& d, TileInfo* tiles,
                        int32_t* n_tiles, int32_t* status, cudaStream_t st);
cudaError_t launch_gate(const PathArgs& a, cudaStream_t st);
cudaError_t launch_fixed_gate(const PathArgs& a, const float* fg, cudaStream_t st);
cudaError_t launch_simt_gemm1(const PathArgs& a, cudaStream_t st);
cudaError_t launch_simt_gemm2(const PathArgs& a, cudaStream_t st);

// tcgen05 path. GEMM1: source K/V load maps, W1 load map and the A2 store map
// (box 64 x 32 x 1); GEMM2: A2 load map (box 64 x 128 x 1) and W2 load map.
constexpr int kUmmaN = 256;   // N of one accumulator tile
constexpr int kUmmaK = 64;    // K per pipeline stage (one 128-byte swizzle row)
bool umma_supported(const Dims& d);
cudaError_t launch_umma_gemm1(const PathArgs& a, const CUtensorMap& tmK, const CUtensorMap& tmV,
                              const CUtensorMap& tmW1, const CUtensorMap& tmA2st, int num_sms,
                              cudaStream_t st);
cudaError_t launch_umma_gemm2(const PathArgs& a, const CUtensorMap& tmA2, const CUtensorMap& tmW2,
                              const CUtensorMap& tmG16, const CUtensorMap& tmB2t, int num_sms,
                              cudaStream_t st);

// 2-SM variant (umma2.cu): CTA pairs, tcgen05.mma.cta_group::2 on 256 x 256
// tiles. The W maps here have 64 x 128 boxes (each CTA loads half of B).
cudaError_t launch_umma2_gemm1(const PathArgs& a, const CUtensorMap& tmK, const CUtensorMap& tmV,
                               const CUtensorMap& tmW1h, const CUtensorMap& tmA2st, int num_sms,
                               cudaStream_t st);
cudaError_t launch_umma2_gemm2(const PathArgs& a, const CUtensorMap& tmA2, const CUtensorMap& tmW2h,
                               const CUtensorMap& tmG16, const CUtensorMap& tmB2th, int num_sms,
                               cudaStream_t st);

// Gate on the tensor cores (gate_mma.cu): the source K/V load maps (box
// 64 x 128) and a map over wg16 = [G * 16][D_s] bf16 (box 64 x 16), the gate
// weights zero-padded to 16 rows per group.
cudaError_t launch_gate_mma(const PathArgs& a, const CUtensorMap& tmK, const CUtensorMap& tmV,
                            const CUtensorMap& tmWg, int num_sms, cudaStream_t st);

// Sparse routing launchers (sparse.cu); the GEMMs are the pair kernels of
// umma2.cu over the packed rows: GEMM1 reads the zp map (box 64 x 128 over
// [H_s * R][d_s]) and stores A2p through a 32 x 32 x 1 box over [1][R][H];
// GEMM2 reads A2p (box 64 x 128 x 1) and gate16p (box 64 x 128 x 1 over [1][R][64]).
// step 0: bucket sizes; 1: packed layout and pair-tile list; 2: bucket rows.
cudaError_t launch_route(const PathArgs& a, const SparseArgs& s, int step, cudaStream_t st);
cudaError_t launch_pack(const PathArgs& a, const SparseArgs& s, cudaStream_t st);
cudaError_t launch_combine(const PathArgs& a, const SparseArgs& s, cudaStream_t st);
cudaError_t launch_umma2_sparse_gemm1(const PathArgs& a, const SparseArgs& s,
                                      const CUtensorMap& tmZp, const CUtensorMap& tmW1h,
                                      const CUtensorMap& tmA2pst, int num_sms, cudaStream_t st);
cudaError_t launch_umma2_sparse_gemm2(const PathArgs& a, const SparseArgs& s,
                                      const CUtensorMap& tmA2p, const CUtensorMap& tmW2h,
                                      const CUtensorMap& tmG16p, const CUtensorMap& tmB2th,
                                      int num_sms, cudaStream_t st);

// MoT-h (App. C.5) projection on CTA pairs: K | V = a_hat [W^K; W^V]^T, bf16.
// a.d holds the target cache dims; act_width = d_at (a multiple of 64).
cudaError_t launch_umma2_proj(const PathArgs& a, const CUtensorMap& tmAct,
                              const CUtensorMap& tmWkv, int act_width, int num_sms,
                              cudaStream_t st);

// On-chip translation on CTA pairs for D_s <= 128, D_t = 256 (onchip.cu):
// GEMM1, GELU * gate and GEMM2 in one persistent launch over all groups, the
// hidden activations kept in shared memory. W1 map: box 64 x 64 (half of a
// 128-row chunk); W2 and b2t maps: box 64 x 128; gate16: box 64 x 128 x 1.
bool onchip_supported(const Dims& d);
cudaError_t launch_onchip(const PathArgs& a, const CUtensorMap& tmK, const CUtensorMap& tmV,
                          const CUtensorMap& tmW1q, const CUtensorMap& tmW2h,
                          const CUtensorMap& tmG16, const CUtensorMap& tmB2th, int num_sms,
                          cudaStream_t st);

// On-chip translation for D_t = 512 (wide.cu): clusters of two CTA pairs, pair
// p owning output columns [256 p, 256 p + 256); the pairs split GEMM1's hidden
// chunks and exchange them through distributed shared memory. Same maps as the
// on-chip kernel.
bool wide_supported(const Dims& d);
cudaError_t launch_wide(const PathArgs& a, const CUtensorMap& tmK, const CUtensorMap& tmV,
                        const CUtensorMap& tmW1q, const CUtensorMap& tmW2h,
                        const CUtensorMap& tmG16, const CUtensorMap& tmB2th, int num_sms,
                        cudaStream_t st);

// Fused persistent kernel: both GEMMs of a pass in one launch (fused.cu).
// `counters` holds fused_counter_ints(d, gp) int32 (zeroed by the launcher).
int fused_block_tiles(const Dims& d, int num_sms);
size_t fused_counter_ints(const Dims& d, int gp);
cudaError_t launch_fused(const PathArgs& a, const CUtensorMap& tmK, const CUtensorMap& tmV,
                         const CUtensorMap& tmW1, const CUtensorMap& tmA2,
                         const CUtensorMap& tmW2, const CUtensorMap& tmA2st,
                         const CUtensorMap& tmG16, const CUtensorMap& tmB2t, int32_t* counters,
                         int num_sms, cudaStream_t st);

}  // namespace mot
