// Internal declarations shared by the C-ABI layer and the kernel files.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "mot.h"

namespace mot {

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

// ---------------------------------------------------------------- backbone translators
//
// The App. C.2 backbone inside the gated mixture (bt.cu). Per token, the rows
// of the channel window are the source cache's P = H_s heads of each slot; the
// kernels work on a row space of R = B * S * P rows, row ((b * S + s) * P + p),
// one row space per group g = x * E + m (K/V block x, backbone m). The row layer
// norms' affines are applied where the rows are written; LN_in's and LN_out's
// are folded into W_in and W_out at load.
constexpr int kBtMaxSlots = 32;
constexpr int kBtMaxP = 16;

struct BtDims {
  int32_t L_s, P, d_s, L_t, H_t, d_t, E, top_k, B, S;
  int32_t Ds, Dt;
  int32_t N, q0, d, na, df;   // window slots, first window layer, width, heads, FFN width
  int32_t G;                  // 2 * E groups
  int32_t tau;                // tokens per row tile (128 / P, rounded down)
  int32_t tiles_b;            // row tiles per batch entry: ceil(S / tau)
  int64_t R;                  // rows of one group's row space: B * S * P
};

struct BtArgs {
  BtDims d;
  const void* src[2];
  void* dst[2];
  const int32_t* seq_lens;
  int32_t batch;
  int32_t slot;                         // r of this launch
  int32_t src_layer[kBtMaxSlots];       // source layer of each window slot
  // folded weights (fp32 vectors; bf16 matrices are read through tensor maps)
  const void* wg;        // [2][E][N * Ds] bf16
  const float* bg;       // [2][E]
  const float* s_in;     // [G][d]  row sums of the folded W_in (hi + lo)
  const float* ln_q;     // [G][N][2][d] gamma, beta of LN_Q of each slot
  const float* ln_c;     // [G][N][2][d] LN_C
  const float* ln_f;     // [G][N][2][d] LN_F
  const float* c_in;     // [G][d]
  const float* c_q;      // [G][N][d]
  const float* c_kv;     // [G][N][2d]
  const float* c_o;      // [G][N][d]
  const float* c_f1;     // [G][N][df]
  const float* c_f2;     // [G][N][d]
  const float* c_out;    // [G][Dt]
  const float* s_out;    // [G][Dt]  row sums of the folded W_out
  // workspace, [G][R][...] per group
  float* gate;           // [2][B * S][E] kept, renormalised gate weights
  void* xz;              // bf16 normalised z_r rows          [d]
  void* xq;              // bf16 normalised h_{r-1} rows      [d]
  float* h;              // fp32 state h                       [d]
  float* ht;             // fp32 h~ (after the attention)     [d]
  void* q;               // bf16 queries                       [d]
  void* kv;              // bf16 keys | values                 [2d]
  void* o;               // bf16 attention output              [d]
  void* xf;              // bf16 normalised h~ rows            [d]
  void* f;               // bf16 FFN hidden                    [df]
  void* xo;              // bf16 h_r (raw)                     [d] (= [B * S][P * d])
  float2* rstat;         // [G][R] (mean, M2) of each h_r row over its d values
  int32_t* status;
  long long wait_limit;
};

// GEMM modes of bt_gemm (the epilogue each one runs).
enum BtMode : int {
  kBtIn = 0,    // z = GELU(LN-folded W_in x + c); xz = LN_C(z); slot 0: h = z, xq = LN_Q(z)
  kBtQ = 1,     // q = W_Q xq + b_Q
  kBtKV = 2,    // k | v = W_KV xz + b_KV
  kBtO = 3,     // ht = h + W_O o + b_O; xf = LN_F(ht)
  kBtF1 = 4,    // f = GELU(W_F1 xf + b_F1)
  kBtF2 = 5,    // h = ht + W_F2 f + b_F2; xq = LN_Q(h); xo = bf16(h); row statistics
  kBtOut = 6,   // dst = sum_m gtilde_m GELU(LN-folded W_out' xo_m + c_m)
};

bool bt_supported(const BtDims& d);
cudaError_t launch_bt_gate(const BtArgs& a, cudaStream_t st);
cudaError_t launch_bt_attn(const BtArgs& a, cudaStream_t st);
// tmA: the mode's A operand map (kBtIn: the source K and V maps, tmA and tmA2);
// tmB: its weight map.
cudaError_t launch_bt_gemm(int mode, const BtArgs& a, const CUtensorMap& tmA,
                           const CUtensorMap& tmA2, const CUtensorMap& tmB, int num_sms,
                           cudaStream_t st);
// FFN1 + GELU + FFN2 in one kernel (d_f % 128 == 0): xf map (box 64 x 128), W_F1
// map with box 64 x 128, W_F2 map with box 64 x d; ends with kBtF2's row epilogue.
cudaError_t launch_bt_ffn(const BtArgs& a, const CUtensorMap& tmXf, const CUtensorMap& tmW1,
                          const CUtensorMap& tmW2, int num_sms, cudaStream_t st);

// ---------------------------------------------------------------- replay attention
//
// App. C.4 (replay.cu): one target layer's attention over the replay cache,
// full causal for layers below L_Full, else over the Top-S positions of the
// source guidance map's causal row. Layouts: q / out [B][Hq][N][d], k / v
// [B][Hkv][N][d], guide [B][N][N] (bf16), sel [B][N][S] int32 (ascending
// positions, -1 after the row's count).
struct ReplayDims {
  int32_t B, N, Hq, Hkv, d, S, n_full;
};
struct ReplayArgs {
  ReplayDims d;
  const void* q;
  const void* k;
  const void* v;
  const void* guide;
  void* out;
  int32_t* sel;
  const int32_t* seq_lens;
  int32_t batch;
  int32_t full;   // 1: attend to every position 0..u
  int32_t* status;
};
bool replay_supported(const ReplayDims& d);
// Full causal attention on the tensor cores: maps over q [B*Hq*N][d], k
// [B*Hkv*N][d] (box 64 x 128) and V^T [B*Hkv*d][N] (box 64 x d), the last
// written by launch_replay_vt into `vt`.
bool replay_fmha_supported(const ReplayDims& d);
cudaError_t launch_replay_vt(const ReplayArgs& a, void* vt, cudaStream_t st);
cudaError_t launch_replay_fmha(const ReplayArgs& a, const CUtensorMap& tmQ, const CUtensorMap& tmK,
                               const CUtensorMap& tmVt, cudaStream_t st);
cudaError_t launch_replay_select(const ReplayArgs& a, cudaStream_t st);
cudaError_t launch_replay_attn(const ReplayArgs& a, cudaStream_t st);

// Kernel launchers (each returns the launch's cudaError_t).
cudaError_t launch_bf16_to_f16_inplace(void* buf, size_t n, cudaStream_t st);
cudaError_t launch_build_b2t(const float* b2, void* b2t, int G, int E, int Dt, cudaStream_t st);
cudaError_t launch_build_wg16(const void* wg, void* wg16, int G, int E, int Ds, cudaStream_t st);
cudaError_t launch_f32_to_f16(const float* src, void* dst, size_t n, cudaStream_t st);
cudaError_t launch_prep(const int32_t* seq_lens, int32_t batch, const Dims& d, TileInfo* tiles,
                        int32_t* n_tiles, int32_t* status, cudaStream_t st);
cudaError_t launch_gate(const PathArgs& a, cudaStream_t st);
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
