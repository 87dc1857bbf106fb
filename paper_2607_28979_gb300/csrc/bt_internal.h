// Internal declarations of the backbone translators (bt.cu), shared with the C-ABI layer.
#pragma once

#include "mot_internal.h"

namespace mot {

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
  // Top-1 routing (token buckets): group g's row space holds only the tokens
  // that chose backbone g % E, packed in token order: row (pos * P + p) for
  // bucket position pos < cnt[g], whose token slot b * S + s is list[g][pos].
  int32_t routed;
  const int32_t* cnt;         // [G] tokens per bucket
  const int32_t* list;        // [G][B * S] token slot of each bucket position
  const int32_t* rpre;        // [2][G + 1] prefix sums of row tiles per bucket: tau-token
                              // tiles, then 128-token tiles (the output projection)
  const void* xs;             // [G][R][d_s] bf16 source rows of the slot, packed per bucket
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
// Top-1 routing: bucket lists and tile prefixes from the gate (cnt, list, rpre),
// then per window slot the bucket tokens' source rows packed into xs.
cudaError_t launch_bt_route(const BtArgs& a, int32_t* cnt, int32_t* list, int32_t* rpre,
                            cudaStream_t st);
cudaError_t launch_bt_pack(const BtArgs& a, void* xs, cudaStream_t st);
cudaError_t launch_bt_attn(const BtArgs& a, cudaStream_t st);
// tmA: the mode's A operand map (kBtIn: the source K and V maps, tmA and tmA2;
// routed, the packed source rows xs in tmA); tmB: its weight map.
cudaError_t launch_bt_gemm(int mode, const BtArgs& a, const CUtensorMap& tmA,
                           const CUtensorMap& tmA2, const CUtensorMap& tmB, int num_sms,
                           cudaStream_t st);
// FFN1 + GELU + FFN2 in one kernel (d_f % 128 == 0): xf map (box 64 x 128), W_F1
// map with box 64 x 128, W_F2 map with box 64 x d; ends with kBtF2's row epilogue.
cudaError_t launch_bt_ffn(const BtArgs& a, const CUtensorMap& tmXf, const CUtensorMap& tmW1,
                          const CUtensorMap& tmW2, int num_sms, cudaStream_t st);

}  // namespace mot
