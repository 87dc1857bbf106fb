// Internal declarations of the replay attention (replay.cu, replay_fmha.cu,
// replay_gattn.cu), shared with the C-ABI layer.
#pragma once

#include "mot_internal.h"

namespace mot {

// ---------------------------------------------------------------- replay attention
//
// App. C.4: one target layer's attention over the replay cache,
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
  long long wait_limit;   // bound of every pipeline wait (SM cycles)
  int32_t stall_test;     // test hook: the guided kernel's first CTA stalls its first MMA barrier
};
bool replay_supported(const ReplayDims& d);
// Full causal attention on the tensor cores: maps over k [B*Hkv*N][d] (box
// 64 x 128) and V^T [B*Hkv*d][N] (box 64 x d), the latter written by
// launch_replay_vt into `vt`; the query rows are read from a.q (16-byte aligned).
bool replay_fmha_supported(const ReplayDims& d);
cudaError_t launch_replay_vt(const ReplayArgs& a, void* vt, cudaStream_t st);
cudaError_t launch_replay_fmha(const ReplayArgs& a, const CUtensorMap& tmK,
                               const CUtensorMap& tmVt, cudaStream_t st);
cudaError_t launch_replay_select(const ReplayArgs& a, cudaStream_t st);
// Guided layers on the tensor cores (d = 128, GQA groups of up to 16, S <= 128):
// persistent CTAs, as many per SM as fit.
bool replay_gattn_supported(const ReplayDims& d);
cudaError_t launch_replay_gattn(const ReplayArgs& a, int num_sms, cudaStream_t st);
cudaError_t launch_replay_attn(const ReplayArgs& a, cudaStream_t st);

}  // namespace mot
