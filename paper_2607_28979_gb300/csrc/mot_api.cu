// C ABI of libmot.so: handle lifetime, weight repacking, argument checking and
// the launch sequence of one translation (see include/mot.h).
#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>
#include <string.h>

#include <algorithm>
#include <cmath>
#include <new>
#include <string>
#include <vector>

#include "bt_internal.h"
#include "mot_internal.h"
#include "replay_internal.h"

using namespace mot;

namespace {

// Upper bound on the A2 workspace; groups are translated in passes of `gp`
// groups so that gp * tpad * E*H elements fit in it.
constexpr size_t kA2Budget = size_t(8) << 30;

// Chunks of target layers the host-buffer entry point pipelines over.
constexpr int kHostChunks = 16;   // most chunks of layers of the host-buffer pipeline

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}

// 16-bit tensor map (bf16, or fp16 when `f16`) with 128-byte swizzle (64-byte
// when `swizzle64`); dims[0] is the contiguous one.
bool encode_bf16(CUtensorMap* map, const void* base, int rank, const uint64_t* dims,
                 const uint64_t* strides_bytes, const uint32_t* box, bool f16 = false,
                 bool swizzle64 = false) {
  EncodeTiledFn fn = encode_fn();
  if (!fn) return false;
  cuuint64_t gd[5], gs[4];
  cuuint32_t bx[5], es[5];
  for (int i = 0; i < rank; ++i) {
    gd[i] = dims[i];
    bx[i] = box[i];
    es[i] = 1;
  }
  for (int i = 0; i < rank - 1; ++i) gs[i] = strides_bytes[i];
  CUresult r = fn(map, f16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), gd, gs, bx,
                  es, CU_TENSOR_MAP_INTERLEAVE_NONE,
                  swizzle64 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_128B,
                  CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

struct Ev {
  cudaEvent_t a, b;
  int kind;
};

}  // namespace

// Backbone-translator handles (kind 2): folded weights, the per-group row
// space workspace and the tensor maps over them (bt.cu has the layouts).
struct BtState {
  BtDims d{};
  int32_t src_layer[kBtMaxSlots] = {};
  void* wg = nullptr;     // [2][E][N * Ds] bf16
  float* bg = nullptr;    // [2][E]
  float *s_in = nullptr, *c_in = nullptr, *c_q = nullptr, *c_kv = nullptr, *c_o = nullptr,
        *c_f1 = nullptr, *c_f2 = nullptr, *c_out = nullptr, *s_out = nullptr, *ln_q = nullptr,
        *ln_c = nullptr, *ln_f = nullptr;
  // bf16 matrices: win [G][d][2 d_s] (hi | lo), wq [G][N][d][d], wkv [G][N][2d][d], wo [G][N][d][d],
  // wf1 [G][N][df][d], wf2 [G][N][d][df], wout [G][Dt][P d]
  void *win = nullptr, *wq = nullptr, *wkv = nullptr, *wo = nullptr, *wf1 = nullptr,
       *wf2 = nullptr, *wout = nullptr;
  float *gate = nullptr, *h = nullptr, *ht = nullptr;
  void *xz = nullptr, *xq = nullptr, *q = nullptr, *kv = nullptr, *o = nullptr, *xf = nullptr,
       *f = nullptr, *xo = nullptr;
  float2* rstat = nullptr;
  // Top-1 routing (token buckets): counts, lists, tile prefixes, packed source rows
  int32_t *rcnt = nullptr, *rlist = nullptr, *rpre = nullptr;
  void* xs = nullptr;   // [G][R][d_s] bf16
  CUtensorMap tm_win{}, tm_wq{}, tm_wkv{}, tm_wo{}, tm_wf1{}, tm_wf2{}, tm_wout{}, tm_wf1c{};
  CUtensorMap tm_xz{}, tm_xq{}, tm_o{}, tm_xf{}, tm_f{}, tm_xo{};
  CUtensorMap tm_xs{}, tm_wout_r{};   // routed: packed source rows, W_out with 256-row boxes

  void free_all() {
    void* ptrs[] = {wg, bg, s_in, c_in, c_q, c_kv, c_o, c_f1, c_f2, c_out, s_out, ln_q, ln_c,
                    ln_f, win, wq, wkv, wo, wf1, wf2, wout, gate, h, ht, xz, xq, q, kv, o, xf,
                    f, xo, rstat, rcnt, rlist, rpre, xs};
    for (void* p : ptrs)
      if (p) cudaFree(p);
  }
};

struct mot_ctx {
  mot_config cfg{};
  std::vector<int32_t> layer_map;
  Dims d{};
  int device = 0;
  int num_sms = 0;
  bool use_umma = false;
  int schedule = 2;           // tcgen05 path: 0 split, 1 fused, 2 split on CTA pairs, 3 on-chip,
                              // 4 on-chip on clusters of two pairs (D_t = 512)
  long long wait_limit = 4000000000LL;   // bound of every pipeline wait (SM cycles)
  int stall_test = 0;                    // test hook, see mot_debug_set
  const float* fixed_gate = nullptr;     // test hook, see mot_debug_fixed_gate
  bool weights_loaded = false;
  int gp_max = 1;
  std::vector<GroupInfo> groups_h;

  // weights (library layout, see PathArgs)
  void* wg = nullptr;
  float* bg = nullptr;
  void* w1 = nullptr;
  float* b1 = nullptr;
  void* b1h = nullptr;   // fp16 copy of b1 (tensor-core path)
  void* w2 = nullptr;    // dtype on the SIMT path, fp16 on the tensor-core path
  float* b2 = nullptr;
  GroupInfo* groups = nullptr;
  // workspace
  float* gate = nullptr;
  void* gate16 = nullptr;   // fp16 gate rows padded to 64 (tensor-core path)
  void* b2t = nullptr;      // fp16 b2 transposed, padded to 64 (tensor-core path)
  void* wg16 = nullptr;     // bf16 gate weights padded to 16 rows per group (tensor-core path)
  void* a2 = nullptr;
  TileInfo* tiles = nullptr;
  int32_t* n_tiles = nullptr;
  int32_t* status = nullptr;
  int32_t* counters = nullptr;   // fused schedule: item counter + per-tile completions
  // tensor maps that do not depend on the caller's buffers
  CUtensorMap tm_w1{}, tm_w2{}, tm_a2{}, tm_a2_st{}, tm_w1h{}, tm_w2h{}, tm_w1q{};
  CUtensorMap tm_g16{}, tm_b2t{}, tm_b2th{}, tm_wg16{};
  // MoT-h (App. C.5): kind 1 handles translate activations; `d` then holds the
  // mixture's dims (one-head source of width d_as, one-head output of width
  // d_at) and `hd` the target cache the projections restore.
  int kind = 0;
  int32_t act_tgt = 0;
  Dims hd{};
  int gp_h = 1;                 // groups (layers) per pass; a_hat slot = group % gp_h
  void* wkv = nullptr;          // [G][2 D_t][d_at] bf16: W^K then W^V of each layer
  void* ahat = nullptr;         // [gp_h][B][S][d_at] bf16 translated activations
  int32_t* proj_layer = nullptr;   // [G] target layer of each group
  CUtensorMap tm_wkv{}, tm_ahat{};
  // backbone translators (App. C.2): kind 2
  BtState* bt = nullptr;
  // replay attention (App. C.4): kind 3
  ReplayDims rd{};
  int32_t* rsel = nullptr;   // [B][N][S] selection workspace
  void* rvt = nullptr;       // [B][Hkv][d][N] bf16: V^T for the tensor-core full attention
  // Top-K routing (tensor-core path, 0 < top_k < E): token buckets per expert
  bool sparse_ok = false;   // the shapes support it
  int routing = 0;          // 0 dense compute with a zeroed gate, 1 token buckets
  int gp_sparse = 1;        // groups per routed pass
  uint32_t* sel = nullptr;  // [G][tpad] Top-K choices per row
  SparseArgs sp{};
  bool counts_valid = false;
  CUtensorMap tm_zp{}, tm_a2p{}, tm_a2p_st{}, tm_g16p{};
  // host-buffer staging for mot_translate_host (allocated on first use)
  void* st_src[2] = {nullptr, nullptr};
  void* st_dst[2] = {nullptr, nullptr};
  int32_t* st_len = nullptr;
  cudaStream_t copy_h2d = nullptr, copy_d2h = nullptr;   // created on first use
  cudaEvent_t ev_h2d[kHostChunks] = {}, ev_comp[kHostChunks] = {};
  cudaEvent_t ev_prev_compute = nullptr, ev_prev_d2h = nullptr;
  // profiling
  bool profile = false;
  std::vector<Ev> ev_used, ev_free;
  std::vector<std::string> kind_names;
  int64_t launches = 0;
};

namespace {

size_t esize(const Dims& d) { return d.dtype == 0 ? 2 : 4; }
size_t src_bytes(const Dims& d) {
  return size_t(d.L_s) * d.B * d.H_s * size_t(d.S) * d.d_s * esize(d);
}
size_t dst_bytes(const Dims& d) {
  return size_t(d.L_t) * d.B * d.H_t * size_t(d.S) * d.d_t * esize(d);
}
size_t group_elems(const Dims& d) {
  const size_t E = d.E, Ds = d.Ds, Dt = d.Dt, H = d.H;
  return E * Ds + E + E * (H * Ds + H + Dt * H + Dt);
}

void free_all(mot_ctx* h) {
  void* ptrs[] = {h->wg, h->bg, h->w1, h->b1, h->b1h, h->w2, h->b2, h->groups, h->gate, h->gate16,
                  h->b2t, h->wg16, h->a2, h->tiles, h->sel, h->sp.counts, h->sp.counts_all,
                  h->sp.row0, h->sp.plan, h->sp.pairs, h->sp.ltok, h->sp.lslot, h->sp.gatep,
                  h->sp.gate16p, h->sp.zp, h->sp.a2p, h->sp.ybuf, h->wkv, h->ahat,
                  h->proj_layer,
                  h->rsel, h->rvt,
                  h->n_tiles, h->status, h->counters, h->st_src[0], h->st_src[1], h->st_dst[0],
                  h->st_dst[1], h->st_len};
  for (void* p : ptrs)
    if (p) cudaFree(p);
  if (h->bt) {
    h->bt->free_all();
    delete h->bt;
    h->bt = nullptr;
  }
  for (auto& e : h->ev_used) { cudaEventDestroy(e.a); cudaEventDestroy(e.b); }
  for (int c = 0; c < kHostChunks; ++c) {
    if (h->ev_h2d[c]) cudaEventDestroy(h->ev_h2d[c]);
    if (h->ev_comp[c]) cudaEventDestroy(h->ev_comp[c]);
  }
  if (h->ev_prev_compute) cudaEventDestroy(h->ev_prev_compute);
  if (h->ev_prev_d2h) cudaEventDestroy(h->ev_prev_d2h);
  if (h->copy_h2d) cudaStreamDestroy(h->copy_h2d);
  if (h->copy_d2h) cudaStreamDestroy(h->copy_d2h);
  for (auto& e : h->ev_free) { cudaEventDestroy(e.a); cudaEventDestroy(e.b); }
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool overlap(const void* a, size_t na, const void* b, size_t nb) {
  const uintptr_t x = reinterpret_cast<uintptr_t>(a), y = reinterpret_cast<uintptr_t>(b);
  return x < y + nb && y < x + na;
}

int kind_id(mot_ctx* h, const char* name) {
  for (size_t i = 0; i < h->kind_names.size(); ++i)
    if (h->kind_names[i] == name) return static_cast<int>(i);
  h->kind_names.emplace_back(name);
  return static_cast<int>(h->kind_names.size() - 1);
}

// Launch wrapper: counts the launch and, when profiling, brackets it with events.
template <class F>
cudaError_t timed(mot_ctx* h, const char* name, cudaStream_t st, F&& launch) {
  NvtxRange range(name);
  Ev ev{};
  if (h->profile) {
    if (!h->ev_free.empty()) {
      ev = h->ev_free.back();
      h->ev_free.pop_back();
    } else {
      if (cudaEventCreate(&ev.a) != cudaSuccess || cudaEventCreate(&ev.b) != cudaSuccess)
        return cudaErrorMemoryAllocation;
    }
    ev.kind = kind_id(h, name);
    cudaEventRecord(ev.a, st);
  }
  cudaError_t e = launch();
  ++h->launches;
  if (h->profile) {
    cudaEventRecord(ev.b, st);
    h->ev_used.push_back(ev);
  }
  return e;
}

mot_status validate(const mot_config* c) {
  if (c->n_layers_src <= 0 || c->src_kv_heads <= 0 || c->src_head_dim <= 0 ||
      c->n_layers_tgt <= 0 || c->tgt_kv_heads <= 0 || c->tgt_head_dim <= 0 ||
      c->n_translators <= 0 || c->hidden <= 0 || c->max_batch <= 0 || c->max_seq <= 0)
    return MOT_ERR_INVALID_ARG;
  if (c->top_k < 0 || c->top_k > c->n_translators) return MOT_ERR_INVALID_ARG;
  if (c->dtype != MOT_BF16 && c->dtype != MOT_FP32) return MOT_ERR_INVALID_ARG;
  if (c->layer_map)
    for (int l = 0; l < c->n_layers_tgt; ++l)
      if (c->layer_map[l] < -1 || c->layer_map[l] >= c->n_layers_src) return MOT_ERR_INVALID_ARG;
  if (c->n_translators > kMaxE || c->max_batch > 4096) return MOT_ERR_UNSUPPORTED;
  // index arithmetic inside the kernels uses 32-bit tile and row counts
  const long long tiles = (long long)c->max_batch * ((c->max_seq + kTileM - 1) / kTileM);
  if (tiles * kTileM > INT32_MAX / 2) return MOT_ERR_UNSUPPORTED;
  if ((long long)c->n_translators * c->hidden > (1 << 24)) return MOT_ERR_UNSUPPORTED;
  // TMA row coordinates of the caches are 32-bit
  if ((long long)c->n_layers_src * c->max_batch * c->src_kv_heads * c->max_seq > INT32_MAX / 2)
    return MOT_ERR_UNSUPPORTED;
  return MOT_OK;
}

// Depth-ratio channel map (App. C.3): round(l*(L_s-1)/(L_t-1)), halves up.
void depth_ratio(int L_s, int L_t, std::vector<int32_t>& out) {
  out.resize(L_t);
  for (int l = 0; l < L_t; ++l) {
    if (L_t == 1) { out[l] = 0; continue; }
    const long long num = (long long)l * (L_s - 1), den = L_t - 1;
    out[l] = static_cast<int32_t>((2 * num + den) / (2 * den));
  }
}

PathArgs path_args(mot_ctx* h) {
  PathArgs a{};
  a.d = h->d;
  a.tiles = h->tiles;
  a.n_tiles = h->n_tiles;
  a.groups = h->groups;
  a.wg = h->wg;
  a.bg = h->bg;
  a.w1 = h->w1;
  a.b1 = h->b1;
  a.b1h = h->b1h;
  a.w2 = h->w2;
  a.b2 = h->b2;
  a.gate = h->gate;
  a.gate16 = h->use_umma ? h->gate16 : nullptr;
  a.b2t = h->b2t;
  a.a2 = h->a2;
  a.status = h->status;
  a.wait_limit = h->wait_limit;
  a.stall_test = h->stall_test;
  return a;
}

#define MOT_CUDA_TRY(x)                 \
  do {                                  \
    if ((x) != cudaSuccess) {           \
      cudaGetLastError();               \
      return MOT_ERR_CUDA;              \
    }                                   \
  } while (0)

// Translate groups [g_begin, g_end) (group 2r + x: r-th translated target
// layer, x = K/V) on `st`; `do_prep` builds the tile list from seq_lens first.
mot_status run_translate(mot_ctx* h, const void* src_k, const void* src_v, const int32_t* seq_lens,
                         int32_t batch, void* dst_k, void* dst_v, cudaStream_t st, int g_begin,
                         int g_end, bool do_prep) {
  const Dims& d = h->d;
  if (batch == 0 || g_end <= g_begin) return MOT_OK;
  PathArgs a = path_args(h);
  a.src[0] = src_k;
  a.src[1] = src_v;
  a.dst[0] = dst_k;
  a.dst[1] = dst_v;

  CUtensorMap tmK{}, tmV{};
  if (h->use_umma) {
    // the source cache as rows of d_s elements: row ((l * B + b) * H_s + h) * S + s
    const uint64_t dims[2] = {uint64_t(d.d_s), uint64_t(d.L_s) * d.B * d.H_s * d.S};
    const uint64_t st_b[1] = {uint64_t(d.d_s) * 2};
    const uint32_t box[2] = {uint32_t(kUmmaK), uint32_t(kTileM)};
    if (!encode_bf16(&tmK, src_k, 2, dims, st_b, box) ||
        !encode_bf16(&tmV, src_v, 2, dims, st_b, box))
      return MOT_ERR_CUDA;
  }

  if (do_prep)
    MOT_CUDA_TRY(timed(h, "prep_tiles", st, [&] {
      return launch_prep(seq_lens, batch, d, h->tiles, h->n_tiles, h->status, st);
    }));
  a.g0 = g_begin;
  a.gp = g_end - g_begin;
  const bool routed = h->use_umma && h->sparse_ok && h->routing == 1;
  a.sel = routed ? h->sel : nullptr;
  if (h->fixed_gate) {   // test hook: the caller's gate rows replace the gate
    if (routed) return MOT_ERR_UNSUPPORTED;
    MOT_CUDA_TRY(timed(h, "gate_fixed", st, [&] { return launch_fixed_gate(a, h->fixed_gate, st); }));
  } else {
    MOT_CUDA_TRY(timed(h, "gate", st, [&] {
      return h->use_umma ? launch_gate_mma(a, tmK, tmV, h->tm_wg16, h->num_sms, st)
                         : launch_gate(a, st);
    }));
  }
  if (routed) {   // Top-K: per-expert token buckets, passes of gp_sparse groups
    const SparseArgs& sp = h->sp;
    for (int g0 = g_begin; g0 < g_end; g0 += h->gp_sparse) {
      a.g0 = g0;
      a.gp = std::min(h->gp_sparse, g_end - g0);
      MOT_CUDA_TRY(timed(h, "route_count", st, [&] { return launch_route(a, sp, 0, st); }));
      MOT_CUDA_TRY(timed(h, "route_plan", st, [&] { return launch_route(a, sp, 1, st); }));
      MOT_CUDA_TRY(timed(h, "route_fill", st, [&] { return launch_route(a, sp, 2, st); }));
      MOT_CUDA_TRY(timed(h, "pack", st, [&] { return launch_pack(a, sp, st); }));
      MOT_CUDA_TRY(timed(h, "umma2_sparse_gemm1", st, [&] {
        return launch_umma2_sparse_gemm1(a, sp, h->tm_zp, h->tm_w1h, h->tm_a2p_st, h->num_sms, st);
      }));
      MOT_CUDA_TRY(timed(h, "umma2_sparse_gemm2", st, [&] {
        return launch_umma2_sparse_gemm2(a, sp, h->tm_a2p, h->tm_w2h, h->tm_g16p, h->tm_b2th,
                                         h->num_sms, st);
      }));
      if (d.top_k > 1)   // top_k = 1: GEMM2 stored the target rows
        MOT_CUDA_TRY(timed(h, "combine", st, [&] { return launch_combine(a, sp, st); }));
    }
    h->counts_valid = true;
    return MOT_OK;
  }
  if (h->use_umma && h->schedule == 4) {   // one launch; no A2 workspace, so no passes
    MOT_CUDA_TRY(timed(h, "umma2_wide_translate", st, [&] {
      return launch_wide(a, tmK, tmV, h->tm_w1q, h->tm_w2h, h->tm_g16, h->tm_b2th, h->num_sms, st);
    }));
    return MOT_OK;
  }
  if (h->use_umma && h->schedule == 3) {   // one launch; no A2 workspace, so no passes
    MOT_CUDA_TRY(timed(h, "umma2_onchip_translate", st, [&] {
      return launch_onchip(a, tmK, tmV, h->tm_w1q, h->tm_w2h, h->tm_g16, h->tm_b2th, h->num_sms,
                           st);
    }));
    return MOT_OK;
  }
  for (int g0 = g_begin; g0 < g_end; g0 += h->gp_max) {
    a.g0 = g0;
    a.gp = std::min(h->gp_max, g_end - g0);
    if (h->use_umma && h->schedule == 2) {
      MOT_CUDA_TRY(timed(h, "umma2_gemm1_gelu_gate", st, [&] {
        return launch_umma2_gemm1(a, tmK, tmV, h->tm_w1h, h->tm_a2_st, h->num_sms, st);
      }));
      MOT_CUDA_TRY(timed(h, "umma2_gemm2_combine_store", st, [&] {
        return launch_umma2_gemm2(a, h->tm_a2, h->tm_w2h, h->tm_g16, h->tm_b2th, h->num_sms, st);
      }));
    } else if (h->use_umma && h->schedule == 1) {
      MOT_CUDA_TRY(timed(h, "umma_fused_translate", st, [&] {
        return launch_fused(a, tmK, tmV, h->tm_w1, h->tm_a2, h->tm_w2, h->tm_a2_st, h->tm_g16,
                            h->tm_b2t, h->counters, h->num_sms, st);
      }));
    } else if (h->use_umma) {
      MOT_CUDA_TRY(timed(h, "umma_gemm1_gelu_gate", st, [&] {
        return launch_umma_gemm1(a, tmK, tmV, h->tm_w1, h->tm_a2_st, h->num_sms, st);
      }));
      MOT_CUDA_TRY(timed(h, "umma_gemm2_combine_store", st, [&] {
        return launch_umma_gemm2(a, h->tm_a2, h->tm_w2, h->tm_g16, h->tm_b2t, h->num_sms, st);
      }));
    } else {
      MOT_CUDA_TRY(timed(h, "simt_gemm1_gelu_gate", st, [&] { return launch_simt_gemm1(a, st); }));
      MOT_CUDA_TRY(timed(h, "simt_gemm2_combine_store", st, [&] { return launch_simt_gemm2(a, st); }));
    }
  }
  return MOT_OK;
}

// Copy the real-token rows (s < lens[b], every head, batch entries b < batch)
// of layers [l0, l1) of a cache laid out [L][B][H][S][d] between host and
// device staging. Equal lengths make each layer (and, with the whole batch, a
// run of layers) one strided 2-D copy; ragged lengths copy per batch entry.
cudaError_t copy_real_rows(void* dst, const void* src, int l0, int l1, int B, int H, int S, int dd,
                           size_t es, const int32_t* lens, int batch, cudaMemcpyKind kind,
                           cudaStream_t st) {
  bool uniform = true;
  for (int b = 1; b < batch; ++b) uniform = uniform && lens[b] == lens[0];
  const size_t pitch = size_t(S) * dd * es;
  char* dp = static_cast<char*>(dst);
  const char* sp = static_cast<const char*>(src);
  if (uniform) {
    const size_t width = size_t(lens[0]) * dd * es;
    if (width == 0) return cudaSuccess;
    if (batch == B) {
      const size_t off = size_t(l0) * B * H * pitch;
      return cudaMemcpy2DAsync(dp + off, pitch, sp + off, pitch, width,
                               size_t(l1 - l0) * B * H, kind, st);
    }
    for (int l = l0; l < l1; ++l) {
      const size_t off = size_t(l) * B * H * pitch;
      cudaError_t e = cudaMemcpy2DAsync(dp + off, pitch, sp + off, pitch, width, size_t(batch) * H,
                                        kind, st);
      if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
  }
  for (int l = l0; l < l1; ++l)
    for (int b = 0; b < batch; ++b) {
      const size_t width = size_t(lens[b]) * dd * es;
      if (width == 0) continue;
      const size_t off = (size_t(l) * B + b) * H * pitch;
      cudaError_t e = cudaMemcpy2DAsync(dp + off, pitch, sp + off, pitch, width, H, kind, st);
      if (e != cudaSuccess) return e;
    }
  return cudaSuccess;
}

mot_status check_translate_args(mot_ctx* h, const void* src_k, const void* src_v,
                                const int32_t* seq_lens, int32_t batch, const void* dst_k,
                                const void* dst_v) {
  if (!h || h->kind != 0) return MOT_ERR_INVALID_ARG;   // MoT-h handles: mot_translate_h
  if (batch < 0 || batch > h->d.B) return MOT_ERR_INVALID_ARG;
  if (!src_k || !src_v || !dst_k || !dst_v || (batch > 0 && !seq_lens)) return MOT_ERR_INVALID_ARG;
  if (!aligned16(src_k) || !aligned16(src_v) || !aligned16(dst_k) || !aligned16(dst_v))
    return MOT_ERR_INVALID_ARG;
  const size_t sb = src_bytes(h->d), db = dst_bytes(h->d);
  if (overlap(dst_k, db, dst_v, db) || overlap(dst_k, db, src_k, sb) ||
      overlap(dst_k, db, src_v, sb) || overlap(dst_v, db, src_k, sb) ||
      overlap(dst_v, db, src_v, sb))
    return MOT_ERR_INVALID_ARG;
  if (!h->weights_loaded) return MOT_ERR_NO_WEIGHTS;
  return MOT_OK;
}

}  // namespace

extern "C" {

const char* mot_status_string(mot_status s) {
  switch (s) {
    case MOT_OK: return "MOT_OK";
    case MOT_ERR_INVALID_ARG: return "MOT_ERR_INVALID_ARG";
    case MOT_ERR_UNSUPPORTED: return "MOT_ERR_UNSUPPORTED";
    case MOT_ERR_NO_WEIGHTS: return "MOT_ERR_NO_WEIGHTS";
    case MOT_ERR_WEIGHTS_SIZE: return "MOT_ERR_WEIGHTS_SIZE";
    case MOT_ERR_OOM: return "MOT_ERR_OOM";
    case MOT_ERR_CUDA: return "MOT_ERR_CUDA";
    case MOT_ERR_SEQ_LEN: return "MOT_ERR_SEQ_LEN";
    case MOT_ERR_TIMEOUT: return "MOT_ERR_TIMEOUT";
  }
  return "MOT_ERR_UNKNOWN";
}

}  // extern "C"

namespace {

// MoT-h extras of a handle: the translated activation width and the target
// cache the projections fill.
struct HSpec {
  int32_t act_tgt, H_t, d_t;
};

mot_status create_impl(const mot_config* cfg, const HSpec* hs, mot_handle* out) {
  if (!out) return MOT_ERR_INVALID_ARG;
  *out = nullptr;
  if (!cfg) return MOT_ERR_INVALID_ARG;
  mot_status vs = validate(cfg);
  if (vs != MOT_OK) return vs;

  mot_ctx* h = new (std::nothrow) mot_ctx();
  if (!h) return MOT_ERR_OOM;
  h->cfg = *cfg;
  if (cfg->layer_map)
    h->layer_map.assign(cfg->layer_map, cfg->layer_map + cfg->n_layers_tgt);
  else
    depth_ratio(cfg->n_layers_src, cfg->n_layers_tgt, h->layer_map);
  h->cfg.layer_map = nullptr;

  Dims& d = h->d;
  d.L_s = cfg->n_layers_src; d.H_s = cfg->src_kv_heads; d.d_s = cfg->src_head_dim;
  d.L_t = cfg->n_layers_tgt; d.H_t = cfg->tgt_kv_heads; d.d_t = cfg->tgt_head_dim;
  d.E = cfg->n_translators; d.top_k = cfg->top_k; d.H = cfg->hidden;
  d.B = cfg->max_batch; d.S = cfg->max_seq;
  d.Ds = d.H_s * d.d_s; d.Dt = d.H_t * d.d_t; d.EH = d.E * d.H;
  d.dtype = cfg->dtype == MOT_BF16 ? 0 : 1;
  d.tiles_max = d.B * ((d.S + kTileM - 1) / kTileM);
  d.tpad = d.tiles_max * kTileM;
  std::vector<int32_t> proj_h;
  if (hs) {   // MoT-h: one group per translated layer; its a_hat slot is group % gp_h
    h->kind = 1;
    h->act_tgt = hs->act_tgt;
    h->hd = d;
    h->hd.H_t = hs->H_t;
    h->hd.d_t = hs->d_t;
    h->hd.Dt = hs->H_t * hs->d_t;
    for (int l = 0; l < d.L_t; ++l)
      if (h->layer_map[l] >= 0) proj_h.push_back(l);
    const size_t G = proj_h.size();
    const size_t per = size_t(d.B) * d.S * hs->act_tgt * 2;
    h->gp_h = static_cast<int>(std::max<size_t>(1, std::min<size_t>(G ? G : 1, kA2Budget / per)));
    if (G) {
      const int passes = static_cast<int>((G + h->gp_h - 1) / h->gp_h);
      h->gp_h = static_cast<int>((G + passes - 1) / passes);
    }
    for (size_t g = 0; g < G; ++g)
      h->groups_h.push_back(
          GroupInfo{static_cast<int32_t>(g % h->gp_h), h->layer_map[proj_h[g]], 0, 0});
  } else {
    for (int l = 0; l < d.L_t; ++l)
      if (h->layer_map[l] >= 0)
        for (int x = 0; x < 2; ++x) h->groups_h.push_back(GroupInfo{l, h->layer_map[l], x, 0});
  }
  d.G = static_cast<int32_t>(h->groups_h.size());

  int dev = 0, cc_major = 0, cc_minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&cc_major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&cc_minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess) {
    cudaGetLastError();
    delete h;
    return MOT_ERR_CUDA;
  }
  h->device = dev;
  if (cc_major != 10 || cc_minor != 3) {   // the kernels are built for sm_103a only
    delete h;
    return MOT_ERR_UNSUPPORTED;
  }
  h->use_umma = umma_supported(d) && encode_fn() != nullptr;
  if (hs && !(h->use_umma && h->hd.Dt % kUmmaN == 0 && h->hd.d_t % 32 == 0)) {
    delete h;   // MoT-h runs on the tensor-core path only
    return MOT_ERR_UNSUPPORTED;
  }
  if (h->use_umma && onchip_supported(d)) h->schedule = 3;

  const size_t es = esize(d), G = d.G, E = d.E, EH = d.EH;
  const size_t a2_row = EH * (h->use_umma ? 2 : 4);
  const size_t per_group_a2 = size_t(d.tpad) * a2_row;
  h->gp_max = static_cast<int>(std::max<size_t>(1, std::min<size_t>(G ? G : 1, kA2Budget / per_group_a2)));
  if (G) {   // balance the passes
    const int passes = (d.G + h->gp_max - 1) / h->gp_max;
    h->gp_max = (d.G + passes - 1) / passes;
  }
  // Top-K routing workspace: per group, K * tpad routed rows plus each bucket's
  // padding to whole pair tiles (under 256 rows per bucket)
  h->sparse_ok = h->use_umma && d.top_k > 0 && d.top_k < d.E && d.H % kUmmaN == 0 && G > 0;
  h->routing = h->sparse_ok ? 1 : 0;
  size_t sp_rows_g = 0, sp_pairs_g = 0;
  if (h->sparse_ok) {
    const size_t K = d.top_k;
    sp_rows_g = K * d.tpad + E * 2 * kTileM;
    sp_pairs_g = (K * d.tpad + 2 * kTileM - 1) / (2 * kTileM) + E;
    const size_t per_g = sp_rows_g * (size_t(d.Ds) * 2 + size_t(d.H) * 2 + 64 * 2 + 12) +
                         (K > 1 ? size_t(d.tpad) * K * d.Dt * 4 : 0);
    h->gp_sparse = static_cast<int>(std::max<size_t>(1, std::min<size_t>(G, kA2Budget / per_g)));
    const int passes = (d.G + h->gp_sparse - 1) / h->gp_sparse;
    h->gp_sparse = (d.G + passes - 1) / passes;
    h->sp.R = static_cast<int32_t>(sp_rows_g * h->gp_sparse);
    h->sp.max_pairs = static_cast<int32_t>(sp_pairs_g * h->gp_sparse);
  }
  const size_t spR = h->sparse_ok ? size_t(h->sp.R) : 1, spGP = h->sparse_ok ? h->gp_sparse : 1;
  struct A { void** p; size_t n; } allocs[] = {
      {(void**)&h->sel, h->sparse_ok ? G * size_t(d.tpad) * 4 : 16},
      {(void**)&h->sp.counts, spGP * E * 4}, {(void**)&h->sp.counts_all, G * E * 4},
      {(void**)&h->sp.row0, spGP * E * 4}, {(void**)&h->sp.plan, 16},
      {(void**)&h->sp.pairs, h->sparse_ok ? size_t(h->sp.max_pairs) * sizeof(SparsePair) : 16},
      {(void**)&h->sp.ltok, spR * 4}, {(void**)&h->sp.lslot, spR * 4},
      {(void**)&h->sp.gatep, spR * 4}, {&h->sp.gate16p, spR * 64 * 2},
      {&h->sp.zp, h->sparse_ok ? spR * d.Ds * 2 : 16},
      {&h->sp.a2p, h->sparse_ok ? spR * d.H * 2 : 16},
      {(void**)&h->sp.ybuf,
       h->sparse_ok && d.top_k > 1 ? spGP * d.tpad * size_t(d.top_k) * d.Dt * 4 : 16},
      {&h->wkv, hs ? G * 2 * size_t(h->hd.Dt) * hs->act_tgt * 2 : 16},
      {&h->ahat, hs ? size_t(h->gp_h) * d.B * d.S * hs->act_tgt * 2 : 16},
      {(void**)&h->proj_layer, std::max<size_t>(G, 1) * 4},
      {&h->wg, G * E * d.Ds * es}, {(void**)&h->bg, G * E * 4},
      {&h->w1, G * EH * d.Ds * es}, {(void**)&h->b1, G * EH * 4}, {&h->b1h, G * EH * 2},
      {&h->w2, G * d.Dt * EH * es}, {(void**)&h->b2, G * E * d.Dt * 4},
      {(void**)&h->groups, std::max<size_t>(G, 1) * sizeof(GroupInfo)},
      {(void**)&h->gate, G * size_t(d.tpad) * E * 4},
      {&h->gate16, h->use_umma ? G * size_t(d.tpad) * 64 * 2 : 16},
      {&h->b2t, h->use_umma ? G * size_t(d.Dt) * 64 * 2 : 16},
      {&h->wg16, h->use_umma ? G * 16 * size_t(d.Ds) * 2 : 16},
      {&h->a2, size_t(h->gp_max) * per_group_a2},
      {(void**)&h->tiles, size_t(d.tiles_max) * sizeof(TileInfo)},
      {(void**)&h->n_tiles, 16}, {(void**)&h->status, 16},
      {(void**)&h->counters, fused_counter_ints(d, h->gp_max) * sizeof(int32_t)}};
  for (auto& a : allocs) {
    if (cudaMalloc(a.p, std::max<size_t>(a.n, 16)) != cudaSuccess) {
      cudaGetLastError();
      free_all(h);
      delete h;
      return MOT_ERR_OOM;
    }
  }
  if ((hs && G &&
       cudaMemcpy(h->proj_layer, proj_h.data(), G * 4, cudaMemcpyHostToDevice) != cudaSuccess) ||
      cudaMemset(h->status, 0, 16) != cudaSuccess || cudaMemset(h->n_tiles, 0, 16) != cudaSuccess ||
      (G && cudaMemcpy(h->groups, h->groups_h.data(), G * sizeof(GroupInfo),
                       cudaMemcpyHostToDevice) != cudaSuccess)) {
    cudaGetLastError();
    free_all(h);
    delete h;
    return MOT_ERR_CUDA;
  }
  if (h->use_umma && G) {
    bool ok = true;
    {  // W1cat: [G*EH rows][Ds], box 64 x 256
      const uint64_t dims[2] = {uint64_t(d.Ds), uint64_t(G * EH)};
      const uint64_t st_b[1] = {uint64_t(d.Ds) * 2};
      const uint32_t box[2] = {uint32_t(kUmmaK), uint32_t(kUmmaN)};
      ok = ok && encode_bf16(&h->tm_w1, h->w1, 2, dims, st_b, box);
      const uint32_t box_h[2] = {uint32_t(kUmmaK), uint32_t(kUmmaN / 2)};   // one CTA of a pair
      ok = ok && encode_bf16(&h->tm_w1h, h->w1, 2, dims, st_b, box_h);
      const uint32_t box_q[2] = {uint32_t(kUmmaK), 64};   // one CTA's half of a 128-row chunk
      ok = ok && encode_bf16(&h->tm_w1q, h->w1, 2, dims, st_b, box_q);
    }
    {  // W2cat: [G*Dt rows][EH], box 64 x 256
      const uint64_t dims[2] = {uint64_t(EH), uint64_t(G * d.Dt)};
      const uint64_t st_b[1] = {uint64_t(EH) * 2};
      const uint32_t box[2] = {uint32_t(kUmmaK), uint32_t(kUmmaN)};
      ok = ok && encode_bf16(&h->tm_w2, h->w2, 2, dims, st_b, box, /*f16=*/true);
      const uint32_t box_h[2] = {uint32_t(kUmmaK), uint32_t(kUmmaN / 2)};
      ok = ok && encode_bf16(&h->tm_w2h, h->w2, 2, dims, st_b, box_h, /*f16=*/true);
    }
    {  // A2: [gp][tpad][EH], box 64 x 128 x 1
      const uint64_t dims[3] = {uint64_t(EH), uint64_t(d.tpad), uint64_t(h->gp_max)};
      const uint64_t st_b[2] = {uint64_t(EH) * 2, uint64_t(d.tpad) * EH * 2};
      const uint32_t box[3] = {uint32_t(kUmmaK), uint32_t(kTileM), 1};
      ok = ok && encode_bf16(&h->tm_a2, h->a2, 3, dims, st_b, box, /*f16=*/true);
      const uint32_t box_st[3] = {32, 32, 1};   // one epilogue warp's 32 x 32 store tile
      ok = ok && encode_bf16(&h->tm_a2_st, h->a2, 3, dims, st_b, box_st, /*f16=*/true,
                             /*swizzle64=*/true);
    }
    {  // gate16: [G][tpad][64], box 64 x 128 x 1 (GEMM2's bias K block, A side)
      const uint64_t dims[3] = {64, uint64_t(d.tpad), uint64_t(G)};
      const uint64_t st_b[2] = {128, uint64_t(d.tpad) * 128};
      const uint32_t box[3] = {64, uint32_t(kTileM), 1};
      ok = ok && encode_bf16(&h->tm_g16, h->gate16, 3, dims, st_b, box, /*f16=*/true);
    }
    if (h->sparse_ok) {   // routed rows: zp [H_s * R][d_s], A2p [1][R][H], gate16p [1][R][64]
      const uint64_t R = uint64_t(h->sp.R);
      const uint64_t zd[2] = {uint64_t(d.d_s), uint64_t(d.H_s) * R};
      const uint64_t zs[1] = {uint64_t(d.d_s) * 2};
      const uint32_t zb[2] = {uint32_t(kUmmaK), uint32_t(kTileM)};
      ok = ok && encode_bf16(&h->tm_zp, h->sp.zp, 2, zd, zs, zb);
      const uint64_t ad[3] = {uint64_t(d.H), R, 1};
      const uint64_t as[2] = {uint64_t(d.H) * 2, R * d.H * 2};
      const uint32_t ab[3] = {uint32_t(kUmmaK), uint32_t(kTileM), 1}, ab_st[3] = {32, 32, 1};
      ok = ok && encode_bf16(&h->tm_a2p, h->sp.a2p, 3, ad, as, ab, /*f16=*/true);
      ok = ok && encode_bf16(&h->tm_a2p_st, h->sp.a2p, 3, ad, as, ab_st, /*f16=*/true,
                             /*swizzle64=*/true);
      const uint64_t gd[3] = {64, R, 1};
      const uint64_t gs[2] = {128, R * 128};
      const uint32_t gb[3] = {64, uint32_t(kTileM), 1};
      ok = ok && encode_bf16(&h->tm_g16p, h->sp.gate16p, 3, gd, gs, gb, /*f16=*/true);
    }
    if (hs) {   // MoT-h: [W^K; W^V] per layer [G * 2 D_t][d_at] and a_hat [gp_h * B * S][d_at]
      const uint64_t wd[2] = {uint64_t(hs->act_tgt), uint64_t(G) * 2 * h->hd.Dt};
      const uint64_t ws[1] = {uint64_t(hs->act_tgt) * 2};
      const uint32_t box[2] = {uint32_t(kUmmaK), uint32_t(kTileM)};
      ok = ok && encode_bf16(&h->tm_wkv, h->wkv, 2, wd, ws, box);
      const uint64_t ad[2] = {uint64_t(hs->act_tgt), uint64_t(h->gp_h) * d.B * d.S};
      ok = ok && encode_bf16(&h->tm_ahat, h->ahat, 2, ad, ws, box);
    }
    {  // wg16: [G * 16][Ds], box 64 x 16 (the gate MMA's B side)
      const uint64_t dims[2] = {uint64_t(d.Ds), uint64_t(G) * 16};
      const uint64_t st_b[1] = {uint64_t(d.Ds) * 2};
      const uint32_t box[2] = {uint32_t(kUmmaK), 16};
      ok = ok && encode_bf16(&h->tm_wg16, h->wg16, 2, dims, st_b, box);
    }
    {  // b2t: [G * Dt][64], boxes 64 x 256 and 64 x 128 (B side)
      const uint64_t dims[2] = {64, uint64_t(G * d.Dt)};
      const uint64_t st_b[1] = {128};
      const uint32_t box[2] = {64, uint32_t(kUmmaN)}, box_h[2] = {64, uint32_t(kUmmaN / 2)};
      ok = ok && encode_bf16(&h->tm_b2t, h->b2t, 2, dims, st_b, box, /*f16=*/true);
      ok = ok && encode_bf16(&h->tm_b2th, h->b2t, 2, dims, st_b, box_h, /*f16=*/true);
    }
    if (!ok) {
      free_all(h);
      delete h;
      return MOT_ERR_CUDA;
    }
  }
  *out = h;
  return MOT_OK;
}

}  // namespace

namespace {

// ---------------------------------------------------------------- backbone translators

float bf16_bits_to_float(uint16_t b) {
  const uint32_t u = uint32_t(b) << 16;
  float f;
  memcpy(&f, &u, 4);
  return f;
}

uint16_t float_to_bf16_bits(float f) {   // round to nearest even (finite values)
  uint32_t u;
  memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return static_cast<uint16_t>(u >> 16);
}

// Elements of one K/V block of the backbone blob (see include/mot.h).
size_t bt_block_elems(const BtDims& d) {
  const size_t ds = d.d_s, D = d.d, df = d.df, P = d.P, Dt = d.Dt;
  const size_t slot = 4 * D + 4 * (D * D + D) + 2 * D + (df * D + df) + (D * df + D);
  const size_t expert = 2 * ds + D * ds + D + size_t(d.N) * slot + 2 * P * D + Dt * P * D + Dt;
  return size_t(d.E) * d.N * d.Ds + d.E + d.E * expert;
}

mot_status bt_create(const mot_config* cfg, const mot_bt_config* bc, mot_handle* out) {
  if (!out) return MOT_ERR_INVALID_ARG;
  *out = nullptr;
  if (!cfg || !bc) return MOT_ERR_INVALID_ARG;
  const mot_config& c = *cfg;
  if (c.n_layers_src <= 0 || c.src_kv_heads <= 0 || c.src_head_dim <= 0 || c.n_layers_tgt <= 0 ||
      c.tgt_kv_heads <= 0 || c.tgt_head_dim <= 0 || c.n_translators <= 0 || c.max_batch <= 0 ||
      c.max_seq <= 0 || c.top_k < 0 || c.top_k > c.n_translators)
    return MOT_ERR_INVALID_ARG;
  if (bc->win_len <= 0 || bc->win_start < 0 || bc->win_start + bc->win_len > c.n_layers_tgt ||
      bc->width <= 0 || bc->heads <= 0 || bc->ffn <= 0 || bc->width % bc->heads)
    return MOT_ERR_INVALID_ARG;
  if (c.dtype != MOT_BF16 && c.dtype != MOT_FP32) return MOT_ERR_INVALID_ARG;
  std::vector<int32_t> map;
  if (c.layer_map) {
    for (int l = 0; l < c.n_layers_tgt; ++l)
      if (c.layer_map[l] < -1 || c.layer_map[l] >= c.n_layers_src) return MOT_ERR_INVALID_ARG;
    map.assign(c.layer_map, c.layer_map + c.n_layers_tgt);
  } else {
    depth_ratio(c.n_layers_src, c.n_layers_tgt, map);
  }
  if (c.dtype != MOT_BF16 || bc->win_len > kBtMaxSlots || c.max_batch > 4096)
    return MOT_ERR_UNSUPPORTED;
  for (int r = 0; r < bc->win_len; ++r)
    if (map[bc->win_start + r] < 0) return MOT_ERR_UNSUPPORTED;   // every window layer mapped

  BtDims bd{};
  bd.L_s = c.n_layers_src; bd.P = c.src_kv_heads; bd.d_s = c.src_head_dim;
  bd.L_t = c.n_layers_tgt; bd.H_t = c.tgt_kv_heads; bd.d_t = c.tgt_head_dim;
  bd.E = c.n_translators; bd.top_k = c.top_k; bd.B = c.max_batch; bd.S = c.max_seq;
  bd.Ds = bd.P * bd.d_s; bd.Dt = bd.H_t * bd.d_t;
  bd.N = bc->win_len; bd.q0 = bc->win_start; bd.d = bc->width; bd.na = bc->heads; bd.df = bc->ffn;
  bd.G = 2 * bd.E;
  bd.tau = 128 / std::max(bd.P, 1);
  bd.tiles_b = (bd.S + std::max(bd.tau, 1) - 1) / std::max(bd.tau, 1);
  bd.R = int64_t(bd.B) * bd.S * bd.P;
  if (!bt_supported(bd)) return MOT_ERR_UNSUPPORTED;
  // tensor-map row coordinates are 32-bit
  if (int64_t(bd.G) * bd.R > INT32_MAX / 2 ||
      int64_t(bd.L_s) * bd.B * bd.P > INT32_MAX / 2)
    return MOT_ERR_UNSUPPORTED;

  mot_ctx* h = new (std::nothrow) mot_ctx();
  if (!h) return MOT_ERR_OOM;
  h->bt = new (std::nothrow) BtState();
  if (!h->bt) {
    delete h;
    return MOT_ERR_OOM;
  }
  h->kind = 2;
  h->cfg = c;
  h->cfg.layer_map = nullptr;
  h->layer_map = map;
  Dims& d = h->d;   // the cache shapes, for the argument checks
  d.L_s = bd.L_s; d.H_s = bd.P; d.d_s = bd.d_s; d.L_t = bd.L_t; d.H_t = bd.H_t; d.d_t = bd.d_t;
  d.E = bd.E; d.top_k = bd.top_k; d.B = bd.B; d.S = bd.S; d.Ds = bd.Ds; d.Dt = bd.Dt;
  d.dtype = 0;
  BtState& bt = *h->bt;
  bt.d = bd;
  for (int r = 0; r < bd.N; ++r) bt.src_layer[r] = map[bd.q0 + r];

  int dev = 0, cc_major = 0, cc_minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&cc_major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&cc_minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess) {
    cudaGetLastError();
    free_all(h);
    delete h;
    return MOT_ERR_CUDA;
  }
  h->device = dev;
  if (cc_major != 10 || cc_minor != 3 || !encode_fn()) {
    free_all(h);
    delete h;
    return MOT_ERR_UNSUPPORTED;
  }
  h->use_umma = true;

  const size_t G = bd.G, N = bd.N, D = bd.d, df = bd.df, R = size_t(bd.R), E = bd.E;
  struct A { void** p; size_t n; } allocs[] = {
      {&bt.wg, 2 * E * N * bd.Ds * 2}, {(void**)&bt.bg, 2 * E * 4},
      {(void**)&bt.s_in, G * D * 4}, {(void**)&bt.c_in, G * D * 4},
      {(void**)&bt.c_q, G * N * D * 4}, {(void**)&bt.c_kv, G * N * 2 * D * 4},
      {(void**)&bt.c_o, G * N * D * 4}, {(void**)&bt.c_f1, G * N * df * 4},
      {(void**)&bt.c_f2, G * N * D * 4}, {(void**)&bt.c_out, G * bd.Dt * 4},
      {(void**)&bt.s_out, G * bd.Dt * 4}, {(void**)&bt.rstat, G * R * 8},
      {(void**)&bt.ln_q, G * N * 2 * D * 4}, {(void**)&bt.ln_c, G * N * 2 * D * 4},
      {(void**)&bt.ln_f, G * N * 2 * D * 4},
      {&bt.win, G * D * 2 * bd.d_s * 2}, {&bt.wq, G * N * D * D * 2}, {&bt.wkv, G * N * 2 * D * D * 2},
      {&bt.wo, G * N * D * D * 2}, {&bt.wf1, G * N * df * D * 2}, {&bt.wf2, G * N * D * df * 2},
      {&bt.wout, G * bd.Dt * bd.P * D * 2},
      {(void**)&bt.gate, 2 * size_t(bd.B) * bd.S * E * 4},
      {(void**)&bt.h, G * R * D * 4}, {(void**)&bt.ht, G * R * D * 4},
      {&bt.xz, G * R * D * 2}, {&bt.xq, G * R * D * 2}, {&bt.q, G * R * D * 2},
      {&bt.kv, G * R * 2 * D * 2}, {&bt.o, G * R * D * 2}, {&bt.xf, G * R * D * 2},
      {&bt.f, G * R * df * 2}, {&bt.xo, G * R * D * 2},
      {(void**)&bt.rcnt, 64 * 4}, {(void**)&bt.rlist, G * size_t(bd.B) * bd.S * 4},
      {(void**)&bt.rpre, (2 * G + 2) * 4},
      {&bt.xs, bd.top_k == 1 ? G * R * bd.d_s * 2 : 16},
      {(void**)&h->status, 16}};
  for (auto& a : allocs) {
    if (cudaMalloc(a.p, std::max<size_t>(a.n, 16)) != cudaSuccess) {
      cudaGetLastError();
      free_all(h);
      delete h;
      return MOT_ERR_OOM;
    }
  }
  if (cudaMemset(h->status, 0, 16) != cudaSuccess) {
    cudaGetLastError();
    free_all(h);
    delete h;
    return MOT_ERR_CUDA;
  }
  bool ok = true;
  auto map2 = [&](CUtensorMap* m, void* base, uint64_t inner, uint64_t rows, uint32_t box_rows) {
    const uint64_t dims[2] = {inner, rows};
    const uint64_t st_b[1] = {inner * 2};
    const uint32_t box[2] = {64, box_rows};
    ok = ok && encode_bf16(m, base, 2, dims, st_b, box);
  };
  // weights (B operands): box 64 x N-tile rows
  const uint32_t nt_f1 = df <= 256 ? uint32_t(df) : 256u;
  uint32_t nt_out = 256 / bd.E;
  nt_out -= nt_out % 32;
  while (nt_out > 32 && bd.Dt % nt_out) nt_out -= 32;
  map2(&bt.tm_win, bt.win, 2 * bd.d_s, G * D, uint32_t(D));
  map2(&bt.tm_wq, bt.wq, D, G * N * D, uint32_t(D));
  map2(&bt.tm_wkv, bt.wkv, D, G * N * 2 * D, uint32_t(2 * D));
  map2(&bt.tm_wo, bt.wo, D, G * N * D, uint32_t(D));
  map2(&bt.tm_wf1, bt.wf1, D, G * N * df, nt_f1);
  map2(&bt.tm_wf1c, bt.wf1, D, G * N * df, 128);   // 128-row chunks for the fused FFN
  map2(&bt.tm_wf2, bt.wf2, df, G * N * D, uint32_t(D));
  map2(&bt.tm_wout, bt.wout, uint64_t(bd.P) * D, G * bd.Dt, nt_out);
  // activations (A operands): box 64 x 128 rows
  map2(&bt.tm_xz, bt.xz, D, G * R, 128);
  map2(&bt.tm_xq, bt.xq, D, G * R, 128);
  map2(&bt.tm_o, bt.o, D, G * R, 128);
  map2(&bt.tm_xf, bt.xf, D, G * R, 128);
  map2(&bt.tm_f, bt.f, df, G * R, 128);
  map2(&bt.tm_xo, bt.xo, uint64_t(bd.P) * D, G * size_t(bd.B) * bd.S, 128);
  if (bd.top_k == 1) {   // Top-1 routing (the default for these handles): token buckets
    uint32_t nt_r = 256;
    while (nt_r > 32 && bd.Dt % nt_r) nt_r -= 32;
    map2(&bt.tm_wout_r, bt.wout, uint64_t(bd.P) * D, G * bd.Dt, nt_r);
    map2(&bt.tm_xs, bt.xs, bd.d_s, G * R, uint32_t(bd.tau * bd.P));
    h->routing = 1;
  }
  if (!ok) {
    free_all(h);
    delete h;
    return MOT_ERR_CUDA;
  }
  *out = h;
  return MOT_OK;
}

// Parse the backbone blob and upload it. LN_in and LN_out, whose inputs the
// GEMMs read raw (the source cache, the bf16 state rows), are folded into the
// map after them: for y = W LN(x) + b with LN(x) = gamma * xhat + beta,
// y = W' xhat + c with W' = W diag(gamma), c = b + W beta. W_in' is kept as two
// bf16 matrices hi + lo (hi = bf16(W'), lo = bf16(W' - hi)), so its product is
// exact to about 2^-17; W_out' is rounded to bf16 once. The other layer norms'
// gamma and beta are applied by the epilogues that write their rows, so W_Q,
// W_K, W_V and W_F1 stay the blob's values.
mot_status bt_load(mot_ctx* h, const void* host_blob, size_t bytes) {
  BtState& bt = *h->bt;
  const BtDims& d = bt.d;
  const size_t blk = bt_block_elems(d);
  if (bytes != 2 * blk * 2) return MOT_ERR_WEIGHTS_SIZE;
  if (cudaSetDevice(h->device) != cudaSuccess) return MOT_ERR_CUDA;
  const uint16_t* blob = static_cast<const uint16_t*>(host_blob);
  const size_t E = d.E, N = d.N, D = d.d, df = d.df, ds = d.d_s, P = d.P, Dt = d.Dt;
  const size_t G = d.G, WD = N * d.Ds;
  std::vector<uint16_t> wg(2 * E * WD), win(G * D * 2 * ds), wq(G * N * D * D),
      wkv(G * N * 2 * D * D), wo(G * N * D * D), wf1(G * N * df * D), wf2(G * N * D * df),
      wout(G * Dt * P * D);
  std::vector<float> bg(2 * E), s_in(G * D), c_in(G * D), c_q(G * N * D), c_kv(G * N * 2 * D),
      c_o(G * N * D), c_f1(G * N * df), c_f2(G * N * D), c_out(G * Dt), s_out(G * Dt),
      ln_q(G * N * 2 * D), ln_c(G * N * 2 * D), ln_f(G * N * 2 * D);
  auto f = [&](size_t i) { return double(bf16_bits_to_float(blob[i])); };
  // Folded rows: W'[n][k] = W[n][k] gamma[k] as hi (and lo, when w_lo is set)
  // with row stride `ld`; c[n] = b[n] + sum_k W[n][k] beta[k]; rowsum = sum of
  // the stored parts.
  auto fold = [&](size_t o_g, size_t o_w, size_t o_b, size_t n_out, size_t n_in, size_t ld,
                  uint16_t* w_hi, uint16_t* w_lo, float* c_dst, float* rowsum) {
    for (size_t n = 0; n < n_out; ++n) {
      double cb = f(o_b + n);
      double rs = 0.0;
      for (size_t k = 0; k < n_in; ++k) {
        const double w = f(o_w + n * n_in + k);
        const double wp = w * f(o_g + k);
        const uint16_t hi = float_to_bf16_bits(float(wp));
        w_hi[n * ld + k] = hi;
        rs += bf16_bits_to_float(hi);
        if (w_lo) {
          const uint16_t lo = float_to_bf16_bits(float(wp - bf16_bits_to_float(hi)));
          w_lo[n * ld + k] = lo;
          rs += bf16_bits_to_float(lo);
        }
        cb += w * f(o_g + n_in + k);
      }
      c_dst[n] = float(cb);
      if (rowsum) rowsum[n] = float(rs);
    }
  };
  auto copy = [&](size_t o_w, size_t o_b, size_t n_out, size_t n_in, uint16_t* w_dst, float* b_dst) {
    memcpy(w_dst, blob + o_w, n_out * n_in * 2);
    for (size_t n = 0; n < n_out; ++n) b_dst[n] = float(f(o_b + n));
  };
  auto ln = [&](size_t o_g, float* dst) {   // gamma[D], beta[D]
    for (size_t k = 0; k < 2 * D; ++k) dst[k] = float(f(o_g + k));
  };
  for (size_t x = 0; x < 2; ++x) {
    size_t off = x * blk;
    memcpy(&wg[x * E * WD], blob + off, E * WD * 2);
    off += E * WD;
    for (size_t m = 0; m < E; ++m) bg[x * E + m] = float(f(off + m));
    off += E;
    for (size_t m = 0; m < E; ++m) {
      const size_t g = x * E + m;
      const size_t o_lnin = off, o_win = o_lnin + 2 * ds, o_bin = o_win + D * ds;
      uint16_t* wi = &win[g * D * 2 * ds];
      fold(o_lnin, o_win, o_bin, D, ds, 2 * ds, wi, wi + ds, &c_in[g * D], &s_in[g * D]);
      off = o_bin + D;
      for (size_t r = 0; r < N; ++r) {
        const size_t gr = g * N + r;
        const size_t o_lnq = off, o_lnc = off + 2 * D, o_wq = off + 4 * D, o_bq = o_wq + D * D;
        const size_t o_wk = o_bq + D, o_bk = o_wk + D * D, o_wv = o_bk + D, o_bv = o_wv + D * D;
        const size_t o_wo = o_bv + D, o_bo = o_wo + D * D, o_lnf = o_bo + D;
        const size_t o_wf1 = o_lnf + 2 * D, o_bf1 = o_wf1 + df * D, o_wf2 = o_bf1 + df;
        const size_t o_bf2 = o_wf2 + D * df;
        ln(o_lnq, &ln_q[gr * 2 * D]);
        ln(o_lnc, &ln_c[gr * 2 * D]);
        ln(o_lnf, &ln_f[gr * 2 * D]);
        copy(o_wq, o_bq, D, D, &wq[gr * D * D], &c_q[gr * D]);
        copy(o_wk, o_bk, D, D, &wkv[gr * 2 * D * D], &c_kv[gr * 2 * D]);
        copy(o_wv, o_bv, D, D, &wkv[gr * 2 * D * D + D * D], &c_kv[gr * 2 * D + D]);
        copy(o_wo, o_bo, D, D, &wo[gr * D * D], &c_o[gr * D]);
        copy(o_wf1, o_bf1, df, D, &wf1[gr * df * D], &c_f1[gr * df]);
        copy(o_wf2, o_bf2, D, df, &wf2[gr * D * df], &c_f2[gr * D]);
        off = o_bf2 + D;
      }
      const size_t o_lnout = off, o_wout = o_lnout + 2 * P * D, o_bout = o_wout + Dt * P * D;
      fold(o_lnout, o_wout, o_bout, Dt, P * D, P * D, &wout[g * Dt * P * D], nullptr,
           &c_out[g * Dt], &s_out[g * Dt]);
      off = o_bout + Dt;
    }
    if (off != (x + 1) * blk) return MOT_ERR_WEIGHTS_SIZE;   // layout bookkeeping check
  }
  struct U { void* dst; const void* src; size_t n; } ups[] = {
      {bt.wg, wg.data(), wg.size() * 2}, {bt.bg, bg.data(), bg.size() * 4},
      {bt.win, win.data(), win.size() * 2}, {bt.s_in, s_in.data(), s_in.size() * 4},
      {bt.c_in, c_in.data(), c_in.size() * 4}, {bt.wq, wq.data(), wq.size() * 2},
      {bt.c_q, c_q.data(), c_q.size() * 4}, {bt.wkv, wkv.data(), wkv.size() * 2},
      {bt.c_kv, c_kv.data(), c_kv.size() * 4}, {bt.wo, wo.data(), wo.size() * 2},
      {bt.c_o, c_o.data(), c_o.size() * 4}, {bt.wf1, wf1.data(), wf1.size() * 2},
      {bt.c_f1, c_f1.data(), c_f1.size() * 4}, {bt.wf2, wf2.data(), wf2.size() * 2},
      {bt.c_f2, c_f2.data(), c_f2.size() * 4}, {bt.wout, wout.data(), wout.size() * 2},
      {bt.c_out, c_out.data(), c_out.size() * 4}, {bt.s_out, s_out.data(), s_out.size() * 4},
      {bt.ln_q, ln_q.data(), ln_q.size() * 4}, {bt.ln_c, ln_c.data(), ln_c.size() * 4},
      {bt.ln_f, ln_f.data(), ln_f.size() * 4}};
  for (auto& u : ups) MOT_CUDA_TRY(cudaMemcpy(u.dst, u.src, u.n, cudaMemcpyHostToDevice));
  MOT_CUDA_TRY(cudaDeviceSynchronize());
  h->weights_loaded = true;
  return MOT_OK;
}

}  // namespace

extern "C" {

mot_status mot_create(const mot_config* cfg, mot_handle* out) {
  return create_impl(cfg, nullptr, out);
}

mot_status mot_create_h(const mot_h_config* cfg, mot_handle* out) {
  if (!out) return MOT_ERR_INVALID_ARG;
  *out = nullptr;
  if (!cfg || cfg->src_act_dim <= 0 || cfg->tgt_act_dim <= 0 || cfg->tgt_kv_heads <= 0 ||
      cfg->tgt_head_dim <= 0)
    return MOT_ERR_INVALID_ARG;
  mot_config mc{};
  mc.n_layers_src = cfg->n_layers_src;
  mc.src_kv_heads = 1;
  mc.src_head_dim = cfg->src_act_dim;
  mc.n_layers_tgt = cfg->n_layers_tgt;
  mc.tgt_kv_heads = 1;
  mc.tgt_head_dim = cfg->tgt_act_dim;
  mc.n_translators = cfg->n_translators;
  mc.top_k = cfg->top_k;
  mc.hidden = cfg->hidden;
  mc.max_batch = cfg->max_batch;
  mc.max_seq = cfg->max_seq;
  mc.dtype = cfg->dtype;
  mc.layer_map = cfg->layer_map;
  if (mc.dtype != MOT_BF16) return MOT_ERR_UNSUPPORTED;
  const HSpec hs{cfg->tgt_act_dim, cfg->tgt_kv_heads, cfg->tgt_head_dim};
  return create_impl(&mc, &hs, out);
}

mot_status mot_load_weights(mot_handle h, const void* host_blob, size_t bytes) {
  if (!h || !host_blob) return MOT_ERR_INVALID_ARG;
  if (h->kind == 2) return bt_load(h, host_blob, bytes);
  const Dims& d = h->d;
  const size_t es = esize(d), gsz = group_elems(d);
  // MoT-h blocks: the mixture, then the layer's W^K and W^V [D_t][d_at]
  const size_t proj = h->kind == 1 ? 2 * size_t(h->hd.Dt) * h->act_tgt : 0;
  const size_t stride = gsz + proj;
  if (bytes != size_t(d.G) * stride * es) return MOT_ERR_WEIGHTS_SIZE;
  if (cudaSetDevice(h->device) != cudaSuccess) return MOT_ERR_CUDA;
  const size_t E = d.E, Ds = d.Ds, Dt = d.Dt, H = d.H, EH = d.EH;
  const char* blob = static_cast<const char*>(host_blob);
  auto to_f = [&](const char* p, size_t i) -> float {
    if (d.dtype == 1) {
      float f;
      memcpy(&f, p + 4 * i, 4);
      return f;
    }
    uint16_t b;
    memcpy(&b, p + 2 * i, 2);
    uint32_t u = uint32_t(b) << 16;
    float f;
    memcpy(&f, &u, 4);
    return f;
  };
  std::vector<float> bg(d.G * E), b1(d.G * EH), b2(d.G * E * Dt);
  char* wg = static_cast<char*>(h->wg);
  char* w1 = static_cast<char*>(h->w1);
  char* w2 = static_cast<char*>(h->w2);
  for (size_t g = 0; g < size_t(d.G); ++g) {
    const char* p = blob + g * stride * es;
    if (proj)
      MOT_CUDA_TRY(cudaMemcpy(static_cast<char*>(h->wkv) + g * proj * es, p + gsz * es,
                              proj * es, cudaMemcpyHostToDevice));
    size_t off = 0;
    MOT_CUDA_TRY(cudaMemcpy(wg + g * E * Ds * es, p, E * Ds * es, cudaMemcpyHostToDevice));
    off += E * Ds;
    for (size_t m = 0; m < E; ++m) bg[g * E + m] = to_f(p, off + m);
    off += E;
    for (size_t m = 0; m < E; ++m) {
      // W1_m -> rows [m*H, (m+1)*H) of W1cat
      MOT_CUDA_TRY(cudaMemcpy(w1 + (g * EH + m * H) * Ds * es, p + off * es, H * Ds * es,
                              cudaMemcpyHostToDevice));
      off += H * Ds;
      for (size_t j = 0; j < H; ++j) b1[g * EH + m * H + j] = to_f(p, off + j);
      off += H;
      // W2_m [Dt][H] -> columns [m*H, (m+1)*H) of W2cat [Dt][EH]
      MOT_CUDA_TRY(cudaMemcpy2D(w2 + (g * Dt * EH + m * H) * es, EH * es, p + off * es, H * es,
                                H * es, Dt, cudaMemcpyHostToDevice));
      off += Dt * H;
      for (size_t i = 0; i < Dt; ++i) b2[(g * E + m) * Dt + i] = to_f(p, off + i);
      off += Dt;
    }
  }
  if (d.G) {
    MOT_CUDA_TRY(cudaMemcpy(h->bg, bg.data(), bg.size() * 4, cudaMemcpyHostToDevice));
    MOT_CUDA_TRY(cudaMemcpy(h->b1, b1.data(), b1.size() * 4, cudaMemcpyHostToDevice));
    MOT_CUDA_TRY(cudaMemcpy(h->b2, b2.data(), b2.size() * 4, cudaMemcpyHostToDevice));
    if (h->use_umma) {
      // GEMM2 runs fp16 x fp16: W2 to fp16 in place, b1 copied to fp16
      MOT_CUDA_TRY(launch_bf16_to_f16_inplace(h->w2, size_t(d.G) * Dt * EH, 0));
      MOT_CUDA_TRY(launch_f32_to_f16(h->b1, h->b1h, b1.size(), 0));
      MOT_CUDA_TRY(launch_build_b2t(h->b2, h->b2t, d.G, d.E, d.Dt, 0));
      MOT_CUDA_TRY(launch_build_wg16(h->wg, h->wg16, d.G, d.E, d.Ds, 0));
    }
  }
  MOT_CUDA_TRY(cudaDeviceSynchronize());
  h->weights_loaded = true;
  return MOT_OK;
}

mot_status mot_translate(mot_handle h, const void* src_k, const void* src_v,
                         const int32_t* seq_lens, int32_t batch, void* dst_k, void* dst_v,
                         mot_stream_t stream) {
  NvtxRange range("mot_translate");
  mot_status s = check_translate_args(h, src_k, src_v, seq_lens, batch, dst_k, dst_v);
  if (s != MOT_OK) return s;
  return run_translate(h, src_k, src_v, seq_lens, batch, dst_k, dst_v,
                       reinterpret_cast<cudaStream_t>(stream), 0, h->d.G, true);
}

mot_status mot_translate_host(mot_handle h, const void* src_k, const void* src_v,
                              const int32_t* seq_lens, int32_t batch, void* dst_k, void* dst_v,
                              mot_stream_t stream) {
  NvtxRange range("mot_translate_host");
  if (!h || h->kind != 0) return MOT_ERR_INVALID_ARG;   // MoT-h handles: mot_translate_h
  if (batch < 0 || batch > h->d.B) return MOT_ERR_INVALID_ARG;
  if (!src_k || !src_v || !dst_k || !dst_v || (batch > 0 && !seq_lens)) return MOT_ERR_INVALID_ARG;
  if (!h->weights_loaded) return MOT_ERR_NO_WEIGHTS;
  const Dims& d = h->d;
  for (int b = 0; b < batch; ++b)
    if (seq_lens[b] < 0 || seq_lens[b] > d.S) return MOT_ERR_SEQ_LEN;
  if (batch == 0 || d.G == 0) return MOT_OK;
  if (!h->st_src[0]) {
    const size_t sb = src_bytes(d), db = dst_bytes(d);
    void** ps[5] = {&h->st_src[0], &h->st_src[1], &h->st_dst[0], &h->st_dst[1], (void**)&h->st_len};
    const size_t ns[5] = {sb, sb, db, db, size_t(d.B) * 4};
    for (int i = 0; i < 5; ++i)
      if (cudaMalloc(ps[i], ns[i]) != cudaSuccess) {
        cudaGetLastError();
        for (int k = 0; k < 5; ++k)
          if (*ps[k]) { cudaFree(*ps[k]); *ps[k] = nullptr; }
        return MOT_ERR_OOM;
      }
  }
  if (!h->copy_h2d) {
    if (cudaStreamCreateWithFlags(&h->copy_h2d, cudaStreamNonBlocking) != cudaSuccess ||
        cudaStreamCreateWithFlags(&h->copy_d2h, cudaStreamNonBlocking) != cudaSuccess) {
      cudaGetLastError();
      return MOT_ERR_CUDA;
    }
    for (auto* e : {&h->ev_prev_compute, &h->ev_prev_d2h})
      if (cudaEventCreateWithFlags(e, cudaEventDisableTiming) != cudaSuccess) return MOT_ERR_CUDA;
    for (int c = 0; c < kHostChunks; ++c)
      if (cudaEventCreateWithFlags(&h->ev_h2d[c], cudaEventDisableTiming) != cudaSuccess ||
          cudaEventCreateWithFlags(&h->ev_comp[c], cudaEventDisableTiming) != cudaSuccess)
        return MOT_ERR_CUDA;
    MOT_CUDA_TRY(cudaEventRecord(h->ev_prev_compute, h->copy_h2d));
    MOT_CUDA_TRY(cudaEventRecord(h->ev_prev_d2h, h->copy_d2h));
  }
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const size_t es = esize(d);
  // Pipeline over chunks of translated target layers: the copies of chunk c's
  // source layers (stream copy_h2d), the translation of chunk c (`stream`) and
  // the copies of chunk c's target layers back (stream copy_d2h) overlap with
  // the neighbouring chunks. Only real tokens (s < seq_len[b]) are copied.
  std::vector<int> tl;   // translated target layers, ascending (group 2r + x)
  for (int l = 0; l < d.L_t; ++l)
    if (h->layer_map[l] >= 0) tl.push_back(l);
  const int n_tl = static_cast<int>(tl.size());
  // chunk boundaries: the first and last chunks are small (1, then 2 layers),
  // so the pipeline fills and drains quickly; the middle chunks hold about 4
  // (more when there are more than 4 * (kHostChunks - 4) of them)
  std::vector<int> cb{0};
  if (n_tl <= 6) {
    for (int r = 1; r <= n_tl; ++r) cb.push_back(r);
  } else {
    cb.push_back(1);
    cb.push_back(3);
    const int mid = n_tl - 6, nm = std::min((mid + 3) / 4, kHostChunks - 4);
    for (int i = 1; i <= nm; ++i) cb.push_back(3 + i * mid / nm);
    cb.push_back(n_tl - 1);
    cb.push_back(n_tl);
  }
  const int nc = static_cast<int>(cb.size()) - 1;   // <= kHostChunks
  // the previous call's translation read the source staging and its copies
  // read the target staging: order this call after both
  MOT_CUDA_TRY(cudaStreamWaitEvent(h->copy_h2d, h->ev_prev_compute, 0));
  MOT_CUDA_TRY(cudaStreamWaitEvent(st, h->ev_prev_d2h, 0));
  MOT_CUDA_TRY(cudaMemcpyAsync(h->st_len, seq_lens, size_t(batch) * 4, cudaMemcpyHostToDevice, st));
  std::vector<char> copied(d.L_s, 0);
  for (int c = 0; c < nc; ++c) {
    const int r0 = cb[c], r1 = cb[c + 1];
    // source layers first needed by this chunk, copied in runs of consecutive layers
    std::vector<char> need(d.L_s, 0);
    for (int r = r0; r < r1; ++r) {
      const int ls = h->layer_map[tl[r]];
      if (!copied[ls]) need[ls] = copied[ls] = 1;
    }
    for (int l0 = 0; l0 < d.L_s;) {
      if (!need[l0]) { ++l0; continue; }
      int l1 = l0;
      while (l1 < d.L_s && need[l1]) ++l1;
      for (int x = 0; x < 2; ++x)
        MOT_CUDA_TRY(copy_real_rows(h->st_src[x], x ? src_v : src_k, l0, l1, d.B, d.H_s, d.S, d.d_s,
                                    es, seq_lens, batch, cudaMemcpyHostToDevice, h->copy_h2d));
      l0 = l1;
    }
    MOT_CUDA_TRY(cudaEventRecord(h->ev_h2d[c], h->copy_h2d));
    MOT_CUDA_TRY(cudaStreamWaitEvent(st, h->ev_h2d[c], 0));
    mot_status s = run_translate(h, h->st_src[0], h->st_src[1], h->st_len, batch, h->st_dst[0],
                                 h->st_dst[1], st, 2 * r0, 2 * r1, c == 0);
    if (s != MOT_OK) return s;
    MOT_CUDA_TRY(cudaEventRecord(h->ev_comp[c], st));
    MOT_CUDA_TRY(cudaStreamWaitEvent(h->copy_d2h, h->ev_comp[c], 0));
    // this chunk's target layers back, in runs of consecutive layers
    for (int r = r0; r < r1;) {
      int r2 = r + 1;
      while (r2 < r1 && tl[r2] == tl[r2 - 1] + 1) ++r2;
      for (int x = 0; x < 2; ++x)
        MOT_CUDA_TRY(copy_real_rows(x ? dst_v : dst_k, h->st_dst[x], tl[r], tl[r2 - 1] + 1, d.B,
                                    d.H_t, d.S, d.d_t, es, seq_lens, batch,
                                    cudaMemcpyDeviceToHost, h->copy_d2h));
      r = r2;
    }
  }
  MOT_CUDA_TRY(cudaEventRecord(h->ev_prev_compute, st));
  MOT_CUDA_TRY(cudaEventRecord(h->ev_prev_d2h, h->copy_d2h));
  // `stream` completes only after the last copy back
  MOT_CUDA_TRY(cudaStreamWaitEvent(st, h->ev_prev_d2h, 0));
  return MOT_OK;
}

mot_status mot_get_device_status(mot_handle h, mot_stream_t stream) {
  if (!h) return MOT_ERR_INVALID_ARG;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  MOT_CUDA_TRY(cudaStreamSynchronize(st));
  int32_t v = 0;
  MOT_CUDA_TRY(cudaMemcpy(&v, h->status, 4, cudaMemcpyDeviceToHost));
  MOT_CUDA_TRY(cudaMemset(h->status, 0, 4));
  if (v & kStatusTimeout) return MOT_ERR_TIMEOUT;
  if (v & kStatusSeqLen) return MOT_ERR_SEQ_LEN;
  return MOT_OK;
}

mot_status mot_destroy(mot_handle h) {
  if (!h) return MOT_ERR_INVALID_ARG;
  cudaSetDevice(h->device);
  cudaDeviceSynchronize();
  free_all(h);
  cudaGetLastError();
  delete h;
  return MOT_OK;
}

mot_status mot_get_layer_map(mot_handle h, int32_t* out, int32_t n) {
  if (!h || !out || n != h->d.L_t) return MOT_ERR_INVALID_ARG;
  for (int l = 0; l < n; ++l) out[l] = h->layer_map[l];
  return MOT_OK;
}

mot_status mot_get_path(mot_handle h, int32_t* path) {
  if (!h || !path) return MOT_ERR_INVALID_ARG;
  *path = h->use_umma ? 1 : 0;
  return MOT_OK;
}

mot_status mot_set_schedule(mot_handle h, int32_t schedule) {
  if (!h || schedule < 0 || schedule > 4) return MOT_ERR_INVALID_ARG;
  if (schedule == 3 && !(h->use_umma && onchip_supported(h->d))) return MOT_ERR_UNSUPPORTED;
  if (schedule == 4 && !(h->kind == 0 && h->use_umma && wide_supported(h->d)))
    return MOT_ERR_UNSUPPORTED;
  h->schedule = schedule;
  return MOT_OK;
}

mot_status mot_get_schedule(mot_handle h, int32_t* schedule) {
  if (!h || !schedule) return MOT_ERR_INVALID_ARG;
  *schedule = h->schedule;
  return MOT_OK;
}

mot_status mot_debug_set(mot_handle h, int32_t stall_test, int64_t wait_limit_cycles) {
  if (!h || stall_test < 0 || stall_test > 1 || wait_limit_cycles < 0) return MOT_ERR_INVALID_ARG;
  h->stall_test = stall_test;
  h->wait_limit = wait_limit_cycles > 0 ? wait_limit_cycles : 4000000000LL;
  return MOT_OK;
}

mot_status mot_debug_fixed_gate(mot_handle h, const float* gate) {
  if (!h || h->kind != 0) return MOT_ERR_INVALID_ARG;
  if (gate && (reinterpret_cast<uintptr_t>(gate) & 3u)) return MOT_ERR_INVALID_ARG;
  h->fixed_gate = gate;
  return MOT_OK;
}

mot_status mot_profile_enable(mot_handle h, int32_t enable) {
  if (!h) return MOT_ERR_INVALID_ARG;
  h->profile = enable != 0;
  return MOT_OK;
}

mot_status mot_profile_read(mot_handle h, mot_kernel_stat* out, int32_t cap, int32_t* n) {
  if (!h || !n || (cap > 0 && !out)) return MOT_ERR_INVALID_ARG;
  std::vector<mot_kernel_stat> stats(h->kind_names.size());
  for (size_t i = 0; i < stats.size(); ++i) {
    memset(&stats[i], 0, sizeof(mot_kernel_stat));
    strncpy(stats[i].name, h->kind_names[i].c_str(), sizeof(stats[i].name) - 1);
  }
  mot_status rs = MOT_OK;
  for (auto& e : h->ev_used) {
    float ms = 0.f;
    if (cudaEventSynchronize(e.b) != cudaSuccess || cudaEventElapsedTime(&ms, e.a, e.b) != cudaSuccess) {
      cudaGetLastError();
      rs = MOT_ERR_CUDA;
    }
    stats[e.kind].launches += 1;
    stats[e.kind].total_ms += ms;
    h->ev_free.push_back(e);
  }
  h->ev_used.clear();
  int32_t k = 0;
  for (size_t i = 0; i < stats.size(); ++i) {
    if (stats[i].launches == 0) continue;
    if (k < cap) out[k] = stats[i];
    ++k;
  }
  *n = std::min(k, cap);
  return rs;
}

mot_status mot_get_launch_count(mot_handle h, int64_t* count) {
  if (!h || !count) return MOT_ERR_INVALID_ARG;
  *count = h->launches;
  return MOT_OK;
}

mot_status mot_translate_h(mot_handle h, const void* src_act, const int32_t* seq_lens,
                           int32_t batch, void* dst_k, void* dst_v, mot_stream_t stream) {
  NvtxRange range("mot_translate_h");
  if (!h || h->kind != 1) return MOT_ERR_INVALID_ARG;
  const Dims& d = h->d;
  if (batch < 0 || batch > d.B) return MOT_ERR_INVALID_ARG;
  if (!src_act || !dst_k || !dst_v || (batch > 0 && !seq_lens)) return MOT_ERR_INVALID_ARG;
  if (!aligned16(src_act) || !aligned16(dst_k) || !aligned16(dst_v)) return MOT_ERR_INVALID_ARG;
  const size_t sb = src_bytes(d), db = dst_bytes(h->hd);
  if (overlap(dst_k, db, dst_v, db) || overlap(dst_k, db, src_act, sb) ||
      overlap(dst_v, db, src_act, sb))
    return MOT_ERR_INVALID_ARG;
  if (!h->weights_loaded) return MOT_ERR_NO_WEIGHTS;
  if (cudaSetDevice(h->device) != cudaSuccess) return MOT_ERR_CUDA;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (batch == 0 || d.G == 0) return MOT_OK;
  for (int g0 = 0; g0 < d.G; g0 += h->gp_h) {
    const int g1 = std::min(d.G, g0 + h->gp_h);
    // the mixture of this pass's layers into their a_hat slots
    mot_status r = run_translate(h, src_act, src_act, seq_lens, batch, h->ahat, h->ahat, st, g0,
                                 g1, g0 == 0);
    if (r != MOT_OK) return r;
    // K | V = a_hat [W^K; W^V]^T into the target caches
    PathArgs a = path_args(h);
    a.d = h->hd;
    a.dst[0] = dst_k;
    a.dst[1] = dst_v;
    a.proj_layer = h->proj_layer;
    a.g0 = g0;
    a.gp = g1 - g0;
    MOT_CUDA_TRY(timed(h, "umma2_proj", st, [&] {
      return launch_umma2_proj(a, h->tm_ahat, h->tm_wkv, h->act_tgt, h->num_sms, st);
    }));
  }
  return MOT_OK;
}

mot_status mot_create_bt(const mot_config* cfg, const mot_bt_config* bt, mot_handle* out) {
  return bt_create(cfg, bt, out);
}

mot_status mot_translate_bt(mot_handle h, const void* src_k, const void* src_v,
                            const int32_t* seq_lens, int32_t batch, void* dst_k, void* dst_v,
                            mot_stream_t stream) {
  NvtxRange range("mot_translate_bt");
  if (!h || h->kind != 2) return MOT_ERR_INVALID_ARG;
  const Dims& dd = h->d;
  if (batch < 0 || batch > dd.B) return MOT_ERR_INVALID_ARG;
  if (!src_k || !src_v || !dst_k || !dst_v || (batch > 0 && !seq_lens)) return MOT_ERR_INVALID_ARG;
  if (!aligned16(src_k) || !aligned16(src_v) || !aligned16(dst_k) || !aligned16(dst_v))
    return MOT_ERR_INVALID_ARG;
  const size_t sb = src_bytes(dd), db = dst_bytes(dd);
  if (overlap(dst_k, db, dst_v, db) || overlap(dst_k, db, src_k, sb) ||
      overlap(dst_k, db, src_v, sb) || overlap(dst_v, db, src_k, sb) ||
      overlap(dst_v, db, src_v, sb))
    return MOT_ERR_INVALID_ARG;
  if (!h->weights_loaded) return MOT_ERR_NO_WEIGHTS;
  if (cudaSetDevice(h->device) != cudaSuccess) return MOT_ERR_CUDA;
  if (batch == 0) return MOT_OK;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  BtState& bt = *h->bt;
  const BtDims& d = bt.d;
  BtArgs a{};
  a.d = d;
  a.src[0] = src_k;
  a.src[1] = src_v;
  a.dst[0] = dst_k;
  a.dst[1] = dst_v;
  a.seq_lens = seq_lens;
  a.batch = batch;
  for (int r = 0; r < d.N; ++r) a.src_layer[r] = bt.src_layer[r];
  a.wg = bt.wg; a.bg = bt.bg; a.s_in = bt.s_in; a.c_in = bt.c_in; a.c_q = bt.c_q;
  a.c_kv = bt.c_kv; a.c_o = bt.c_o; a.c_f1 = bt.c_f1; a.c_f2 = bt.c_f2; a.c_out = bt.c_out;
  a.s_out = bt.s_out; a.rstat = bt.rstat;
  a.ln_q = bt.ln_q; a.ln_c = bt.ln_c; a.ln_f = bt.ln_f;
  a.gate = bt.gate; a.xz = bt.xz; a.xq = bt.xq; a.h = bt.h; a.ht = bt.ht; a.q = bt.q;
  a.kv = bt.kv; a.o = bt.o; a.xf = bt.xf; a.f = bt.f; a.xo = bt.xo;
  a.status = h->status;
  a.wait_limit = h->wait_limit;
  // the source caches as 3-D tensors (d_s, S, L_s * B * H_s), box (64, tau, P)
  CUtensorMap tmK{}, tmV{};
  {
    const uint64_t dims[3] = {uint64_t(d.d_s), uint64_t(d.S), uint64_t(d.L_s) * d.B * d.P};
    const uint64_t st_b[2] = {uint64_t(d.d_s) * 2, uint64_t(d.S) * d.d_s * 2};
    const uint32_t box[3] = {64, uint32_t(d.tau), uint32_t(d.P)};
    if (!encode_bf16(&tmK, src_k, 3, dims, st_b, box) ||
        !encode_bf16(&tmV, src_v, 3, dims, st_b, box))
      return MOT_ERR_CUDA;
  }
  MOT_CUDA_TRY(timed(h, "bt_gate", st, [&] { return launch_bt_gate(a, st); }));
  // Top-1 routing: each backbone runs on its own tokens only (packed row spaces)
  const bool routed = h->routing == 1 && d.top_k == 1;
  if (routed) {
    a.routed = 1;
    a.cnt = bt.rcnt;
    a.list = bt.rlist;
    a.rpre = bt.rpre;
    a.xs = bt.xs;
    MOT_CUDA_TRY(timed(h, "bt_route", st, [&] {
      return launch_bt_route(a, bt.rcnt, bt.rlist, bt.rpre, st);
    }));
  }
  for (int r = 0; r < d.N; ++r) {
    a.slot = r;
    if (routed)
      MOT_CUDA_TRY(timed(h, "bt_pack", st, [&] { return launch_bt_pack(a, bt.xs, st); }));
    MOT_CUDA_TRY(timed(h, "bt_in_ln_gelu", st, [&] {
      return routed ? launch_bt_gemm(kBtIn, a, bt.tm_xs, bt.tm_xs, bt.tm_win, h->num_sms, st)
                    : launch_bt_gemm(kBtIn, a, tmK, tmV, bt.tm_win, h->num_sms, st);
    }));
    MOT_CUDA_TRY(timed(h, "bt_q", st, [&] {
      return launch_bt_gemm(kBtQ, a, bt.tm_xq, bt.tm_xq, bt.tm_wq, h->num_sms, st);
    }));
    MOT_CUDA_TRY(timed(h, "bt_kv", st, [&] {
      return launch_bt_gemm(kBtKV, a, bt.tm_xz, bt.tm_xz, bt.tm_wkv, h->num_sms, st);
    }));
    MOT_CUDA_TRY(timed(h, "bt_attn", st, [&] { return launch_bt_attn(a, st); }));
    MOT_CUDA_TRY(timed(h, "bt_o_residual_ln", st, [&] {
      return launch_bt_gemm(kBtO, a, bt.tm_o, bt.tm_o, bt.tm_wo, h->num_sms, st);
    }));
    if (d.df % 128 == 0) {   // FFN1, GELU and FFN2 with the hidden kept on the SM
      MOT_CUDA_TRY(timed(h, "bt_ffn_fused", st, [&] {
        return launch_bt_ffn(a, bt.tm_xf, bt.tm_wf1c, bt.tm_wf2, h->num_sms, st);
      }));
    } else {
      MOT_CUDA_TRY(timed(h, "bt_ffn1_gelu", st, [&] {
        return launch_bt_gemm(kBtF1, a, bt.tm_xf, bt.tm_xf, bt.tm_wf1, h->num_sms, st);
      }));
      MOT_CUDA_TRY(timed(h, "bt_ffn2_residual_ln", st, [&] {
        return launch_bt_gemm(kBtF2, a, bt.tm_f, bt.tm_f, bt.tm_wf2, h->num_sms, st);
      }));
    }
    MOT_CUDA_TRY(timed(h, "bt_out_gelu_combine", st, [&] {
      return launch_bt_gemm(kBtOut, a, bt.tm_xo, bt.tm_xo, routed ? bt.tm_wout_r : bt.tm_wout,
                            h->num_sms, st);
    }));
  }
  if (routed) h->counts_valid = true;
  return MOT_OK;
}

mot_status mot_create_replay(const mot_replay_config* cfg, mot_handle* out) {
  if (!out) return MOT_ERR_INVALID_ARG;
  *out = nullptr;
  if (!cfg || cfg->q_heads <= 0 || cfg->kv_heads <= 0 || cfg->head_dim <= 0 ||
      cfg->max_batch <= 0 || cfg->max_seq <= 0 || cfg->top_s <= 0 || cfg->n_full < 0 ||
      cfg->q_heads % cfg->kv_heads)
    return MOT_ERR_INVALID_ARG;
  ReplayDims rd{cfg->max_batch, cfg->max_seq, cfg->q_heads, cfg->kv_heads, cfg->head_dim,
                cfg->top_s, cfg->n_full};
  if (!replay_supported(rd) || int64_t(rd.B) * rd.N > INT32_MAX / 2) return MOT_ERR_UNSUPPORTED;
  mot_ctx* h = new (std::nothrow) mot_ctx();
  if (!h) return MOT_ERR_OOM;
  h->kind = 3;
  h->rd = rd;
  int dev = 0, cc_major = 0, cc_minor = 0;
  if (cudaGetDevice(&dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&h->num_sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&cc_major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
      cudaDeviceGetAttribute(&cc_minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess) {
    cudaGetLastError();
    delete h;
    return MOT_ERR_CUDA;
  }
  h->device = dev;
  if (cc_major != 10 || cc_minor != 3) {
    delete h;
    return MOT_ERR_UNSUPPORTED;
  }
  const size_t vt_bytes = replay_fmha_supported(rd) ? size_t(rd.B) * rd.Hkv * rd.d * rd.N * 2 : 16;
  if (cudaMalloc(&h->rsel, size_t(rd.B) * rd.N * rd.S * 4) != cudaSuccess ||
      cudaMalloc(&h->rvt, vt_bytes) != cudaSuccess ||
      cudaMalloc(&h->status, 16) != cudaSuccess || cudaMemset(h->status, 0, 16) != cudaSuccess) {
    cudaGetLastError();
    free_all(h);
    delete h;
    return MOT_ERR_OOM;
  }
  h->weights_loaded = true;   // nothing to load
  *out = h;
  return MOT_OK;
}

namespace {

mot_status replay_args(mot_handle h, const void* q, const void* k, const void* v,
                       const void* guide, const int32_t* seq_lens, int32_t batch, void* out,
                       bool need_qkv, ReplayArgs& a) {
  if (!h || h->kind != 3) return MOT_ERR_INVALID_ARG;
  const ReplayDims& d = h->rd;
  if (batch < 0 || batch > d.B || (batch > 0 && !seq_lens)) return MOT_ERR_INVALID_ARG;
  if (need_qkv && (!q || !k || !v || !out || !aligned16(q) || !aligned16(k) || !aligned16(v) ||
                   !aligned16(out)))
    return MOT_ERR_INVALID_ARG;
  if (need_qkv) {
    const size_t qb = size_t(d.B) * d.Hq * d.N * d.d * 2, kb = size_t(d.B) * d.Hkv * d.N * d.d * 2;
    if (overlap(out, qb, q, qb) || overlap(out, qb, k, kb) || overlap(out, qb, v, kb))
      return MOT_ERR_INVALID_ARG;
  }
  a = ReplayArgs{};
  a.d = d;
  a.q = q;
  a.k = k;
  a.v = v;
  a.guide = guide;
  a.out = out;
  a.sel = h->rsel;
  a.seq_lens = seq_lens;
  a.batch = batch;
  a.status = h->status;
  a.wait_limit = h->wait_limit;
  a.stall_test = h->stall_test;
  return MOT_OK;
}

}  // namespace

mot_status mot_replay_select(mot_handle h, const void* guide, const int32_t* seq_lens,
                             int32_t batch, int32_t* sel, mot_stream_t stream) {
  ReplayArgs a;
  mot_status r = replay_args(h, nullptr, nullptr, nullptr, guide, seq_lens, batch, nullptr,
                             false, a);
  if (r != MOT_OK) return r;
  if (!guide || !sel || !aligned16(guide)) return MOT_ERR_INVALID_ARG;
  if (cudaSetDevice(h->device) != cudaSuccess) return MOT_ERR_CUDA;
  if (batch == 0) return MOT_OK;
  a.sel = sel;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  MOT_CUDA_TRY(timed(h, "replay_select", st, [&] { return launch_replay_select(a, st); }));
  return MOT_OK;
}

mot_status mot_replay_attention(mot_handle h, int32_t layer, const void* q, const void* k,
                                const void* v, const void* guide, const int32_t* seq_lens,
                                int32_t batch, void* out, mot_stream_t stream) {
  NvtxRange range("mot_replay_attention");
  ReplayArgs a;
  mot_status r = replay_args(h, q, k, v, guide, seq_lens, batch, out, true, a);
  if (r != MOT_OK) return r;
  if (layer < 0) return MOT_ERR_INVALID_ARG;
  const bool full = layer < h->rd.n_full;
  if (!full && (!guide || !aligned16(guide))) return MOT_ERR_INVALID_ARG;
  if (cudaSetDevice(h->device) != cudaSuccess) return MOT_ERR_CUDA;
  if (batch == 0) return MOT_OK;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  a.full = full ? 1 : 0;
  const ReplayDims& d = h->rd;
  if (full && replay_fmha_supported(d) && encode_fn()) {
    // tensor-core causal attention: V^T first, then one launch over all query tiles
    CUtensorMap tmK{}, tmVt{};
    const uint64_t kd[2] = {uint64_t(d.d), uint64_t(d.B) * d.Hkv * d.N};
    const uint64_t vd[2] = {uint64_t(d.N), uint64_t(d.B) * d.Hkv * d.d};
    const uint64_t ks[1] = {uint64_t(d.d) * 2}, vs[1] = {uint64_t(d.N) * 2};
    const uint32_t box[2] = {64, 128}, vbox[2] = {64, uint32_t(d.d)};
    if (!encode_bf16(&tmK, k, 2, kd, ks, box) || !encode_bf16(&tmVt, h->rvt, 2, vd, vs, vbox))
      return MOT_ERR_CUDA;
    MOT_CUDA_TRY(timed(h, "replay_vt", st, [&] { return launch_replay_vt(a, h->rvt, st); }));
    MOT_CUDA_TRY(timed(h, "replay_fmha_full", st,
                       [&] { return launch_replay_fmha(a, tmK, tmVt, st); }));
    return MOT_OK;
  }
  if (!full && replay_gattn_supported(d)) {
    // guided layer on the tensor cores: selection, then the gathered-row attention
    MOT_CUDA_TRY(timed(h, "replay_select", st, [&] { return launch_replay_select(a, st); }));
    MOT_CUDA_TRY(timed(h, "replay_attn_sparse", st,
                       [&] { return launch_replay_gattn(a, h->num_sms, st); }));
    return MOT_OK;
  }
  if (!full)
    MOT_CUDA_TRY(timed(h, "replay_select", st, [&] { return launch_replay_select(a, st); }));
  MOT_CUDA_TRY(timed(h, full ? "replay_attn_full" : "replay_attn_sparse", st,
                     [&] { return launch_replay_attn(a, st); }));
  return MOT_OK;
}

mot_status mot_set_routing(mot_handle h, int32_t routing) {
  if (!h || routing < 0 || routing > 1) return MOT_ERR_INVALID_ARG;
  const bool bt_top1 = h->kind == 2 && h->bt && h->bt->d.top_k == 1;
  if (routing == 1 && !h->sparse_ok && !bt_top1) return MOT_ERR_UNSUPPORTED;
  h->routing = routing;
  return MOT_OK;
}

mot_status mot_get_routing(mot_handle h, int32_t* routing) {
  if (!h || !routing) return MOT_ERR_INVALID_ARG;
  *routing = h->routing;
  return MOT_OK;
}

mot_status mot_get_expert_counts(mot_handle h, int32_t* counts, int32_t n, mot_stream_t stream) {
  if (h && h->kind == 2 && h->bt) {   // backbone buckets: [2][E], block x then backbone
    if (!counts || n != h->bt->d.G) return MOT_ERR_INVALID_ARG;
    if (!(h->routing == 1 && h->bt->d.top_k == 1 && h->counts_valid)) return MOT_ERR_UNSUPPORTED;
    if (cudaSetDevice(h->device) != cudaSuccess) return MOT_ERR_CUDA;
    cudaStream_t st = static_cast<cudaStream_t>(stream);
    if (cudaMemcpyAsync(counts, h->bt->rcnt, size_t(n) * 4, cudaMemcpyDeviceToHost, st) !=
            cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess) {
      cudaGetLastError();
      return MOT_ERR_CUDA;
    }
    return MOT_OK;
  }
  if (!h || !counts || n != h->d.G * h->d.E) return MOT_ERR_INVALID_ARG;
  if (!(h->sparse_ok && h->routing == 1 && h->counts_valid)) return MOT_ERR_UNSUPPORTED;
  if (cudaSetDevice(h->device) != cudaSuccess) return MOT_ERR_CUDA;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (cudaMemcpyAsync(counts, h->sp.counts_all, size_t(n) * 4, cudaMemcpyDeviceToHost, st) !=
          cudaSuccess ||
      cudaStreamSynchronize(st) != cudaSuccess) {
    cudaGetLastError();
    return MOT_ERR_CUDA;
  }
  return MOT_OK;
}

mot_status mot_expert_usage(const int32_t* counts, int32_t n, double* cv2, double* entropy) {
  if (!counts || !cv2 || !entropy || n <= 0) return MOT_ERR_INVALID_ARG;
  double sum = 0.0;
  for (int32_t i = 0; i < n; ++i) {
    if (counts[i] < 0) return MOT_ERR_INVALID_ARG;
    sum += counts[i];
  }
  const double mean = sum / n;
  double var = 0.0;
  for (int32_t i = 0; i < n; ++i) var += (counts[i] - mean) * (counts[i] - mean);
  var /= n;
  *cv2 = mean > 0.0 ? var / (mean * mean) : 0.0;
  double h = 0.0;
  if (sum > 0.0)
    for (int32_t i = 0; i < n; ++i)
      if (counts[i] > 0) {
        const double p = counts[i] / sum;
        h -= p * std::log(p);
      }
  *entropy = h;
  return MOT_OK;
}

}  // extern "C"
