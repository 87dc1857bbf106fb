// Replay attention of the post-translation phase (App. C.4) on sm_103a:
// Top-S source-guided sparse attention, and full causal attention for the
// L_Full bottom layers.
//
//   replay_select_kernel  one warp per context row (b, u): the S positions j <= u
//                         with the largest guidance score A[b][u][j] (ties to the
//                         lower position), written in ascending order. It is exact
//                         integer work on the order-preserving 16-bit image of each
//                         score. The row is read once into shared memory as keys,
//                         with its key range; a 256-bin histogram of the top digit
//                         of (key - min), scaled to the row's range, and, when the
//                         range spans more than 256 keys, a histogram of the low bits in the
//                         chosen bin find the key V of the S-th largest (score,
//                         -position) and how many of the positions scoring V it
//                         takes; ballots then keep every score above V and the
//                         lowest positions at V. Rows with u + 1 <= S take every
//                         position. Rows past 4,096 positions take
//   replay_select_stream_kernel, the same selection with the high and low byte as
//                         the two digits, reading the row once per pass.
//   replay_attn_kernel    one warp per (b, key/value head, u), no block barriers:
//                         the query heads of the GQA group attend to the selected
//                         rows (sparse) or to positions 0..u in 128-key chunks
//                         with an online softmax (full). Each lane scores four keys
//                         of the chunk against every query of the group (16-byte
//                         key reads, the pre-scaled queries broadcast from the
//                         warp's shared copy), the softmax runs on warp shuffles in
//                         fp32, and each lane accumulates d / 32 output dimensions
//                         over the chunk's value rows (the warp reads each row
//                         once, coalesced).
//   replay_gattn_kernel   guided layers on the tensor cores (d = 128, S <= 128):
//                         every query head of a GQA group attends to the same
//                         selected rows, so one (b, key/value head, u) item is two
//                         small MMAs. A TMEM-allocating kernel runs one CTA per
//                         SM, so each persistent CTA holds 3 independent lanes of
//                         4 warps that run their items start to finish, while the
//                         SM overlaps the lanes: cp.async gathers of the selected
//                         key and value rows and the group's query rows into
//                         128B-swizzled tiles; S^T = K_sel Q^T (M = 128 keys,
//                         N = 16 heads); per-quarter maxima (redux.sync) traded
//                         through shared memory, P as bf16 into a swizzled tile,
//                         its row sums as exact fixed-point integer reductions;
//                         O^T = V_sel^T P^T (M = 128 dims, the value rows read
//                         MN-major); normalised rows out. Lanes synchronise on
//                         their own named barriers only.
//   replay_fmha_kernel    full causal attention on the tensor cores (layers below
//                         L_Full): one CTA per (b, query head, 128-query tile),
//                         persistent over its key tiles 0..diagonal.
//                           warp 0  TMA: K and V^T tiles (V transposed per layer by
//                                   replay_vt_kernel so both MMAs read K-major
//                                   operands) into 3 stages;
//                           warp 1  S_j = Q K_j^T (M=128, N=128 keys) into double-
//                                   buffered TMEM, up to two key tiles ahead, and
//                                   O += P_j V_j (M=128, N=d + 16) accumulated in
//                                   TMEM; both MMAs take their A operand (Q, P)
//                                   from TMEM. A row of ones below V^T's d rows
//                                   makes column d of O the row's sum of the very
//                                   bf16 probabilities the MMA uses;
//                           warps 4..19 four threads per query row, each a quarter
//                                   of its keys and of its output columns: the
//                                   query row into TMEM once, then per key tile the
//                                   scaled, masked scores from TMEM, the row's
//                                   running max (the quarters' maxima traded through
//                                   shared memory; base-2 exponentials on
//                                   ex2.approx), P as bf16 pairs written back over
//                                   the scores' TMEM columns. The running max rises
//                                   only when a tile's max exceeds it by more than
//                                   2^8, and only then are the O row and its sum in
//                                   TMEM rescaled; O is read from TMEM once, at the end.
//                         Every wait is bounded; on a timeout the roles unwind,
//                         copies and MMAs in flight are drained and TMEM is freed.
#include <cuda_bf16.h>

#include "replay_internal.h"
#include "ptx.cuh"

namespace mot {
namespace {


__device__ __forceinline__ float bf16f(uint16_t b) { return __uint_as_float(uint32_t(b) << 16); }

// 2^x on the special-function unit (PTX ex2.approx.ftz: relative error about 2^-22, results
// below the normal range flushed to 0), for the softmax probabilities that are then rounded
// to bf16.
__device__ __forceinline__ float ex2_fast(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&v);
}

// Order-preserving map of bf16 bits to unsigned 16-bit: larger value -> larger key.
__device__ __forceinline__ uint32_t ord16(uint16_t b) {
  return (b & 0x8000u) ? (~uint32_t(b) & 0xFFFFu) : (uint32_t(b) | 0x8000u);
}

__device__ __forceinline__ int seq_len_of(const ReplayArgs& a, int b) {
  if (b >= a.batch) return 0;
  const int L = a.seq_lens[b];
  return L < 0 ? 0 : (L > a.d.N ? a.d.N : L);
}

constexpr int kSelWarps = 8;         // rows per CTA, one warp each
constexpr int kSelCopies = 4;        // histogram copies per warp

// Warp-wide exclusive prefix of v (and the warp total).
__device__ __forceinline__ int warp_excl_scan(int v, int& total) {
  const int lane = threadIdx.x & 31;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  total = __shfl_sync(0xffffffffu, x, 31);
  return x - v;
}

// The bin of a warp's histogram (C copies of 256 bins) that holds the
// k-th largest counted key, scanning from bin 255 down: lane 0 sums the top 8
// bins, lane 31 the bottom 8. On return k is the rank left inside that bin.
template <int C = kSelCopies>
__device__ __forceinline__ uint32_t kth_bin(const int (*h)[256], int& k) {
  const int lane = threadIdx.x & 31;
  int c[8], t = 0;
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    c[e] = 0;
#pragma unroll
    for (int cp = 0; cp < C; ++cp) c[e] += h[cp][(31 - lane) * 8 + (7 - e)];
    t += c[e];
  }
  int tot;
  const int before = warp_excl_scan(t, tot);
  int found = -1, krem = 0, acc = before;
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    if (found < 0 && acc + c[e] >= k) {
      found = (31 - lane) * 8 + (7 - e);
      krem = k - acc;
    }
    acc += c[e];
  }
  const int src = __ffs(__ballot_sync(0xffffffffu, found >= 0)) - 1;
  k = __shfl_sync(0xffffffffu, krem, src);
  return uint32_t(__shfl_sync(0xffffffffu, found, src));
}

// Order-preserving keys of two bf16 scores packed in a word (low half first):
// a negative score's bits are inverted, a positive score's sign bit is set.
__device__ __forceinline__ uint32_t ord16x2(uint32_t q) {
  return q ^ ((((q >> 15) & 0x00010001u) * 0xFFFFu) | 0x80008000u);
}

// Selection for any max_seq. One warp per context row (b, u). With o = the
// order-preserving 16 bits of a score, the S-th largest (o, -j) key is found in
// two histogram passes over o (high byte, then low byte): V = its score bits, k =
// how many positions with o == V it takes. The selection is then every o > V plus
// the k lowest positions with o == V, compacted in ascending order by warp scans.
// Each lane reads 8 consecutive scores per step (16-byte loads when max_seq % 8
// == 0); every pass reads the row again.
__global__ void __launch_bounds__(32 * kSelWarps) replay_select_stream_kernel(const ReplayArgs a) {
  __shared__ int hist[kSelWarps][kSelCopies][256];   // copy lane % kSelCopies: fewer same-bin collisions
  const ReplayDims& d = a.d;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = blockIdx.x * kSelWarps + w;
  if (row >= d.B * d.N) return;
  const int b = row / d.N, u = row - b * d.N;
  if (u >= seq_len_of(a, b)) return;
  int32_t* out = a.sel + int64_t(row) * d.S;
  const int n = u + 1;
  if (n <= d.S) {
    for (int j = lane; j < d.S; j += 32) out[j] = j < n ? j : -1;
    return;
  }
  const uint16_t* A = static_cast<const uint16_t*>(a.guide) + int64_t(row) * d.N;
  const bool vec = (d.N & 7) == 0;   // then every 8-score group of the row is 16-byte aligned
  // the 8 order-preserving scores at positions j8 .. j8 + 7 (0 past n; never counted)
  auto load8 = [&](int j8, uint32_t (&o)[8]) {
    if (vec) {
      const uint4 q = __ldg(reinterpret_cast<const uint4*>(A + j8));
      const uint32_t qq[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        o[2 * e] = ord16(qq[e] & 0xFFFFu);
        o[2 * e + 1] = ord16(qq[e] >> 16);
      }
    } else {
#pragma unroll
      for (int e = 0; e < 8; ++e) o[e] = j8 + e < n ? ord16(__ldg(A + j8 + e)) : 0u;
    }
  };
  int* hw = hist[w][lane % kSelCopies];
  int k = d.S;
  uint32_t hi = 0, V = 0;
  for (int pass = 0; pass < 2; ++pass) {
    for (int i = lane; i < kSelCopies * 256; i += 32) hist[w][0][i] = 0;
    __syncwarp();
    for (int j8 = lane * 8; j8 - lane * 8 < n; j8 += 256) {   // warp-uniform trip count
      uint32_t o[8];
      if (j8 < n) load8(j8, o);
      if (pass == 0) {
#pragma unroll
        for (int e = 0; e < 8; ++e)
          if (j8 + e < n) atomicAdd(&hw[o[e] >> 8], 1);
      } else {
        // only the scores in bin `hi` count, spread over 256 low bytes
#pragma unroll
        for (int e = 0; e < 8; ++e)
          if (j8 + e < n && (o[e] >> 8) == hi) atomicAdd(&hw[o[e] & 0xFFu], 1);
      }
    }
    __syncwarp();
    const uint32_t bin = kth_bin(hist[w], k);
    if (pass == 0)
      hi = bin;
    else
      V = (hi << 8) | bin;   // k: positions with o == V to take, lowest first
    __syncwarp();
  }
  // compaction in ascending position order, 256 positions per round
  int base = 0, eq_taken = 0;
  for (int j8 = lane * 8; j8 - lane * 8 < n; j8 += 256) {
    uint32_t o[8];
    if (j8 < n) load8(j8, o);
    int n_eq = 0;
#pragma unroll
    for (int e = 0; e < 8; ++e) n_eq += (j8 + e < n && o[e] == V);
    int eq_tot;
    int eq_rank = eq_taken + warp_excl_scan(n_eq, eq_tot);
    bool sel[8];
    int n_sel = 0;
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const bool in = j8 + e < n;
      const bool eq = in && o[e] == V;
      sel[e] = in && (o[e] > V || (eq && eq_rank < k));
      eq_rank += eq;
      n_sel += sel[e];
    }
    int sel_tot;
    int pos = base + warp_excl_scan(n_sel, sel_tot);
#pragma unroll
    for (int e = 0; e < 8; ++e)
      if (sel[e]) out[pos++] = j8 + e;
    base += sel_tot;
    eq_taken += eq_tot;
  }
}

// Selection for max_seq <= 4096, with the row's keys cached in shared memory.
// One warp per context row (b, u): the row is read once and turned into
// order-preserving keys o (lane L holds positions 256 r + 8 L + e, as one 16-byte
// word of packed keys per round r), together with its key range [omin, omax].
// The S-th largest (o, -j) key is then found by a radix selection over o - omin:
// a 256-bin histogram of the top digit (o - omin) >> sh, sh the smallest shift
// that fits the row's range into 256 bins, then, when sh > 0, a histogram of the
// low sh bits among the keys of the chosen bin. That gives V, the threshold key,
// and k, how many positions with o == V are taken. The compaction keeps every
// o > V and the k lowest positions with o == V, in ascending order. The digits
// follow the row's own range, so increments spread over many bins even when the
// scores share a few binades.
constexpr int kSelCacheWarps = 4;    // rows per CTA
constexpr int kSelCacheRounds = 16;  // 256-position rounds cached per row: max_seq <= 4096
constexpr int kSelCacheCopies = 1;   // histogram copies per warp (36 KB per CTA: 6 CTAs per SM)

__global__ void __launch_bounds__(32 * kSelCacheWarps) replay_select_kernel(const ReplayArgs a) {
  __shared__ int hist[kSelCacheWarps][kSelCacheCopies][256];   // copy lane % kSelCacheCopies
  __shared__ uint4 keys[kSelCacheWarps][kSelCacheRounds][32];
  const ReplayDims& d = a.d;
  const int w = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int row = blockIdx.x * kSelCacheWarps + w;
  if (row >= d.B * d.N) return;
  const int b = row / d.N, u = row - b * d.N;
  if (u >= seq_len_of(a, b)) return;
  int32_t* out = a.sel + int64_t(row) * d.S;
  const int n = u + 1;
  if (n <= d.S) {
    for (int j = lane; j < d.S; j += 32) out[j] = j < n ? j : -1;
    return;
  }
  const uint16_t* A = static_cast<const uint16_t*>(a.guide) + int64_t(row) * d.N;
  const bool vec = (d.N & 7) == 0;   // then every 8-score group of the row is 16-byte aligned
  const int nr = (n + 255) >> 8;     // rounds holding positions < n (<= kSelCacheRounds)
  uint4 (*kc)[32] = keys[w];
  uint32_t lo = 0xFFFFu, hi = 0u;
  // Rounds r < nfull hold n's positions on every lane (no per-position test there).
  const int nfull = n >> 8;
  int r0 = 0;
  if (vec) {
    uint32_t lo1 = 0xFFFFu, hi1 = 0u;
#pragma unroll 4
    for (; r0 < nfull; ++r0) {
      const uint4 v = __ldg(reinterpret_cast<const uint4*>(A + r0 * 256 + lane * 8));
      const uint32_t q[4] = {ord16x2(v.x), ord16x2(v.y), ord16x2(v.z), ord16x2(v.w)};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        lo = min(lo, q[i] & 0xFFFFu);
        hi = max(hi, q[i] & 0xFFFFu);
        lo1 = min(lo1, q[i] >> 16);
        hi1 = max(hi1, q[i] >> 16);
      }
      kc[r0][lane] = make_uint4(q[0], q[1], q[2], q[3]);
    }
    lo = min(lo, lo1);
    hi = max(hi, hi1);
  }
#pragma unroll 4
  for (int r = r0; r < nr; ++r) {
    const int j8 = r * 256 + lane * 8;
    const int lim = min(n - j8, 8);   // this lane's positions < n in the round (may be <= 0)
    uint32_t q[4] = {0u, 0u, 0u, 0u};
    if (lim > 0) {
      if (vec) {
        const uint4 v = __ldg(reinterpret_cast<const uint4*>(A + j8));
        q[0] = v.x;
        q[1] = v.y;
        q[2] = v.z;
        q[3] = v.w;
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e)
          if (e < lim) q[e >> 1] |= uint32_t(__ldg(A + j8 + e)) << (16 * (e & 1));
      }
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      q[i] = ord16x2(q[i]);
      const uint32_t o0 = q[i] & 0xFFFFu, o1 = q[i] >> 16;
      if (2 * i < lim) {
        lo = min(lo, o0);
        hi = max(hi, o0);
      }
      if (2 * i + 1 < lim) {
        lo = min(lo, o1);
        hi = max(hi, o1);
      }
    }
    kc[r][lane] = make_uint4(q[0], q[1], q[2], q[3]);
  }
  const uint32_t omin = __reduce_min_sync(0xffffffffu, lo);
  const uint32_t range = __reduce_max_sync(0xffffffffu, hi) - omin;   // < 65536
  const int sh = range > 255u ? 24 - __clz(range) : 0;   // (range >> sh) <= 255, sh <= 8
  int* hw = hist[w][lane % kSelCacheCopies];
  int k = d.S;
  // key e (0..7) of a lane's 16-byte word
  auto key_of = [](const uint4& v, int e) -> uint32_t {
    const uint32_t x = e < 2 ? v.x : e < 4 ? v.y : e < 6 ? v.z : v.w;
    return (e & 1) ? x >> 16 : x & 0xFFFFu;
  };
  // Every key is at least omin, so subtracting omin from both halves of a packed word
  // borrows nothing across them: each half holds its own o - omin.
  const uint32_t omin2 = omin * 0x10001u;
  // top digit
  for (int i = lane; i < kSelCacheCopies * 256; i += 32) hist[w][0][i] = 0;
  __syncwarp();
  for (int r = 0; r < nfull; ++r) {
    const uint4 v = kc[r][lane];
    const uint32_t wd[4] = {v.x - omin2, v.y - omin2, v.z - omin2, v.w - omin2};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      atomicAdd(&hw[(wd[i] & 0xFFFFu) >> sh], 1);
      atomicAdd(&hw[wd[i] >> (16 + sh)], 1);
    }
  }
  if (nfull < nr) {
    const int lim = min(n - (nfull * 256 + lane * 8), 8);
    const uint4 v = kc[nfull][lane];
#pragma unroll
    for (int e = 0; e < 8; ++e)
      if (e < lim) atomicAdd(&hw[(key_of(v, e) - omin) >> sh], 1);
  }
  __syncwarp();
  const uint32_t top = kth_bin<kSelCacheCopies>(hist[w], k);
  uint32_t V = omin + (top << sh);
  if (sh > 0) {   // the low sh bits among the keys of bin `top`: o - omin in [top << sh, + 2^sh)
    __syncwarp();
    for (int i = lane; i < kSelCacheCopies * 256; i += 32) hist[w][0][i] = 0;
    __syncwarp();
    const uint32_t msk = (1u << sh) - 1u, lo_b = top << sh;
    for (int r = 0; r < nfull; ++r) {
      const uint4 v = kc[r][lane];
      const uint32_t wd[4] = {v.x - omin2, v.y - omin2, v.z - omin2, v.w - omin2};
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const uint32_t a = wd[i] & 0xFFFFu, c = wd[i] >> 16;
        if (a - lo_b <= msk) atomicAdd(&hw[a & msk], 1);
        if (c - lo_b <= msk) atomicAdd(&hw[c & msk], 1);
      }
    }
    if (nfull < nr) {
      const int lim = min(n - (nfull * 256 + lane * 8), 8);
      const uint4 v = kc[nfull][lane];
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        const uint32_t o = key_of(v, e) - omin;
        if (e < lim && (o >> sh) == top) atomicAdd(&hw[o & msk], 1);
      }
    }
    __syncwarp();
    V += kth_bin<kSelCacheCopies>(hist[w], k);
  }
  // compaction in ascending position order; bit e of a lane's masks is position 256 r + 8 lane + e
  int base = 0, eq_taken = 0;
  for (int r = 0; r < nr && base < d.S; ++r) {   // warp-uniform
    const int j8 = r * 256 + lane * 8;
    const uint4 v = kc[r][lane];
    uint32_t gt = 0u, eq = 0u;
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      const uint32_t o = key_of(v, e);
      gt |= uint32_t(o > V) << e;
      eq |= uint32_t(o == V) << e;
    }
    if (r == nfull) {   // the partial round: positions past n never count
      const int lim = min(n - j8, 8);
      const uint32_t in = lim <= 0 ? 0u : (1u << lim) - 1u;
      gt &= in;
      eq &= in;
    }
    uint32_t sel = gt;
    if (__any_sync(0xffffffffu, eq != 0u)) {   // the k lowest positions at the threshold are taken
      int eq_tot;
      int take = k - (eq_taken + warp_excl_scan(__popc(eq), eq_tot));
      for (uint32_t m = eq; m != 0u && take > 0; m &= m - 1u, --take) sel |= m & (0u - m);
      eq_taken += eq_tot;
    }
    int sel_tot;
    int pos = base + warp_excl_scan(__popc(sel), sel_tot);
    for (uint32_t m = sel; m != 0u; m &= m - 1u) out[pos++] = j8 + __ffs(m) - 1;
    base += sel_tot;
  }
}

constexpr int kAttnWarps = 4;   // (b, key/value head, u) items per CTA, one warp each

// Shared memory of one warp: the group's pre-scaled queries [G][D], the chunk's
// probabilities [G][128] and its key positions [128].
template <int D, int G>
__host__ __device__ constexpr int attn_warp_floats() { return G * D + G * 128 + 128; }

// Residency floor per group size: the gathers are latency-bound, so small groups
// trade a few spilled registers for more resident warps.
__host__ __device__ constexpr int attn_min_blocks(int g) { return g <= 8 ? 4 : 1; }

template <int D, int G>
__global__ void __launch_bounds__(32 * kAttnWarps, attn_min_blocks(G))
    replay_attn_kernel(const ReplayArgs a) {
  constexpr int DL = D / 32;   // output dimensions per lane
  extern __shared__ float4 attn_smem4[];
  const ReplayDims& d = a.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t item = int64_t(blockIdx.x) * kAttnWarps + warp;
  if (item >= int64_t(d.B) * d.Hkv * d.N) return;
  const int u = static_cast<int>(item % d.N);
  const int bh = static_cast<int>(item / d.N);
  const int hk = bh % d.Hkv, b = bh / d.Hkv;
  if (u >= seq_len_of(a, b)) return;
  float* ws = reinterpret_cast<float*>(attn_smem4) + warp * attn_warp_floats<D, G>();
  float* qs = ws;                        // [G][D]
  float* ps = ws + G * D;                // [G][128]
  int32_t* ix = reinterpret_cast<int32_t*>(ps + G * 128);   // [128]
  const float scale = rsqrtf(float(D));
  for (int i = lane; i < G * D; i += 32) {
    const int g = i / D, c = i - g * D;
    qs[i] = bf16f(static_cast<const uint16_t*>(a.q)[((int64_t(b) * d.Hq + hk * G + g) * d.N + u) * D + c]) *
            scale;
  }
  const bool full = a.full != 0;
  const int n_keys = full ? u + 1 : min(d.S, u + 1);
  const int32_t* sel = a.sel + (int64_t(b) * d.N + u) * d.S;
  const uint16_t* kb = static_cast<const uint16_t*>(a.k) + (int64_t(b) * d.Hkv + hk) * d.N * D;
  const uint16_t* vb = static_cast<const uint16_t*>(a.v) + (int64_t(b) * d.Hkv + hk) * d.N * D;
  float m[G], l[G], acc[G][DL];
#pragma unroll
  for (int g = 0; g < G; ++g) {
    m[g] = -INFINITY;
    l[g] = 0.f;
#pragma unroll
    for (int e = 0; e < DL; ++e) acc[g][e] = 0.f;
  }
  __syncwarp();
  for (int c0 = 0; c0 < n_keys; c0 += 128) {
    const int nc = min(128, n_keys - c0);
    // this lane's keys: chunk positions lane, lane + 32, lane + 64, lane + 96
    int j[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int t = lane + 32 * i;
      j[i] = t < nc ? (full ? c0 + t : sel[c0 + t]) : -1;
      ix[t] = j[i];
    }
    float s[4][G];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
      for (int g = 0; g < G; ++g) s[i][g] = 0.f;
#pragma unroll 2
    for (int c = 0; c < D / 8; ++c) {
      float kf[4][8];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        uint4 w = make_uint4(0u, 0u, 0u, 0u);
        if (j[i] >= 0) w = __ldg(reinterpret_cast<const uint4*>(kb + int64_t(j[i]) * D) + c);
        kf[i][0] = __uint_as_float(w.x << 16); kf[i][1] = __uint_as_float(w.x & 0xFFFF0000u);
        kf[i][2] = __uint_as_float(w.y << 16); kf[i][3] = __uint_as_float(w.y & 0xFFFF0000u);
        kf[i][4] = __uint_as_float(w.z << 16); kf[i][5] = __uint_as_float(w.z & 0xFFFF0000u);
        kf[i][6] = __uint_as_float(w.w << 16); kf[i][7] = __uint_as_float(w.w & 0xFFFF0000u);
      }
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const float4 q0 = *reinterpret_cast<const float4*>(qs + g * D + 8 * c);
        const float4 q1 = *reinterpret_cast<const float4*>(qs + g * D + 8 * c + 4);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          float x = s[i][g];
          x = fmaf(q0.x, kf[i][0], x); x = fmaf(q0.y, kf[i][1], x);
          x = fmaf(q0.z, kf[i][2], x); x = fmaf(q0.w, kf[i][3], x);
          x = fmaf(q1.x, kf[i][4], x); x = fmaf(q1.y, kf[i][5], x);
          x = fmaf(q1.z, kf[i][6], x); x = fmaf(q1.w, kf[i][7], x);
          s[i][g] = x;
        }
      }
    }
    // online softmax per query of the group (warp reductions only)
#pragma unroll
    for (int g = 0; g < G; ++g) {
      float mx = -INFINITY;
#pragma unroll
      for (int i = 0; i < 4; ++i)
        if (j[i] >= 0) mx = fmaxf(mx, s[i][g]);
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
      const float mnew = fmaxf(m[g], mx);
      const float corr = m[g] == -INFINITY ? 0.f : expf(m[g] - mnew);
      float sum = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const float pv = j[i] >= 0 ? expf(s[i][g] - mnew) : 0.f;
        ps[g * 128 + lane + 32 * i] = pv;
        sum += pv;
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
      l[g] = l[g] * corr + sum;
      m[g] = mnew;
#pragma unroll
      for (int e = 0; e < DL; ++e) acc[g][e] *= corr;
    }
    __syncwarp();
    // weighted value rows: this lane's DL dimensions of every selected row
    for (int t0 = 0; t0 < nc; t0 += 4) {
      float pq[G][4];
#pragma unroll
      for (int g = 0; g < G; ++g) {
        const float4 p4 = *reinterpret_cast<const float4*>(ps + g * 128 + t0);
        pq[g][0] = p4.x; pq[g][1] = p4.y; pq[g][2] = p4.z; pq[g][3] = p4.w;
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        if (t0 + i >= nc) break;
        const uint16_t* vr = vb + int64_t(ix[t0 + i]) * D + lane * DL;
        float vv[DL];
        if constexpr (DL == 4) {
          const uint2 w = __ldg(reinterpret_cast<const uint2*>(vr));
          vv[0] = __uint_as_float(w.x << 16); vv[1] = __uint_as_float(w.x & 0xFFFF0000u);
          vv[2] = __uint_as_float(w.y << 16); vv[3] = __uint_as_float(w.y & 0xFFFF0000u);
        } else {
          const uint32_t w = __ldg(reinterpret_cast<const uint32_t*>(vr));
          vv[0] = __uint_as_float(w << 16); vv[1] = __uint_as_float(w & 0xFFFF0000u);
        }
#pragma unroll
        for (int g = 0; g < G; ++g)
#pragma unroll
          for (int e = 0; e < DL; ++e) acc[g][e] = fmaf(pq[g][i], vv[e], acc[g][e]);
      }
    }
    __syncwarp();
  }
  uint16_t* o = static_cast<uint16_t*>(a.out);
#pragma unroll
  for (int g = 0; g < G; ++g) {
    const float inv = 1.f / l[g];
    uint16_t* orow = o + ((int64_t(b) * d.Hq + hk * G + g) * d.N + u) * D + lane * DL;
    if constexpr (DL == 4) {
      *reinterpret_cast<uint2*>(orow) = make_uint2(pack_bf16(acc[g][0] * inv, acc[g][1] * inv),
                                                   pack_bf16(acc[g][2] * inv, acc[g][3] * inv));
    } else {
      *reinterpret_cast<uint32_t*>(orow) = pack_bf16(acc[g][0] * inv, acc[g][1] * inv);
    }
  }
}

// ---------------------------------------------------------------- V^T for the tensor-core path

// vt[(b * Hkv + hk) * d + i][j] = v[(b * Hkv + hk) * N + j][i], 32 x 32 tiles through SMEM.
__global__ void __launch_bounds__(256) replay_vt_kernel(const uint16_t* __restrict__ v,
                                                         uint16_t* __restrict__ vt, int N, int D) {
  __shared__ uint16_t tile[32][33];
  const int bh = blockIdx.z;
  const int j0 = blockIdx.x * 32, i0 = blockIdx.y * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;   // 32 x 8
  const uint16_t* src = v + int64_t(bh) * N * D;
  uint16_t* dst = vt + int64_t(bh) * D * N;
  for (int r = ty; r < 32; r += 8) {
    const int j = j0 + r, i = i0 + tx;
    tile[r][tx] = (j < N && i < D) ? src[int64_t(j) * D + i] : 0;
  }
  __syncthreads();
  for (int r = ty; r < 32; r += 8) {
    const int i = i0 + r, j = j0 + tx;
    if (i < D && j < N) dst[int64_t(i) * N + j] = tile[tx][r];
  }
}

// ---------------------------------------------------------------- tensor-core causal attention

template <int D>
struct Fa {
  static constexpr int kK = 128 * D * 2;      // K tile: D/64 blocks of 128 rows x 128 B
  static constexpr int kVtRows = D + 16;     // V^T rows: d, then a row of ones and 15 of zeros
  static constexpr int kVtBlk = kVtRows * 128;   // one V^T block: kVtRows rows x 64 keys
  static constexpr int kVt = 2 * kVtBlk;      // V^T tile: 128 keys
  static constexpr int kVtCopy = 2 * D * 128; // bytes the copies of a V^T tile write (rows 0 .. d - 1)
  static constexpr int kStages = 3;           // K / V^T stages
  static constexpr int kQcol = 256 + kVtRows; // TMEM: S buffers 0 / 128, O (kVtRows columns) 256, Q
  static constexpr int kBytes = kStages * (kK + kVt);
  static constexpr int kXch = 2 * 4 * 128 * 4;   // partial maxima [parity][key quarter][row]
  static constexpr int kSmem = kBytes + 256 + kXch + 1024;
  static constexpr int kSmWarps = 16;         // softmax warps: four per TMEM lane quarter
  static constexpr int kThreads = 32 * (4 + kSmWarps);
};
static_assert(Fa<128>::kSmem <= 232448, "shared memory budget");
static_assert(Fa<128>::kQcol + 64 <= 512 && Fa<64>::kQcol + 32 <= 512, "TMEM columns");
static_assert(Fa<64>::kThreads == Fa<128>::kThreads, "one launch size for both head widths");

// Named barrier `id` over `n` threads, returning the AND of `p`.
__device__ __forceinline__ bool lane_and_n(int id, int n, bool p) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred a, q;\n\t"
      "setp.ne.u32 a, %1, 0;\n\t"
      "bar.red.and.pred q, %2, %3, a;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(p)), "r"(id), "r"(n)
      : "memory");
  return r != 0;
}

// Each thread of the warp writes 32 (16) consecutive 32-bit columns of its TMEM lane.
__device__ __forceinline__ void tmem_st_32x32b_x32(uint32_t taddr, const uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
      "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15]),
      "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]), "r"(r[22]), "r"(r[23]),
      "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]), "r"(r[29]), "r"(r[30]), "r"(r[31])
      : "memory");
}

__device__ __forceinline__ void tmem_st_32x32b_x16(uint32_t taddr, const uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
      "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16};" ::"r"(taddr),
      "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7]),
      "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]), "r"(r[15])
      : "memory");
}

__device__ __forceinline__ void tmem_st_32x32b_x8(uint32_t taddr, const uint32_t (&r)[8]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"r"(taddr),
               "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]), "r"(r[7])
               : "memory");
}

__device__ __forceinline__ void tmem_st_wait() {
  asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// mbar_wait for the attention kernel's TMA producer and the softmax warps' lane-0
// waits: each poll may suspend the thread (up to 0.5 us, ended early when the
// phase completes), so waiting warps leave their sub-partition's issue slots to
// the softmax warps. The MMA issuer keeps the polling mbar_wait.
__device__ __forceinline__ bool mbar_try_wait_sleep(uint32_t bar_addr, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar_addr), "r"(parity), "r"(500u)
      : "memory");
  return ok != 0;
}

__device__ __forceinline__ bool mbar_wait_sleep(uint64_t* bar, uint32_t parity, volatile int* abort_flag,
                                                long long limit) {
  const uint32_t a = smem_u32(bar);
  const long long t0 = clock64();
  while (!mbar_try_wait_sleep(a, parity)) {
    if (*abort_flag) return false;
    if (clock64() - t0 > limit) {
      *abort_flag = 1;
      return false;
    }
  }
  return true;
}

__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// Packed pairs of fp32 (sm_100 family): d = a * b + c per lane.
__device__ __forceinline__ uint64_t f32x2(float lo, float hi) {
  return (static_cast<uint64_t>(__float_as_uint(hi)) << 32) | __float_as_uint(lo);
}
__device__ __forceinline__ uint64_t ffma_x2(uint64_t a, uint64_t b, uint64_t c) {
  uint64_t d;
  asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(d) : "l"(a), "l"(b), "l"(c));
  return d;
}

// One 32-key chunk (keys k0 .. k0 + 31 of the tile) of a query row's scores v, in
// its softmax: the running maxima of 8 independent chains (two keys per step), and
// the bf16 pairs of P = exp2(s * sl2 - m). DIAG: the diagonal tile, whose keys past
// the row r are masked (on other tiles every key counts, with no per-key test).
template <bool DIAG>
__device__ __forceinline__ void chunk_max(const uint32_t (&v)[32], int k0, int r, float (&mk)[8]) {
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    const float a0 = (!DIAG || k0 + 2 * k <= r) ? __uint_as_float(v[2 * k]) : -INFINITY;
    const float a1 = (!DIAG || k0 + 2 * k + 1 <= r) ? __uint_as_float(v[2 * k + 1]) : -INFINITY;
    mk[k & 7] = fmax3(mk[k & 7], a0, a1);
  }
}

template <bool DIAG>
__device__ __forceinline__ void chunk_p(const uint32_t (&v)[32], int k0, int r, float sl2, float m,
                                        uint32_t (&pk)[16]) {
  const uint64_t s2 = f32x2(sl2, sl2), nm2 = f32x2(-m, -m);
#pragma unroll
  for (int k = 0; k < 16; ++k) {
    const uint64_t x = ffma_x2((static_cast<uint64_t>(v[2 * k + 1]) << 32) | v[2 * k], s2, nm2);
    const float p0 = (!DIAG || k0 + 2 * k <= r) ? ex2_fast(__uint_as_float(static_cast<uint32_t>(x))) : 0.f;
    const float p1 = (!DIAG || k0 + 2 * k + 1 <= r) ? ex2_fast(__uint_as_float(static_cast<uint32_t>(x >> 32))) : 0.f;
    __nv_bfloat162 pb = __floats2bfloat162_rn(p0, p1);
    pk[k] = *reinterpret_cast<uint32_t*>(&pb);
  }
}

// One 32-bit TMEM column of the thread's lane (warp-collective, 32x32b shape).
__device__ __forceinline__ void tmem_st_x1(uint32_t taddr, uint32_t v) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x1.b32 [%0], {%1};" ::"r"(taddr), "r"(v) : "memory");
}

__device__ __forceinline__ uint32_t tmem_ld_x1(uint32_t taddr) {
  uint32_t v;
  asm volatile("tcgen05.ld.sync.aligned.32x32b.x1.b32 {%0}, [%1];" : "=r"(v) : "r"(taddr) : "memory");
  asm volatile("tcgen05.wait::ld.sync.aligned;" : "+r"(v)::"memory");
  return v;
}

// D[tmem] (+)= A[tmem] * B[smem]^T, issued by a single thread: A (M = 128 rows,
// 16-bit elements, two consecutive K values per 32-bit column) is read from the
// lanes of the issuing CTA's tensor memory.
__device__ __forceinline__ void umma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t bdesc,
                                             uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
      "r"(a_tmem), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// One CTA per (b, query head, 128-query tile), persistent over key tiles
// 0..diagonal. Tensor memory (512 columns): S of key tile j in buffer j & 1 at
// columns 128 (j & 1); its bf16 probabilities for keys 32 c .. 32 c + 31 written
// over the buffer's columns 32 c .. 32 c + 15 (two keys per 32-bit column); O at
// 256: d output columns, then the row sum (the V^T tile carries a row of ones
// below its d rows, so the second MMA adds up the very bf16 probabilities it
// uses); Q at Fa::kQcol (d / 2 columns, two dimensions per column). Both MMAs
// read their A operand (Q, P) from tensor memory and their B operand (K, V^T)
// from shared memory.
template <int D>
__global__ void __launch_bounds__(Fa<D>::kThreads, 1)
    replay_fmha_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmVt,
                       const ReplayArgs a) {
  constexpr int kS = Fa<D>::kStages;
  constexpr int OC = D / 4;   // output columns (and query dimensions) per softmax thread
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sK = smem;                        // [kS] stages
  uint8_t* sV = sK + kS * Fa<D>::kK;         // [kS] stages
  uint64_t* bars = reinterpret_cast<uint64_t*>(sV + kS * Fa<D>::kVt);
  uint64_t* q_ready = bars;          // Q in TMEM (every softmax warp)
  uint64_t* kv_full = bars + 1;      // [kS]
  uint64_t* kv_empty = bars + 4;     // [kS]
  uint64_t* s_full = bars + 7;       // [2] by S buffer
  uint64_t* p_full = bars + 9;       // [2] by S buffer (every softmax warp)
  uint64_t* pv_done = bars + 11;     // phase j: P_j V_j added into O
  uint64_t* drain = bars + 12;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 13);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  float* xch = reinterpret_cast<float*>(reinterpret_cast<uint8_t*>(bars) + 256);   // Fa::kXch bytes
  static_assert(kS == 3, "barrier block layout");

  const ReplayDims& d = a.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int n_qt = (d.N + 127) / 128;
  const int qt = n_qt - 1 - static_cast<int>(blockIdx.x % n_qt);   // heavy tiles first
  const int bh = static_cast<int>(blockIdx.x / n_qt);
  const int b = bh / d.Hq, h = bh - b * d.Hq;
  const int hk = h / (d.Hq / d.Hkv);
  const int L = seq_len_of(a, b);
  const int q0 = qt * 128;
  if (q0 >= L) return;   // uniform over the CTA: no barrier or TMEM use yet
  const int n_kv = qt + 1;
  const long long wl = a.wait_limit;

  if (threadIdx.x == 0) {
    mbar_init(q_ready, Fa<D>::kSmWarps);
    for (int i = 0; i < kS; ++i) {
      mbar_init(&kv_full[i], 1);
      mbar_init(&kv_empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s_full[i], 1);
      mbar_init(&p_full[i], Fa<D>::kSmWarps);
    }
    mbar_init(pv_done, 1);
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmVt);
  }
  if (warp == 2) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  uint32_t issued_mask = 0, issue_parity = 0;
  bool mma_issued = false;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer: K and V^T tiles, kS stages
      const int krow = (b * d.Hkv + hk) * d.N, vrow = (b * d.Hkv + hk) * D;
      for (int j = 0; j < n_kv; ++j) {
        const int st = j % kS;
        const uint32_t use = static_cast<uint32_t>(j / kS);
        if (!mbar_wait_sleep(&kv_empty[st], (use & 1u) ^ 1u, abort_flag, wl)) break;
        mbar_arrive_expect_tx(&kv_full[st], Fa<D>::kK + Fa<D>::kVtCopy);
        for (int kb = 0; kb < D / 64; ++kb)
          tma_load_2d(sK + st * Fa<D>::kK + kb * 128 * 128, &tmK, &kv_full[st], kb * 64,
                      krow + j * 128);
        for (int kb = 0; kb < 2; ++kb)
          tma_load_2d(sV + st * Fa<D>::kVt + kb * Fa<D>::kVtBlk, &tmVt, &kv_full[st],
                      j * 128 + kb * 64, vrow);
        issued_mask |= 1u << st;
        issue_parity = (issue_parity & ~(1u << st)) | ((use & 1u) << st);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer (warp-uniform, elected lane)
    // S_j = Q K_j^T into buffer j & 1 runs up to two key tiles ahead of the softmax;
    // O += P_j V_j follows each tile's probabilities. S_{j+2} overwrites P_j, and MMAs
    // with different accumulators are not ordered by issue, so it waits until
    // O += P_j V_j is done.
    const uint32_t idS = idesc_bf16_f32(128, 128), idPV = idesc_bf16_f32(128, Fa<D>::kVtRows);
    bool ok = mbar_wait(q_ready, 0, abort_flag, wl);
    tc_fence_after();
    auto issue_s = [&](int j) -> bool {
      const int st = j % kS;
      if (!mbar_wait(&kv_full[st], static_cast<uint32_t>(j / kS) & 1u, abort_flag, wl)) return false;
      tc_fence_after();
      if (elect_one()) {
        for (int kb = 0; kb < D / 64; ++kb) {
          const uint64_t bd = sdesc_k_sw128(smem_u32(sK + st * Fa<D>::kK + kb * 128 * 128));
#pragma unroll
          for (int k = 0; k < 4; ++k)   // dimensions 64 kb + 16 k ..: Q columns kQcol + 32 kb + 8 k
            umma_bf16_ts(tmem + (j & 1) * 128, tmem + Fa<D>::kQcol + kb * 32 + k * 8, bd + 2 * k, idS,
                         (kb | k) != 0);
        }
        umma_commit(&s_full[j & 1]);
      }
      __syncwarp();
      mma_issued = true;
      return true;
    };
    auto issue_pv = [&](int j) -> bool {
      const int st = j % kS;
      if (!mbar_wait(&p_full[j & 1], static_cast<uint32_t>(j >> 1) & 1u, abort_flag, wl)) return false;
      tc_fence_after();
      if (elect_one()) {
        for (int kb = 0; kb < 2; ++kb) {
          const uint64_t bd = sdesc_k_sw128(smem_u32(sV + st * Fa<D>::kVt + kb * Fa<D>::kVtBlk));
#pragma unroll
          for (int k = 0; k < 4; ++k) {   // keys 64 kb + 16 k ..: key quarter 2 kb + k / 2
            const uint32_t pc = static_cast<uint32_t>(32 * (2 * kb + (k >> 1)) + 8 * (k & 1));
            umma_bf16_ts(tmem + 256, tmem + (j & 1) * 128 + pc, bd + 2 * k, idPV, (j | kb | k) != 0);
          }
        }
        umma_commit(pv_done);
        umma_commit(&kv_empty[st]);
      }
      __syncwarp();
      return true;
    };
    if (ok) ok = issue_s(0);
    if (ok && n_kv > 1) ok = issue_s(1);
    for (int j = 0; ok && j < n_kv; ++j) {
      ok = issue_pv(j);
      if (ok && j + 2 < n_kv)
        ok = mbar_wait(pv_done, static_cast<uint32_t>(j) & 1u, abort_flag, wl) && issue_s(j + 2);
    }
  } else if (warp >= 4) {
    // ------------------------------------------------ Q into TMEM, softmax, output rows
    // Warps 4 + 4 c + q (c = 0..3) take TMEM lane quarter q and key quarter c: the
    // four threads of a query row each take 32 of a tile's keys, OC query
    // dimensions and OC output columns. P for their keys goes over the first 16
    // of their own 32 score columns, so no thread writes where another reads. The
    // quarters' partial maxima meet in shared memory (double-buffered by key-tile
    // parity), so all four take the same max and the same rescaling decisions.
    // O, with the row sum in its column d, accumulates in TMEM across key tiles.
    // A row's running max m is raised only when a tile's max exceeds it by more
    // than kTau (base 2), so every probability exp2(s - m) stays below 2^kTau;
    // raising it rescales the row's O columns and sum in TMEM (after the previous
    // tile's PV has landed). The four warps of a lane quarter (one per key
    // quarter) pair on named barrier 1 + q with bar.red.and, which also agrees on
    // their waits, so a timeout stops all four together.
    constexpr float kTau = 8.f;
    const int c4 = (warp - 4) >> 2, q = warp & 3;
    const int r = q * 32 + lane;
    const uint32_t lanes = static_cast<uint32_t>(q * 32) << 16;
    const uint32_t tO = tmem + lanes + 256 + c4 * OC, tL = tmem + lanes + 256 + D;
    float* xm = xch;              // [parity][quarter][row] partial maxima
    const float sl2 = rsqrtf(float(D)) * 1.4426950408889634f;   // scale * log2(e)
    const int k0 = c4 * 32;       // this quarter's first key of a tile
    {
      // the constant rows of every V^T block: row d all ones (bf16 1.0), rows d + 1 .. d + 15
      // zero; the TMA copies write only rows 0 .. d - 1
      const int t = threadIdx.x - 128;   // 0 .. 32 kSmWarps - 1
      for (int e = t; e < kS * 2 * 128; e += 32 * Fa<D>::kSmWarps) {   // 16-byte units, 2 KB per block
        const int blk = e >> 7, u = e & 127;
        const uint32_t w = u < 8 ? 0x3F803F80u : 0u;   // the first 128 bytes are row d
        st_shared_v4(smem_u32(sV + blk * Fa<D>::kVtBlk + D * 128 + u * 16), w, w, w, w);
      }
      fence_proxy_async_smem();
      // dimensions OC c4 .. OC c4 + OC - 1 of this row's query, as bf16 pairs into TMEM
      // columns kQcol + OC c4 / 2 ..
      const int qrow = q0 + r;
      const uint4* src = reinterpret_cast<const uint4*>(static_cast<const uint16_t*>(a.q) +
                                                        ((int64_t(b) * d.Hq + h) * d.N + qrow) * D + OC * c4);
      uint32_t qv[OC / 2];
#pragma unroll
      for (int i = 0; i < OC / 8; ++i) {
        const uint4 u = qrow < d.N ? src[i] : make_uint4(0u, 0u, 0u, 0u);
        qv[4 * i] = u.x;
        qv[4 * i + 1] = u.y;
        qv[4 * i + 2] = u.z;
        qv[4 * i + 3] = u.w;
      }
      const uint32_t tq = tmem + lanes + Fa<D>::kQcol + static_cast<uint32_t>(OC / 2 * c4);
      if constexpr (OC == 32)
        tmem_st_32x32b_x16(tq, qv);
      else
        tmem_st_32x32b_x8(tq, qv);
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(q_ready);
    }
    float m = -INFINITY;
    bool ok = true;
    auto agree = [&](bool p) -> bool { return lane_and_n(1 + q, 128, p); };
    auto wait_lane0 = [&](uint64_t* bar, uint32_t par) -> bool {
      int w = 1;
      if (lane == 0) w = mbar_wait_sleep(bar, par, abort_flag, wl) ? 1 : 0;
      return __shfl_sync(0xffffffffu, w, 0) != 0;
    };
    for (int j = 0; j < n_kv; ++j) {
      const uint32_t tS = tmem + lanes + (j & 1) * 128 + k0;
      const bool okw = wait_lane0(&s_full[j & 1], static_cast<uint32_t>(j >> 1) & 1u);
      const bool diag = j == qt;
      uint32_t v[32];
      float pm = -INFINITY;
      if (okw) {
        tc_fence_after();
        tmem_ld_32x32b_x32(tS, v);
        tmem_ld_wait(v);
        // the maximum of this quarter's masked scores in 8 independent chains
        float mk[8];
#pragma unroll
        for (int e = 0; e < 8; ++e) mk[e] = -INFINITY;
        if (diag)
          chunk_max<true>(v, k0, r, mk);
        else
          chunk_max<false>(v, k0, r, mk);
        pm = fmaxf(fmax3(mk[0], mk[1], mk[2]), fmax3(mk[3], mk[4], fmax3(mk[5], mk[6], mk[7])));
      }
      float* xmj = xm + (j & 1) * 512;
      xmj[c4 * 128 + r] = pm;
      // one barrier trades the quarters' maxima and agrees on the four warps' waits
      if (!agree(okw)) { ok = false; break; }
      // the row's max of the scaled scores (the scale is positive: scaled after the comparison)
      const float mx = fmaxf(fmax3(xmj[r], xmj[128 + r], xmj[256 + r]), xmj[384 + r]) * sl2;
      const bool raise = mx > m + kTau;   // always on the first tile (m = -inf)
      const float alpha = (raise && m != -INFINITY) ? ex2_fast(m - mx) : 1.f;
      // the same for the quarter's four warps: they hold the same 32 rows
      const bool rescale = __any_sync(0xffffffffu, alpha != 1.f);
      if (rescale) {   // needs P_{j-1} V_{j-1} in O
        if (!agree(wait_lane0(pv_done, static_cast<uint32_t>(j - 1) & 1u))) {
          ok = false;
          break;
        }
        tc_fence_after();
        uint32_t o[OC];
        if constexpr (OC == 32) {
          tmem_ld_32x32b_x32(tO, o);
          tmem_ld_wait(o);
        } else {
          tmem_ld_32x32b_x16(tO, o);
          tmem_ld_wait(o);
        }
#pragma unroll
        for (int k = 0; k < OC; ++k) o[k] = __float_as_uint(__uint_as_float(o[k]) * alpha);
        if constexpr (OC == 32)
          tmem_st_32x32b_x32(tO, o);
        else
          tmem_st_32x32b_x16(tO, o);
        if (c4 == 0) tmem_st_x1(tL, __float_as_uint(__uint_as_float(tmem_ld_x1(tL)) * alpha));
      }
      if (raise) m = mx;
      // P = exp2(s - m) as bf16 pairs over the first 16 of this quarter's score columns
      uint32_t pk[16];
      if (diag)
        chunk_p<true>(v, k0, r, sl2, m, pk);
      else
        chunk_p<false>(v, k0, r, sl2, m, pk);
      tmem_st_32x32b_x16(tS, pk);
      tmem_st_wait();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&p_full[j & 1]);
    }
    // the quarter's four warps take part (ok is uniform over them: the loop's exits are agreed)
    const bool done = agree(ok && wait_lane0(pv_done, static_cast<uint32_t>(n_kv - 1) & 1u));
    if (done) {
      tc_fence_after();
      const int qq = q0 + r;
      const float inv = 1.f / __uint_as_float(tmem_ld_x1(tL));   // the row sum
      uint32_t o[OC];
      if constexpr (OC == 32) {
        tmem_ld_32x32b_x32(tO, o);
        tmem_ld_wait(o);
      } else {
        tmem_ld_32x32b_x16(tO, o);
        tmem_ld_wait(o);
      }
      if (qq < L) {
        uint4* dst = reinterpret_cast<uint4*>(static_cast<uint16_t*>(a.out) +
                                              ((int64_t(b) * d.Hq + h) * d.N + qq) * D + c4 * OC);
#pragma unroll
        for (int e8 = 0; e8 < OC / 8; ++e8) {
          uint32_t w4[4];
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            __nv_bfloat162 u = __floats2bfloat162_rn(__uint_as_float(o[8 * e8 + 2 * e]) * inv,
                                                     __uint_as_float(o[8 * e8 + 2 * e + 1]) * inv);
            w4[e] = *reinterpret_cast<uint32_t*>(&u);
          }
          dst[e8] = make_uint4(w4[0], w4[1], w4[2], w4[3]);
        }
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    if (warp == 0 && lane == 0) {
      for (int st = 0; st < kS; ++st)
        if ((issued_mask >> st) & 1u) {
          const uint32_t ad = smem_u32(&kv_full[st]);
          const long long t0 = clock64();
          while (!mbar_try_wait(ad, (issue_parity >> st) & 1u) && clock64() - t0 < wl) {
          }
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
// ---------------------------------------------------------------- tensor-core guided attention

// Shared memory of replay_gattn_kernel (d = 128, GQA groups of up to 16 query
// heads, S <= 128). A kernel that allocates TMEM runs one CTA per SM, so the CTA
// holds kLanes independent 4-warp lanes, each with its own tiles: the item's
// gathered key rows and value rows (each two 16 KB blocks of 128 rows x 64 dims,
// 128B-swizzled), its query rows (two 2 KB blocks of 16 rows x 64 dims) and the
// P tile (two 2 KB blocks of 16 head rows x 64 keys); then each lane's softmax
// exchange words and MMA barriers.
struct Ga {
  static constexpr int kLanes = 3;
  static constexpr int kBlk = 128 * 128;
  static constexpr int kKV = 2 * kBlk;
  static constexpr int kQBlk = 16 * 128;
  static constexpr int kPBlk = 16 * 128;
  static constexpr int kOffV = kKV;
  static constexpr int kOffQ = 2 * kKV;
  static constexpr int kOffP = 2 * kKV + 2 * kQBlk;
  static constexpr int kTiles = kOffP + 2 * kPBlk;           // per lane, a multiple of 1024
  static constexpr int kXch = 2 * 16 * 4 * 4;                 // maxima and sums, [head][quarter]
  static constexpr int kLaneAux = kXch + 4 * 8;               // + barriers: MMA 1, MMA 2, drain, pad
  static constexpr int kSmem = kLanes * (kTiles + kLaneAux) + 16 + 1024;
  static constexpr int kThreads = 128 * kLanes;
  static constexpr int kTmemCols = 128;                       // lane l: S^T at 32 l, O^T at 32 l + 16
};
static_assert(Ga::kSmem <= 232448, "shared memory budget");
static_assert(Ga::kTiles % 1024 == 0, "1024-byte aligned operand tiles");
static_assert(32 * Ga::kLanes <= Ga::kTmemCols, "TMEM columns");

__device__ __forceinline__ void st_shared_u16(uint32_t addr, uint16_t v) {
  asm volatile("st.shared.u16 [%0], %1;" ::"r"(addr), "h"(v) : "memory");
}

// Named barrier `id` over the 128 threads of one lane.
__device__ __forceinline__ void lane_sync(int id) {
  asm volatile("bar.sync %0, 128;" ::"r"(id) : "memory");
}

// The same, returning the AND of `p` over the lane's threads.
__device__ __forceinline__ bool lane_and(int id, bool p) {
  uint32_t r;
  asm volatile(
      "{\n\t.reg .pred a, q;\n\t"
      "setp.ne.u32 a, %1, 0;\n\t"
      "bar.red.and.pred q, %2, 128, a;\n\t"
      "selp.u32 %0, 1, 0, q;\n\t}"
      : "=r"(r)
      : "r"(static_cast<uint32_t>(p)), "r"(id)
      : "memory");
  return r != 0;
}

// G: query heads per key/value head (the N = 16 columns of the MMAs hold G of them).
template <int G>
__global__ void __launch_bounds__(Ga::kThreads, 1) replay_gattn_kernel(const ReplayArgs a) {
  constexpr int D = 128;
  static_assert(G >= 1 && G <= 16, "GQA group of the N = 16 MMA columns");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const int ln = threadIdx.x >> 7;                 // this thread's lane
  const int tid = threadIdx.x & 127;
  const int warp = tid >> 5, lane = threadIdx.x & 31;
  uint8_t* tiles = smem + ln * Ga::kTiles;
  uint8_t* aux = smem + Ga::kLanes * Ga::kTiles + ln * Ga::kLaneAux;
  float* xm = reinterpret_cast<float*>(aux);                       // [16][4]
  uint32_t* xl = reinterpret_cast<uint32_t*>(aux) + 64;            // [16][4]
  uint64_t* bar_s = reinterpret_cast<uint64_t*>(aux + Ga::kXch);   // MMA 1 complete
  uint64_t* bar_o = bar_s + 1;                                     // MMA 2 complete
  uint64_t* drain = bar_s + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + Ga::kLanes * (Ga::kTiles + Ga::kLaneAux));
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
  const int bar_id = 1 + ln;

  const ReplayDims& d = a.d;
  const int64_t n_items = int64_t(d.B) * d.Hkv * d.N;   // <= INT32_MAX (checked at launch)
  const long long wl = a.wait_limit;

  // Zero the operand tiles once: query rows >= G, P rows >= G and key/value rows
  // past a short row's count are never copied, so they hold zeros or finite
  // values from earlier items (whose probabilities are 0).
  {
    uint4* z = reinterpret_cast<uint4*>(smem);
    for (int i = threadIdx.x; i < Ga::kLanes * Ga::kTiles / 16; i += Ga::kThreads)
      z[i] = make_uint4(0u, 0u, 0u, 0u);
    fence_proxy_async_smem();
  }
  if (tid == 0) {
    mbar_init(bar_s, 1);
    mbar_init(bar_o, 1);
    mbar_init(drain, 1);
  }
  if (threadIdx.x == 0) *abort_flag = 0;
  if (tid == 0) fence_barrier_init();
  if (threadIdx.x < 32) {
    tmem_alloc(tmem_slot, Ga::kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot + 32 * ln;   // this lane's S^T (+0) and O^T (+16)

  // gather roles: per copy instruction a warp moves two 256-byte rows (lanes
  // 0-15 one key's row, lanes 16-31 the next key's); warp w takes keys
  // 8 m + kr (m = 0..15, kr = 2 w + half), and lane L holds the position of key
  // 8 (L >> 1) + 2 w + (L & 1). A thread's 16-byte unit q16 of key 8 m + kr lands
  // at the same swizzled column of every 1,024-byte atom (key & 7 == kr), so its
  // destination is a fixed base plus 1,024 m.
  const int half = lane >> 4, q16 = lane & 15;
  const uint32_t sbase = smem_u32(tiles);
  const int my_key = 8 * (lane >> 1) + 2 * warp + (lane & 1);
  const int kr = 2 * warp + half;
  const uint32_t gdst = sbase + static_cast<uint32_t>((q16 >> 3) * Ga::kBlk + kr * 128 + (((q16 & 7) ^ kr) << 4));
  // softmax / output roles: warp w owns keys (S^T rows) and dims (O^T rows) 32 w .. 32 w + 31,
  // TMEM lanes 32 w .. 32 w + 31 (w = the warp's index mod 4)
  const int row = 32 * warp + lane;
  const uint32_t tlanes = static_cast<uint32_t>(32 * warp) << 16;
  const int kk = row & 63;
  const uint32_t prow = sbase + static_cast<uint32_t>(Ga::kOffP + (row >> 6) * Ga::kPBlk);
  const float sl2 = rsqrtf(float(D)) * 1.4426950408889634f;   // scale * log2(e)
  const uint32_t id1 = idesc_bf16_f32(128, 16), id2 = id1 | kIdescAMajorMN;
  bool mma_issued = false;
  uint32_t n = 0;   // items done: the parity of both MMA barriers

  // lane `ln` of CTA `blockIdx.x` takes items v, v + V, .. (v its global lane index);
  // item it = bh * N + u is (b, key/value head) = (bh / Hkv, bh % Hkv) at context
  // position u, kept as (c_bh, c_u) and advanced by V without a division
  struct Item {
    int b, hk, u, c;
  };
  int64_t it = int64_t(blockIdx.x) * Ga::kLanes + ln;
  const int it_step = static_cast<int>(gridDim.x) * Ga::kLanes;
  const int step_bh = it_step / d.N, step_u = it_step - step_bh * d.N;
  int c_bh = static_cast<int>(it / d.N), c_u = static_cast<int>(it - int64_t(c_bh) * d.N);
  auto next_item = [&](Item& x) -> bool {
    while (it < n_items) {
      const int bh = c_bh, u = c_u;
      it += it_step;
      c_bh += step_bh;
      c_u += step_u;
      if (c_u >= d.N) {
        c_u -= d.N;
        ++c_bh;
      }
      const int b = bh / d.Hkv;
      if (u < seq_len_of(a, b)) {
        x.b = b;
        x.hk = bh - b * d.Hkv;
        x.u = u;
        x.c = min(d.S, u + 1);
        return true;
      }
    }
    return false;
  };
  auto load_pos = [&](const Item& x) -> int {
    return my_key < x.c ? min(max(a.sel[(int64_t(x.b) * d.N + x.u) * d.S + my_key], 0), d.N - 1) : 0;
  };
  // the item's selected key rows (which = 0, plus its query rows) or value rows (which = 1)
  auto issue_rows = [&](const Item& x, int my_pos, int which) {
    const char* src = reinterpret_cast<const char*>(static_cast<const uint16_t*>(which ? a.v : a.k) +
                                                    int64_t(x.b * d.Hkv + x.hk) * d.N * D + q16 * 8);
    const uint32_t dst = gdst + static_cast<uint32_t>(which * Ga::kKV);
    const int n_m = x.c - kr;   // key 8 m + kr is selected while 8 m < n_m
#pragma unroll
    for (int m = 0; m < 16; ++m) {
      const int pos = __shfl_sync(0xffffffffu, my_pos, 2 * m + half);   // pos < N <= 65536
      if (8 * m < n_m) cp_async_16(dst + 1024 * m, src + static_cast<uint32_t>(pos) * (2 * D));
    }
    if (which == 0) {
      for (int e = tid; e < G * 16; e += 128) {
        const int h = e >> 4, c16 = e & 15;
        cp_async_16(sbase + Ga::kOffQ + (c16 >> 3) * Ga::kQBlk + h * 128 + (((c16 & 7) ^ (h & 7)) << 4),
                    static_cast<const uint16_t*>(a.q) +
                        ((int64_t(x.b) * d.Hq + x.hk * G + h) * d.N + x.u) * D + c16 * 8);
      }
    }
    cp_async_commit();
  };

  // Per item i the lane issues the first MMA, then finishes item i - 1 (waits
  // for its second MMA, copies item i's value rows into the freed tile, writes
  // item i - 1's output rows), then runs item i's softmax (copying item i + 1's
  // key and query rows into the freed tiles) and issues its second MMA without
  // waiting for it. Commit groups run KQ(0), V(0), KQ(1), V(1), ..
  auto output_rows = [&](const Item& x) {   // O^T row = this thread's dim, normalised per head
    uint32_t v[16];
    tmem_ld_32x32b_x16(tmem + tlanes + 16, v);
    tmem_ld_wait(v);
    uint16_t* o = static_cast<uint16_t*>(a.out) + ((int64_t(x.b) * d.Hq + x.hk * G) * d.N + x.u) * D + row;
#pragma unroll
    for (int h = 0; h < 16; ++h) {
      if (h < G) {
        const uint4 l4 = *reinterpret_cast<const uint4*>(xl + h * 4);
        // l >= 1 (the row maximum's probability is 1), so the fast division is exact to 2 ulp
        const float l = __uint2float_rn(l4.x + l4.y + l4.z + l4.w) * (1.f / 16777216.f);
        o[int64_t(h) * d.N * D] = __bfloat16_as_ushort(__float2bfloat16_rn(__fdividef(__uint_as_float(v[h]), l)));
      }
    }
  };
  Item cur, nxt, prev;
  bool have = next_item(cur), have_prev = false, ok = true;
  int pos_cur = have ? load_pos(cur) : 0;
  if (have) issue_rows(cur, pos_cur, 0);
  while (have) {
    const bool have_nxt = next_item(nxt);
    const int pos_nxt = have_nxt ? load_pos(nxt) : 0;
    cp_async_wait_group<0>();   // KQ(cur) landed
    fence_proxy_async_smem();   // this thread's copies, visible to the tensor core
    tc_fence_before();
    lane_sync(bar_id);
    // ---- MMA 1: S^T = K_sel Q^T (M = 128 keys, N = 16 heads, K = d)
    if (warp == 0) {
      tc_fence_after();
      if (elect_one()) {
#pragma unroll
        for (int blk = 0; blk < 2; ++blk) {
          const uint64_t ad = sdesc_k_sw128(sbase + blk * Ga::kBlk);
          const uint64_t bd = sdesc_k_sw128(sbase + Ga::kOffQ + blk * Ga::kQBlk);
#pragma unroll
          for (int k4 = 0; k4 < 4; ++k4) umma_bf16(tmem, ad + 2 * k4, bd + 2 * k4, id1, (blk | k4) != 0);
        }
        // test hook: the first item of CTA 0's lane 0 never signals, so its wait runs out
        if (!(a.stall_test && blockIdx.x == 0 && ln == 0 && n == 0)) umma_commit(bar_s);
      }
      __syncwarp();
      mma_issued = true;
    }
    // ---- finish the previous item while the first MMA runs
    if (have_prev) {
      if (!lane_and(bar_id, tid != 0 || mbar_wait(bar_o, (n - 1) & 1u, abort_flag, wl))) {
        ok = false;
        break;
      }
      tc_fence_after();
    }
    issue_rows(cur, pos_cur, 1);   // the value tile (and the P tile) are free again
    if (have_prev) output_rows(prev);
    if (!lane_and(bar_id, tid != 0 || mbar_wait(bar_s, n & 1u, abort_flag, wl))) {
      ok = false;
      break;
    }
    tc_fence_after();
    // ---- softmax over the keys of each head (TMEM lane = key)
    const bool valid = row < cur.c;
    float sc[16];
    {
      uint32_t v[16];
      tmem_ld_32x32b_x16(tmem + tlanes, v);
      tmem_ld_wait(v);
#pragma unroll
      for (int h = 0; h < 16; ++h) sc[h] = __uint_as_float(v[h]) * sl2;
    }
    if (have_nxt) issue_rows(nxt, pos_nxt, 0);   // the key and query tiles are free again
    else cp_async_commit();
#pragma unroll
    for (int h = 0; h < 16; ++h) {
      if (h < G) {
        const float m = redux_max_f32(valid ? sc[h] : -INFINITY);
        if (lane == h) xm[h * 4 + warp] = m;
      }
    }
    lane_sync(bar_id);   // maxima traded; every thread's output rows of the previous item read xl
#pragma unroll
    for (int h = 0; h < 16; ++h) {
      if (h < G) {
        const float4 m4 = *reinterpret_cast<const float4*>(xm + h * 4);
        const float m = fmaxf(fmaxf(m4.x, m4.y), fmaxf(m4.z, m4.w));
        const __nv_bfloat16 pb16 = __float2bfloat16_rn(valid ? ex2_fast(sc[h] - m) : 0.f);
        st_shared_u16(prow + h * 128 + (((kk >> 3) ^ (h & 7)) << 4) + (kk & 7) * 2, __bfloat16_as_ushort(pb16));
        // the row sum of the rounded probabilities the MMA uses, in exact 2^-24 units
        const uint32_t sum = redux_add_u32(__float2uint_rn(__bfloat162float(pb16) * 16777216.f));
        if (lane == h) xl[h * 4 + warp] = sum;
      }
    }
    cp_async_wait_group<1>();   // V(cur) landed (KQ(nxt) may still be in flight)
    fence_proxy_async_smem();   // the P tile and the value rows, visible to the tensor core
    tc_fence_before();
    lane_sync(bar_id);
    // ---- MMA 2: O^T = V_sel^T P^T (M = 128 dims, value rows read MN-major, N = 16 heads)
    if (warp == 0) {
      tc_fence_after();
      if (elect_one()) {
        const int n_ks = (cur.c + 15) >> 4;   // 16-key steps holding the row's keys
        for (int ks = 0; ks < n_ks; ++ks) {
          const uint64_t ad = sdesc_mn_sw128(sbase + Ga::kOffV + ks * 2048, Ga::kBlk);
          const uint64_t bd = sdesc_k_sw128(sbase + Ga::kOffP + (ks >> 2) * Ga::kPBlk) + 2 * (ks & 3);
          umma_bf16(tmem + 16, ad, bd, id2, ks != 0);
        }
        umma_commit(bar_o);
      }
      __syncwarp();
    }
    ++n;
    prev = cur;
    have_prev = true;
    cur = nxt;
    pos_cur = pos_nxt;
    have = have_nxt;
  }
  if (ok && have_prev) {   // the last item's output rows
    if (lane_and(bar_id, tid != 0 || mbar_wait(bar_o, (n - 1) & 1u, abort_flag, wl))) {
      tc_fence_after();
      output_rows(prev);
    }
  }

  cp_async_wait_group<0>();
  if (warp == 0 && mma_issued && *abort_flag) {   // this lane's MMAs may be in flight after a timeout
    if (elect_one()) umma_commit(drain);
    __syncwarp();
    const uint32_t ad = smem_u32(drain);
    const long long t0 = clock64();
    while (!mbar_try_wait(ad, 0) && clock64() - t0 < wl) {
    }
  }
  tc_fence_before();
  __syncthreads();
  if (threadIdx.x < 32) {
    tc_fence_after();
    tmem_dealloc(*tmem_slot, Ga::kTmemCols);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicOr(a.status, kStatusTimeout);
}
}  // namespace

// GQA group sizes with an instantiated attention kernel
__host__ __device__ constexpr bool group_ok(int g) {
  return (g >= 1 && g <= 8) || g == 12 || g == 16;
}

bool replay_supported(const ReplayDims& d) {
  return d.Hkv > 0 && d.Hq % d.Hkv == 0 && group_ok(d.Hq / d.Hkv) &&
         (d.d == 64 || d.d == 128) && d.S >= 1 && d.S <= 4096 && d.N >= 1 && d.N <= 65536;
}

cudaError_t launch_replay_select(const ReplayArgs& a, cudaStream_t st) {
  const int rows = a.d.B * a.d.N;
  if (rows <= 0) return cudaSuccess;
  if (a.d.N <= 256 * kSelCacheRounds)
    replay_select_kernel<<<(rows + kSelCacheWarps - 1) / kSelCacheWarps, 32 * kSelCacheWarps, 0, st>>>(a);
  else
    replay_select_stream_kernel<<<(rows + kSelWarps - 1) / kSelWarps, 32 * kSelWarps, 0, st>>>(a);
  return cudaGetLastError();
}

bool replay_fmha_supported(const ReplayDims& d) {
  return (d.d == 64 || d.d == 128) && d.N % 8 == 0;
}

cudaError_t launch_replay_vt(const ReplayArgs& a, void* vt, cudaStream_t st) {
  const ReplayDims& d = a.d;
  dim3 grid((d.N + 31) / 32, (d.d + 31) / 32, d.B * d.Hkv);
  replay_vt_kernel<<<grid, 256, 0, st>>>(static_cast<const uint16_t*>(a.v),
                                         static_cast<uint16_t*>(vt), d.N, d.d);
  return cudaGetLastError();
}

cudaError_t launch_replay_fmha(const ReplayArgs& a, const CUtensorMap& tmK,
                               const CUtensorMap& tmVt, cudaStream_t st) {
  const ReplayDims& d = a.d;
  static bool attr[2] = {false, false};
  const int di = d.d == 128 ? 1 : 0;
  auto kern = d.d == 128 ? replay_fmha_kernel<128> : replay_fmha_kernel<64>;
  const int smem = d.d == 128 ? Fa<128>::kSmem : Fa<64>::kSmem;
  if (!attr[di]) {
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (e != cudaSuccess) return e;
    attr[di] = true;
  }
  const int n_qt = (d.N + 127) / 128;
  kern<<<d.B * d.Hq * n_qt, Fa<128>::kThreads, smem, st>>>(tmK, tmVt, a);
  return cudaGetLastError();
}

bool replay_gattn_supported(const ReplayDims& d) {
  const int G = d.Hq / d.Hkv;
  return d.d == 128 && group_ok(G) && G <= 16 && d.S >= 1 && d.S <= 128 &&
         int64_t(d.B) * d.Hkv * d.N <= INT32_MAX && int64_t(d.B) * d.Hq <= INT32_MAX;
}

template <int G>
cudaError_t launch_gattn_g(const ReplayArgs& a, int num_sms, cudaStream_t st) {
  static bool attr = false;
  if (!attr) {
    cudaError_t e = cudaFuncSetAttribute(replay_gattn_kernel<G>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, Ga::kSmem);
    if (e != cudaSuccess) return e;
    attr = true;
  }
  const int64_t lanes = (int64_t(a.d.B) * a.d.Hkv * a.d.N + Ga::kLanes - 1) / Ga::kLanes;
  const int g = static_cast<int>(lanes < num_sms ? lanes : num_sms);   // persistent, one CTA per SM
  if (g <= 0) return cudaSuccess;
  replay_gattn_kernel<G><<<g, Ga::kThreads, Ga::kSmem, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_replay_gattn(const ReplayArgs& a, int num_sms, cudaStream_t st) {
  switch (a.d.Hq / a.d.Hkv) {
    case 1: return launch_gattn_g<1>(a, num_sms, st);
    case 2: return launch_gattn_g<2>(a, num_sms, st);
    case 3: return launch_gattn_g<3>(a, num_sms, st);
    case 4: return launch_gattn_g<4>(a, num_sms, st);
    case 5: return launch_gattn_g<5>(a, num_sms, st);
    case 6: return launch_gattn_g<6>(a, num_sms, st);
    case 7: return launch_gattn_g<7>(a, num_sms, st);
    case 8: return launch_gattn_g<8>(a, num_sms, st);
    case 12: return launch_gattn_g<12>(a, num_sms, st);
    case 16: return launch_gattn_g<16>(a, num_sms, st);
    default: return cudaErrorInvalidValue;
  }
}

template <int D, int G>
cudaError_t launch_attn_dg(const ReplayArgs& a, cudaStream_t st) {
  const size_t smem = size_t(kAttnWarps) * attn_warp_floats<D, G>() * 4;
  static bool attr = false;
  if (!attr && smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(replay_attn_kernel<D, G>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    if (e != cudaSuccess) return e;
  }
  attr = true;
  const int64_t items = int64_t(a.d.B) * a.d.Hkv * a.d.N;
  const unsigned grid = static_cast<unsigned>((items + kAttnWarps - 1) / kAttnWarps);
  replay_attn_kernel<D, G><<<grid, 32 * kAttnWarps, smem, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_replay_attn(const ReplayArgs& a, cudaStream_t st) {
  const int G = a.d.Hq / a.d.Hkv;
#define MOT_RP_CASE(GG)                                                             \
  case GG:                                                                          \
    return a.d.d == 128 ? launch_attn_dg<128, GG>(a, st) : launch_attn_dg<64, GG>(a, st);
  switch (G) {
    MOT_RP_CASE(1) MOT_RP_CASE(2) MOT_RP_CASE(3) MOT_RP_CASE(4) MOT_RP_CASE(5)
    MOT_RP_CASE(6) MOT_RP_CASE(7) MOT_RP_CASE(8) MOT_RP_CASE(12) MOT_RP_CASE(16)
    default: return cudaErrorInvalidValue;
  }
#undef MOT_RP_CASE
}

}  // namespace mot
