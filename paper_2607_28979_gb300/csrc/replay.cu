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
//   replay_vt_kernel      V -> V^T per layer for the full-attention kernel.
//   The tensor-core kernels are in replay_fmha.cu (full causal attention) and
//   replay_gattn.cu (guided attention).
#include "replay_common.cuh"

namespace mot {
namespace {

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
}  // namespace

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

cudaError_t launch_replay_vt(const ReplayArgs& a, void* vt, cudaStream_t st) {
  const ReplayDims& d = a.d;
  dim3 grid((d.N + 31) / 32, (d.d + 31) / 32, d.B * d.Hkv);
  replay_vt_kernel<<<grid, 256, 0, st>>>(static_cast<const uint16_t*>(a.v),
                                         static_cast<uint16_t*>(vt), d.N, d.d);
  return cudaGetLastError();
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
