// 2-SM (cta_group::2) variant of the two translation GEMMs (see umma.cu for
// what each computes). A cluster of two CTAs computes a 256 x 256 tile: token
// tiles 2*mp (leader, cluster rank 0) and 2*mp + 1 (peer), against one
// 256-column slice of W1cat / W2cat. Each CTA stages only its own 128 rows of
// A and its own 128 rows of B per K block (32 KB instead of 48 KB for the
// same tensor-core work per SM), so six stages fit where four did, and every
// SM pulls two thirds of the operand bytes through L2 and its TMA unit.
//
// Roles per CTA (same warp layout as umma.cu):
//   warp 0 lane 0 (both CTAs)  TMA loads of its A rows and B half; the
//                              transaction bytes of both CTAs complete on the
//                              leader's stage barrier;
//   warp 1 lane 0 (leader)     tcgen05.mma.cta_group::2 M=256 N=256 K=16;
//                              commits arrive on both CTAs' barriers;
//   warp 2 (both CTAs)         allocates the pair's TMEM together;
//   warps 4.. (both CTAs)      epilogue of its own 128 accumulator rows, then
//                              an arrive on the leader's accumulator-free
//                              barrier.
// A token tile past the last one (odd tile count) is computed from arbitrary
// in-bounds rows and never stored. Every wait is bounded; a timeout unwinds and raises
// kStatusTimeout.
#include "umma_common.cuh"

namespace mot {
namespace {

constexpr int kStages2 = 6;
constexpr int kABytes2 = UM * UK * 2;         // 16 KB: this CTA's 128 rows of A
constexpr int kBBytes2 = (UN / 2) * UK * 2;   // 16 KB: this CTA's 128 rows of B
constexpr int kStageBytes2 = kABytes2 + kBBytes2;
constexpr int kBarBytes2 = 256;
__host__ __device__ constexpr int epi_warps2(int mode) { return mode == 1 ? 8 : 4; }
__host__ __device__ constexpr int threads2(int mode) { return 32 * (4 + epi_warps2(mode)); }
__host__ __device__ constexpr int store_bytes2(int mode) {
  return mode == 1 ? epi_warps2(mode) * kStoreTileBytes : 0;
}
__host__ __device__ constexpr int smem_bytes2(int mode) {
  return kStages2 * kStageBytes2 + store_bytes2(mode) + kBarBytes2 + 1024;
}
static_assert(smem_bytes2(1) <= 232448 && smem_bytes2(2) <= 232448, "shared memory budget");

struct Umma2Args {
  PathArgs p;
  SparseArgs sp;      // sparse routing: the packed rows and their pair-tile list
  int32_t nk;         // K blocks per tile
  int32_t n_tiles_n;  // 256-column tiles per group (per expert when sparse)
  int32_t b_rows;     // rows of B per group (E*H for GEMM1, D_t for GEMM2)
};

// One work item: a pair tile and a 256-column tile n. Dense: token tiles
// 2 mp and 2 mp + 1 of group grp; sparse: a pair tile of bucket (group, expert
// em) at packed rows p_own (this CTA's half). `live` = this CTA's tile has rows.
struct Work {
  int gl, grp, m_own, n, em, p_own, rows_own;
  bool live;
};

// Sparse GEMM2 epilogue of one warp: row 32 q + lane of the pair tile's half
// at packed row p_own; its fp32 result goes to the token's slot row.
__device__ __forceinline__ void epilogue_gemm2_sparse(const PathArgs& p, const SparseArgs& sp,
                                                      uint32_t tbase, int q, int lane, int gl,
                                                      int p_own, int rows_own, int n0) {
  const Dims& d = p.d;
  const int r = q * 32 + lane;
  const bool valid = r < rows_own;
  float* out = nullptr;              // top_k > 1: the token's slot row (fp32)
  __nv_bfloat16* tgt = nullptr;      // top_k = 1: the target cache row, head 0
  if (valid) {
    const int tok = sp.ltok[p_own + r], slot = sp.lslot[p_own + r];
    if (d.top_k == 1) {
      const GroupInfo gi = p.groups[p.g0 + gl];
      const TileInfo ti = p.tiles[tok / UM];
      tgt = static_cast<__nv_bfloat16*>(p.dst[gi.x]) +
            ((static_cast<size_t>(gi.tgt_layer) * d.B + ti.b) * d.H_t * d.S + ti.s0 + tok % UM) *
                d.d_t;
    } else {
      out = sp.ybuf + ((static_cast<size_t>(gl) * d.tpad + tok) * d.top_k + slot) * d.Dt + n0;
    }
  }
#pragma unroll 1
  for (int ch = 0; ch < UN / 32; ++ch) {
    uint32_t v[32];
    tmem_ld_32x32b_x32(tbase + ch * 32, v);
    tmem_ld_wait(v);
    if (valid && tgt) {   // channel c of head c / d_t, d_t a multiple of 32
      const int c = n0 + ch * 32, h = c / d.d_t, i0 = c - h * d.d_t;
      uint4* o4 = reinterpret_cast<uint4*>(tgt + static_cast<size_t>(h) * d.S * d.d_t + i0);
#pragma unroll
      for (int j = 0; j < 4; ++j)
        o4[j] = make_uint4(pack_bf16x2(__uint_as_float(v[8 * j + 0]), __uint_as_float(v[8 * j + 1])),
                           pack_bf16x2(__uint_as_float(v[8 * j + 2]), __uint_as_float(v[8 * j + 3])),
                           pack_bf16x2(__uint_as_float(v[8 * j + 4]), __uint_as_float(v[8 * j + 5])),
                           pack_bf16x2(__uint_as_float(v[8 * j + 6]), __uint_as_float(v[8 * j + 7])));
    } else if (valid) {
      float4* o4 = reinterpret_cast<float4*>(out + ch * 32);
#pragma unroll
      for (int j = 0; j < 8; ++j)
        o4[j] = make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                            __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3]));
    }
  }
}

// Spin about `cycles` SM cycles (used only while unwinding after a timeout).
__device__ __forceinline__ void spin_cycles(long long cycles) {
  const long long t0 = clock64();
  while (clock64() - t0 < cycles) {
  }
}

// MoT-h projection epilogue of one warp (App. C.5): output columns
// n0 .. n0 + 255 of [K | V] = a_hat [W^K; W^V]^T for row 32 q + lane of token
// tile m, stored as bf16 into the target cache of the group's target layer
// (columns below D_t into dst[0] = K, the rest into dst[1] = V). D_t is a
// multiple of 256, so a tile never straddles the two.
__device__ __forceinline__ void epilogue_proj(const PathArgs& p, uint32_t tbase, int q, int lane,
                                              int grp, int m, int n0) {
  const Dims& d = p.d;
  const int row = q * 32 + lane;
  const TileInfo ti = p.tiles[m];
  const bool valid = row < ti.rows;
  const int x = n0 >= d.Dt ? 1 : 0;
  const int c0 = n0 - x * d.Dt;
  __nv_bfloat16* dst = static_cast<__nv_bfloat16*>(p.dst[x]);
  const size_t s = static_cast<size_t>(ti.s0) + row;
  const size_t lbase = (static_cast<size_t>(p.proj_layer[grp]) * d.B + ti.b) * d.H_t;
#pragma unroll 1
  for (int ch = 0; ch < UN / 32; ++ch) {
    uint32_t r[32];
    tmem_ld_32x32b_x32(tbase + ch * 32, r);
    tmem_ld_wait(r);
    if (valid) {
      const int c = c0 + ch * 32, h = c / d.d_t, i0 = c - h * d.d_t;
      uint4* o4 = reinterpret_cast<uint4*>(dst + ((lbase + h) * d.S + s) * d.d_t + i0);
#pragma unroll
      for (int v = 0; v < 4; ++v)
        o4[v] = make_uint4(pack_bf16x2(__uint_as_float(r[8 * v + 0]), __uint_as_float(r[8 * v + 1])),
                           pack_bf16x2(__uint_as_float(r[8 * v + 2]), __uint_as_float(r[8 * v + 3])),
                           pack_bf16x2(__uint_as_float(r[8 * v + 4]), __uint_as_float(r[8 * v + 5])),
                           pack_bf16x2(__uint_as_float(r[8 * v + 6]), __uint_as_float(r[8 * v + 7])));
    }
  }
}

// MODE 1 = GEMM1 (A = source cache, or the packed rows when SPARSE), 2 = GEMM2
// (A = A2), 3 = the MoT-h projection (A = translated activation, bf16).
// SPARSE: work items come from the routing's pair-tile list and B is the
// bucket expert's slice of W1cat / W2cat.
template <int MODE, bool SPARSE>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(threads2(MODE), 1)
    umma2_gemm_kernel(const __grid_constant__ CUtensorMap tmA0,
                      const __grid_constant__ CUtensorMap tmA1,
                      const __grid_constant__ CUtensorMap tmB,
                      const __grid_constant__ CUtensorMap tmS, const Umma2Args ua) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + kStages2 * kABytes2;
  uint8_t* sOut = smem + kStages2 * kStageBytes2;
  uint64_t* full = reinterpret_cast<uint64_t*>(sOut + store_bytes2(MODE));
  uint64_t* empty = full + kStages2;
  uint64_t* tfull = empty + kStages2;   // [2]
  uint64_t* tempty = tfull + 2;         // [2] (used in the leader)
  uint64_t* drain = tempty + 2;         // [1]
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const PathArgs& p = ua.p;
  const Dims& d = p.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages2; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], 2 * epi_warps2(MODE));
    }
    mbar_init(drain, 1);
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmA0);
    tma_prefetch_desc(&tmA1);
    tma_prefetch_desc(&tmB);
    tma_prefetch_desc(&tmS);
  }
  if (warp == 2) {
    tmem_alloc_pair(tmem_slot, kTmemCols);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();   // barrier inits and the TMEM address are visible in both CTAs
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int n_m = min(*p.n_tiles, d.tiles_max);
  const int n_mp = (n_m + 1) / 2;
  const int per_grp = n_mp * ua.n_tiles_n;
  const int total = SPARSE ? ua.sp.plan[0] * ua.n_tiles_n : p.gp * per_grp;
  const int pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;
  auto decode = [&](int t) {
    Work w;
    if (SPARSE) {
      const int pe = t / ua.n_tiles_n;
      w.n = t - pe * ua.n_tiles_n;
      const SparsePair sp = ua.sp.pairs[pe];
      w.gl = sp.vg / d.E;
      w.em = sp.vg - w.gl * d.E;
      w.grp = p.g0 + w.gl;
      w.m_own = 0;
      w.p_own = sp.p0 + static_cast<int>(rank) * UM;
      w.rows_own = rank ? sp.rows1 : sp.rows0;
      w.live = w.rows_own > 0;
    } else {
      w.gl = t / per_grp;
      const int rem = t - w.gl * per_grp;
      const int mp = rem / ua.n_tiles_n;
      w.n = rem - mp * ua.n_tiles_n;
      w.grp = p.g0 + w.gl;
      w.m_own = 2 * mp + static_cast<int>(rank);
      w.em = 0;
      w.p_own = 0;
      w.rows_own = 0;
      w.live = w.m_own < n_m;
    }
    return w;
  };

  uint32_t issued_mask = 0, issue_parity = 0;
  bool mma_issued = false;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer (both CTAs)
      int stage = 0;
      uint32_t phase = 0;
      for (int t = pair; t < total; t += n_pairs) {
        const Work w = decode(t);
        const int gl = w.gl, n = w.n, grp = w.grp, m_own = w.m_own;
        TileInfo ti;
        GroupInfo gi;
        if ((MODE == 1 || MODE == 3) && !SPARSE) {
          gi = p.groups[grp];
          if (m_own < n_m) {
            ti = p.tiles[m_own];
          } else {   // no such tile: load any in-bounds rows; they are never stored
            ti.b = 0;
            ti.s0 = 0;
          }
        }
        bool ok = true;
        for (int kb = 0; kb < ua.nk; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, p.wait_limit)) { ok = false; break; }
          if (leader) mbar_arrive_expect_tx(&full[stage], 2 * kStageBytes2);
          const uint32_t bar = leader_addr(&full[stage]);
          const int b_row = grp * ua.b_rows + (MODE == 1 ? w.em * d.H : 0) + n * UN +
                            static_cast<int>(rank) * (UN / 2);
          if (MODE == 3) {   // projection: the translated activation rows of slot gl
            tma_load_2d_pair(sA + stage * kABytes2, &tmA0, bar, kb * UK,
                             (gl * d.B + ti.b) * d.S + ti.s0);
            tma_load_2d_pair(sB + stage * kBBytes2, &tmB, bar, kb * UK, b_row);
          } else if (MODE == 1 && SPARSE) {   // packed rows: [H_s][R][d_s]
            const int k = kb * UK, h = k / d.d_s, d0 = k - h * d.d_s;
            tma_load_2d_pair(sA + stage * kABytes2, &tmA0, bar, d0, h * ua.sp.R + w.p_own);
            tma_load_2d_pair(sB + stage * kBBytes2, &tmB, bar, kb * UK, b_row);
          } else if (MODE == 1) {
            const int k = kb * UK, h = k / d.d_s, d0 = k - h * d.d_s;
            tma_load_2d_pair(sA + stage * kABytes2, gi.x ? &tmA1 : &tmA0, bar, d0,
                             ((gi.src_layer * d.B + ti.b) * d.H_s + h) * d.S + ti.s0);
            tma_load_2d_pair(sB + stage * kBBytes2, &tmB, bar, kb * UK, b_row);
          } else if (kb < ua.nk - 1) {   // A2 x W2cat (sparse: the expert's K range of W2cat)
            if (SPARSE)
              tma_load_3d_pair(sA + stage * kABytes2, &tmA0, bar, kb * UK, w.p_own, 0);
            else
              tma_load_3d_pair(sA + stage * kABytes2, &tmA0, bar, kb * UK, m_own * UM, gl);
            tma_load_2d_pair(sB + stage * kBBytes2, &tmB, bar, w.em * d.H + kb * UK, b_row);
          } else {                       // last K block: gate16 x b2t (the combine biases)
            if (SPARSE)
              tma_load_3d_pair(sA + stage * kABytes2, &tmA1, bar, 0, w.p_own, 0);
            else
              tma_load_3d_pair(sA + stage * kABytes2, &tmA1, bar, 0, m_own * UM, grp);
            tma_load_2d_pair(sB + stage * kBBytes2, &tmS, bar, 0, b_row);
          }
          issued_mask |= 1u << stage;
          issue_parity = (issue_parity & ~(1u << stage)) | (phase << stage);
          if (++stage == kStages2) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
      }
    }
  } else if (warp == 1) {
    if (lane == 0 && leader) {
      // ------------------------------------------------ MMA issuer (leader)
      const uint32_t idesc = MODE == 2 ? idesc_f16_f32(2 * UM, UN) : idesc_bf16_f32(2 * UM, UN);
      int stage = 0, acc = 0;
      uint32_t phase = 0, acc_phase = 0;
      for (int t = pair; t < total; t += n_pairs) {
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, p.wait_limit)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * UN);
        bool ok = true;
        for (int kb = 0; kb < ua.nk; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag, p.wait_limit)) { ok = false; break; }
          tc_fence_after();
          const uint64_t adesc = sdesc_k_sw128(smem_u32(sA + stage * kABytes2));
          const uint64_t bdesc = sdesc_k_sw128(smem_u32(sB + stage * kBBytes2));
#pragma unroll
          for (int k = 0; k < UK / 16; ++k)   // +32 bytes of K per step = +2 in the address field
            umma_pair(d_tmem, adesc + 2 * k, bdesc + 2 * k, idesc, (kb | k) != 0);
          mma_issued = true;
          umma_commit_pair(&empty[stage]);
          if (++stage == kStages2) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        umma_commit_pair(&tfull[acc]);
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
      }
    }
  } else if (warp >= 4) {
    // ------------------------------------------------ epilogue (both CTAs)
    const int e = warp - 4;
    const int q = e & 3;
    int acc = 0;
    uint32_t acc_phase = 0;
    // GEMM1: the gate value of this thread's row for the next tile, fetched ahead
    auto tile_coords = [&](int tt, int& gl, int& grp, int& m_own, int& n) {
      gl = tt / per_grp;
      const int rem = tt - gl * per_grp;
      const int mp = rem / ua.n_tiles_n;
      n = rem - mp * ua.n_tiles_n;
      grp = p.g0 + gl;
      m_own = 2 * mp + static_cast<int>(rank);
    };
    float gate_next = 0.f;
    if (MODE == 1 && !SPARSE && pair < total) {
      int gl, grp, m_own, n;
      tile_coords(pair, gl, grp, m_own, n);
      if (m_own < n_m) gate_next = gemm1_prefetch(p, q, lane, grp, m_own, n * UN, (e >> 2) * 128);
    }
    for (int t = pair; t < total; t += n_pairs) {
      const float gate_cur = gate_next;
      if (MODE == 1 && !SPARSE && t + n_pairs < total) {
        int gl, grp, m_own, n;
        tile_coords(t + n_pairs, gl, grp, m_own, n);
        if (m_own < n_m) gate_next = gemm1_prefetch(p, q, lane, grp, m_own, n * UN, (e >> 2) * 128);
      }
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&tfull[acc], acc_phase, abort_flag, p.wait_limit) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      tc_fence_after();
      const Work w = decode(t);
      const int gl = w.gl, n = w.n, grp = w.grp, m_own = w.m_own;
      const uint32_t tbase = tmem_base + static_cast<uint32_t>(acc * UN) +
                             (static_cast<uint32_t>(q * 32) << 16);
      if (w.live) {
        if (MODE == 1 && SPARSE)   // bias of expert em; A2 rows are the packed rows
          epilogue_gemm1(p, &tmS, tbase, sOut + e * kStoreTileBytes, q, lane, grp,
                         w.em * d.H + n * UN, n * UN, w.p_own, 0, (e >> 2) * 128, 2,
                         ua.sp.gatep[w.p_own + q * 32 + lane]);
        else if (MODE == 1)   // 8 warps: this warp owns columns 128 * (e / 4) .. +127
          epilogue_gemm1(p, &tmS, tbase, sOut + e * kStoreTileBytes, q, lane, grp, n * UN,
                         n * UN, m_own * UM, gl, (e >> 2) * 128, 2, gate_cur);
        else if (MODE == 3)
          epilogue_proj(p, tbase, q, lane, grp, m_own, n * UN);
        else if (SPARSE)
          epilogue_gemm2_sparse(p, ua.sp, tbase, q, lane, gl, w.p_own, w.rows_own, n * UN);
        else             // 4 warps: all 256 columns
          epilogue_gemm2(p, tbase, q, lane, grp, m_own, n * UN, 0, UN / 32);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(&tempty[acc], 0);
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
    if (MODE == 1 && lane == 0) bulk_wait_group<0>();
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    // Unwinding after a timed-out wait (bounded): copies this CTA started
    // complete on the leader's barriers, so give them time to land; the
    // leader also waits for its issued MMAs.
    if (warp == 0 && lane == 0 && issued_mask) {
      if (leader) {
        for (int s = 0; s < kStages2; ++s)
          if ((issued_mask >> s) & 1u) {
            const uint32_t a = smem_u32(&full[s]);
            const long long t0 = clock64();
            while (!mbar_try_wait(a, (issue_parity >> s) & 1u) &&
                   clock64() - t0 < p.wait_limit) {
            }
          }
      } else {
        spin_cycles(20000000LL);
      }
    }
    if (warp == 1 && lane == 0 && leader && mma_issued) {
      umma_commit_pair(drain);
      const uint32_t a = smem_u32(drain);
      const long long t0 = clock64();
      while (!mbar_try_wait(a, 0) && clock64() - t0 < p.wait_limit) {
      }
    }
    __syncthreads();
  }
  tc_fence_before();
  cluster_sync();   // the leader's MMAs no longer read this CTA's shared memory or TMEM
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kTmemCols);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicOr(p.status, kStatusTimeout);
}

template <int MODE, bool SPARSE>
cudaError_t launch_umma2(const PathArgs& a, const SparseArgs* sp, const CUtensorMap& A0,
                         const CUtensorMap& A1, const CUtensorMap& B, const CUtensorMap& S, int nk,
                         int n_tiles_n, int b_rows, int num_sms, cudaStream_t st) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(umma2_gemm_kernel<MODE, SPARSE>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         smem_bytes2(MODE));
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  Umma2Args ua{};
  ua.p = a;
  if (sp) ua.sp = *sp;
  ua.nk = nk;
  ua.n_tiles_n = n_tiles_n;
  ua.b_rows = b_rows;
  const long long pairs =
      static_cast<long long>(SPARSE ? sp->max_pairs : a.gp * ((a.d.tiles_max + 1) / 2)) *
      n_tiles_n;
  const long long max_pairs = num_sms / 2;
  const int grid = 2 * static_cast<int>(pairs < max_pairs ? pairs : max_pairs);
  if (grid <= 0) return cudaSuccess;
  umma2_gemm_kernel<MODE, SPARSE>
      <<<grid, threads2(MODE), smem_bytes2(MODE), st>>>(A0, A1, B, S, ua);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_umma2_gemm1(const PathArgs& a, const CUtensorMap& tmK, const CUtensorMap& tmV,
                               const CUtensorMap& tmW1h, const CUtensorMap& tmA2st, int num_sms,
                               cudaStream_t st) {
  return launch_umma2<1, false>(a, nullptr, tmK, tmV, tmW1h, tmA2st, a.d.Ds / UK, a.d.EH / UN,
                                a.d.EH, num_sms, st);
}

// Sparse GEMM1: A = packed rows (zp), B = the bucket expert's H rows of W1cat,
// stores A2p rows; n runs over the expert's H / 256 column tiles.
cudaError_t launch_umma2_sparse_gemm1(const PathArgs& a, const SparseArgs& s,
                                      const CUtensorMap& tmZp, const CUtensorMap& tmW1h,
                                      const CUtensorMap& tmA2pst, int num_sms, cudaStream_t st) {
  return launch_umma2<1, true>(a, &s, tmZp, tmZp, tmW1h, tmA2pst, a.d.Ds / UK, a.d.H / UN, a.d.EH,
                               num_sms, st);
}

// Sparse GEMM2: A = A2p rows (K = H) and gate16p for the bias block, B = the
// expert's K range of W2cat and b2t; fp32 slot rows into ybuf.
cudaError_t launch_umma2_sparse_gemm2(const PathArgs& a, const SparseArgs& s,
                                      const CUtensorMap& tmA2p, const CUtensorMap& tmW2h,
                                      const CUtensorMap& tmG16p, const CUtensorMap& tmB2th,
                                      int num_sms, cudaStream_t st) {
  return launch_umma2<2, true>(a, &s, tmA2p, tmG16p, tmW2h, tmB2th, a.d.H / UK + 1, a.d.Dt / UN,
                               a.d.Dt, num_sms, st);
}

// GEMM2's map slots: A0 = A2, A1 = gate16, B = W2cat half, S = b2t half (last K block).
cudaError_t launch_umma2_gemm2(const PathArgs& a, const CUtensorMap& tmA2, const CUtensorMap& tmW2h,
                               const CUtensorMap& tmG16, const CUtensorMap& tmB2th, int num_sms,
                               cudaStream_t st) {
  return launch_umma2<2, false>(a, nullptr, tmA2, tmG16, tmW2h, tmB2th, a.d.EH / UK + 1,
                                a.d.Dt / UN, a.d.Dt, num_sms, st);
}

// MoT-h projection: A = translated activations [slots * B * S][d_at] (box
// 64 x 128), B = [W^K; W^V] per group [G * 2 D_t][d_at] (box 64 x 128).
cudaError_t launch_umma2_proj(const PathArgs& a, const CUtensorMap& tmAct,
                              const CUtensorMap& tmWkv, int act_width, int num_sms,
                              cudaStream_t st) {
  return launch_umma2<3, false>(a, nullptr, tmAct, tmAct, tmWkv, tmWkv, act_width / UK,
                                2 * a.d.Dt / UN, 2 * a.d.Dt, num_sms, st);
}

}  // namespace mot
