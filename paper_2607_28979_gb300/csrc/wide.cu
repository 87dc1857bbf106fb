// On-chip translation for D_t = 512 (schedule 4): GEMM1 -> GELU * gate ->
// GEMM2 with the hidden activations kept in shared memory, for translators
// whose output is too wide for one CTA pair's tensor memory.
//
// A pair's accumulator for 256 token rows and D_t = 512 output columns would
// fill all 512 TMEM columns of each SM, leaving none for GEMM1. So a cluster
// of four CTAs -- two CTA pairs -- shares one 256-row pair tile (token tiles
// 2 mp and 2 mp + 1 of one (target layer, K/V) group): pair p accumulates
// output columns [256 p, 256 p + 256) of Y = A2 * W2cat^T in TMEM (256
// columns) and keeps two 128-column GEMM1 accumulators. The concatenated
// hidden dimension E*H is walked in 128-column chunks; chunk c's GEMM1
//   U_c = Z * W1cat[128 c .. 128 c + 127]^T     (M = 256, N = 128, K = D_s)
// runs on pair c % 2 only, whose epilogue writes A2_c = fp16(GELU(U_c + b1) *
// gtilde_m) into its pair's shared-memory slot in the tcgen05 operand layout,
// and each epilogue warp copies its 4 KB of rows (cp.async.bulk, shared::cta ->
// shared::cluster) into the same slot of the other pair's CTA that holds the
// same token rows. Both pairs run
//   Y_p += A2_c * W2cat[256 p .. 256 p + 255, 128 c .. 128 c + 127]^T
// for every chunk; after the last chunk, Y_p += gate16 * b2t adds the
// gate-weighted biases sum_m gtilde_m b2_m (Def. 3.1) as one more K block,
// and the epilogue stores Y_p as bf16 into the target cache. A2 never leaves
// the chip, and each pair does half of both GEMMs' tensor-core work.
//
// Shared memory per CTA: a ring of 4 stages of 24 KB (a 16 KB block of this
// CTA's 128 source rows and the 8 KB block of its half of the chunk's W1
// rows, K = 64 each), a ring of 2 W2 stages of 16 KB (this CTA's 128 of its
// pair's 256 rows of W2cat, K = 64; the tile's b2t block takes one stage
// too), 2 A2 slots of 32 KB and 16 KB of gate16 rows. Slot q holds the chunks
// that pair q computes (c % 2 == q), so a slot is only ever written by one
// pair's epilogue, which waits for every use of it in order: no barrier phase
// of a slot can pass unobserved by its writer.
// TMEM per CTA (512 columns): acc2 in [0, 256), acc1[0] in [256, 384),
// acc1[1] in [384, 512).
//
// Roles per CTA (13 warps):
//   warp 0 lane 0      TMA loads of the source / W1 ring (own chunks only);
//   warp 1 lane 0      TMA loads of the W2 ring, the b2t block and gate16;
//   warp 2             TMEM allocation of the pair, then (lane 0) the relay:
//                      for an own chunk it waits for this CTA's epilogue and
//                      tells the pair leader the slot is full; for the other
//                      pair's chunk it waits for the copies to land and tells
//                      the pair leader;
//   warp 3 (leader)    GEMM1 issue (one elected lane);
//   warp 4 (leader)    GEMM2 and bias issue (one elected lane); every GEMM2
//                      commit arrives on slot-free barriers in all four CTAs;
//   warps 5..12        epilogue: warp 5 + 4 hh + q owns rows 32 q .. 32 q + 31,
//                      chunk columns 64 hh .. 64 hh + 63 and output columns
//                      128 hh .. 128 hh + 127 of its pair's 256.
// Every wait is bounded; a timeout unwinds every role and raises
// kStatusTimeout.
#include "umma_common.cuh"

namespace mot {
namespace {

constexpr int kWPairs = 2;                    // CTA pairs per cluster (D_t = 256 * kWPairs)
constexpr int kWCtas = 2 * kWPairs;
constexpr int kWChunk = 128;                  // hidden columns per chunk
constexpr int kWBlk = UM * UK * 2;            // 16 KB: 128 rows x 64 K, 16-bit
constexpr int kWW1Blk = (kWChunk / 2) * UK * 2;   // 8 KB: 64 rows x 64 K
constexpr int kWStage1 = kWBlk + kWW1Blk;     // source block + W1 block
constexpr int kWStages1 = 4;
constexpr int kWStages2 = 2;
constexpr int kWSlots = kWPairs;              // slot q: the chunks pair q computes
constexpr int kWSlotBytes = 2 * kWBlk;        // 128 rows x 128 K
constexpr int kWOffW2 = kWStages1 * kWStage1;
constexpr int kWOffA2 = kWOffW2 + kWStages2 * kWBlk;
constexpr int kWOffG = kWOffA2 + kWSlots * kWSlotBytes;
constexpr int kWOffBar = kWOffG + kWBlk;
constexpr int kWEpiWarps = 8;
constexpr int kWThreads = 32 * (5 + kWEpiWarps);
constexpr int kWSmemBytes = kWOffBar + 512 + 1024;
static_assert(kWSmemBytes <= 232448, "shared memory budget");
static_assert(kWOffW2 % 1024 == 0 && kWOffA2 % 1024 == 0 && kWOffG % 1024 == 0, "alignment");
constexpr uint32_t kWAcc1Col = UN;            // acc1[b] at column 256 + 128 b
constexpr uint32_t kWTmemAlloc = 512;
constexpr uint32_t kWSlotTx = kWSlotBytes;    // bytes of one slot's copies (8 x 4 KB)
constexpr uint32_t kWPieceBytes = 32 * 128;   // one epilogue warp's rows of one K block

struct WBars {
  uint64_t zfull[kWStages1], zempty[kWStages1];   // source / W1 ring
  uint64_t w2full[kWStages2], w2empty[kWStages2]; // W2 ring
  uint64_t gfull, gempty;                         // gate16 rows of the tile
  uint64_t a1full[2];     // GEMM1 of an own chunk done (commit, both CTAs of the pair)
  uint64_t acc1free[2];   // its acc1 read out (pair leader; 2 x 8 warp arrivals)
  uint64_t epidone[kWSlots];  // this CTA's A2 rows of an own chunk written (8 warp arrivals)
  uint64_t rx[kWSlots];       // the other pair's chunk copied in (1 arrival + 8 x 4 KB)
  uint64_t a2full[kWSlots];   // both CTAs' rows of a chunk present (pair leader; 2 arrivals)
  uint64_t slotfree[kWSlots]; // every pair's GEMM2 of the slot's chunk done (kWPairs commits;
                              // waited only by the slot's writers, at every use)
  uint64_t acc2full;      // a tile's GEMM2 + bias done (commit, both CTAs of the pair)
  uint64_t acc2empty;     // acc2 read out (pair leader; 2 x 8 warp arrivals)
  uint64_t drain, drain2;
  uint32_t tmem_slot;
  int abort_flag;
};
static_assert(sizeof(WBars) <= 512, "barrier block");

struct WideArgs {
  PathArgs p;
  int32_t nk1;   // 64-wide K blocks of GEMM1 (D_s / 64)
  int32_t nc;    // chunks per tile (E*H / 128)
};

__device__ __forceinline__ void wide_spin(long long cycles) {
  const long long t0 = clock64();
  while (clock64() - t0 < cycles) {
  }
}

// Row r's 16-byte chunks 4 s .. 4 s + 3 of a 64-wide K block at `blk` (128B swizzle).
__device__ __forceinline__ void wide_store_a2(uint32_t blk, int r, int s, const uint32_t (&pk)[16]) {
  const uint32_t row = blk + static_cast<uint32_t>(r * 128);
#pragma unroll
  for (int v = 0; v < 4; ++v)
    st_shared_v4(row + static_cast<uint32_t>(((4 * s + v) ^ (r & 7)) << 4), pk[4 * v],
                 pk[4 * v + 1], pk[4 * v + 2], pk[4 * v + 3]);
}

__device__ __forceinline__ void wide_gelu_cols(const uint32_t (&acc)[32], const uint4 (&b)[4],
                                               __half2 half_g, uint32_t (&pk)[16]) {
#pragma unroll
  for (int v = 0; v < 4; ++v) {
    const uint32_t bw[4] = {b[v].x, b[v].y, b[v].z, b[v].w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const int j = v * 8 + 2 * k;
      pk[4 * v + k] = gelu_gate_pair(acc[j], acc[j + 1], bw[k], half_g);
    }
  }
}

__device__ __forceinline__ void wide_store_out(const uint32_t (&acc)[32], __nv_bfloat16* o) {
  uint4* o4 = reinterpret_cast<uint4*>(o);
#pragma unroll
  for (int v = 0; v < 4; ++v)
    o4[v] = make_uint4(pack_bf16x2(__uint_as_float(acc[8 * v + 0]), __uint_as_float(acc[8 * v + 1])),
                       pack_bf16x2(__uint_as_float(acc[8 * v + 2]), __uint_as_float(acc[8 * v + 3])),
                       pack_bf16x2(__uint_as_float(acc[8 * v + 4]), __uint_as_float(acc[8 * v + 5])),
                       pack_bf16x2(__uint_as_float(acc[8 * v + 6]), __uint_as_float(acc[8 * v + 7])));
}

__global__ void __cluster_dims__(kWCtas, 1, 1) __launch_bounds__(kWThreads, 1)
    wide_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                const __grid_constant__ CUtensorMap tmW1q, const __grid_constant__ CUtensorMap tmW2h,
                const __grid_constant__ CUtensorMap tmG16,
                const __grid_constant__ CUtensorMap tmB2th, const WideArgs wa) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sZW = smem;
  uint8_t* sW2 = smem + kWOffW2;
  uint8_t* sA2 = smem + kWOffA2;
  uint8_t* sG = smem + kWOffG;
  WBars* bars = reinterpret_cast<WBars*>(smem + kWOffBar);
  volatile int* abort_flag = &bars->abort_flag;

  const PathArgs& p = wa.p;
  const Dims& d = p.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const uint32_t half = rank & 1u;            // which 128 rows of the pair tile
  const uint32_t pr = rank >> 1;              // which CTA pair: output columns 256 pr ..
  const uint32_t lead = rank & ~1u;           // the pair's leader CTA
  const bool leader = half == 0;
  const uint16_t pair_mask = static_cast<uint16_t>(3u << (2 * pr));
  const uint16_t all_mask = static_cast<uint16_t>((1u << kWCtas) - 1u);
  const int nc = wa.nc, nk1 = wa.nk1;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kWStages1; ++i) {
      mbar_init(&bars->zfull[i], 1);
      mbar_init(&bars->zempty[i], 1);
    }
    for (int i = 0; i < kWStages2; ++i) {
      mbar_init(&bars->w2full[i], 1);
      mbar_init(&bars->w2empty[i], 1);
    }
    mbar_init(&bars->gfull, 1);
    mbar_init(&bars->gempty, 1);
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->a1full[i], 1);
      mbar_init(&bars->acc1free[i], 2 * kWEpiWarps);
    }
    for (int i = 0; i < kWSlots; ++i) {
      mbar_init(&bars->epidone[i], kWEpiWarps);
      mbar_init(&bars->rx[i], 1);
      mbar_init(&bars->a2full[i], 2);
      mbar_init(&bars->slotfree[i], kWPairs);
    }
    mbar_init(&bars->acc2full, 1);
    mbar_init(&bars->acc2empty, 2 * kWEpiWarps);
    mbar_init(&bars->drain, 1);
    mbar_init(&bars->drain2, 1);
    bars->abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
    tma_prefetch_desc(&tmW1q);
    tma_prefetch_desc(&tmW2h);
    tma_prefetch_desc(&tmG16);
    tma_prefetch_desc(&tmB2th);
  }
  if (warp == 2) {
    tmem_alloc_pair(&bars->tmem_slot, kWTmemAlloc);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();   // barrier inits and TMEM addresses visible in all four CTAs
  tc_fence_after();
  const uint32_t tmem_base = bars->tmem_slot;

  const int n_m = min(*p.n_tiles, d.tiles_max);
  const int n_mp = (n_m + 1) / 2;
  const int total = p.gp * n_mp;
  const int cl = blockIdx.x / kWCtas, n_cl = gridDim.x / kWCtas;
  // own chunks of a tile: c = pr, pr + kWPairs, ...
  const int n_own = (nc - static_cast<int>(pr) + kWPairs - 1) / kWPairs;

  // unwinding state: loads in flight (bit i: zfull 0-2, w2full 3-4, gfull 5)
  uint32_t pend_mask = 0, pend_par = 0;
  bool mma_issued = false;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ source / W1 loads (own chunks)
      int s = 0;
      uint32_t ph = 0;
      bool ok = true;
      for (int t = cl; ok && t < total; t += n_cl) {
        const int gl = t / n_mp, mp = t - gl * n_mp;
        const int grp = p.g0 + gl;
        const GroupInfo gi = p.groups[grp];
        const int m_own = 2 * mp + static_cast<int>(half);
        TileInfo ti;
        if (m_own < n_m) {
          ti = p.tiles[m_own];
        } else {   // no such tile: any in-bounds rows; they are never stored
          ti.b = 0;
          ti.s0 = 0;
        }
        const int zrow = ((gi.src_layer * d.B + ti.b) * d.H_s) * d.S + ti.s0;
        for (int c = static_cast<int>(pr); ok && c < nc; c += kWPairs) {
          const int wrow = grp * d.EH + c * kWChunk + static_cast<int>(half) * (kWChunk / 2);
          for (int kb = 0; kb < nk1; ++kb) {
            if (!mbar_wait(&bars->zempty[s], ph ^ 1u, abort_flag, p.wait_limit)) { ok = false; break; }
            if (leader) mbar_arrive_expect_tx(&bars->zfull[s], 2 * kWStage1);
            const uint32_t bar = leader_addr(&bars->zfull[s]);
            const int kk = kb * UK, h = kk / d.d_s, d0 = kk - h * d.d_s;
            uint8_t* st = sZW + s * kWStage1;
            tma_load_2d_pair(st, gi.x ? &tmV : &tmK, bar, d0, zrow + h * d.S);
            tma_load_2d_pair(st + kWBlk, &tmW1q, bar, kk, wrow);
            pend_mask |= 1u << s;
            pend_par = (pend_par & ~(1u << s)) | (ph << s);
            if (++s == kWStages1) { s = 0; ph ^= 1u; }
          }
        }
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------ W2 ring, b2t and gate16 loads
      int s = 0;
      uint32_t ph = 0, k = 0;
      bool ok = true;
      const int wrow0 = static_cast<int>(pr) * UN + static_cast<int>(half) * UM;
      auto w2_stage = [&]() -> uint32_t {
        if (!mbar_wait(&bars->w2empty[s], ph ^ 1u, abort_flag, p.wait_limit)) return 0;
        if (leader) mbar_arrive_expect_tx(&bars->w2full[s], 2 * kWBlk);
        return leader_addr(&bars->w2full[s]);
      };
      auto w2_next = [&]() {
        pend_mask |= 1u << (kWStages1 + s);
        pend_par = (pend_par & ~(1u << (kWStages1 + s))) | (ph << (kWStages1 + s));
        if (++s == kWStages2) { s = 0; ph ^= 1u; }
      };
      for (int t = cl; ok && t < total; t += n_cl, ++k) {
        const int gl = t / n_mp, mp = t - gl * n_mp;
        const int grp = p.g0 + gl;
        const int m_own = 2 * mp + static_cast<int>(half);
        for (int c = 0; ok && c < nc; ++c)
          for (int kb = 0; kb < 2; ++kb) {
            const uint32_t bar = w2_stage();
            if (!bar) { ok = false; break; }
            tma_load_2d_pair(sW2 + s * kWBlk, &tmW2h, bar, c * kWChunk + kb * UK,
                             grp * d.Dt + wrow0);
            w2_next();
          }
        if (!ok) break;
        // the tile's bias block: B = b2t rows of this pair's columns, A = gate16 rows
        {
          const uint32_t bar = w2_stage();
          if (!bar) break;
          tma_load_2d_pair(sW2 + s * kWBlk, &tmB2th, bar, 0, grp * d.Dt + wrow0);
          w2_next();
        }
        if (!mbar_wait(&bars->gempty, (k & 1u) ^ 1u, abort_flag, p.wait_limit)) break;
        if (leader) mbar_arrive_expect_tx(&bars->gfull, 2 * kWBlk);
        tma_load_3d_pair(sG, &tmG16, leader_addr(&bars->gfull), 0, m_own * UM, grp);
        pend_mask |= 1u << (kWStages1 + kWStages2);
        pend_par = (pend_par & ~(1u << (kWStages1 + kWStages2))) |
                   ((k & 1u) << (kWStages1 + kWStages2));
      }
    }
  } else if (warp == 2) {
    if (lane == 0) {
      // ------------------------------------------------ relay between the pairs
      // per slot: uses whose epilogue (own) or copies (other pair) were waited for
      uint32_t use_n[kWSlots] = {};
      bool ok = true;
      for (int t = cl; ok && t < total; t += n_cl) {
        for (int c = 0; c < nc; ++c) {
          const int slot = c % kWPairs;
          if (slot == static_cast<int>(pr)) {
            if (!mbar_wait(&bars->epidone[slot], use_n[slot] & 1u, abort_flag, p.wait_limit)) {
              ok = false;
              break;
            }
          } else {
            mbar_arrive_expect_tx(&bars->rx[slot], kWSlotTx);
            if (!mbar_wait_cluster(&bars->rx[slot], use_n[slot] & 1u, abort_flag, p.wait_limit)) {
              ok = false;
              break;
            }
          }
          ++use_n[slot];
          mbar_arrive_release_cluster(&bars->a2full[slot], lead);
        }
      }
    }
  } else if ((warp == 3 || warp == 4) && leader) {
    // ------------------------------------------------ MMA issuers (pair leader)
    auto wait_all = [&](uint64_t* bar, uint32_t parity) -> bool {
      const bool r = mbar_wait(bar, parity, abort_flag, p.wait_limit);
      return __all_sync(0xffffffffu, r) != 0;
    };
    auto wait_all_cluster = [&](uint64_t* bar, uint32_t parity) -> bool {
      const bool r = mbar_wait_cluster(bar, parity, abort_flag, p.wait_limit);
      return __all_sync(0xffffffffu, r) != 0;
    };
    bool ok = true;
    if (warp == 3) {
      // GEMM1 of own chunks: acc1[j % 2] = Z * W1cat[chunk]^T
      constexpr uint32_t idesc1 = idesc_bf16_f32(2 * UM, kWChunk);
      int s = 0;
      uint32_t ph = 0, j = 0;
      for (int t = cl; ok && t < total; t += n_cl) {
        for (int o = 0; ok && o < n_own; ++o, ++j) {
          const uint32_t b = j & 1u;
          if (j >= 2) ok = wait_all(&bars->acc1free[b], ((j >> 1) & 1u) ^ 1u);
          if (!ok) break;
          const uint32_t d1 = tmem_base + kWAcc1Col + b * kWChunk;
          for (int kb = 0; kb < nk1; ++kb) {
            if (!wait_all(&bars->zfull[s], ph)) { ok = false; break; }
            tc_fence_after();
            const uint32_t za = smem_u32(sZW + s * kWStage1);
            if (elect_one()) {
              const uint64_t zdesc = sdesc_k_sw128(za), wdesc = sdesc_k_sw128(za + kWBlk);
#pragma unroll
              for (int kk = 0; kk < UK / 16; ++kk)   // +32 bytes of K = +2 in the address field
                umma_pair(d1, zdesc + 2 * kk, wdesc + 2 * kk, idesc1, (kb | kk) != 0);
              umma_commit_mask(&bars->zempty[s], pair_mask);
            }
            __syncwarp();
            mma_issued = true;
            if (++s == kWStages1) { s = 0; ph ^= 1u; }
          }
          if (!ok) break;
          if (elect_one()) umma_commit_mask(&bars->a1full[b], pair_mask);
          __syncwarp();
        }
      }
    } else {
      // GEMM2 of every chunk into acc2, then the bias block
      constexpr uint32_t idesc2 = idesc_f16_f32(2 * UM, UN);
      int s = 0;
      uint32_t ph = 0, k = 0;
      uint32_t use_n[kWSlots] = {};
      for (int t = cl; ok && t < total; t += n_cl, ++k) {
        for (int c = 0; ok && c < nc; ++c) {
          const int slot = c % kWPairs;
          ok = wait_all_cluster(&bars->a2full[slot], use_n[slot] & 1u);
          ++use_n[slot];
          if (ok && c == 0) ok = wait_all(&bars->acc2empty, (k & 1u) ^ 1u);
          if (!ok) break;
          const uint32_t aa = smem_u32(sA2 + slot * kWSlotBytes);
          for (int kb = 0; kb < 2; ++kb) {
            if (!wait_all(&bars->w2full[s], ph)) { ok = false; break; }
            tc_fence_after();
            if (elect_one()) {
              const uint64_t adesc = sdesc_k_sw128(aa + kb * kWBlk);
              const uint64_t bdesc = sdesc_k_sw128(smem_u32(sW2 + s * kWBlk));
#pragma unroll
              for (int kk = 0; kk < UK / 16; ++kk)
                umma_pair(tmem_base, adesc + 2 * kk, bdesc + 2 * kk, idesc2, (c | kb | kk) != 0);
              umma_commit_mask(&bars->w2empty[s], pair_mask);
            }
            __syncwarp();
            mma_issued = true;
            if (++s == kWStages2) { s = 0; ph ^= 1u; }
          }
          if (!ok) break;
          // the slot is free once every pair's GEMM2 of this chunk is done
          if (elect_one()) umma_commit_mask(&bars->slotfree[slot], all_mask);
          __syncwarp();
        }
        if (!ok) break;
        if (!wait_all(&bars->gfull, k & 1u)) break;
        if (!wait_all(&bars->w2full[s], ph)) break;
        tc_fence_after();
        if (elect_one()) {
          const uint64_t gdesc = sdesc_k_sw128(smem_u32(sG));
          const uint64_t bdesc = sdesc_k_sw128(smem_u32(sW2 + s * kWBlk));
#pragma unroll
          for (int kk = 0; kk < UK / 16; ++kk)
            umma_pair(tmem_base, gdesc + 2 * kk, bdesc + 2 * kk, idesc2, 1u);
          umma_commit_mask(&bars->w2empty[s], pair_mask);
          umma_commit_mask(&bars->gempty, pair_mask);
          umma_commit_mask(&bars->acc2full, pair_mask);
        }
        __syncwarp();
        if (++s == kWStages2) { s = 0; ph ^= 1u; }
      }
    }
  } else if (warp >= 5) {
    // ------------------------------------------------ epilogue (every CTA)
    const int e = warp - 5, q = warp & 3, hh = e >> 2;   // q: the TMEM lane quarter warp % 4 may access
    const int r = q * 32 + lane;
    const uint32_t tq = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
    const __half* b1h = static_cast<const __half*>(p.b1h);
    uint32_t j = 0, k = 0;   // j: own chunks so far = uses of this pair's slot
    bool ok = true;
    const int slot = static_cast<int>(pr);
    const uint32_t peer = (rank ^ 2u);   // the other pair's CTA with the same rows (2 pairs)
    for (int t = cl; ok && t < total; t += n_cl, ++k) {
      const int gl = t / n_mp, mp = t - gl * n_mp;
      const int grp = p.g0 + gl;
      const int m_own = 2 * mp + static_cast<int>(half);
      const bool valid = m_own < n_m;
      const float* grow =
          p.gate + (static_cast<size_t>(grp) * d.tpad + static_cast<size_t>(m_own) * UM + r) * d.E;
      const uint4* bias4 = reinterpret_cast<const uint4*>(b1h + static_cast<size_t>(grp) * d.EH);
      for (int c = static_cast<int>(pr); c < nc; c += kWPairs, ++j) {
        const uint32_t b = j & 1u;
        // this warp's 2 x 32 biases and the row's gate value, fetched before the wait
        uint4 bias[2][4];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
          bias[0][i] = __ldg(bias4 + (c * kWChunk + hh * 64) / 8 + i);
          bias[1][i] = __ldg(bias4 + (c * kWChunk + hh * 64 + 32) / 8 + i);
        }
        const float gate = valid ? __ldg(grow + (c * kWChunk) / d.H) : 0.f;
        int w = 1;
        if (lane == 0) w = mbar_wait(&bars->a1full[b], (j >> 1) & 1u, abort_flag, p.wait_limit);
        if (!__shfl_sync(0xffffffffu, w, 0)) { ok = false; break; }
        tc_fence_after();
        uint32_t pa[16], pb[16];
        {
          uint32_t ra[32], rb[32];
          tmem_ld_32x32b_x32(tq + kWAcc1Col + b * kWChunk + hh * 64, ra);
          tmem_ld_32x32b_x32(tq + kWAcc1Col + b * kWChunk + hh * 64 + 32, rb);
          tmem_ld_wait(ra);
          tmem_ld_wait(rb);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster(&bars->acc1free[b], lead);   // GEMM1(j + 2) may start
          const __half2 hg = __float2half2_rn(0.5f * gate);
          wide_gelu_cols(ra, bias[0], hg, pa);
          wide_gelu_cols(rb, bias[1], hg, pb);
        }
        // every pair's GEMM2 of the slot's previous chunk (use j - 1) must be
        // done reading it, here and in the other pair's CTA this warp copies to
        if (j >= 1) {
          if (lane == 0)
            w = mbar_wait_cluster(&bars->slotfree[slot], (j - 1) & 1u, abort_flag, p.wait_limit);
          if (!__shfl_sync(0xffffffffu, w, 0)) { ok = false; break; }
        }
        uint8_t* piece = sA2 + slot * kWSlotBytes + hh * kWBlk + q * kWPieceBytes;
        const uint32_t a2 = smem_u32(sA2 + slot * kWSlotBytes) + static_cast<uint32_t>(hh * kWBlk);
        wide_store_a2(a2, r, 0, pa);
        wide_store_a2(a2, r, 1, pb);
        fence_proxy_async_smem();   // the MMA and the bulk copy (async proxy) read these stores
        __syncwarp();
        if (lane == 0) {
          bulk_copy_to_cta(piece, piece, kWPieceBytes, &bars->rx[slot], peer);
          mbar_arrive(&bars->epidone[slot]);
        }
      }
      if (!ok) break;
      // output: this pair's columns 256 pr + 128 hh .. + 127 of this warp's rows
      const GroupInfo gi = p.groups[grp];
      TileInfo ti;
      ti.rows = 0;
      if (valid) ti = p.tiles[m_own];
      int w = 1;
      if (lane == 0) w = mbar_wait(&bars->acc2full, k & 1u, abort_flag, p.wait_limit);
      if (!__shfl_sync(0xffffffffu, w, 0)) break;
      tc_fence_after();
      if (valid) {   // warp-uniform: the TMEM loads are warp-collective; stores are per row
        __nv_bfloat16* const dst = static_cast<__nv_bfloat16*>(gi.x ? p.dst[1] : p.dst[0]);
        const size_t s_pos = static_cast<size_t>(ti.s0) + r;
        uint32_t ra[32], rb[32];
#pragma unroll 1
        for (int cc = hh * (UN / 2); cc < (hh + 1) * (UN / 2); cc += 64) {
          tmem_ld_32x32b_x32(tq + cc, ra);
          tmem_ld_32x32b_x32(tq + cc + 32, rb);
          tmem_ld_wait(ra);
          tmem_ld_wait(rb);
          if (r < ti.rows) {
#pragma unroll
            for (int u = 0; u < 2; ++u) {
              const int col = static_cast<int>(pr) * UN + cc + 32 * u;
              const int hd = col / d.d_t, i0 = col - hd * d.d_t;
              __nv_bfloat16* o = dst + ((((static_cast<size_t>(gi.tgt_layer) * d.B + ti.b) * d.H_t +
                                          hd) * d.S + s_pos) * d.d_t + i0);
              wide_store_out(u ? rb : ra, o);
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(&bars->acc2empty, lead);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    // Unwinding after a timed-out wait (bounded): copies this CTA started
    // complete on its pair leader's barriers, so give them time to land; the
    // leader also waits for its issued MMAs.
    if ((warp == 0 || warp == 1) && lane == 0 && pend_mask) {
      if (leader) {
        for (int i = 0; i < kWStages1 + kWStages2 + 1; ++i) {
          if (!((pend_mask >> i) & 1u)) continue;
          uint64_t* fb = i < kWStages1 ? &bars->zfull[i]
                                       : (i < kWStages1 + kWStages2 ? &bars->w2full[i - kWStages1]
                                                                    : &bars->gfull);
          const uint32_t a = smem_u32(fb);
          const long long t0 = clock64();
          while (!mbar_try_wait(a, (pend_par >> i) & 1u) && clock64() - t0 < p.wait_limit) {
          }
        }
      } else {
        wide_spin(20000000LL);
      }
    }
    if ((warp == 3 || warp == 4) && leader && mma_issued) {   // each issuing lane drains its MMAs
      if (elect_one()) {
        uint64_t* dr = warp == 3 ? &bars->drain : &bars->drain2;
        umma_commit_mask(dr, pair_mask);
        const uint32_t a = smem_u32(dr);
        const long long t0 = clock64();
        while (!mbar_try_wait(a, 0) && clock64() - t0 < p.wait_limit) {
        }
      }
      __syncwarp();
    }
    if (warp >= 5 && lane == 0) wide_spin(20000000LL);   // slot copies in flight land
    __syncthreads();
  }
  tc_fence_before();
  cluster_sync();   // no CTA's MMAs, copies or arrivals still touch another CTA
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kWTmemAlloc);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicOr(p.status, kStatusTimeout);
}

}  // namespace

bool wide_supported(const Dims& d) {
  return umma_supported(d) && d.Dt == kWPairs * UN && d.Ds % UK == 0 && d.H % kWChunk == 0 &&
         d.d_t % 32 == 0;
}

cudaError_t launch_wide(const PathArgs& a, const CUtensorMap& tmK, const CUtensorMap& tmV,
                        const CUtensorMap& tmW1q, const CUtensorMap& tmW2h,
                        const CUtensorMap& tmG16, const CUtensorMap& tmB2th, int num_sms,
                        cudaStream_t st) {
  static int max_clusters = 0;
  if (max_clusters == 0) {
    cudaError_t e = cudaFuncSetAttribute(wide_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kWSmemBytes);
    if (e != cudaSuccess) return e;
    // clusters that fit at once (one CTA per SM): the persistent grid's size
    cudaLaunchConfig_t cfg{};
    cfg.gridDim = dim3(kWCtas * (num_sms / kWCtas));
    cfg.blockDim = dim3(kWThreads);
    cfg.dynamicSmemBytes = kWSmemBytes;
    int n = 0;
    e = cudaOccupancyMaxActiveClusters(&n, wide_kernel, &cfg);
    if (e != cudaSuccess) return e;
    max_clusters = n > 0 ? n : 1;
  }
  WideArgs wa;
  wa.p = a;
  wa.nk1 = a.d.Ds / UK;
  wa.nc = a.d.EH / kWChunk;
  const long long items = static_cast<long long>(a.gp) * ((a.d.tiles_max + 1) / 2);
  const long long n_cl = items < max_clusters ? items : max_clusters;
  if (n_cl <= 0) return cudaSuccess;
  wide_kernel<<<static_cast<int>(kWCtas * n_cl), kWThreads, kWSmemBytes, st>>>(
      tmK, tmV, tmW1q, tmW2h, tmG16, tmB2th, wa);
  return cudaGetLastError();
}

}  // namespace mot
