// On-chip translation for D_t = 512, D_s <= 512 (schedule 4): GEMM1 -> GELU *
// gate -> GEMM2 with the hidden activations kept on chip, for translators whose
// output is too wide for one CTA pair's tensor memory.
//
// One pair's GEMM2 accumulator for 256 token rows and D_t = 512 columns fills
// all 512 TMEM columns of each of its SMs, leaving none for GEMM1. So a
// cluster of four CTAs -- two CTA pairs -- works on one 256-row pair tile
// (token tiles 2 mp and 2 mp + 1 of one (target layer, K/V) group) with the
// two GEMMs on different pairs:
//   pair 0 (ranks 0, 1) walks the concatenated hidden dimension E*H in
//     128-column chunks, U_c = Z * W1cat[128 c .. 128 c + 127]^T (M = 256,
//     N = 128, K = D_s) into one of four TMEM accumulators, with the tile's
//     source rows Z resident in shared memory; its epilogue computes
//     A2_c = fp16(GELU(U_c + b1) * gtilde_m) and stores it straight into a
//     shared-memory slot of the pair-1 CTA that holds the same token rows,
//     in the tcgen05 operand layout (st.shared::cluster);
//   pair 1 (ranks 2, 3) accumulates Y += A2_c * W2cat[:, 128 c .. 128 c + 127]^T
//     (M = 256, two N = 256 halves of D_t, K = 128) in TMEM over every chunk,
//     adds the gate-weighted biases sum_m gtilde_m b2_m (Def. 3.1) as one more
//     K block (A = gate16, B = b2t), and stores Y as bf16 into the target
//     cache.
// The two GEMMs have equal work when D_s = D_t. A2 never leaves the chip.
//
// Shared memory per CTA, pair 0: Z as D_s / 64 blocks of 16 KB (128 rows x 64
// K) and a ring of 12 W1 stages of 8 KB (its 64 of a chunk's 128 rows, K = 64);
// pair 1: 3 A2 slots of 32 KB (chunk c in slot c % 3), a ring of 3 W2 stages
// of 32 KB (its 128 rows of each 256-column half, K = 64; the tile's b2t
// block takes one stage too) and 16 KB of gate16 rows.
// TMEM: pair 0 acc1[4] x 128 columns, pair 1 acc2 512 columns.
//
// Roles (13 warps per CTA):
//   pair 0  warp 0 lane 0   TMA loads of Z (once per tile) and of the W1 ring;
//           warp 3 (leader) GEMM1 issue (one elected lane);
//           warps 5..12     chunk epilogue: warp w owns rows 32 (w % 4) ..,
//                           chunk columns 64 hh .. 64 hh + 63 (hh = (w - 5) / 4);
//   pair 1  warp 1 lane 0   TMA loads of the W2 ring, b2t and gate16;
//           warp 4 (leader) GEMM2 and bias issue (one elected lane); the commit
//                           after each chunk frees its slot (arrives in pair 0);
//           warps 5..12     output epilogue: rows 32 (w % 4) .., columns
//                           256 hh .. 256 hh + 255;
//   both    warp 2          TMEM allocation of the pair.
// Every slot use is written by pair 0's epilogue, which waits for the slot's
// previous use to be freed before every write, so no barrier phase can pass
// unobserved. Every wait is bounded; a timeout unwinds every role and raises
// kStatusTimeout.
#include "umma_common.cuh"

namespace mot {
namespace {

constexpr int kWCtas = 4;                     // two CTA pairs per cluster
constexpr int kWChunk = 128;                  // hidden columns per chunk
constexpr int kWBlk = UM * UK * 2;            // 16 KB: 128 rows x 64 K, 16-bit
constexpr int kWW1Blk = (kWChunk / 2) * UK * 2;   // 8 KB: 64 rows x 64 K
constexpr int kWMaxZ = 8;                     // Z blocks: D_s <= 512
constexpr int kWStagesW1 = 12;
constexpr int kWStagesW2 = 3;
constexpr int kWW2Stage = 2 * kWBlk;          // both 256-column halves, K = 64
constexpr int kWSlots = 3;
constexpr int kWSlotBytes = 2 * kWBlk;        // 128 rows x 128 K
constexpr int kWAcc1 = 4;                     // GEMM1 accumulators of 128 columns
// pair 0 layout
constexpr int kWOffW1 = kWMaxZ * kWBlk;
constexpr int kWEnd0 = kWOffW1 + kWStagesW1 * kWW1Blk;
// pair 1 layout
constexpr int kWOffW2 = kWSlots * kWSlotBytes;
constexpr int kWOffG = kWOffW2 + kWStagesW2 * kWW2Stage;
constexpr int kWEnd1 = kWOffG + kWBlk;
constexpr int kWOffBar = kWEnd0 > kWEnd1 ? kWEnd0 : kWEnd1;
constexpr int kWEpiWarps = 8;
constexpr int kWThreads = 32 * (5 + kWEpiWarps);
constexpr int kWSmemBytes = kWOffBar + 1024 + 1024;
static_assert(kWSmemBytes <= 232448, "shared memory budget");
static_assert(kWOffW1 % 1024 == 0 && kWOffW2 % 1024 == 0 && kWOffG % 1024 == 0, "alignment");
constexpr uint32_t kWTmemAlloc = 512;

struct WBars {
  // pair 0
  uint64_t zfull[kWMaxZ];        // Z block landed (leader; both CTAs' bytes)
  uint64_t zempty;               // the tile's last GEMM1 done with Z (commit, pair 0)
  uint64_t w1full[kWStagesW1], w1empty[kWStagesW1];
  uint64_t a1full[kWAcc1];       // GEMM1 of a chunk done (commit, pair 0)
  uint64_t acc1free[kWAcc1];     // its accumulator read out (pair-0 leader; 2 x 8 arrivals)
  uint64_t slotfree[kWSlots];    // pair 1's GEMM2 done with the slot (commit, arrives in pair 0)
  // pair 1
  uint64_t a2full[kWSlots];      // a chunk's A2 written into both pair-1 CTAs (pair-1 leader;
                                 // 2 x 8 warp arrivals from pair 0)
  uint64_t w2full[kWStagesW2], w2empty[kWStagesW2];
  uint64_t gfull, gempty;
  uint64_t acc2full;             // a tile's GEMM2 + bias done (commit, pair 1)
  uint64_t acc2empty;            // acc2 read out (pair-1 leader; 2 x 8 arrivals)
  uint64_t drain;
  uint32_t tmem_slot;
  int abort_flag;
};
static_assert(sizeof(WBars) <= 1024, "barrier block");

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

// Row r's 16-byte chunks 4 s .. 4 s + 3 of a 64-wide K block at cluster
// address `blk` (128B swizzle), in another CTA's shared memory.
__device__ __forceinline__ void wide_store_a2_remote(uint32_t blk, int r, int s,
                                                     const uint32_t (&pk)[16]) {
  const uint32_t row = blk + static_cast<uint32_t>(r * 128);
#pragma unroll
  for (int v = 0; v < 4; ++v)
    st_cluster_v4(row + static_cast<uint32_t>(((4 * s + v) ^ (r & 7)) << 4), pk[4 * v],
                  pk[4 * v + 1], pk[4 * v + 2], pk[4 * v + 3]);
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
  WBars* bars = reinterpret_cast<WBars*>(smem + kWOffBar);
  volatile int* abort_flag = &bars->abort_flag;

  const PathArgs& p = wa.p;
  const Dims& d = p.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const uint32_t half = rank & 1u;            // which 128 rows of the pair tile
  const uint32_t pr = rank >> 1;              // 0: GEMM1 pair, 1: GEMM2 pair
  const bool leader = half == 0;
  constexpr uint16_t kMask0 = 0x3, kMask1 = 0xC;   // the CTAs of pair 0 / pair 1
  const int nc = wa.nc, nk1 = wa.nk1;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kWMaxZ; ++i) mbar_init(&bars->zfull[i], 1);
    mbar_init(&bars->zempty, 1);
    for (int i = 0; i < kWStagesW1; ++i) {
      mbar_init(&bars->w1full[i], 1);
      mbar_init(&bars->w1empty[i], 1);
    }
    for (int i = 0; i < kWAcc1; ++i) {
      mbar_init(&bars->a1full[i], 1);
      mbar_init(&bars->acc1free[i], 2 * kWEpiWarps);
    }
    for (int i = 0; i < kWSlots; ++i) {
      mbar_init(&bars->slotfree[i], 1);
      mbar_init(&bars->a2full[i], 2 * kWEpiWarps);
    }
    for (int i = 0; i < kWStagesW2; ++i) {
      mbar_init(&bars->w2full[i], 1);
      mbar_init(&bars->w2empty[i], 1);
    }
    mbar_init(&bars->gfull, 1);
    mbar_init(&bars->gempty, 1);
    mbar_init(&bars->acc2full, 1);
    mbar_init(&bars->acc2empty, 2 * kWEpiWarps);
    mbar_init(&bars->drain, 1);
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

  // unwinding state: loads in flight (bit i: zfull 0-7, w1full 8-19, w2full 20-22, gfull 23)
  uint32_t pend_mask = 0, pend_par = 0;
  auto note = [&](int bit, uint32_t ph) {
    pend_mask |= 1u << bit;
    pend_par = (pend_par & ~(1u << bit)) | (ph << bit);
  };
  bool mma_issued = false;

  if (pr == 0 && warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ Z and W1 loads (pair 0)
      int s = 0;
      uint32_t ph = 0, k = 0;
      bool ok = true;
      for (int t = cl; ok && t < total; t += n_cl, ++k) {
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
        // chunk 0's W1 blocks first (they only need free ring stages), then Z
        // once the previous tile's last GEMM1 is done with it, then the rest
        for (int c = 0; ok && c < nc; ++c) {
          if (c == 1 || nc == 1) {
            if (!mbar_wait(&bars->zempty, (k & 1u) ^ 1u, abort_flag, p.wait_limit)) {
              ok = false;
              break;
            }
            const int zrow = ((gi.src_layer * d.B + ti.b) * d.H_s) * d.S + ti.s0;
            for (int kb = 0; kb < nk1; ++kb) {
              if (leader) mbar_arrive_expect_tx(&bars->zfull[kb], 2 * kWBlk);
              const int kk = kb * UK, h = kk / d.d_s, d0 = kk - h * d.d_s;
              tma_load_2d_pair(smem + kb * kWBlk, gi.x ? &tmV : &tmK,
                               leader_addr(&bars->zfull[kb]), d0, zrow + h * d.S);
              note(kb, k & 1u);
            }
          }
          const int wrow = grp * d.EH + c * kWChunk + static_cast<int>(half) * (kWChunk / 2);
          for (int kb = 0; kb < nk1; ++kb) {
            if (!mbar_wait(&bars->w1empty[s], ph ^ 1u, abort_flag, p.wait_limit)) { ok = false; break; }
            if (leader) mbar_arrive_expect_tx(&bars->w1full[s], 2 * kWW1Blk);
            tma_load_2d_pair(smem + kWOffW1 + s * kWW1Blk, &tmW1q, leader_addr(&bars->w1full[s]),
                             kb * UK, wrow);
            note(kWMaxZ + s, ph);
            if (++s == kWStagesW1) { s = 0; ph ^= 1u; }
          }
        }
      }
    }
  } else if (pr == 1 && warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------ W2 ring, b2t and gate16 loads (pair 1)
      int s = 0;
      uint32_t ph = 0, k = 0;
      bool ok = true;
      const int wrow = static_cast<int>(half) * UM;   // this CTA's rows of each 256-column half
      auto stage = [&]() -> uint32_t {
        if (!mbar_wait(&bars->w2empty[s], ph ^ 1u, abort_flag, p.wait_limit)) return 0;
        if (leader) mbar_arrive_expect_tx(&bars->w2full[s], 2 * kWW2Stage);
        return leader_addr(&bars->w2full[s]);
      };
      auto next = [&]() {
        note(kWMaxZ + kWStagesW1 + s, ph);
        if (++s == kWStagesW2) { s = 0; ph ^= 1u; }
      };
      for (int t = cl; ok && t < total; t += n_cl, ++k) {
        const int gl = t / n_mp, mp = t - gl * n_mp;
        const int grp = p.g0 + gl;
        const int m_own = 2 * mp + static_cast<int>(half);
        for (int c = 0; ok && c < nc; ++c)
          for (int kb = 0; kb < 2; ++kb) {
            const uint32_t bar = stage();
            if (!bar) { ok = false; break; }
            uint8_t* st = smem + kWOffW2 + s * kWW2Stage;
            for (int n = 0; n < 2; ++n)
              tma_load_2d_pair(st + n * kWBlk, &tmW2h, bar, c * kWChunk + kb * UK,
                               grp * d.Dt + n * UN + wrow);
            next();
          }
        if (!ok) break;
        {   // the bias block's B: b2t rows of both halves
          const uint32_t bar = stage();
          if (!bar) break;
          uint8_t* st = smem + kWOffW2 + s * kWW2Stage;
          for (int n = 0; n < 2; ++n)
            tma_load_2d_pair(st + n * kWBlk, &tmB2th, bar, 0, grp * d.Dt + n * UN + wrow);
          next();
        }
        if (!mbar_wait(&bars->gempty, (k & 1u) ^ 1u, abort_flag, p.wait_limit)) break;
        if (leader) mbar_arrive_expect_tx(&bars->gfull, 2 * kWBlk);
        tma_load_3d_pair(smem + kWOffG, &tmG16, leader_addr(&bars->gfull), 0, m_own * UM, grp);
        note(kWMaxZ + kWStagesW1 + kWStagesW2, k & 1u);
      }
    }
  } else if (warp == 3 + static_cast<int>(pr) && leader) {
    // ------------------------------------------------ MMA issue (pair leaders)
    auto wait_all = [&](uint64_t* bar, uint32_t parity) -> bool {
      const bool r = mbar_wait(bar, parity, abort_flag, p.wait_limit);
      return __all_sync(0xffffffffu, r) != 0;
    };
    auto wait_all_cluster = [&](uint64_t* bar, uint32_t parity) -> bool {
      const bool r = mbar_wait_cluster(bar, parity, abort_flag, p.wait_limit);
      return __all_sync(0xffffffffu, r) != 0;
    };
    bool ok = true;
    if (pr == 0) {
      // GEMM1: acc1[cg % 4] = Z * W1cat[chunk]^T
      constexpr uint32_t idesc1 = idesc_bf16_f32(2 * UM, kWChunk);
      int s = 0;
      uint32_t ph = 0, k = 0, cg = 0;
      for (int t = cl; ok && t < total; t += n_cl, ++k) {
        for (int c = 0; ok && c < nc; ++c, ++cg) {
          const uint32_t b = cg % kWAcc1;
          if (cg >= kWAcc1) ok = wait_all(&bars->acc1free[b], ((cg / kWAcc1) & 1u) ^ 1u);
          if (!ok) break;
          const uint32_t d1 = tmem_base + b * kWChunk;
          for (int kb = 0; kb < nk1; ++kb) {
            if (c == 0 && !wait_all(&bars->zfull[kb], k & 1u)) { ok = false; break; }
            if (!wait_all(&bars->w1full[s], ph)) { ok = false; break; }
            tc_fence_after();
            if (elect_one()) {
              const uint64_t zdesc = sdesc_k_sw128(smem_u32(smem + kb * kWBlk));
              const uint64_t wdesc = sdesc_k_sw128(smem_u32(smem + kWOffW1 + s * kWW1Blk));
#pragma unroll
              for (int kk = 0; kk < UK / 16; ++kk)   // +32 bytes of K = +2 in the address field
                umma_pair(d1, zdesc + 2 * kk, wdesc + 2 * kk, idesc1, (kb | kk) != 0);
              umma_commit_mask(&bars->w1empty[s], kMask0);
            }
            __syncwarp();
            mma_issued = true;
            if (++s == kWStagesW1) { s = 0; ph ^= 1u; }
          }
          if (!ok) break;
          if (elect_one()) {
            umma_commit_mask(&bars->a1full[b], kMask0);
            if (c == nc - 1) umma_commit_mask(&bars->zempty, kMask0);
          }
          __syncwarp();
        }
      }
    } else {
      // GEMM2: acc2[0, 512) += A2_c * W2cat[:, chunk]^T over every chunk, then the bias block
      constexpr uint32_t idesc2 = idesc_f16_f32(2 * UM, UN);
      int s = 0;
      uint32_t ph = 0, k = 0, cg = 0;
      for (int t = cl; ok && t < total; t += n_cl, ++k) {
        for (int c = 0; ok && c < nc; ++c, ++cg) {
          const uint32_t slot = cg % kWSlots, use = cg / kWSlots;
          ok = wait_all_cluster(&bars->a2full[slot], use & 1u);
          if (ok && c == 0) ok = wait_all(&bars->acc2empty, (k & 1u) ^ 1u);
          if (!ok) break;
          const uint32_t aa = smem_u32(smem + slot * kWSlotBytes);
          for (int kb = 0; kb < 2; ++kb) {
            if (!wait_all(&bars->w2full[s], ph)) { ok = false; break; }
            tc_fence_after();
            if (elect_one()) {
              const uint64_t adesc = sdesc_k_sw128(aa + kb * kWBlk);
              const uint32_t ba = smem_u32(smem + kWOffW2 + s * kWW2Stage);
#pragma unroll
              for (int n = 0; n < 2; ++n) {
                const uint64_t bdesc = sdesc_k_sw128(ba + n * kWBlk);
#pragma unroll
                for (int kk = 0; kk < UK / 16; ++kk)
                  umma_pair(tmem_base + n * UN, adesc + 2 * kk, bdesc + 2 * kk, idesc2,
                            (c | kb | kk) != 0);
              }
              umma_commit_mask(&bars->w2empty[s], kMask1);
            }
            __syncwarp();
            mma_issued = true;
            if (++s == kWStagesW2) { s = 0; ph ^= 1u; }
          }
          if (!ok) break;
          if (elect_one()) umma_commit_mask(&bars->slotfree[slot], kMask0);   // pair 0 may refill it
          __syncwarp();
        }
        if (!ok) break;
        if (!wait_all(&bars->gfull, k & 1u)) break;
        if (!wait_all(&bars->w2full[s], ph)) break;
        tc_fence_after();
        if (elect_one()) {
          const uint64_t gdesc = sdesc_k_sw128(smem_u32(smem + kWOffG));
          const uint32_t ba = smem_u32(smem + kWOffW2 + s * kWW2Stage);
#pragma unroll
          for (int n = 0; n < 2; ++n) {
            const uint64_t bdesc = sdesc_k_sw128(ba + n * kWBlk);
#pragma unroll
            for (int kk = 0; kk < UK / 16; ++kk)
              umma_pair(tmem_base + n * UN, gdesc + 2 * kk, bdesc + 2 * kk, idesc2, 1u);
          }
          umma_commit_mask(&bars->w2empty[s], kMask1);
          umma_commit_mask(&bars->gempty, kMask1);
          umma_commit_mask(&bars->acc2full, kMask1);
        }
        __syncwarp();
        if (++s == kWStagesW2) { s = 0; ph ^= 1u; }
      }
    }
  } else if (warp >= 5) {
    const int e = warp - 5, q = warp & 3, hh = e >> 2;   // q: the TMEM lane quarter warp % 4 may access
    const int r = q * 32 + lane;
    const uint32_t tq = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
    bool ok = true;
    if (pr == 0) {
      // ------------------------------------------------ chunk epilogue (pair 0)
      const __half* b1h = static_cast<const __half*>(p.b1h);
      const uint32_t peer = rank + 2u;   // the pair-1 CTA with the same token rows
      const uint32_t a2_remote = mapa_cluster(smem, peer);
      uint32_t cg = 0;
      for (int t = cl; ok && t < total; t += n_cl) {
        const int gl = t / n_mp, mp = t - gl * n_mp;
        const int grp = p.g0 + gl;
        const int m_own = 2 * mp + static_cast<int>(half);
        const bool valid = m_own < n_m;
        const float* grow = p.gate + (static_cast<size_t>(grp) * d.tpad +
                                      static_cast<size_t>(m_own) * UM + r) * d.E;
        const uint4* bias4 = reinterpret_cast<const uint4*>(b1h + static_cast<size_t>(grp) * d.EH);
        for (int c = 0; c < nc; ++c, ++cg) {
          const uint32_t b = cg % kWAcc1, slot = cg % kWSlots, use = cg / kWSlots;
          // this warp's 2 x 32 biases and the row's gate value, fetched before the wait
          uint4 bias[2][4];
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            bias[0][i] = __ldg(bias4 + (c * kWChunk + hh * 64) / 8 + i);
            bias[1][i] = __ldg(bias4 + (c * kWChunk + hh * 64 + 32) / 8 + i);
          }
          const float gate = valid ? __ldg(grow + (c * kWChunk) / d.H) : 0.f;
          int w = 1;
          if (lane == 0) w = mbar_wait(&bars->a1full[b], (cg / kWAcc1) & 1u, abort_flag, p.wait_limit);
          if (!__shfl_sync(0xffffffffu, w, 0)) { ok = false; break; }
          tc_fence_after();
          uint32_t pa[16], pb[16];
          {
            uint32_t ra[32], rb[32];
            tmem_ld_32x32b_x32(tq + b * kWChunk + hh * 64, ra);
            tmem_ld_32x32b_x32(tq + b * kWChunk + hh * 64 + 32, rb);
            tmem_ld_wait(ra);
            tmem_ld_wait(rb);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(&bars->acc1free[b], 0);   // GEMM1(cg + 4) may start
            const __half2 hg = __float2half2_rn(0.5f * gate);
            wide_gelu_cols(ra, bias[0], hg, pa);
            wide_gelu_cols(rb, bias[1], hg, pb);
          }
          // pair 1's GEMM2 of the slot's previous chunk must be done reading it
          if (use >= 1) {
            if (lane == 0)
              w = mbar_wait_cluster(&bars->slotfree[slot], (use - 1) & 1u, abort_flag, p.wait_limit);
            if (!__shfl_sync(0xffffffffu, w, 0)) { ok = false; break; }
          }
          const uint32_t blk = a2_remote + slot * kWSlotBytes + static_cast<uint32_t>(hh * kWBlk);
          wide_store_a2_remote(blk, r, 0, pa);
          wide_store_a2_remote(blk, r, 1, pb);
          fence_proxy_async_cluster();   // pair 1's tensor core (async proxy) reads these stores
          __syncwarp();
          if (lane == 0) mbar_arrive_release_cluster(&bars->a2full[slot], 2u);
        }
      }
    } else {
      // ------------------------------------------------ output epilogue (pair 1)
      uint32_t k = 0;
      for (int t = cl; t < total; t += n_cl, ++k) {
        const int gl = t / n_mp, mp = t - gl * n_mp;
        const int grp = p.g0 + gl;
        const int m_own = 2 * mp + static_cast<int>(half);
        const bool valid = m_own < n_m;
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
          for (int cc = hh * UN; cc < (hh + 1) * UN; cc += 64) {
            tmem_ld_32x32b_x32(tq + cc, ra);
            tmem_ld_32x32b_x32(tq + cc + 32, rb);
            tmem_ld_wait(ra);
            tmem_ld_wait(rb);
            if (r < ti.rows) {
#pragma unroll
              for (int u = 0; u < 2; ++u) {
                const int col = cc + 32 * u;
                const int hd = col / d.d_t, i0 = col - hd * d.d_t;
                __nv_bfloat16* o = dst + ((((static_cast<size_t>(gi.tgt_layer) * d.B + ti.b) *
                                            d.H_t + hd) * d.S + s_pos) * d.d_t + i0);
                wide_store_out(u ? rb : ra, o);
              }
            }
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(&bars->acc2empty, 2);
      }
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
        for (int i = 0; i < kWMaxZ + kWStagesW1 + kWStagesW2 + 1; ++i) {
          if (!((pend_mask >> i) & 1u)) continue;
          uint64_t* fb = i < kWMaxZ ? &bars->zfull[i]
                       : i < kWMaxZ + kWStagesW1 ? &bars->w1full[i - kWMaxZ]
                       : i < kWMaxZ + kWStagesW1 + kWStagesW2
                           ? &bars->w2full[i - kWMaxZ - kWStagesW1]
                           : &bars->gfull;
          const uint32_t a = smem_u32(fb);
          const long long t0 = clock64();
          while (!mbar_try_wait(a, (pend_par >> i) & 1u) && clock64() - t0 < p.wait_limit) {
          }
        }
      } else {
        wide_spin(20000000LL);
      }
    }
    if (warp == 3 + static_cast<int>(pr) && leader && mma_issued) {   // drain its MMAs
      if (elect_one()) {
        umma_commit_mask(&bars->drain, pr ? kMask1 : kMask0);
        const uint32_t a = smem_u32(&bars->drain);
        const long long t0 = clock64();
        while (!mbar_try_wait(a, 0) && clock64() - t0 < p.wait_limit) {
        }
      }
      __syncwarp();
    }
    __syncthreads();
  }
  tc_fence_before();
  cluster_sync();   // no CTA's MMAs, stores or arrivals still touch another CTA
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kWTmemAlloc);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicOr(p.status, kStatusTimeout);
}

}  // namespace

bool wide_supported(const Dims& d) {
  return umma_supported(d) && d.Dt == 2 * UN && d.Ds % UK == 0 && d.Ds <= kWMaxZ * UK &&
         d.H % kWChunk == 0 && d.d_t % 32 == 0;
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
