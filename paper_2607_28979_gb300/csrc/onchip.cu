// On-chip translation for narrow translators (D_s <= 128, D_t = 256) on CTA
// pairs: GEMM1 -> GELU * gate -> GEMM2 with the hidden activations kept in
// shared memory and TMEM, so the A2 intermediate (E*H fp16 values per token
// row, 7.5 GB for the Qwen2.5-0.5B -> 1.5B shapes) never goes through HBM.
//
// A cluster of two CTAs owns a 256-row pair tile (token tiles 2*mp, 2*mp + 1
// of one (target layer, K/V) group) and walks the concatenated hidden
// dimension E*H in chunks of 128 columns. For chunk j:
//   U_j  = Z * W1cat[128 j .. 128 j + 127]^T       tcgen05 M=256 N=128 K=D_s -> TMEM acc1[c % 2]
//   A2_j = fp16( GELU(U_j + b1) * gtilde_m )        epilogue warps, into shared memory in the
//                                                  K-major 128B-swizzled operand layout
//   Y   += A2_j * W2cat[:, 128 j .. 128 j + 127]^T  tcgen05 M=256 N=256 K=128 -> TMEM acc2
// (c counts chunks across tiles; m = 128 j / H is the chunk's expert, as
// H % 128 == 0). After the last chunk Y += gate16 * b2t adds the
// gate-weighted biases sum_m gtilde_m b2_m (Def. 3.1), and the epilogue
// stores Y as bf16 into the target cache.
//
// TMEM per CTA (512 columns): acc2 in [0, 256), acc1[0] in [256, 384),
// acc1[1] in [384, 512). Shared memory per CTA: Z 2 x 32 KB (the next tile's
// rows load during the current tile; after its last GEMM1 a tile's buffer
// holds b2t and gate16 for the bias MMA), W1 ring 2 x 16 KB, W2 ring
// 2 x 32 KB, A2 2 x 32 KB.
//
// Roles per CTA:
//   warp 0 lane 0 (both)    TMA loads of its Z rows and its halves of W1 / W2;
//                           transaction bytes complete on the leader's barriers;
//   warp 1 (leader)         GEMM1 issue (one elected lane), up to two chunks ahead;
//   warp 3 (leader)         GEMM2 and bias-MMA issue (one elected lane);
//   warp 2 (both)           TMEM allocation of the pair;
//   warps 4..19 (both)      epilogue: warp 4 + 4 p + q owns rows 32 q .. 32 q + 31; of
//                           every chunk it evaluates columns 32 p .. 32 p + 31, and at the
//                           end of a tile it stores output columns 64 p .. 64 p + 63.
// With two acc1 buffers the chunk epilogue is on the MMA's critical path, so it
// is kept short: all sixteen warps share each chunk, take its biases into
// registers before its accumulator is ready, and release acc1 as soon as it is
// read (GEMM1 two chunks ahead is issued then, ahead of GEMM2 of this chunk);
// the A2 stores then wait only for GEMM2 two chunks back.
// Every wait is bounded; a timeout unwinds and raises kStatusTimeout.
#include "umma_common.cuh"

namespace mot {
namespace {

constexpr int kChunk = 128;                              // hidden columns per chunk
constexpr int kBlk16 = UM * UK * 2;                      // 16 KB: 128 rows x 64 K, 16-bit
constexpr int kZBytes = 2 * kBlk16;                      // Z: 128 rows x D_s (<= 128)
constexpr int kW1Blk = (kChunk / 2) * UK * 2;            // 8 KB: 64 rows x 64 K
constexpr int kW1Bytes = 2 * kW1Blk;
constexpr int kW2Bytes = 2 * kBlk16;                     // 128 rows x 128 K
constexpr int kA2Bytes = 2 * kBlk16;                     // 128 rows x 128 K
constexpr int kOffW1 = 2 * kZBytes;
constexpr int kOffW2 = kOffW1 + 2 * kW1Bytes;
constexpr int kOffA2 = kOffW2 + 2 * kW2Bytes;
constexpr int kOffBar = kOffA2 + 2 * kA2Bytes;
constexpr int kEpiWarps = 16;
constexpr int kThreads = 32 * (4 + kEpiWarps);
constexpr int kSmemBytes = kOffBar + 256 + 1024;
static_assert(kSmemBytes <= 232448, "shared memory budget");
constexpr uint32_t kAcc1Col = UN;   // acc1[b] at column 256 + 128 b
constexpr uint32_t kTmemAlloc = 512;

// Each tcgen05.commit costs the tensor pipe several hundred cycles, so a chunk
// has two: a1full (GEMM1 done: its acc1 is ready and its W1 slot free) and
// a2empty (GEMM2 done: its A2 buffer and its W2 slot free). The ring slots of
// W1, W2, acc1 and A2 are all indexed by the chunk counter c, so one commit
// serves both waiters; the tile's bias stage (gate16, b2t) uses the tile's Z
// buffer once its last GEMM1 is done.
struct Bars {
  uint64_t zfull[2], zempty[2], w1full[2], w2full[2], bfull[2];
  uint64_t a1full[2];   // GEMM1 of a chunk done (commit, both CTAs)
  uint64_t acc1free[2]; // the chunk's acc1 read out (leader; 2 x 16 warp arrivals)
  uint64_t a2full[2];   // the chunk's A2 written (leader; 2 x 16 warp arrivals)
  uint64_t a2empty[2];  // GEMM2 of a chunk done reading its A2 (commit, both CTAs)
  uint64_t acc2full;    // a tile's GEMM2 + bias done (commit, both CTAs)
  uint64_t acc2empty;   // acc2 read out (leader; 2 x 16 warp arrivals)
  uint64_t drain, drain2;
  uint32_t tmem_slot;
  int abort_flag;
};
static_assert(sizeof(Bars) <= 256, "barrier block");

struct OnchipArgs {
  PathArgs p;
  int32_t nk1;   // 64-wide K blocks of GEMM1 (D_s / 64)
  int32_t nc;    // chunks per tile (E*H / 128)
};

__device__ __forceinline__ void spin_cycles(long long cycles) {
  const long long t0 = clock64();
  while (clock64() - t0 < cycles) {
  }
}

// GELU(u + b) * g on 32 accumulator columns (`acc`, fp32 bits) with their
// fp16 biases in `b` (four 16-byte vectors): fp16 pairs for the A2 operand.
__device__ __forceinline__ void gelu_cols(const uint32_t (&acc)[32], const uint4* b, __half2 half_g,
                                          uint32_t (&pk)[16]) {
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

// Row r's 16-byte chunks 4 s .. 4 s + 3 of a 64-wide K block at `blk`, each at
// chunk position (index ^ (r % 8)) of its 128-byte row (the 128B swizzle).
__device__ __forceinline__ void store_a2(uint32_t blk, int r, int s, const uint32_t (&pk)[16]) {
  const uint32_t row = blk + static_cast<uint32_t>(r * 128);
#pragma unroll
  for (int v = 0; v < 4; ++v)
    st_shared_v4(row + static_cast<uint32_t>(((4 * s + v) ^ (r & 7)) << 4), pk[4 * v],
                 pk[4 * v + 1], pk[4 * v + 2], pk[4 * v + 3]);
}

// 32 fp32 accumulator columns -> 32 bf16 channels at `o` (64 bytes), as two
// 32-byte stores (`o` 32-byte aligned) or four 16-byte stores.
__device__ __forceinline__ void store_out32(const uint32_t (&acc)[32], __nv_bfloat16* o) {
  uint32_t w[16];
#pragma unroll
  for (int i = 0; i < 16; ++i)
    w[i] = pack_bf16x2(__uint_as_float(acc[2 * i]), __uint_as_float(acc[2 * i + 1]));
#pragma unroll
  for (int h = 0; h < 2; ++h)
    asm volatile("st.global.v8.b32 [%0], {%1, %2, %3, %4, %5, %6, %7, %8};" ::"l"(o + 16 * h),
                 "r"(w[8 * h]), "r"(w[8 * h + 1]), "r"(w[8 * h + 2]), "r"(w[8 * h + 3]),
                 "r"(w[8 * h + 4]), "r"(w[8 * h + 5]), "r"(w[8 * h + 6]), "r"(w[8 * h + 7])
                 : "memory");
}

__device__ __forceinline__ void store_out(const uint32_t (&acc)[32], __nv_bfloat16* o) {
  uint4* o4 = reinterpret_cast<uint4*>(o);
#pragma unroll
  for (int v = 0; v < 4; ++v)
    o4[v] = make_uint4(pack_bf16x2(__uint_as_float(acc[8 * v + 0]), __uint_as_float(acc[8 * v + 1])),
                       pack_bf16x2(__uint_as_float(acc[8 * v + 2]), __uint_as_float(acc[8 * v + 3])),
                       pack_bf16x2(__uint_as_float(acc[8 * v + 4]), __uint_as_float(acc[8 * v + 5])),
                       pack_bf16x2(__uint_as_float(acc[8 * v + 6]), __uint_as_float(acc[8 * v + 7])));
}

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    onchip_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                  const __grid_constant__ CUtensorMap tmW1q,
                  const __grid_constant__ CUtensorMap tmW2h,
                  const __grid_constant__ CUtensorMap tmG16,
                  const __grid_constant__ CUtensorMap tmB2th, const OnchipArgs oa) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sZ = smem;
  uint8_t* sW1 = smem + kOffW1;
  uint8_t* sW2 = smem + kOffW2;
  uint8_t* sA2 = smem + kOffA2;
  Bars* bars = reinterpret_cast<Bars*>(smem + kOffBar);
  volatile int* abort_flag = &bars->abort_flag;

  const PathArgs& p = oa.p;
  const Dims& d = p.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int nc = oa.nc, nk1 = oa.nk1;

  if (threadIdx.x == 0) {
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars->zfull[i], 1);
      mbar_init(&bars->zempty[i], 1);
      mbar_init(&bars->w1full[i], 1);
      mbar_init(&bars->w2full[i], 1);
      mbar_init(&bars->bfull[i], 1);
      mbar_init(&bars->a1full[i], 1);
      mbar_init(&bars->acc1free[i], 2 * kEpiWarps);
      mbar_init(&bars->a2full[i], 2 * kEpiWarps);
      mbar_init(&bars->a2empty[i], 1);
    }
    mbar_init(&bars->acc2full, 1);
    mbar_init(&bars->acc2empty, 2 * kEpiWarps);
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
    tmem_alloc_pair(&bars->tmem_slot, kTmemAlloc);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  cluster_sync();
  tc_fence_after();
  const uint32_t tmem_base = bars->tmem_slot;

  const int n_m = min(*p.n_tiles, d.tiles_max);
  const int n_mp = (n_m + 1) / 2;
  const int total = p.gp * n_mp;
  const int pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;

  // unwinding state: full barriers with loads in flight (bit i: zfull 0-1,
  // w1full 2-3, w2full 4-5, bfull 6-7) and the parity of each one's last phase
  uint32_t pend_mask = 0, pend_par = 0;
  bool mma_issued = false;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer (both CTAs)
      auto note = [&](int bit, uint32_t ph) {
        pend_mask |= 1u << bit;
        pend_par = (pend_par & ~(1u << bit)) | (ph << bit);
      };
      auto load_z = [&](int t, uint32_t k) -> bool {
        const int zb = k & 1;
        const uint32_t ph = (k >> 1) & 1u;
        if (!mbar_wait(&bars->zempty[zb], ph ^ 1u, abort_flag, p.wait_limit)) return false;
        const int gl = t / n_mp, mp = t - gl * n_mp;
        const GroupInfo gi = p.groups[p.g0 + gl];
        const int m_own = 2 * mp + static_cast<int>(rank);
        TileInfo ti;
        if (m_own < n_m) {
          ti = p.tiles[m_own];
        } else {   // no such tile: any in-bounds rows; they are never stored
          ti.b = 0;
          ti.s0 = 0;
        }
        if (leader) mbar_arrive_expect_tx(&bars->zfull[zb], 2 * nk1 * kBlk16);
        const uint32_t bar = leader_addr(&bars->zfull[zb]);
        for (int kb = 0; kb < nk1; ++kb) {
          const int kk = kb * UK, h = kk / d.d_s, d0 = kk - h * d.d_s;
          tma_load_2d_pair(sZ + zb * kZBytes + kb * kBlk16, gi.x ? &tmV : &tmK, bar, d0,
                           ((gi.src_layer * d.B + ti.b) * d.H_s + h) * d.S + ti.s0);
        }
        note(zb, ph);
        return true;
      };
      // W1 rows of chunk c (column block j of group grp) into slot c % 2, once
      // GEMM1(c - 2) has released it
      auto load_w1 = [&](int grp, int j, uint32_t c) -> bool {
        const int s = c & 1;
        const uint32_t ph = (c >> 1) & 1u;
        if (!mbar_wait(&bars->a1full[s], ph ^ 1u, abort_flag, p.wait_limit)) return false;
        if (leader) mbar_arrive_expect_tx(&bars->w1full[s], 2 * nk1 * kW1Blk);
        const uint32_t bar = leader_addr(&bars->w1full[s]);
        const int row = grp * d.EH + j * kChunk + static_cast<int>(rank) * (kChunk / 2);
        for (int kb = 0; kb < nk1; ++kb)
          tma_load_2d_pair(sW1 + s * kW1Bytes + kb * kW1Blk, &tmW1q, bar, kb * UK, row);
        note(2 + s, ph);
        return true;
      };
      // W2 columns of chunk c into slot c % 2, once GEMM2(c - 2) has released it
      auto load_w2 = [&](int grp, int j, uint32_t c) -> bool {
        const int s = c & 1;
        const uint32_t ph = (c >> 1) & 1u;
        if (!mbar_wait(&bars->a2empty[s], ph ^ 1u, abort_flag, p.wait_limit)) return false;
        if (leader) mbar_arrive_expect_tx(&bars->w2full[s], 2 * kW2Bytes);
        const uint32_t bar = leader_addr(&bars->w2full[s]);
        const int row = grp * d.Dt + static_cast<int>(rank) * (UN / 2);
        uint8_t* dst = sW2 + s * kW2Bytes;
        tma_load_2d_pair(dst, &tmW2h, bar, j * kChunk, row);
        tma_load_2d_pair(dst + kBlk16, &tmW2h, bar, j * kChunk + UK, row);
        note(4 + s, ph);
        return true;
      };
      // the tile's bias stage into its Z buffer once GEMM1 of its last chunk
      // c_last is done: B = b2t half, A = gate16 rows of this CTA's token tile
      auto load_bias = [&](int grp, int m_own, uint32_t k, uint32_t c_last) -> bool {
        const int zb = k & 1;
        const uint32_t ph = (k >> 1) & 1u;
        if (!mbar_wait(&bars->a1full[c_last & 1], (c_last >> 1) & 1u, abort_flag, p.wait_limit))
          return false;
        if (leader) mbar_arrive_expect_tx(&bars->bfull[zb], 2 * kZBytes);
        const uint32_t bar = leader_addr(&bars->bfull[zb]);
        const int row = grp * d.Dt + static_cast<int>(rank) * (UN / 2);
        tma_load_2d_pair(sZ + zb * kZBytes, &tmB2th, bar, 0, row);
        tma_load_3d_pair(sZ + zb * kZBytes + kBlk16, &tmG16, bar, 0, m_own * UM, grp);
        note(6 + zb, ph);
        return true;
      };
      uint32_t k = 0, c0 = 0;
      for (int t = pair; t < total; t += n_pairs, ++k, c0 += nc) {
        const int gl = t / n_mp, mp = t - gl * n_mp;
        const int grp = p.g0 + gl;
        const int m_own = 2 * mp + static_cast<int>(rank);
        bool ok = true;
        if (k == 0) ok = load_z(t, 0);
        ok = ok && load_w1(grp, 0, c0);
        if (nc > 1) ok = ok && load_w1(grp, 1, c0 + 1);
        if (t + n_pairs < total) ok = ok && load_z(t + n_pairs, k + 1);
        for (int j = 0; ok && j < nc; ++j) {   // the MMA's order: GEMM1(j + 2), then GEMM2(j)
          if (j + 2 < nc) ok = load_w1(grp, j + 2, c0 + j + 2);
          ok = ok && load_w2(grp, j, c0 + j);
        }
        ok = ok && load_bias(grp, m_own, k, c0 + nc - 1);
        if (!ok) break;
      }
    }
  } else if ((warp == 1 || warp == 3) && leader) {
    // ------------------------------------------------ MMA issuers (leader)
    // GEMM1 (warp 1) and GEMM2 + bias (warp 3) write different accumulators,
    // so each has its own issuing warp: issuing costs tens of cycles per MMA,
    // and one warp issuing both would serialise that with its waits. The
    // loops, waits and descriptors are warp-uniform; one elected lane issues
    // each warp's MMAs and commits (a commit tracks its own thread's MMAs).
    auto wait_all = [&](uint64_t* bar, uint32_t parity) -> bool {
      const bool r = mbar_wait(bar, parity, abort_flag, p.wait_limit);
      return __all_sync(0xffffffffu, r) != 0;
    };
    uint32_t c0 = 0, k = 0;
    bool ok = true;
    if (warp == 1) {
      constexpr uint32_t idesc1 = idesc_bf16_f32(2 * UM, kChunk);
      for (int t = pair; ok && t < total; t += n_pairs, ++k, c0 += nc) {
        const int zb = k & 1;
        if (!wait_all(&bars->zfull[zb], (k >> 1) & 1u)) break;
        tc_fence_after();
        const uint32_t zaddr = smem_u32(sZ + zb * kZBytes);
        for (int j = 0; ok && j < nc; ++j) {
          const uint32_t c = c0 + j, b = c & 1u;
          // acc1[b] is free once the epilogue of chunk c - 2 has read it
          if (c >= 2) ok = wait_all(&bars->acc1free[b], ((c >> 1) & 1u) ^ 1u);
          ok = ok && wait_all(&bars->w1full[b], (c >> 1) & 1u);
          if (!ok) break;
          tc_fence_after();
          const uint32_t waddr = smem_u32(sW1 + b * kW1Bytes);
          if (elect_one()) {
            for (int kb = 0; kb < nk1; ++kb) {
              const uint64_t zdesc = sdesc_k_sw128(zaddr + kb * kBlk16);
              const uint64_t wdesc = sdesc_k_sw128(waddr + kb * kW1Blk);
#pragma unroll
              for (int kk = 0; kk < UK / 16; ++kk)   // +32 bytes of K = +2 in the address field
                umma_pair(tmem_base + kAcc1Col + b * kChunk, zdesc + 2 * kk, wdesc + 2 * kk, idesc1,
                          (kb | kk) != 0);
            }
            umma_commit_pair(&bars->a1full[b]);
          }
          __syncwarp();
          mma_issued = true;
        }
      }
    } else {
      constexpr uint32_t idesc2 = idesc_f16_f32(2 * UM, UN);
      for (int t = pair; ok && t < total; t += n_pairs, ++k, c0 += nc) {
        const int zb = k & 1;
        for (int j = 0; ok && j < nc; ++j) {
          const uint32_t c = c0 + j, b = c & 1u;
          ok = wait_all(&bars->a2full[b], (c >> 1) & 1u);
          if (ok && j == 0) ok = wait_all(&bars->acc2empty, (k & 1u) ^ 1u);
          ok = ok && wait_all(&bars->w2full[b], (c >> 1) & 1u);
          if (!ok) break;
          tc_fence_after();
          const uint32_t aaddr = smem_u32(sA2 + b * kA2Bytes), baddr = smem_u32(sW2 + b * kW2Bytes);
          if (elect_one()) {
#pragma unroll
            for (int kb = 0; kb < 2; ++kb) {
              const uint64_t adesc = sdesc_k_sw128(aaddr + kb * kBlk16);
              const uint64_t bdesc = sdesc_k_sw128(baddr + kb * kBlk16);
#pragma unroll
              for (int kk = 0; kk < UK / 16; ++kk)
                umma_pair(tmem_base, adesc + 2 * kk, bdesc + 2 * kk, idesc2, (j | kb | kk) != 0);
            }
            umma_commit_pair(&bars->a2empty[b]);
          }
          __syncwarp();
          mma_issued = true;
        }
        if (!ok) break;
        // gate-weighted biases from the tile's Z buffer (loaded there once the
        // tile's last GEMM1 is done): A = gate16, B = b2t
        if (!wait_all(&bars->bfull[zb], (k >> 1) & 1u)) break;
        tc_fence_after();
        const uint32_t zaddr = smem_u32(sZ + zb * kZBytes);
        if (elect_one()) {
          const uint64_t gdesc = sdesc_k_sw128(zaddr + kBlk16);
          const uint64_t bdesc = sdesc_k_sw128(zaddr);
#pragma unroll
          for (int kk = 0; kk < UK / 16; ++kk)
            umma_pair(tmem_base, gdesc + 2 * kk, bdesc + 2 * kk, idesc2, 1u);
          umma_commit_pair(&bars->zempty[zb]);
          umma_commit_pair(&bars->acc2full);
        }
        __syncwarp();
      }
    }
  } else if (warp >= 4) {
    // ------------------------------------------------ epilogue (both CTAs)
    const int e = warp - 4, q = e & 3, hh = e >> 2;   // rows 32 q.., chunk columns 32 hh..
    const int r = q * 32 + lane;
    const uint32_t tq = tmem_base + (static_cast<uint32_t>(q * 32) << 16);
    const uint32_t a2_addr = smem_u32(sA2) + static_cast<uint32_t>((hh >> 1) * kBlk16);
    const __half* b1h = static_cast<const __half*>(p.b1h);
    uint32_t c = 0, k = 0;
    bool ok = true;
    for (int t = pair; ok && t < total; t += n_pairs, ++k) {
      const int gl = t / n_mp, mp = t - gl * n_mp;
      const int grp = p.g0 + gl;
      const int m_own = 2 * mp + static_cast<int>(rank);
      const bool valid = m_own < n_m;
      const float* grow =
          p.gate + (static_cast<size_t>(grp) * d.tpad + static_cast<size_t>(m_own) * UM + r) * d.E;
      const uint4* bias4 = reinterpret_cast<const uint4*>(b1h + static_cast<size_t>(grp) * d.EH) +
                           hh * 4;
      for (int j = 0; j < nc; ++j, ++c) {
        const uint32_t b = c & 1u;
        // this warp's 32 biases and the row's gate value, fetched before the wait
        uint4 bias[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) bias[i] = __ldg(bias4 + j * (kChunk / 8) + i);
        const float gate = valid ? __ldg(grow + (j * kChunk) / d.H) : 0.f;
        int w = 1;
        if (lane == 0) w = mbar_wait(&bars->a1full[b], (c >> 1) & 1u, abort_flag, p.wait_limit);
        if (!__shfl_sync(0xffffffffu, w, 0)) { ok = false; break; }
        tc_fence_after();
        uint32_t pa[16];
        {
          uint32_t ra[32];
          tmem_ld_32x32b_x32(tq + kAcc1Col + b * kChunk + hh * 32, ra);
          tmem_ld_wait(ra);
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster(&bars->acc1free[b], 0);   // GEMM1(c + 2) may start
          gelu_cols(ra, bias, __float2half2_rn(0.5f * gate), pa);
        }
        // GEMM2(c - 2) must be done reading this A2 buffer
        if (lane == 0) w = mbar_wait(&bars->a2empty[b], ((c >> 1) & 1u) ^ 1u, abort_flag, p.wait_limit);
        if (!__shfl_sync(0xffffffffu, w, 0)) { ok = false; break; }
        store_a2(a2_addr + b * kA2Bytes, r, hh & 1, pa);
        fence_proxy_async_smem();   // the MMA (async proxy) reads these stores
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(&bars->a2full[b], 0);
      }
      if (!ok) break;
      // output: columns 64 hh .. 64 hh + 63 of this warp's rows
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
        const bool wide = (reinterpret_cast<uintptr_t>(dst) & 31u) == 0;   // 32-byte stores
        const size_t s_pos = static_cast<size_t>(ti.s0) + r;
        auto out = [&](int col) {
          const int h = col / d.d_t, i0 = col - h * d.d_t;
          return dst + ((((static_cast<size_t>(gi.tgt_layer) * d.B + ti.b) * d.H_t + h) * d.S +
                         s_pos) * d.d_t + i0);
        };
        uint32_t ra[32], rb[32];
#pragma unroll 1
        for (int cc = hh * (UN / 4); cc < (hh + 1) * (UN / 4); cc += 64) {
          tmem_ld_32x32b_x32(tq + cc, ra);
          tmem_ld_32x32b_x32(tq + cc + 32, rb);
          tmem_ld_wait(ra);
          tmem_ld_wait(rb);
          if (r < ti.rows) {
            if (wide) {
              store_out32(ra, out(cc));
              store_out32(rb, out(cc + 32));
            } else {
              store_out(ra, out(cc));
              store_out(rb, out(cc + 32));
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive_cluster(&bars->acc2empty, 0);
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    // Unwinding after a timed-out wait (bounded): copies this CTA started
    // complete on the leader's barriers, so give them time to land; the
    // leader also waits for its issued MMAs.
    if (warp == 0 && lane == 0 && pend_mask) {
      if (leader) {
        uint64_t* fulls[8] = {&bars->zfull[0],  &bars->zfull[1],  &bars->w1full[0],
                              &bars->w1full[1], &bars->w2full[0], &bars->w2full[1],
                              &bars->bfull[0],  &bars->bfull[1]};
#pragma unroll
        for (int i = 0; i < 8; ++i)
          if ((pend_mask >> i) & 1u) {
            const uint32_t a = smem_u32(fulls[i]);
            const long long t0 = clock64();
            while (!mbar_try_wait(a, (pend_par >> i) & 1u) && clock64() - t0 < p.wait_limit) {
            }
          }
      } else {
        spin_cycles(20000000LL);
      }
    }
    if ((warp == 1 || warp == 3) && leader && mma_issued) {   // each issuing lane drains its MMAs
      if (elect_one()) {
        uint64_t* dr = warp == 1 ? &bars->drain : &bars->drain2;
        umma_commit_pair(dr);
        const uint32_t a = smem_u32(dr);
        const long long t0 = clock64();
        while (!mbar_try_wait(a, 0) && clock64() - t0 < p.wait_limit) {
        }
      }
      __syncwarp();
    }
    __syncthreads();
  }
  tc_fence_before();
  cluster_sync();   // the leader's MMAs no longer read this CTA's shared memory or TMEM
  if (warp == 2) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, kTmemAlloc);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicOr(p.status, kStatusTimeout);
}

}  // namespace

bool onchip_supported(const Dims& d) {
  return umma_supported(d) && d.Dt == UN && d.Ds <= 2 * UK && d.H % kChunk == 0;
}

cudaError_t launch_onchip(const PathArgs& a, const CUtensorMap& tmK, const CUtensorMap& tmV,
                          const CUtensorMap& tmW1q, const CUtensorMap& tmW2h,
                          const CUtensorMap& tmG16, const CUtensorMap& tmB2th, int num_sms,
                          cudaStream_t st) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(onchip_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         kSmemBytes);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  OnchipArgs oa;
  oa.p = a;
  oa.nk1 = a.d.Ds / UK;
  oa.nc = a.d.EH / kChunk;
  const long long pairs = static_cast<long long>(a.gp) * ((a.d.tiles_max + 1) / 2);
  const long long max_pairs = num_sms / 2;
  const int grid = 2 * static_cast<int>(pairs < max_pairs ? pairs : max_pairs);
  if (grid <= 0) return cudaSuccess;
  onchip_kernel<<<grid, kThreads, kSmemBytes, st>>>(tmK, tmV, tmW1q, tmW2h, tmG16, tmB2th, oa);
  return cudaGetLastError();
}

}  // namespace mot
