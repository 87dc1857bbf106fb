// Gate logits on the tensor cores (Def. 3.1). For one 128-token tile of one
// (target layer, K/V) group the logits are L = Z Wg^T, a [128 x E] product
// with K = D_s: a skinny GEMM whose cost is reading Z from the source cache.
// The source rows stream through a TMA ring exactly as GEMM1's A operand
// does; the group's gate weights, zero-padded to 16 rows (wg16), are the
// B operand, so tcgen05.mma M=128 N=16 accumulates the logits in TMEM. The
// epilogue adds bg, takes the max-subtracted softmax (then Top-K and its
// renormalisation) in fp32 and writes the fp32 gate row [E] and the fp16
// gate16 row [64] used by GEMM2's bias block.
//
// Persistent kernel, one CTA per SM over the work items (group, tile):
//   warp 0 lane 0  TMA producer: per K block, 16 KB of Z and 2 KB of wg16
//                  into an 8-stage ring;
//   warp 1         MMA issue (one elected lane), two TMEM accumulators;
//   warp 2         TMEM allocation (64 columns: accumulator b at 32 b);
//   warps 4..7     epilogue: warp 4 + q owns rows 32 q .. 32 q + 31.
// Every wait is bounded; a timeout unwinds and raises kStatusTimeout.
#include "umma_common.cuh"

namespace mot {
namespace {

constexpr int kGStages = 8;
constexpr int kGN = 16;                              // gate rows of the MMA (E <= 16)
constexpr int kGABytes = UM * UK * 2;                // 16 KB of Z per K block
constexpr int kGBBytes = kGN * UK * 2;               // 2 KB of wg16 per K block
constexpr int kGStageBytes = kGABytes + kGBBytes;    // 18 KB, a multiple of 1024
constexpr int kGThreads = 32 * 8;
constexpr int kGSmem = kGStages * kGStageBytes + 256 + 1024;
constexpr uint32_t kGTmemCols = 64;
static_assert(kGStageBytes % 1024 == 0, "stages keep the 1024-byte swizzle alignment");
static_assert(kGSmem <= 232448, "shared memory budget");

struct GBars {
  uint64_t full[kGStages], empty[kGStages], tfull[2], tempty[2], drain;
  uint32_t tmem_slot;
  int abort_flag;
};
static_assert(sizeof(GBars) <= 256, "barrier block");

__global__ void __launch_bounds__(kGThreads, 1)
    gate_mma_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                    const __grid_constant__ CUtensorMap tmWg, const PathArgs p) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  GBars* bars = reinterpret_cast<GBars*>(smem + kGStages * kGStageBytes);
  volatile int* abort_flag = &bars->abort_flag;
  const Dims& d = p.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kGStages; ++s) {
      mbar_init(&bars->full[s], 1);
      mbar_init(&bars->empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&bars->tfull[a], 1);
      mbar_init(&bars->tempty[a], 4);
    }
    mbar_init(&bars->drain, 1);
    bars->abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
    tma_prefetch_desc(&tmWg);
  }
  if (warp == 2) {
    tmem_alloc(&bars->tmem_slot, kGTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = bars->tmem_slot;

  const int n_m = min(*p.n_tiles, d.tiles_max);
  const int total = p.gp * n_m;
  const int nk = d.Ds / UK;
  uint32_t issued_mask = 0, issue_parity = 0;
  bool mma_issued = false;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer
      int stage = 0;
      uint32_t phase = 0;
      bool ok = true;
      for (int t = blockIdx.x; ok && t < total; t += gridDim.x) {
        const int gl = t / n_m, m = t - gl * n_m, grp = p.g0 + gl;
        const TileInfo ti = p.tiles[m];
        const GroupInfo gi = p.groups[grp];
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait(&bars->empty[stage], phase ^ 1u, abort_flag, p.wait_limit)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&bars->full[stage], kGStageBytes);
          uint8_t* st = smem + stage * kGStageBytes;
          const int k = kb * UK, h = k / d.d_s, d0 = k - h * d.d_s;
          tma_load_2d(st, gi.x ? &tmV : &tmK, &bars->full[stage], d0,
                      ((gi.src_layer * d.B + ti.b) * d.H_s + h) * d.S + ti.s0);
          tma_load_2d(st + kGABytes, &tmWg, &bars->full[stage], k, grp * kGN);
          issued_mask |= 1u << stage;
          issue_parity = (issue_parity & ~(1u << stage)) | (phase << stage);
          if (++stage == kGStages) { stage = 0; phase ^= 1u; }
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------ MMA issuer (warp-uniform, elected lane)
    constexpr uint32_t idesc = idesc_bf16_f32(UM, kGN);
    auto wait_all = [&](uint64_t* bar, uint32_t parity) -> bool {
      const bool r = mbar_wait(bar, parity, abort_flag, p.wait_limit);
      return __all_sync(0xffffffffu, r) != 0;
    };
    int stage = 0, acc = 0;
    uint32_t phase = 0, acc_phase = 0;
    bool ok = true;
    for (int t = blockIdx.x; ok && t < total; t += gridDim.x) {
      if (!wait_all(&bars->tempty[acc], acc_phase ^ 1u)) break;
      tc_fence_after();
      for (int kb = 0; kb < nk; ++kb) {
        if (!wait_all(&bars->full[stage], phase)) { ok = false; break; }
        tc_fence_after();
        const uint32_t sa = smem_u32(smem + stage * kGStageBytes);
        if (elect_one()) {
          const uint64_t adesc = sdesc_k_sw128(sa), bdesc = sdesc_k_sw128(sa + kGABytes);
#pragma unroll
          for (int kk = 0; kk < UK / 16; ++kk)
            umma_bf16(tmem_base + acc * 32, adesc + 2 * kk, bdesc + 2 * kk, idesc, (kb | kk) != 0);
          umma_commit(&bars->empty[stage]);
        }
        __syncwarp();
        mma_issued = true;
        if (++stage == kGStages) { stage = 0; phase ^= 1u; }
      }
      if (!ok) break;
      if (elect_one()) umma_commit(&bars->tfull[acc]);
      __syncwarp();
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
  } else if (warp >= 4) {
    // ------------------------------------------------ epilogue: softmax and Top-K per row
    const int q = warp - 4, r = q * 32 + lane;
    const int E = d.E;
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int t = blockIdx.x; t < total; t += gridDim.x) {
      const int gl = t / n_m, m = t - gl * n_m, grp = p.g0 + gl;
      const TileInfo ti = p.tiles[m];
      float bias[kGN];
#pragma unroll
      for (int e = 0; e < kGN; ++e) bias[e] = e < E ? __ldg(p.bg + grp * E + e) : 0.f;
      int w = 1;
      if (lane == 0) w = mbar_wait(&bars->tfull[acc], acc_phase, abort_flag, p.wait_limit) ? 1 : 0;
      if (!__shfl_sync(0xffffffffu, w, 0)) break;
      tc_fence_after();
      uint32_t raw[32];
      tmem_ld_32x32b_x32(tmem_base + acc * 32 + (static_cast<uint32_t>(q * 32) << 16), raw);
      tmem_ld_wait(raw);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&bars->tempty[acc]);
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;

      float g[kGN];
#pragma unroll
      for (int e = 0; e < kGN; ++e) g[e] = 0.f;
      uint32_t chosen = 0;   // the row's Top-K choices (sparse routing)
      if (r < ti.rows) {
        float mx = -INFINITY;
#pragma unroll
        for (int e = 0; e < kGN; ++e)
          if (e < E) {
            g[e] = __uint_as_float(raw[e]) + bias[e];
            mx = fmaxf(mx, g[e]);
          }
        float sum = 0.f;
#pragma unroll
        for (int e = 0; e < kGN; ++e)
          if (e < E) {
            g[e] = expf(g[e] - mx);
            sum += g[e];
          }
        const float inv = 1.f / sum;
#pragma unroll
        for (int e = 0; e < kGN; ++e) g[e] = e < E ? g[e] * inv : 0.f;
        if (d.top_k > 0 && d.top_k < E) {   // keep the top_k largest; ties: lower index
          uint32_t keep = 0;
          for (int kk = 0; kk < d.top_k; ++kk) {
            int best = -1;
            float bv = 0.f;
#pragma unroll
            for (int e = 0; e < kGN; ++e)
              if (e < E && !((keep >> e) & 1u) && (best < 0 || g[e] > bv)) {
                best = e;
                bv = g[e];
              }
            keep |= 1u << best;
          }
          float ks = 0.f;
#pragma unroll
          for (int e = 0; e < kGN; ++e)
            if (e < E && ((keep >> e) & 1u)) ks += g[e];
          const float kinv = 1.f / ks;
#pragma unroll
          for (int e = 0; e < kGN; ++e) g[e] = (e < E && ((keep >> e) & 1u)) ? g[e] * kinv : 0.f;
          chosen = keep;
        }
      }
      const size_t row = static_cast<size_t>(grp) * d.tpad + static_cast<size_t>(m) * UM + r;
      if (p.sel) p.sel[row] = chosen;
      float* __restrict__ gout = p.gate + row * E;
#pragma unroll
      for (int e = 0; e < kGN; ++e)
        if (e < E) gout[e] = g[e];
      if (p.gate16) {   // columns 0 .. 15 carry gtilde (zeros past E), 16 .. 63 are zero
        uint4* out = reinterpret_cast<uint4*>(static_cast<uint16_t*>(p.gate16) + row * 64);
#pragma unroll
        for (int v = 0; v < 2; ++v) {
          uint32_t wv[4];
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const __half2 hv = __floats2half2_rn(g[8 * v + 2 * k], g[8 * v + 2 * k + 1]);
            wv[k] = *reinterpret_cast<const uint32_t*>(&hv);
          }
          out[v] = make_uint4(wv[0], wv[1], wv[2], wv[3]);
        }
#pragma unroll
        for (int v = 2; v < 8; ++v) out[v] = make_uint4(0, 0, 0, 0);
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    // Unwinding after a timed-out wait (bounded): copies in flight land and
    // issued MMAs finish before TMEM is freed.
    if (warp == 0 && lane == 0) {
      for (int s = 0; s < kGStages; ++s)
        if ((issued_mask >> s) & 1u) {
          const uint32_t a = smem_u32(&bars->full[s]);
          const long long t0 = clock64();
          while (!mbar_try_wait(a, (issue_parity >> s) & 1u) && clock64() - t0 < p.wait_limit) {
          }
        }
    }
    if (warp == 1 && mma_issued) {
      if (elect_one()) {
        umma_commit(&bars->drain);
        const uint32_t a = smem_u32(&bars->drain);
        const long long t0 = clock64();
        while (!mbar_try_wait(a, 0) && clock64() - t0 < p.wait_limit) {
        }
      }
      __syncwarp();
    }
    __syncthreads();
  }
  if (warp == 2) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, kGTmemCols);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicOr(p.status, kStatusTimeout);
}

}  // namespace

cudaError_t launch_gate_mma(const PathArgs& a, const CUtensorMap& tmK, const CUtensorMap& tmV,
                            const CUtensorMap& tmWg, int num_sms, cudaStream_t st) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e =
        cudaFuncSetAttribute(gate_mma_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kGSmem);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  const long long items = static_cast<long long>(a.gp) * a.d.tiles_max;
  const int grid = static_cast<int>(items < num_sms ? items : num_sms);
  if (grid <= 0) return cudaSuccess;
  gate_mma_kernel<<<grid, kGThreads, kGSmem, st>>>(tmK, tmV, tmWg, a);
  return cudaGetLastError();
}

}  // namespace mot
