// Fused persistent translation kernel (tcgen05 / TMEM / TMA, bf16 in, fp32 acc).
//
// One launch runs both GEMMs of a pass (see umma.cu for the two GEMMs) as a
// single stream of work items claimed dynamically with an atomic counter in
// the order of schedule.h: 256-column GEMM1 items (source tile x W1cat ->
// GELU * gate -> A2) and 256-column GEMM2 items (A2 x W2cat -> + gate-weighted
// bias -> target cache), skewed so that a GEMM2 item is issued about one block
// of tiles after the GEMM1 items it reads. Compared with two launches:
//   - A2 rows are consumed within microseconds of being written, from L2;
//   - GEMM1's elementwise epilogue overlaps GEMM2's long main loops on the
//     same SM instead of bounding a kernel of its own;
//   - one tail per pass instead of two.
//
// Roles (384 threads): warp 0 lane 0 claims items and drives TMA loads; warp 1
// lane 0 issues tcgen05.mma into two 256-column TMEM accumulators; warp 2
// owns TMEM; warps 4-11 are the epilogue (two per TMEM lane quarter, 128
// columns each). Claimed item ids reach the MMA and epilogue warps through a
// 4-deep shared-memory ring guarded by mbarriers.
//
// Cross-CTA dependency: every epilogue warp, once the TMA stores of its part
// of a GEMM1 item have completed, adds 1 to done[f] of the item's token tile
// with release semantics (after a proxy fence); the producer of a GEMM2 item
// spins (bounded, acquire) until done[f] == n1 * 8, then fences the async
// proxy before its TMA loads of A2. A warp signals an item when it reads the
// next item id, so it never sits on a signal while waiting for more work.
// Every wait is bounded; a timeout unwinds all roles and raises
// kStatusTimeout.
#include "schedule.h"
#include "umma_common.cuh"

namespace mot {
namespace {

constexpr int kEpiWarps = 8;
constexpr int kThreads = 32 * (4 + kEpiWarps);
constexpr int kRing = 4;
constexpr int kBarBytes = 512;
constexpr int kSmemBytes = kStages * kStageBytes + kEpiWarps * kStoreTileBytes + kBarBytes + 1024;
static_assert(kSmemBytes <= 232448, "shared memory budget");

struct FusedArgs {
  PathArgs p;
  int32_t n1, n2;     // 256-column tiles of E*H and of D_t
  int32_t nk1, nk2;   // 64-element K blocks of D_s and of E*H (+1: the bias block)
  int32_t mb;         // token tiles per schedule block
  int32_t* counters;  // [0] item counter, [1 + f] GEMM1 completions of flat tile f
};

__device__ __forceinline__ int ld_acquire(const int32_t* p) {
  int v;
  asm volatile("ld.acquire.gpu.global.s32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ void fence_proxy_async_global() {
  asm volatile("fence.proxy.async.global;" ::: "memory");
}

// Publish one epilogue warp's completed GEMM1 stores for flat tile f.
__device__ __forceinline__ void signal_done(int32_t* ctr) {
  bulk_wait_group<0>();          // this thread's TMA stores are complete
  fence_proxy_async_global();    // order them before the release below
  asm volatile("red.release.gpu.global.add.s32 [%0], 1;" ::"l"(ctr) : "memory");
}

// Bounded acquire-spin until *ctr >= target; then order the async proxy.
__device__ __forceinline__ bool wait_done(const int32_t* ctr, int target,
                                          volatile int* abort_flag, long long limit) {
  const long long t0 = clock64();
  for (;;) {
    if (ld_acquire(ctr) >= target) {
      fence_proxy_async_global();
      return true;
    }
    if (*abort_flag) return false;
    if (clock64() - t0 > limit) {
      *abort_flag = 1;
      return false;
    }
    __nanosleep(128);
  }
}

__global__ void __launch_bounds__(kThreads, 1)
    mot_fused_kernel(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV,
                     const __grid_constant__ CUtensorMap tmW1,
                     const __grid_constant__ CUtensorMap tmA2,
                     const __grid_constant__ CUtensorMap tmW2,
                     const __grid_constant__ CUtensorMap tmS,
                     const __grid_constant__ CUtensorMap tmG16,
                     const __grid_constant__ CUtensorMap tmB2t, const FusedArgs fa) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + kStages * kABytes;
  uint8_t* sOut = smem + kStages * kStageBytes;
  uint64_t* full = reinterpret_cast<uint64_t*>(sOut + kEpiWarps * kStoreTileBytes);
  uint64_t* empty = full + kStages;
  uint64_t* tfull = empty + kStages;   // [2]
  uint64_t* tempty = tfull + 2;        // [2]
  uint64_t* drain = tempty + 2;        // [1]
  uint64_t* ifull = drain + 1;         // [kRing]
  uint64_t* iempty = ifull + kRing;    // [kRing]
  volatile int32_t* ring = reinterpret_cast<volatile int32_t*>(iempty + kRing);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(const_cast<int32_t*>(ring) + kRing);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const PathArgs& p = fa.p;
  const Dims& d = p.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], kEpiWarps);
    }
    mbar_init(drain, 1);
    for (int r = 0; r < kRing; ++r) {
      mbar_init(&ifull[r], 1);
      mbar_init(&iempty[r], 1 + kEpiWarps);
    }
    *abort_flag = 0;
    fence_barrier_init();
  }
  if (warp == 0 && lane == 0) {
    tma_prefetch_desc(&tmK);
    tma_prefetch_desc(&tmV);
    tma_prefetch_desc(&tmW1);
    tma_prefetch_desc(&tmA2);
    tma_prefetch_desc(&tmW2);
    tma_prefetch_desc(&tmS);
    tma_prefetch_desc(&tmG16);
    tma_prefetch_desc(&tmB2t);
  }
  if (warp == 2) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int n_m = min(*p.n_tiles, d.tiles_max);
  Schedule sch;
  sch.F = p.gp * n_m;
  sch.n1 = fa.n1;
  sch.n2 = fa.n2;
  sch.MB = fa.mb;
  const int total = sch.total();
  int32_t* done = fa.counters + 1;
  const int done_target = fa.n1 * kEpiWarps;

  uint32_t issued_mask = 0, issue_parity = 0;
  bool mma_issued = false;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ claim items + TMA producer
      int stage = 0, slot = 0;
      uint32_t phase = 0, sphase = 0;
      for (;;) {
        if (!mbar_wait(&iempty[slot], sphase ^ 1u, abort_flag, p.wait_limit)) break;
        int i = atomicAdd(fa.counters, 1);
        if (i >= total) i = -1;
        ring[slot] = i;
        mbar_arrive(&ifull[slot]);
        if (++slot == kRing) { slot = 0; sphase ^= 1u; }
        if (i < 0) break;
        const Item it = schedule_item(sch, i);
        const int gl = it.f / n_m, m = it.f - gl * n_m, grp = p.g0 + gl;
        if (it.type == 2 && !wait_done(done + it.f, done_target, abort_flag, p.wait_limit)) break;
        TileInfo ti;
        GroupInfo gi;
        if (it.type == 1) {
          ti = p.tiles[m];
          gi = p.groups[grp];
        }
        const int nk = it.type == 1 ? fa.nk1 : fa.nk2;
        bool ok = true;
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, p.wait_limit)) { ok = false; break; }
          mbar_arrive_expect_tx(&full[stage], kStageBytes);
          if (it.type == 1) {
            const int k = kb * UK, h = k / d.d_s, d0 = k - h * d.d_s;
            tma_load_2d(sA + stage * kABytes, gi.x ? &tmV : &tmK, &full[stage], d0,
                        ((gi.src_layer * d.B + ti.b) * d.H_s + h) * d.S + ti.s0);
            tma_load_2d(sB + stage * kBBytes, &tmW1, &full[stage], kb * UK,
                        grp * d.EH + it.n * UN);
          } else if (kb < nk - 1) {   // A2 x W2cat
            tma_load_3d(sA + stage * kABytes, &tmA2, &full[stage], kb * UK, m * UM, gl);
            tma_load_2d(sB + stage * kBBytes, &tmW2, &full[stage], kb * UK,
                        grp * d.Dt + it.n * UN);
          } else {                    // last K block: gate16 x b2t (the combine biases)
            tma_load_3d(sA + stage * kABytes, &tmG16, &full[stage], 0, m * UM, grp);
            tma_load_2d(sB + stage * kBBytes, &tmB2t, &full[stage], 0, grp * d.Dt + it.n * UN);
          }
          issued_mask |= 1u << stage;
          issue_parity = (issue_parity & ~(1u << stage)) | (phase << stage);
          if (++stage == kStages) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      // ------------------------------------------------ MMA issuer
      const uint32_t idesc1 = idesc_bf16_f32(UM, UN);   // bf16 source x bf16 W1
      const uint32_t idesc2 = idesc_f16_f32(UM, UN);    // fp16 A2 x fp16 W2
      int stage = 0, slot = 0, acc = 0;
      uint32_t phase = 0, sphase = 0, acc_phase = 0;
      for (;;) {
        if (!mbar_wait(&ifull[slot], sphase, abort_flag, p.wait_limit)) break;
        const int i = ring[slot];
        mbar_arrive(&iempty[slot]);
        if (++slot == kRing) { slot = 0; sphase ^= 1u; }
        if (i < 0) break;
        const Item it = schedule_item(sch, i);
        const int nk = it.type == 1 ? fa.nk1 : fa.nk2;
        const uint32_t idesc = it.type == 1 ? idesc1 : idesc2;
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, p.wait_limit)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * UN);
        bool ok = true;
        for (int kb = 0; kb < nk; ++kb) {
          if (!mbar_wait(&full[stage], phase, abort_flag, p.wait_limit)) { ok = false; break; }
          tc_fence_after();
          const uint64_t adesc = sdesc_k_sw128(smem_u32(sA + stage * kABytes));
          const uint64_t bdesc = sdesc_k_sw128(smem_u32(sB + stage * kBBytes));
#pragma unroll
          for (int k = 0; k < UK / 16; ++k)   // +32 bytes of K per step = +2 in the address field
            umma_bf16(d_tmem, adesc + 2 * k, bdesc + 2 * k, idesc, (kb | k) != 0);
          mma_issued = true;
          umma_commit(&empty[stage]);
          if (++stage == kStages) { stage = 0; phase ^= 1u; }
        }
        if (!ok) break;
        umma_commit(&tfull[acc]);
        acc ^= 1;
        if (acc == 0) acc_phase ^= 1u;
      }
    }
  } else if (warp >= 4) {
    // ------------------------------------------------ epilogue
    const int e = warp - 4;
    const int q = e & 3;   // TMEM lane quarter (= warp % 4)
    uint8_t* tile = sOut + e * kStoreTileBytes;
    int slot = 0, acc = 0, pending_f = -1;
    uint32_t sphase = 0, acc_phase = 0;
    for (;;) {
      int ok = 1, i = 0;
      if (lane == 0) {
        ok = mbar_wait(&ifull[slot], sphase, abort_flag, p.wait_limit) ? 1 : 0;
        if (ok) i = ring[slot];
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      i = __shfl_sync(0xffffffffu, i, 0);
      if (lane == 0) mbar_arrive(&iempty[slot]);
      if (++slot == kRing) { slot = 0; sphase ^= 1u; }
      if (pending_f >= 0) {
        if (lane == 0) signal_done(done + pending_f);
        pending_f = -1;
      }
      if (i < 0) break;
      const Item it = schedule_item(sch, i);
      const int gl = it.f / n_m, m = it.f - gl * n_m, grp = p.g0 + gl;
      if (lane == 0) ok = mbar_wait(&tfull[acc], acc_phase, abort_flag, p.wait_limit) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      tc_fence_after();
      const uint32_t tbase = tmem_base + static_cast<uint32_t>(acc * UN) +
                             (static_cast<uint32_t>(q * 32) << 16);
      if (it.type == 1) {
        epilogue_gemm1(p, &tmS, tbase, tile, q, lane, grp, it.n * UN, it.n * UN, m * UM, gl,
                       (e >> 2) * 128, 2,
                       gemm1_prefetch(p, q, lane, grp, m, it.n * UN, (e >> 2) * 128));
        pending_f = it.f;
      } else {
        epilogue_gemm2(p, tbase, q, lane, grp, m, it.n * UN, (e >> 2) * 128, 4);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
    if (lane == 0) bulk_wait_group<0>();
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    // Unwinding after a timed-out wait: let every copy the producer started
    // land and every MMA already issued finish before TMEM is freed.
    if (warp == 0 && lane == 0) {
      for (int s = 0; s < kStages; ++s)
        if ((issued_mask >> s) & 1u) {
          const uint32_t a = smem_u32(&full[s]);
          const long long t0 = clock64();
          while (!mbar_try_wait(a, (issue_parity >> s) & 1u) && clock64() - t0 < p.wait_limit) {
          }
        }
    }
    if (warp == 1 && lane == 0 && mma_issued) {
      umma_commit(drain);
      const uint32_t a = smem_u32(drain);
      const long long t0 = clock64();
      while (!mbar_try_wait(a, 0) && clock64() - t0 < p.wait_limit) {
      }
    }
    __syncthreads();
  }
  if (warp == 2) {
    __syncwarp();
    tc_fence_after();
    tmem_dealloc(tmem_base, kTmemCols);
  }
  if (threadIdx.x == 0 && *abort_flag) atomicOr(p.status, kStatusTimeout);
}

}  // namespace

// Token tiles per schedule block: enough GEMM1 items between a GEMM2 item and
// its producers that the producers have finished (about 1.5 items per SM).
int fused_block_tiles(const Dims& d, int num_sms) {
  const int n1 = d.EH / UN;
  return max(1, (3 * num_sms / 2 + n1 - 1) / n1);
}

size_t fused_counter_ints(const Dims& d, int gp) { return 1 + size_t(gp) * d.tiles_max; }

cudaError_t launch_fused(const PathArgs& a, const CUtensorMap& tmK, const CUtensorMap& tmV,
                         const CUtensorMap& tmW1, const CUtensorMap& tmA2,
                         const CUtensorMap& tmW2, const CUtensorMap& tmA2st,
                         const CUtensorMap& tmG16, const CUtensorMap& tmB2t, int32_t* counters,
                         int num_sms, cudaStream_t st) {
  static bool attr_set = false;
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(mot_fused_kernel,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemBytes);
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  cudaError_t e = cudaMemsetAsync(counters, 0, fused_counter_ints(a.d, a.gp) * sizeof(int32_t), st);
  if (e != cudaSuccess) return e;
  FusedArgs fa;
  fa.p = a;
  fa.n1 = a.d.EH / UN;
  fa.n2 = a.d.Dt / UN;
  fa.nk1 = a.d.Ds / UK;
  fa.nk2 = a.d.EH / UK + 1;   // + the combine-bias K block
  fa.mb = fused_block_tiles(a.d, num_sms);
  fa.counters = counters;
  const long long upper = static_cast<long long>(a.gp) * a.d.tiles_max * (fa.n1 + fa.n2);
  const int grid = static_cast<int>(upper < num_sms ? upper : num_sms);
  if (grid <= 0) return cudaSuccess;
  mot_fused_kernel<<<grid, kThreads, kSmemBytes, st>>>(tmK, tmV, tmW1, tmA2, tmW2, tmA2st, tmG16,
                                                       tmB2t, fa);
  return cudaGetLastError();
}

}  // namespace mot
