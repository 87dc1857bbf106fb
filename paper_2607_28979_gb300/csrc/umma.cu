// tcgen05 / TMEM / TMA translation GEMMs for sm_103a (fp32 accumulate; GEMM1
// bf16 x bf16, GEMM2 fp16 x fp16 on the fp16 intermediate and fp16 W2).
//
// The MoT combine (Eq. mot_definition) is a K-reduction once the experts are
// concatenated: with W1cat = [W1_1; ...; W1_E] (E*H x D_s) and
// W2cat = [W2_1, ..., W2_E] (D_t x E*H),
//   GEMM1:  A2 = fp16( GELU(Z W1cat^T + b1cat) (.) gtilde_expand )      [T, E*H]
//   GEMM2:  Y  = A2 W2cat^T + gate16 b2t^T                                [T, D_t]
//           (the last K block adds sum_m gtilde_m b2_m: gate16 holds gtilde, b2t = b2^T)
// so sum_m gtilde_m W2_m GELU(W1_m z + b1_m) is exactly GEMM2's sum over E*H.
//
// One persistent, warp-specialised kernel template runs both GEMMs:
//   warp 0 (one lane)  TMA producer: A and B K-blocks (64 bf16 = one 128-byte
//                      swizzle row) into a 4-stage shared-memory ring;
//   warp 1 (one lane)  MMA issuer: tcgen05.mma M=128, N=256, K=16, fp32
//                      accumulator in TMEM, two accumulator buffers (512 cols);
//   warp 2             TMEM allocator;
//   warps 4..          epilogue: tcgen05.ld of the accumulator (warp w reads
//                      lanes 32*(w%4)...), fused bias / GELU / gate / combine.
//                      GEMM1 runs 8 epilogue warps (two per lane quarter, each
//                      owning 128 of the 256 columns) and writes A2 through a
//                      128B-swizzled shared-memory tile and a TMA store; GEMM2
//                      runs 4 and stores 16-byte vectors straight into the
//                      target cache rows (only rows inside the sequence).
// The epilogue of tile i overlaps the MMAs of tile i+1. Every wait is bounded
// (mot::mbar_wait); on a timeout all roles unwind, in-flight copies and MMAs
// are drained, TMEM is freed and kStatusTimeout is raised.
//
// GEMM1's A operand is read straight from the source cache [L_s][B][H_s][S][d_s]
// through a 2-D tensor map over its rows (inner dim d_s, row
// ((l * B + b) * H_s + h) * S + s) with box (64, 128): K-block kb is head
// kb*64 / d_s, dims (kb*64) % d_s .. +63, of 128 consecutive positions of one
// batch entry. In a short last tile the rows past S are the next head's (or,
// at the end of the cache, zeros); rows past the tile's length are computed
// but never stored.
#include "umma_common.cuh"

namespace mot {
namespace {

constexpr int kBarBytes = 256;
__host__ __device__ constexpr int epi_warps(int mode) { return mode == 1 ? 8 : 4; }
__host__ __device__ constexpr int threads_of(int mode) { return 32 * (4 + epi_warps(mode)); }
__host__ __device__ constexpr int store_bytes(int mode) {
  return mode == 1 ? epi_warps(mode) * kStoreTileBytes : 0;
}
__host__ __device__ constexpr int smem_bytes(int mode) {
  return kStages * kStageBytes + store_bytes(mode) + kBarBytes + 1024;   // + alignment slack
}
static_assert(smem_bytes(1) <= 232448 && smem_bytes(2) <= 232448, "shared memory budget");

struct UmmaArgs {
  PathArgs p;
  int32_t nk;        // K blocks per tile
  int32_t n_tiles_n; // N tiles per group
  int32_t b_rows;    // rows of B per group (E*H for GEMM1, D_t for GEMM2)
};

template <int MODE>   // 1 = GEMM1 (A = source cache), 2 = GEMM2 (A = A2)
__global__ void __launch_bounds__(threads_of(MODE), 1)
    umma_gemm_kernel(const __grid_constant__ CUtensorMap tmA0,
                     const __grid_constant__ CUtensorMap tmA1,
                     const __grid_constant__ CUtensorMap tmB,
                     const __grid_constant__ CUtensorMap tmS, const UmmaArgs ua) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  uint8_t* sA = smem;
  uint8_t* sB = smem + kStages * kABytes;
  uint8_t* sOut = smem + kStages * kStageBytes;   // GEMM1: one store tile per epilogue warp
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes + store_bytes(MODE));
  uint64_t* empty = full + kStages;
  uint64_t* tfull = empty + kStages;    // [2]
  uint64_t* tempty = tfull + 2;         // [2]
  uint64_t* drain = tempty + 2;         // [1] used only when unwinding
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain + 1);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const PathArgs& p = ua.p;
  const Dims& d = p.d;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    for (int a = 0; a < 2; ++a) {
      mbar_init(&tfull[a], 1);
      mbar_init(&tempty[a], epi_warps(MODE));
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
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;

  const int n_m = min(*p.n_tiles, d.tiles_max);
  const int per_grp = n_m * ua.n_tiles_n;
  const int total = p.gp * per_grp;
  // Unwind bookkeeping: TMA loads issued per stage and their phase parity
  // (producer lane), and whether any MMA was issued (MMA lane).
  uint32_t issued_mask = 0, issue_parity = 0;
  bool mma_issued = false;

  if (warp == 0) {
    if (lane == 0) {
      // ------------------------------------------------ TMA producer
      int stage = 0;
      uint32_t phase = 0;
      for (int t = blockIdx.x; t < total; t += gridDim.x) {
        const int gl = t / per_grp, rem = t - gl * per_grp;
        const int m = rem / ua.n_tiles_n, n = rem - m * ua.n_tiles_n;
        const int grp = p.g0 + gl;
        TileInfo ti;
        GroupInfo gi;
        if (MODE == 1) {
          ti = p.tiles[m];
          gi = p.groups[grp];
        }
        bool ok = true;
        for (int kb = 0; kb < ua.nk; ++kb) {
          if (!mbar_wait(&empty[stage], phase ^ 1u, abort_flag, p.wait_limit)) { ok = false; break; }
          if (MODE == 1 && p.stall_test && blockIdx.x == 0 && t == 0 && kb == 0) {
            // test hook: this stage is never filled, so the MMA wait on it runs out
            if (++stage == kStages) { stage = 0; phase ^= 1u; }
            continue;
          }
          mbar_arrive_expect_tx(&full[stage], kStageBytes);
          if (MODE == 1) {
            const int k = kb * UK, h = k / d.d_s, d0 = k - h * d.d_s;
            tma_load_2d(sA + stage * kABytes, gi.x ? &tmA1 : &tmA0, &full[stage], d0,
                        ((gi.src_layer * d.B + ti.b) * d.H_s + h) * d.S + ti.s0);
            tma_load_2d(sB + stage * kBBytes, &tmB, &full[stage], kb * UK,
                        grp * ua.b_rows + n * UN);
          } else if (kb < ua.nk - 1) {   // A2 x W2cat
            tma_load_3d(sA + stage * kABytes, &tmA0, &full[stage], kb * UK, m * UM, gl);
            tma_load_2d(sB + stage * kBBytes, &tmB, &full[stage], kb * UK,
                        grp * ua.b_rows + n * UN);
          } else {                       // last K block: gate16 x b2t (the combine biases)
            tma_load_3d(sA + stage * kABytes, &tmA1, &full[stage], 0, m * UM, grp);
            tma_load_2d(sB + stage * kBBytes, &tmS, &full[stage], 0, grp * ua.b_rows + n * UN);
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
      // GEMM1: bf16 source x bf16 W1; GEMM2: fp16 A2 x fp16 W2
      const uint32_t idesc = MODE == 1 ? idesc_bf16_f32(UM, UN) : idesc_f16_f32(UM, UN);
      int stage = 0;
      uint32_t phase = 0;
      int acc = 0;
      uint32_t acc_phase = 0;
      for (int t = blockIdx.x; t < total; t += gridDim.x) {
        if (!mbar_wait(&tempty[acc], acc_phase ^ 1u, abort_flag, p.wait_limit)) break;
        tc_fence_after();
        const uint32_t d_tmem = tmem_base + static_cast<uint32_t>(acc * UN);
        bool ok = true;
        for (int kb = 0; kb < ua.nk; ++kb) {
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
    const int q = e & 3;                // TMEM lane quarter of this warp (= warp % 4)
    int acc = 0;
    uint32_t acc_phase = 0;
    for (int t = blockIdx.x; t < total; t += gridDim.x) {
      int ok = 1;
      if (lane == 0) ok = mbar_wait(&tfull[acc], acc_phase, abort_flag, p.wait_limit) ? 1 : 0;
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (!ok) break;
      tc_fence_after();
      const int gl = t / per_grp, rem = t - gl * per_grp;
      const int m = rem / ua.n_tiles_n, n = rem - m * ua.n_tiles_n;
      const int grp = p.g0 + gl;
      const uint32_t tbase = tmem_base + static_cast<uint32_t>(acc * UN) +
                             (static_cast<uint32_t>(q * 32) << 16);
      if (MODE == 1)   // 8 warps: this warp owns columns 128 * (e / 4) .. +127
        epilogue_gemm1(p, &tmS, tbase, sOut + e * kStoreTileBytes, q, lane, grp, n * UN, n * UN,
                       m * UM, gl, (e >> 2) * 128, 2,
                       gemm1_prefetch(p, q, lane, grp, m, n * UN, (e >> 2) * 128));
      else             // 4 warps: all 256 columns
        epilogue_gemm2(p, tbase, q, lane, grp, m, n * UN, 0, UN / 32);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty[acc]);
      acc ^= 1;
      if (acc == 0) acc_phase ^= 1u;
    }
    if (MODE == 1 && lane == 0) bulk_wait_group<0>();   // A2 stores complete before exit
  }

  tc_fence_before();
  __syncthreads();
  if (*abort_flag) {
    // Unwinding after a timed-out wait: let every copy the producer started
    // land and every MMA already issued finish before TMEM is freed and the
    // CTA exits. These waits are bounded as well.
    if (warp == 0 && lane == 0) {
      for (int s = 0; s < kStages; ++s)
        if ((issued_mask >> s) & 1u) {
          const uint32_t a = smem_u32(&full[s]);
          const long long t0 = clock64();
          while (!mbar_try_wait(a, (issue_parity >> s) & 1u) &&
                 clock64() - t0 < p.wait_limit) {
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

template <int MODE>
cudaError_t launch_umma(const PathArgs& a, const CUtensorMap& A0, const CUtensorMap& A1,
                        const CUtensorMap& B, const CUtensorMap& S, int nk, int n_tiles_n,
                        int b_rows, int num_sms, cudaStream_t st) {
  static bool attr_set = false;   // per process; the attribute is per function
  if (!attr_set) {
    cudaError_t e = cudaFuncSetAttribute(umma_gemm_kernel<MODE>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         smem_bytes(MODE));
    if (e != cudaSuccess) return e;
    attr_set = true;
  }
  UmmaArgs ua;
  ua.p = a;
  ua.nk = nk;
  ua.n_tiles_n = n_tiles_n;
  ua.b_rows = b_rows;
  const long long upper = static_cast<long long>(a.gp) * a.d.tiles_max * n_tiles_n;
  const int grid = static_cast<int>(upper < num_sms ? upper : num_sms);
  if (grid <= 0) return cudaSuccess;
  umma_gemm_kernel<MODE><<<grid, threads_of(MODE), smem_bytes(MODE), st>>>(A0, A1, B, S, ua);
  return cudaGetLastError();
}

}  // namespace

bool umma_supported(const Dims& d) {
  return d.dtype == 0 && d.d_s % UK == 0 && d.Ds % UK == 0 && d.H % UN == 0 && d.EH % UK == 0 &&
         d.Dt % UN == 0 && d.d_t % 32 == 0 && d.E <= kMaxE;
}

cudaError_t launch_umma_gemm1(const PathArgs& a, const CUtensorMap& tmK, const CUtensorMap& tmV,
                              const CUtensorMap& tmW1, const CUtensorMap& tmA2st, int num_sms,
                              cudaStream_t st) {
  return launch_umma<1>(a, tmK, tmV, tmW1, tmA2st, a.d.Ds / UK, a.d.EH / UN, a.d.EH, num_sms, st);
}

// GEMM2's map slots: A0 = A2, A1 = gate16, B = W2cat, S = b2t (last K block).
cudaError_t launch_umma_gemm2(const PathArgs& a, const CUtensorMap& tmA2, const CUtensorMap& tmW2,
                              const CUtensorMap& tmG16, const CUtensorMap& tmB2t, int num_sms,
                              cudaStream_t st) {
  return launch_umma<2>(a, tmA2, tmG16, tmW2, tmB2t, a.d.EH / UK + 1, a.d.Dt / UN, a.d.Dt, num_sms,
                        st);
}

}  // namespace mot
