// Top-S source-guided attention of the replay phase (App. C.4) on the tensor cores
// (sm_103a), for the layers at and above L_Full (the selection is in replay.cu):
//
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
//                         Every wait is bounded; on a timeout the roles unwind,
//                         copies and MMAs in flight are drained and TMEM is freed.
#include "replay_common.cuh"

namespace mot {
namespace {

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
}  // namespace mot
