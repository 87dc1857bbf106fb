// Full causal attention of the replay phase (App. C.4) on sm_103a, for the layers
// below L_Full:
//
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
#include "replay_common.cuh"

namespace mot {
namespace {

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
}  // namespace

bool replay_fmha_supported(const ReplayDims& d) {
  return (d.d == 64 || d.d == 128) && d.N % 8 == 0;
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
}  // namespace mot
