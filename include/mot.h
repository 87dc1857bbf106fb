/*
 * mot.h -- C ABI of the GB300 (sm_103a) Mixture-of-Translators KV-cache
 * translation library (libmot.so).
 *
 * The library maps a source LLM's per-layer context KV cache into a target
 * LLM's cache space (Sec. 2.1, "Translation": KV^{Src,Ctx} -> KV^{Tgt,Ctx}).
 * For every translated target layer l it reads source layer pi(l) (a channel
 * (pi(l), l), Sec. 2.1 "Communication"; depth-ratio default, App. C.3), and
 * for every token u and X in {K, V} (translated independently, App. C.2):
 *
 *   g(z_u)         = softmax(Wg z_u + bg)                          (Def. 3.1)
 *   gtilde         = g renormalised over its Top-K entries         (Def. 3.1)
 *   Tr_m(z_u)      = W2_m GELU(W1_m z_u + b1_m) + b2_m
 *   Tr_MoT(z_u)    = sum_{m in Top-K} gtilde_m Tr_m(z_u)            (Eq. mot_definition)
 *
 * and writes the result into the target cache in the target's head layout,
 * with no positional re-encoding (the paper prescribes none).
 *
 * Layouts (all row-major, contiguous, caller-owned device memory):
 *   source cache  src_X[L_s][max_batch][H_s][max_seq][d_s]
 *   target cache  dst_X[L_t][max_batch][H_t][max_seq][d_t]
 *   A token vector is its heads concatenated: channel c = h*d + i.
 *   Element type: bf16 (MOT_BF16) or fp32 (MOT_FP32), the same for caches
 *   and weights.
 *
 * Every call returns a mot_status. Nothing in this library traps, asserts on
 * the device or spins without a bound: device-side anomalies (a sequence
 * length outside [0, max_seq], a pipeline wait that exceeded its limit) set a
 * sticky status word that mot_get_device_status reports.
 */
#ifndef MOT_H_
#define MOT_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t; NULL is the legacy default stream. */
struct CUstream_st;
typedef struct CUstream_st* mot_stream_t;

typedef enum {
  MOT_OK = 0,
  MOT_ERR_INVALID_ARG = 1,   /* NULL / misaligned pointer, bad size or config value */
  MOT_ERR_UNSUPPORTED = 2,   /* valid but outside what this build implements */
  MOT_ERR_NO_WEIGHTS = 3,    /* mot_translate before mot_load_weights */
  MOT_ERR_WEIGHTS_SIZE = 4,  /* blob byte count differs from the config's */
  MOT_ERR_OOM = 5,           /* device allocation failed */
  MOT_ERR_CUDA = 6,          /* a CUDA runtime/driver call failed (incl. no GPU) */
  MOT_ERR_SEQ_LEN = 7,       /* a sequence length was outside [0, max_seq] */
  MOT_ERR_TIMEOUT = 8        /* a bounded device-side pipeline wait gave up */
} mot_status;

typedef enum { MOT_BF16 = 0, MOT_FP32 = 1 } mot_dtype;

/*
 * Shapes of one translation (source model -> target model).
 * D_s = src_kv_heads * src_head_dim, D_t = tgt_kv_heads * tgt_head_dim.
 */
typedef struct {
  int32_t n_layers_src, src_kv_heads, src_head_dim;
  int32_t n_layers_tgt, tgt_kv_heads, tgt_head_dim;
  int32_t n_translators;     /* E = N_Tr, 1..16 (Def. 3.1) */
  int32_t top_k;             /* 0 or E: dense softmax gate; 1..E-1: Top-K (Def. 3.1) */
  int32_t hidden;            /* H, translator MLP width */
  int32_t max_batch;         /* B: batch capacity of the caches, 1..4096 */
  int32_t max_seq;           /* S_max: sequence capacity of the caches */
  mot_dtype dtype;           /* caches and weights */
  const int32_t* layer_map;  /* host [n_layers_tgt]: source layer of each target layer,
                                -1 = not translated; NULL = depth-ratio map (App. C.3)
                                pi(l) = round(l*(L_s-1)/(L_t-1)), halves up. Copied. */
} mot_config;

typedef struct mot_ctx* mot_handle;

/*
 * Validate `cfg` and create a handle on the CURRENT CUDA device. Allocates the
 * device weight storage and the translation workspace (the translate calls
 * allocate nothing). Config errors are reported before any CUDA call.
 * Errors: MOT_ERR_INVALID_ARG (cfg/out NULL, non-positive sizes, top_k outside
 * [0, E], a layer_map entry outside [-1, L_s)), MOT_ERR_UNSUPPORTED (E > 16,
 * max_batch > 4096), MOT_ERR_CUDA (no usable device), MOT_ERR_OOM.
 * On error *out is set to NULL.
 */
mot_status mot_create(const mot_config* cfg, mot_handle* out);

/*
 * Upload the translator weights from a host blob (synchronous; the blob may
 * be freed on return). Blob layout, all elements in cfg.dtype, for every
 * translated target layer l in ascending order, then X = K, V:
 *   Wg[E][D_s], bg[E],
 *   then for m = 0..E-1:  W1[H][D_s], b1[H], W2[D_t][H], b2[D_t]
 * (nn.Linear (out, in) convention). `bytes` must equal that size exactly.
 * The library repacks the weights into its own device layout.
 * Errors: MOT_ERR_INVALID_ARG, MOT_ERR_WEIGHTS_SIZE, MOT_ERR_CUDA.
 */
mot_status mot_load_weights(mot_handle h, const void* host_blob, size_t bytes);

/*
 * Translate (Eq. mot_definition) the source caches into the target caches.
 * src_k, src_v, dst_k, dst_v: device pointers, 16-byte aligned, in the layouts
 * above. seq_lens: DEVICE int32[batch], batch <= max_batch; token (b, s) is
 * translated for s < seq_lens[b]. Only those positions of translated layers
 * are written; padding positions, batch entries >= batch and untranslated
 * layers keep their contents. A length outside [0, max_seq] is clamped into
 * that range and reported later by mot_get_device_status (MOT_ERR_SEQ_LEN).
 * Asynchronous on `stream`: no host synchronisation, no allocation. One
 * handle must not run two translations concurrently (shared workspace).
 * Errors: MOT_ERR_INVALID_ARG (NULL/misaligned pointers, batch outside
 * [0, max_batch], dst aliasing src), MOT_ERR_NO_WEIGHTS, MOT_ERR_CUDA.
 */
mot_status mot_translate(mot_handle h, const void* src_k, const void* src_v,
                         const int32_t* seq_lens, int32_t batch, void* dst_k, void* dst_v,
                         mot_stream_t stream);

/*
 * The same translation with HOST buffers (pinned memory recommended): copies
 * the real tokens of src_k/src_v and seq_lens (host int32[batch]) to
 * library-owned device staging, translates, and copies the translated
 * positions back into dst_k/dst_v. The work is pipelined over chunks of target
 * layers on `stream` and two library-owned copy streams, so the copies of one
 * chunk overlap the translation of its neighbours; `stream` is made to wait
 * for the last copy back. The call returns once the work is enqueued;
 * synchronise `stream` before reading dst. The staging buffers, copy streams
 * and events are created on the first call and freed by mot_destroy.
 * Errors: as mot_translate, plus MOT_ERR_SEQ_LEN for a host length outside
 * [0, max_seq] (nothing is enqueued then) and MOT_ERR_OOM.
 */
mot_status mot_translate_host(mot_handle h, const void* src_k, const void* src_v,
                              const int32_t* seq_lens, int32_t batch, void* dst_k, void* dst_v,
                              mot_stream_t stream);

/*
 * Synchronise `stream`, then report and clear the sticky device status word:
 * MOT_ERR_SEQ_LEN, MOT_ERR_TIMEOUT, or MOT_OK. MOT_ERR_CUDA if the stream
 * reports an error.
 */
mot_status mot_get_device_status(mot_handle h, mot_stream_t stream);

/* Free every device resource of the handle (synchronises the device first). */
mot_status mot_destroy(mot_handle h);

/* Static, human-readable name of a status code. */
const char* mot_status_string(mot_status s);

/*
 * Allocation-free translation (the paper has no counterpart: this is a service
 * for callers that cannot call cudaMalloc, such as a process whose device
 * memory is divided up front by its own pool allocator and forbids further
 * allocations, or a host that must not grow its device footprint per call).
 * No handle: `cfg` is as for mot_create (layer_map NULL = depth-ratio map),
 * `weights` is the packed blob of mot_load_weights already in the caller's
 * DEVICE memory (16-byte aligned, cfg.dtype), and the caches and device
 * seq_lens are as for mot_translate. Nothing is allocated: the per-call
 * intermediates live in one 64 MiB __device__ scratch array
 * (MOT_STATIC_SCRATCH_BYTES) that every GPU which loads this library holds
 * until the process exits. A call needs
 *   256-rounded(batch * S_pad * E * 4) + batch * S_pad * E * H * 4 bytes,
 *   S_pad = max_seq rounded up to 64,
 * and returns MOT_ERR_UNSUPPORTED, before any CUDA call, when that exceeds the
 * array (or when max_seq > INT32_MAX - 63). dst_k and dst_v may overlap
 * neither each other, nor src_k / src_v, nor the weight blob
 * (MOT_ERR_INVALID_ARG, before any CUDA call). The first call on a device
 * looks up the array's device address (cudaGetSymbolAddress, with that device
 * current) and keeps it for the life of the process; make that first call
 * before any stream capture. The kept address belongs to the device's primary
 * context (the one the CUDA runtime uses): calls from another context on the
 * device, or after cudaDeviceReset, are not supported. All calls share the array and it keeps the last
 * call's contents (nothing in it needs to start at zero): calls that overlap
 * on the GPU, on any streams, race with each other. Lengths outside
 * [0, max_seq] are clamped; there is no status word to report them. The
 * arithmetic is fp32 FFMA throughout (exact-erf GELU), so bf16 results match
 * mot_translate's within the bf16 tolerance and fp32 results to ~1e-6.
 * Asynchronous on `stream`. Errors: MOT_ERR_INVALID_ARG, MOT_ERR_UNSUPPORTED,
 * MOT_ERR_CUDA.
 */
#define MOT_STATIC_SCRATCH_BYTES ((size_t)64 << 20)
mot_status mot_translate_static(const mot_config* cfg, const void* weights, const void* src_k,
                                const void* src_v, const int32_t* seq_lens, int32_t batch,
                                void* dst_k, void* dst_v, mot_stream_t stream);

/* ---- introspection (no method counterpart; for tests and benchmarks) ------ */

/* The channel map in use: out[n_layers_tgt] (n must equal n_layers_tgt). */
mot_status mot_get_layer_map(mot_handle h, int32_t* out, int32_t n);

/* Which kernel path translate uses: 1 = tcgen05/TMA bf16 GEMMs, 0 = SIMT. */
mot_status mot_get_path(mot_handle h, int32_t* path);

/*
 * Launch schedule of the tcgen05 path (schedules 0-2 have no effect on the
 * SIMT path); all give the same results.
 *   3 (default where supported): one persistent launch on pairs of CTAs that
 *      keeps each token tile's hidden activations GELU(W1 z + b1) * gtilde in
 *      shared memory and TMEM between the two GEMMs, so they never reach HBM.
 *      Supported when D_s <= 128, D_t = 256 and H % 256 == 0 (bf16);
 *      otherwise setting it returns MOT_ERR_UNSUPPORTED.
 *   2 (default otherwise): per pass of groups, GEMM1 then GEMM2 on pairs of
 *      CTAs (two SMs per 256 x 256 tile, tcgen05.mma.cta_group::2), with the
 *      hidden activations in an HBM workspace;
 *   1: one fused persistent launch per pass running both GEMMs as
 *      dependency-ordered work items on single SMs;
 *   0: GEMM1 then GEMM2 on single SMs (128 x 256 tiles).
 */
mot_status mot_set_schedule(mot_handle h, int32_t schedule);
mot_status mot_get_schedule(mot_handle h, int32_t* schedule);

/*
 * Per-kernel timing. While enabled, every kernel that translate launches is
 * bracketed by CUDA events on the launching stream. mot_profile_read
 * synchronises those events, writes up to `cap` records (one per kernel
 * name, in first-launch order) and clears the collected events.
 */
typedef struct {
  char name[32];
  int64_t launches;
  double total_ms;
} mot_kernel_stat;

mot_status mot_profile_enable(mot_handle h, int32_t enable);
mot_status mot_profile_read(mot_handle h, mot_kernel_stat* out, int32_t cap, int32_t* n);

/*
 * Failure-detection test hook. Every device pipeline wait of this handle's
 * kernels gives up after `wait_limit_cycles` SM cycles (0 = the default, about
 * two seconds), sets MOT_ERR_TIMEOUT in the status word and unwinds (copies
 * and MMAs in flight are drained, TMEM is freed). With stall_test = 1, the
 * first CTA of the single-SM GEMM1 kernel (schedule 0) never fills its first
 * pipeline stage, so a wait on it runs out: translations then report
 * MOT_ERR_TIMEOUT through mot_get_device_status and the context stays usable.
 * On a replay handle, stall_test = 1 makes the tensor-core guided attention's
 * first CTA withhold the completion signal of its first MMA, with the same
 * outcome for mot_replay_attention on a guided layer.
 */
mot_status mot_debug_set(mot_handle h, int32_t stall_test, int64_t wait_limit_cycles);

/*
 * Fixed-gate test hook (Def. 3.1 / Eq. mot_definition: the combine is linear
 * in the gate weights). While set, mot_translate uses the caller's gate rows
 * instead of evaluating the gate: gate is device float
 * [G][max_batch][max_seq][E], G = 2 x translated target layers, group 2 r + x
 * for the r-th translated target layer (x = 0 for K, 1 for V); row (g, b, s)
 * is the gtilde of token (b, s) in group g (not renormalised or checked). The
 * buffer must stay valid while set; NULL clears the hook. Dense translation
 * only: a routed translation (mot_set_routing 1) returns MOT_ERR_UNSUPPORTED
 * while the hook is set. MOT_ERR_INVALID_ARG for a MoT-h, backbone or replay
 * handle or a misaligned pointer.
 */
mot_status mot_debug_fixed_gate(mot_handle h, const float* gate);

/*
 * GELU probe (App. C.2: phi = GELU). Evaluates, on the device, the GELU form a
 * kernel family uses, out[i] = GELU(u[i]) * gate[i], so that a test can
 * measure it against the exact erf form:
 *   form 0: the tensor-core MLP epilogue (every schedule): u rounded to fp16,
 *           the tanh form in packed fp16x2 on the hardware tanh unit, times
 *           gate (fp16 of gate / 2, doubled in the form), fp16 result;
 *   form 1: the backbone-translator epilogues: the tanh form in fp32;
 *   form 2: the SIMT path: the exact erf form with erff, fp32.
 * u, gate, out: device float[n]. Asynchronous on `stream`. Errors:
 * MOT_ERR_INVALID_ARG (form outside 0..2, n < 0, NULL buffers with n > 0),
 * MOT_ERR_CUDA.
 */
mot_status mot_debug_gelu(int32_t form, const float* u, const float* gate, int64_t n, float* out,
                           mot_stream_t stream);

/* Number of kernels this handle has launched since it was created. */
mot_status mot_get_launch_count(mot_handle h, int64_t* count);

/*
 * MoT-h (App. C.5): translate the source model's intermediate activation (the
 * input of its attention) instead of K and V, and restore the target cache
 * with the target layer's own projections: for each translated target layer
 * l, with a = src_act[pi(l)][b][s][:],
 *   a_hat = sum_m gtilde_m Tr_m(a)        (the gated mixture above, width d_at),
 *   K = W^K_l a_hat, V = W^V_l a_hat      (no bias, no positional re-encoding),
 * stored head-major into dst_k / dst_v [L_t][B][H_t][S][d_t] like
 * mot_translate. One mixture per layer (not per K/V): about half the
 * translated state of the KV translation.
 *
 * src_act: [L_s][max_batch][max_seq][src_act_dim] bf16, device, 16-byte
 * aligned. The weight blob for mot_load_weights holds, per translated target
 * layer ascending: Wg[E][d_as], bg[E], then for m = 0..E-1 W1[H][d_as], b1[H],
 * W2[d_at][H], b2[d_at]; then W^K[D_t][d_at] and W^V[D_t][d_at] (bf16).
 * Requires bf16, src_act_dim % 64 == 0, tgt_act_dim and D_t = tgt_kv_heads *
 * tgt_head_dim multiples of 256, tgt_head_dim % 32 == 0, hidden % 256 == 0
 * (the tensor-core path); otherwise MOT_ERR_UNSUPPORTED. A MoT-h handle
 * accepts mot_translate_h only (mot_translate returns MOT_ERR_INVALID_ARG);
 * schedules, routing, profiling and status calls work as for KV handles.
 */
typedef struct {
  int32_t n_layers_src, src_act_dim;
  int32_t n_layers_tgt, tgt_act_dim, tgt_kv_heads, tgt_head_dim;
  int32_t n_translators, top_k, hidden;
  int32_t max_batch, max_seq;
  mot_dtype dtype;
  const int32_t* layer_map;   /* as in mot_config */
} mot_h_config;

mot_status mot_create_h(const mot_h_config* cfg, mot_handle* out);
mot_status mot_translate_h(mot_handle h, const void* src_act, const int32_t* seq_lens,
                           int32_t batch, void* dst_k, void* dst_v, mot_stream_t stream);

/*
 * Top-K routing (Def. 3.1 with 0 < top_k < E), tensor-core path.
 *   1 (default where supported): token buckets. The tokens that chose
 *      translator m are gathered per (layer, K/V) group and m's MLP runs on
 *      them only (top_k / E of the dense MLP FLOPs); the top_k contributions
 *      of a token are summed in a fixed order.
 *   0: dense compute; every translator runs on every token, with the
 *      unselected ones weighted by zero.
 * Both give the translation of Def. 3.1 within rounding. Setting 1 on a
 * handle without top_k < E, without the tensor-core path or with H not a
 * multiple of 256 returns MOT_ERR_UNSUPPORTED.
 * Backbone handles (mot_create_bt) with top_k = 1 route too, and do so by
 * default: each backbone runs on the tokens that chose it only (per window
 * slot their source rows are packed per backbone), with a result bit-identical
 * to the dense schedule; other top_k values take the dense schedule only.
 */
mot_status mot_set_routing(mot_handle h, int32_t routing);
mot_status mot_get_routing(mot_handle h, int32_t* routing);

/*
 * Translator usage of the last routed translation (the counts I_e behind
 * the usage metrics of Sec. 4.3): counts[g * E + m] = tokens of translated
 * group g (2 r + x for the r-th translated target layer, x = 0 for K, 1 for
 * V) that chose translator m. n must equal groups * E. Waits for `stream`.
 * For a backbone handle, counts[x * E + m] = tokens of block x (K, V) that
 * chose backbone m, and n must equal 2 * E. MOT_ERR_UNSUPPORTED unless the
 * last translate ran with routing 1.
 */
mot_status mot_get_expert_counts(mot_handle h, int32_t* counts, int32_t n, mot_stream_t stream);

/*
 * Translator usage statistics of Sec. 4.3 over selection counts I_e
 * (host-only; counts[0..n) as returned by mot_get_expert_counts, all groups
 * pooled): *cv2 = Var(I) / Mean(I)^2 (population variance) and *entropy =
 * -sum_e p_e ln p_e with p_e = I_e / sum I (terms with I_e = 0 contribute 0).
 * Both are 0 when every count is 0. MOT_ERR_INVALID_ARG for NULL pointers,
 * n <= 0 or a negative count.
 */
mot_status mot_expert_usage(const int32_t* counts, int32_t n, double* cv2, double* entropy);

/*
 * Backbone translators (App. C.2) as the experts of the mixture (Def. 3.1).
 * The translation covers one channel window: N consecutive target layers
 * t_r = win_start + r (r = 0..N-1), each paired with source layer pi(t_r)
 * (cfg.layer_map, or the depth-ratio map). For every token u and X in {K, V},
 * slot r's input is the source cache entry X_r = src_X[pi(t_r)][b][:, s, :],
 * a P x d_s matrix with one row per source KV head (P = src_kv_heads), and
 * each backbone m computes, with LN a layer norm (eps 1e-5) and GELU exact:
 *   z_r     = GELU(W_in LN_in(X_r) + b_in)                 row-wise, width d
 *   h_0     = z_1
 *   CAB_r:  a = MHA(LN_Q(h_{r-1}), LN_C(z_r), LN_C(z_r))    n_a heads over the
 *                                                           token's P rows
 *           ht = h_{r-1} + a;  h_r = ht + W_F2 GELU(W_F1 LN_F(ht) + b_F1) + b_F2
 *   Y_r     = GELU(W_out LN_out(flatten(h_r)) + b_out)      width D_t
 * (MHA: queries W_Q . + b_Q, keys W_K . + b_K, values W_V . + b_V, softmax of
 * the scaled dot products over the P rows, output W_O . + b_O). The gate reads
 * the whole window, logit = Wg concat_r(X_r flattened head-major) + bg; the
 * output y_r = sum over kept m of gtilde_m Y_{m,r} goes into target layer t_r
 * head-major, as in mot_translate. Layers outside the window are untouched.
 *
 * Weight blob (bf16), the block for X = K, then the block for X = V:
 *   Wg[E][N * D_s], bg[E], then for each backbone m:
 *     ln_in.gamma[d_s], ln_in.beta[d_s], W_in[d][d_s], b_in[d],
 *     for each slot r: ln_q.gamma[d], ln_q.beta[d], ln_c.gamma[d], ln_c.beta[d],
 *       W_Q[d][d], b_Q[d], W_K[d][d], b_K[d], W_V[d][d], b_V[d], W_O[d][d], b_O[d],
 *       ln_f.gamma[d], ln_f.beta[d], W_F1[d_f][d], b_F1[d_f], W_F2[d][d_f], b_F2[d],
 *     ln_out.gamma[P * d], ln_out.beta[P * d], W_out[D_t][P * d], b_out[D_t].
 * mot_load_weights folds LN_in's and LN_out's affines into W_in and W_out;
 * the other layer norms' affines are applied where their rows are written.
 *
 * cfg.hidden is unused (0). Requires bf16, P <= 16, d_s in {64, 128}, d in
 * {64, 128}, d / n_a in {16, 32, 64}, d_f a multiple of 64 (and of 256 above
 * 256), D_t and d_t multiples of 32, E <= 8, N <= 32, every window layer
 * mapped; otherwise MOT_ERR_UNSUPPORTED (MOT_ERR_INVALID_ARG for a window
 * outside [0, L_t) or non-positive sizes). A backbone handle accepts
 * mot_translate_bt only; routing (top_k = 1), expert counts, profiling, launch
 * counts and status calls work as for KV handles. mot_translate_bt has the arguments, layouts, alignment,
 * sequence-length and stream rules of mot_translate.
 */
typedef struct {
  int32_t win_start;   /* first target layer of the channel window */
  int32_t win_len;     /* N, slots of the window */
  int32_t width;       /* d, translator width of one source-head row */
  int32_t heads;       /* n_a, attention heads (width % heads == 0) */
  int32_t ffn;         /* d_f, FFN hidden width */
} mot_bt_config;

mot_status mot_create_bt(const mot_config* cfg, const mot_bt_config* bt, mot_handle* out);
mot_status mot_translate_bt(mot_handle h, const void* src_k, const void* src_v,
                            const int32_t* seq_lens, int32_t batch, void* dst_k, void* dst_v,
                            mot_stream_t stream);

/*
 * Replay attention (App. C.4): after translation the target model replays the
 * context over its cache, and each layer's attention runs here. For target
 * layer `layer`, batch entry b < batch, context position u < seq_lens[b] and
 * query head h (GQA: key/value head h / (q_heads / kv_heads)):
 *   layer <  n_full:  o = Attn(q_u, K[0..u], V[0..u])                 (full, causal)
 *   layer >= n_full:  N(u) = Top-S(A[b][u][0..u], top_s),  o = Attn(q_u, K[N(u)], V[N(u)])
 * where A is the guidance map of the source layer that guides this layer (the
 * source model's attention averaged over heads), Top-S keeps the top_s
 * positions j <= u with the largest A[b][u][j] (equal values: the lower
 * position first; every position when u + 1 <= top_s), and Attn is the
 * softmax of q . k / sqrt(head_dim) over the set applied to the value rows.
 * Layouts (bf16, device, 16-byte aligned, contiguous): q, out
 * [max_batch][q_heads][max_seq][head_dim]; k, v [max_batch][kv_heads][max_seq]
 * [head_dim] (one layer of the replay cache, e.g. a layer of mot_translate's
 * target cache); guide [max_batch][max_seq][max_seq] (row u, column j; only
 * j <= u is read; guide may be NULL for full layers). Rows u >= seq_lens[b] of
 * out are not written. seq_lens: device int32[batch], clamped to [0, max_seq].
 * Requires head_dim in {64, 128}, q_heads / kv_heads in 1..8, 12 or 16, top_s <= 4096,
 * max_seq <= 65536 (else MOT_ERR_UNSUPPORTED). Asynchronous on `stream`. Guided
 * layers with head_dim 128 and top_s <= 128 run on the tensor cores, full
 * layers with max_seq % 8 == 0 too; other shapes take the SIMT kernels.
 *
 * mot_replay_select writes the selection alone: sel [max_batch][max_seq][top_s]
 * int32, the row's positions ascending, then -1 (rows u >= seq_lens[b] are not
 * written). A replay handle accepts only these two calls and the profiling,
 * launch-count, device-status, test-hook (mot_debug_set) and destroy calls.
 */
typedef struct {
  int32_t q_heads, kv_heads, head_dim;
  int32_t max_batch, max_seq;
  int32_t top_s;    /* S_sparse */
  int32_t n_full;   /* L_Full: layers below it use full causal attention */
} mot_replay_config;

mot_status mot_create_replay(const mot_replay_config* cfg, mot_handle* out);
mot_status mot_replay_attention(mot_handle h, int32_t layer, const void* q, const void* k,
                                const void* v, const void* guide, const int32_t* seq_lens,
                                int32_t batch, void* out, mot_stream_t stream);
mot_status mot_replay_select(mot_handle h, const void* guide, const int32_t* seq_lens,
                             int32_t batch, int32_t* sel, mot_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* MOT_H_ */
