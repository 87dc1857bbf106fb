/*
 * fp64 CPU oracle for the Mixture-of-Translators KV-cache translation pass.
 *
 * TEST INFRASTRUCTURE. Only the tests, the smoke check and the CPU-baseline
 * leg of the benchmark may load or call this code. The product path never
 * does. It shares no code with the CUDA path: the only common inputs are the
 * seeded synthetic buffers.
 *
 * What it computes (plain, per token, in double precision, in the order the
 * method states it):
 *
 *   Channel map (App. C.3, depth-ratio mapping): target layer l reads source
 *   layer pi(l) = round(l * (L_s - 1) / (L_t - 1)), halves rounded up; pi(l) = l
 *   when L_s == L_t. A caller-supplied map may mark a layer untranslated (-1).
 *
 *   For each translated target layer l, each X in {K, V} (translated
 *   independently, App. C.2), each batch entry b and position s < seq_len[b]:
 *     z       = src_X[pi(l)][b][:, s, :] flattened head-major (c = h*d_s + i),
 *               every stored value converted exactly to double;
 *     gate    (Def. 3.1: nonnegative token-level scores; read here as a linear
 *               map followed by a softmax)
 *               logit_m = sum_c Wg[m][c] z[c] + bg[m],  g = softmax(logit);
 *     Top-K   (Def. 3.1) if 0 < top_k < E, keep the top_k largest g (equal
 *               scores: lower index first) and renormalise over the kept set,
 *               otherwise keep all E (the renormalisation is then the identity);
 *     Tr_m    (translator, Linear -> GELU -> Linear; GELU is the activation the
 *               paper names in App. C.2, taken in its exact erf form)
 *               h_j = GELU(sum_c W1_m[j][c] z[c] + b1_m[j]),
 *               y_m[i] = sum_j W2_m[i][j] h_j + b2_m[i];
 *     combine (Eq. mot_definition) y = sum over kept m of gtilde_m * y_m;
 *     store   y[c] goes to dst_X[l][b][c / d_t][s][c % d_t] (head-major,
 *               no positional re-encoding: the paper prescribes none).
 *
 * Weight blob (per translated target layer l ascending, then X = K, V):
 *   Wg[E][D_s], bg[E], then for m = 0..E-1: W1[H][D_s], b1[H], W2[D_t][H], b2[D_t],
 *   all in the storage dtype (bf16 bit patterns or fp32).
 *
 * Pins (tests run without a GPU): depth-ratio values against the printed map
 * for 24 -> 28 layers; GELU against normal-table values of Phi; identity and
 * permutation translators built from GELU(x) - GELU(-x) = x; one-hot gate
 * (proof of Prop. 3.1); gate and Top-K closed forms; E = 1 against a library
 * MLP; linearity in the gate; expert-permutation invariance; brute force on
 * tiny inputs. MoT-h (below): the identity mixture with permutation and scaled
 * projections in closed form, linearity in W^K / W^V, and the mixture part
 * against the KV entry point on the same weights. No function here is unpinned.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
  int32_t L_s, H_s, d_s;   /* source layers, KV heads, head dim */
  int32_t L_t, H_t, d_t;   /* target layers, KV heads, head dim */
  int32_t E;               /* number of translators */
  int32_t top_k;           /* 0 or E: dense; 1..E-1: Top-K */
  int32_t H;               /* translator hidden width */
  int32_t B, S;            /* cache batch capacity and max sequence length */
  int32_t dtype;           /* 0 = bf16 bit patterns, 1 = fp32 */
} oracle_dims;

/* ---- storage decoding (exact) ------------------------------------------ */

double oracle_bf16_to_double(uint16_t bits) {
  uint32_t u = (uint32_t)bits << 16;
  float f;
  memcpy(&f, &u, 4);
  return (double)f;
}

static double ld(const void* p, int dtype, int64_t idx) {
  if (dtype == 0) return oracle_bf16_to_double(((const uint16_t*)p)[idx]);
  return (double)((const float*)p)[idx];
}

static void ld_row(const void* p, int dtype, int64_t idx, int64_t n, double* out) {
  for (int64_t k = 0; k < n; ++k) out[k] = ld(p, dtype, idx + k);
}

static double dot(const double* a, const double* b, int64_t n) {
  double s = 0.0;
  for (int64_t k = 0; k < n; ++k) s += a[k] * b[k];
  return s;
}

/* ---- method pieces --------------------------------------------------------- */

/* Depth-ratio channel map (App. C.3). */
int oracle_depth_ratio_map(int32_t L_s, int32_t L_t, int32_t* out) {
  if (L_s <= 0 || L_t <= 0 || !out) return -1;
  for (int32_t l = 0; l < L_t; ++l) {
    if (L_t == 1) { out[l] = 0; continue; }
    /* round(l*(L_s-1)/(L_t-1)) with halves rounded up, in exact integers */
    int64_t num = (int64_t)l * (L_s - 1), den = (int64_t)(L_t - 1);
    out[l] = (int32_t)((2 * num + den) / (2 * den));
  }
  return 0;
}

/* GELU(x) = x * Phi(x), Phi the standard normal CDF (App. C.2 names GELU). */
double oracle_gelu(double x) { return 0.5 * x * (1.0 + erf(x / sqrt(2.0))); }

/* Softmax over E logits, max-subtracted; then Top-K selection and
 * renormalisation (Def. 3.1). g[m] = 0 for experts that are not kept. */
void oracle_gate_from_logits(const double* logit, int E, int top_k, double* g) {
  double mx = logit[0];
  for (int m = 1; m < E; ++m) if (logit[m] > mx) mx = logit[m];
  double s = 0.0;
  for (int m = 0; m < E; ++m) { g[m] = exp(logit[m] - mx); s += g[m]; }
  for (int m = 0; m < E; ++m) g[m] /= s;
  if (top_k > 0 && top_k < E) {
    int keep[64] = {0};
    for (int k = 0; k < top_k; ++k) {
      int best = -1;
      for (int m = 0; m < E; ++m)
        if (!keep[m] && (best < 0 || g[m] > g[best])) best = m;   /* strict: lower index wins ties */
      keep[best] = 1;
    }
    double ks = 0.0;
    for (int m = 0; m < E; ++m) if (keep[m]) ks += g[m];
    for (int m = 0; m < E; ++m) g[m] = keep[m] ? g[m] / ks : 0.0;
  }
}

static int64_t group_elems(const oracle_dims* d) {
  int64_t E = d->E, Ds = (int64_t)d->H_s * d->d_s, Dt = (int64_t)d->H_t * d->d_t, H = d->H;
  return E * Ds + E + E * (H * Ds + H + Dt * H + Dt);
}

static int check_dims(const oracle_dims* d) {
  if (!d) return -1;
  if (d->L_s <= 0 || d->H_s <= 0 || d->d_s <= 0 || d->L_t <= 0 || d->H_t <= 0 || d->d_t <= 0)
    return -1;
  if (d->E <= 0 || d->E > 64 || d->top_k < 0 || d->top_k > d->E || d->H <= 0) return -1;
  if (d->B <= 0 || d->S <= 0 || (d->dtype != 0 && d->dtype != 1)) return -1;
  return 0;
}

/*
 * One token of one (target layer, X) group. `z` holds the gathered source
 * vector; `w` points at the group's blob block. Writes y[D_t] and the kept,
 * renormalised gate g[E]. If `g_fixed` is non-NULL those gate weights are used
 * instead of the gate's own (all E experts then contribute).
 */
static void translate_one(const oracle_dims* d, const void* w, const double* z,
                          const double* g_fixed, double* y, double* g,
                          double* logit, double* row, double* h, double* ym) {
  const int dt = d->dtype;
  const int64_t E = d->E, Ds = (int64_t)d->H_s * d->d_s, Dt = (int64_t)d->H_t * d->d_t;
  const int64_t H = d->H;
  const int64_t off_wg = 0, off_bg = E * Ds, off_exp = E * Ds + E;
  const int64_t per_exp = H * Ds + H + Dt * H + Dt;

  /* gate */
  if (g_fixed) {
    for (int64_t m = 0; m < E; ++m) g[m] = g_fixed[m];
  } else {
    for (int64_t m = 0; m < E; ++m) {
      ld_row(w, dt, off_wg + m * Ds, Ds, row);
      logit[m] = dot(row, z, Ds) + ld(w, dt, off_bg + m);
    }
    oracle_gate_from_logits(logit, (int)E, d->top_k, g);
  }

  for (int64_t i = 0; i < Dt; ++i) y[i] = 0.0;
  for (int64_t m = 0; m < E; ++m) {
    if (!g_fixed && g[m] == 0.0 && d->top_k > 0 && d->top_k < E) continue;  /* not selected */
    const int64_t base = off_exp + m * per_exp;
    const int64_t o_w1 = base, o_b1 = base + H * Ds, o_w2 = o_b1 + H, o_b2 = o_w2 + Dt * H;
    for (int64_t j = 0; j < H; ++j) {
      ld_row(w, dt, o_w1 + j * Ds, Ds, row);
      h[j] = oracle_gelu(dot(row, z, Ds) + ld(w, dt, o_b1 + j));
    }
    for (int64_t i = 0; i < Dt; ++i) {
      ld_row(w, dt, o_w2 + i * H, H, row);
      ym[i] = dot(row, h, H) + ld(w, dt, o_b2 + i);
    }
    for (int64_t i = 0; i < Dt; ++i) y[i] += g[m] * ym[i];
  }
}

/* The channel map in use: the caller's, validated, or the depth-ratio default.
 * Returns a malloc'd [L_t] array, or NULL on an invalid map. */
static int32_t* resolve_map(const oracle_dims* d, const int32_t* layer_map) {
  int32_t* map = (int32_t*)malloc(sizeof(int32_t) * d->L_t);
  if (!map) return NULL;
  if (layer_map) {
    for (int l = 0; l < d->L_t; ++l) {
      if (layer_map[l] < -1 || layer_map[l] >= d->L_s) { free(map); return NULL; }
      map[l] = layer_map[l];
    }
  } else {
    oracle_depth_ratio_map(d->L_s, d->L_t, map);
  }
  return map;
}

/*
 * Translate a list of tokens (tok_b[t], tok_s[t]) for every translated target
 * layer and X. out: [L_t][2][n_tok][D_t] (channel c = h*d_t + i); rows of
 * untranslated layers are left untouched. gate_out (optional): [L_t][2][n_tok][E].
 * gate_fixed (optional): [L_t][2][n_tok][E] gate weights used instead of the gate.
 * layer_map: [L_t] or NULL for the depth-ratio default.
 * Returns 0, or -1 on invalid arguments.
 */
int oracle_translate_tokens(const oracle_dims* d, const int32_t* layer_map,
                            const void* src_k, const void* src_v, const void* blob,
                            int64_t n_tok, const int32_t* tok_b, const int32_t* tok_s,
                            const double* gate_fixed, double* out, double* gate_out) {
  if (check_dims(d) || !src_k || !src_v || !blob || !out || n_tok < 0) return -1;
  if (n_tok > 0 && (!tok_b || !tok_s)) return -1;
  for (int64_t t = 0; t < n_tok; ++t)
    if (tok_b[t] < 0 || tok_b[t] >= d->B || tok_s[t] < 0 || tok_s[t] >= d->S) return -1;
  int32_t* map = resolve_map(d, layer_map);
  if (!map) return -1;
  const int64_t E = d->E, Ds = (int64_t)d->H_s * d->d_s, Dt = (int64_t)d->H_t * d->d_t;
  const int64_t gsz = group_elems(d);
  const int64_t esz = d->dtype == 0 ? 2 : 4;
  int64_t r = 0;   /* index of the translated layer, in ascending order */
  for (int l = 0; l < d->L_t; ++l) {
    if (map[l] < 0) continue;
    const int sl = map[l];
    for (int X = 0; X < 2; ++X) {
      const void* src = X == 0 ? src_k : src_v;
      const char* w = (const char*)blob + (r * 2 + X) * gsz * esz;
#pragma omp parallel
      {
        int64_t mx = Ds > d->H ? Ds : d->H;
        double* z = (double*)malloc(sizeof(double) * Ds);
        double* row = (double*)malloc(sizeof(double) * mx);
        double* h = (double*)malloc(sizeof(double) * d->H);
        double* ym = (double*)malloc(sizeof(double) * Dt);
        double* y = (double*)malloc(sizeof(double) * Dt);
        double g[64], logit[64];
#pragma omp for schedule(dynamic, 1)
        for (int64_t t = 0; t < n_tok; ++t) {
          const int b = tok_b[t], s = tok_s[t];
          for (int64_t c = 0; c < Ds; ++c) {
            const int64_t hs = c / d->d_s, i = c % d->d_s;
            const int64_t idx = ((((int64_t)sl * d->B + b) * d->H_s + hs) * d->S + s) * d->d_s + i;
            z[c] = ld(src, d->dtype, idx);
          }
          const double* gf = gate_fixed ? gate_fixed + ((l * 2 + X) * n_tok + t) * E : NULL;
          translate_one(d, w, z, gf, y, g, logit, row, h, ym);
          double* o = out + ((l * 2 + X) * n_tok + t) * Dt;
          for (int64_t i = 0; i < Dt; ++i) o[i] = y[i];
          if (gate_out) {
            double* go = gate_out + ((l * 2 + X) * n_tok + t) * E;
            for (int64_t m = 0; m < E; ++m) go[m] = g[m];
          }
        }
        free(z); free(row); free(h); free(ym); free(y);
      }
    }
    ++r;
  }
  free(map);
  return 0;
}

/*
 * Full translation into double caches laid out like the target cache:
 * dst_X[L_t][B][H_t][S][d_t]. Only positions s < seq_lens[b] of translated
 * layers are written; everything else is left untouched.
 */
int oracle_translate_full(const oracle_dims* d, const int32_t* layer_map,
                          const void* src_k, const void* src_v, const void* blob,
                          int32_t batch, const int32_t* seq_lens,
                          double* dst_k, double* dst_v) {
  if (check_dims(d) || !seq_lens || !dst_k || !dst_v || batch < 0 || batch > d->B) return -1;
  int64_t n = 0;
  for (int b = 0; b < batch; ++b) {
    if (seq_lens[b] < 0 || seq_lens[b] > d->S) return -1;
    n += seq_lens[b];
  }
  const int64_t Dt = (int64_t)d->H_t * d->d_t;
  int32_t* tb = (int32_t*)malloc(sizeof(int32_t) * (n > 0 ? n : 1));
  int32_t* ts = (int32_t*)malloc(sizeof(int32_t) * (n > 0 ? n : 1));
  double* rows = (double*)malloc(sizeof(double) * (size_t)(d->L_t * 2 * (n > 0 ? n : 1) * Dt));
  if (!tb || !ts || !rows) { free(tb); free(ts); free(rows); return -1; }
  int64_t t = 0;
  for (int b = 0; b < batch; ++b)
    for (int s = 0; s < seq_lens[b]; ++s) { tb[t] = b; ts[t] = s; ++t; }
  int rc = oracle_translate_tokens(d, layer_map, src_k, src_v, blob, n, tb, ts, NULL, rows, NULL);
  int32_t* map = rc == 0 ? resolve_map(d, layer_map) : NULL;
  if (rc == 0 && map) {
    for (int l = 0; l < d->L_t; ++l) {
      if (map[l] < 0) continue;   /* untranslated layer: left untouched */
      for (int X = 0; X < 2; ++X) {
        double* dst = X == 0 ? dst_k : dst_v;
        for (int64_t k = 0; k < n; ++k) {
          const double* y = rows + ((l * 2 + X) * n + k) * Dt;
          for (int64_t c = 0; c < Dt; ++c) {
            const int64_t ht = c / d->d_t, i = c % d->d_t;
            const int64_t idx = ((((int64_t)l * d->B + tb[k]) * d->H_t + ht) * d->S + ts[k]) * d->d_t + i;
            dst[idx] = y[c];
          }
        }
      }
    }
  }
  free(map); free(tb); free(ts); free(rows);
  return rc;
}

/*
 * MoT-h (App. C.5): the translated representation is the intermediate
 * activation entering the target's attention, not K and V. For each
 * translated target layer l and token:
 *   a       = a_src[pi(l)][b][s][:] (width d_as; the source activation,
 *             passed like a one-head cache: d->H_s = 1, d->d_s = d_as);
 *   a_hat   = sum over kept m of gtilde_m Tr_m(a), the same gated mixture as
 *             above with output width d_at (Def. 3.1);
 *   K, V    = W^K a_hat, W^V a_hat, the target layer's own key and value
 *             projections [D_t][d_at] (App. C.5 writes the restoration as these
 *             plain products: no bias, no positional re-encoding).
 * Weight blob per translated target layer ascending: the mixture block (as a
 * KV group block with D_t replaced by d_at), then W^K, then W^V.
 * out_k, out_v: [L_t][n_tok][D_t] (c = h*d_t + i); act_out (optional):
 * [L_t][n_tok][d_at]. Rows of untranslated layers are left untouched.
 * Returns 0, or -1 on invalid arguments.
 */
int oracle_translate_h_tokens(const oracle_dims* d, int32_t act_tgt, const int32_t* layer_map,
                              const void* src_act, const void* blob, int64_t n_tok,
                              const int32_t* tok_b, const int32_t* tok_s, double* out_k,
                              double* out_v, double* act_out) {
  if (check_dims(d) || d->H_s != 1 || act_tgt <= 0 || !src_act || !blob || !out_k || !out_v ||
      n_tok < 0)
    return -1;
  if (n_tok > 0 && (!tok_b || !tok_s)) return -1;
  for (int64_t t = 0; t < n_tok; ++t)
    if (tok_b[t] < 0 || tok_b[t] >= d->B || tok_s[t] < 0 || tok_s[t] >= d->S) return -1;
  int32_t* map = resolve_map(d, layer_map);
  if (!map) return -1;
  oracle_dims md = *d;   /* the mixture: one head of width d_at out */
  md.H_t = 1;
  md.d_t = act_tgt;
  const int64_t Da = act_tgt, Ds = d->d_s, Dt = (int64_t)d->H_t * d->d_t, E = d->E;
  const int64_t mix = group_elems(&md), block = mix + 2 * Dt * Da;
  const int64_t esz = d->dtype == 0 ? 2 : 4;
  int64_t r = 0;
  for (int l = 0; l < d->L_t; ++l) {
    if (map[l] < 0) continue;
    const int sl = map[l];
    const char* w = (const char*)blob + r * block * esz;
#pragma omp parallel
    {
      int64_t mx = Ds > d->H ? Ds : d->H;
      if (Da > mx) mx = Da;
      double* z = (double*)malloc(sizeof(double) * Ds);
      double* row = (double*)malloc(sizeof(double) * mx);
      double* h = (double*)malloc(sizeof(double) * d->H);
      double* ym = (double*)malloc(sizeof(double) * Da);
      double* ah = (double*)malloc(sizeof(double) * Da);
      double g[64], logit[64];
#pragma omp for schedule(dynamic, 1)
      for (int64_t t = 0; t < n_tok; ++t) {
        const int b = tok_b[t], s = tok_s[t];
        const int64_t zi = (((int64_t)sl * d->B + b) * d->S + s) * Ds;
        ld_row(src_act, d->dtype, zi, Ds, z);
        translate_one(&md, w, z, NULL, ah, g, logit, row, h, ym);
        double* ok = out_k + ((int64_t)l * n_tok + t) * Dt;
        double* ov = out_v + ((int64_t)l * n_tok + t) * Dt;
        for (int64_t i = 0; i < Dt; ++i) {
          ld_row(w, d->dtype, mix + i * Da, Da, row);
          ok[i] = dot(row, ah, Da);
          ld_row(w, d->dtype, mix + Dt * Da + i * Da, Da, row);
          ov[i] = dot(row, ah, Da);
        }
        if (act_out) {
          double* oa = act_out + ((int64_t)l * n_tok + t) * Da;
          for (int64_t i = 0; i < Da; ++i) oa[i] = ah[i];
        }
      }
      free(z); free(row); free(h); free(ym); free(ah);
    }
    ++r;
  }
  free(map);
  (void)E;
  return 0;
}
