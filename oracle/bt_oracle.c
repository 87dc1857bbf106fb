/*
 * fp64 CPU oracle for the backbone-translator variant of the MoT pass
 * (App. C.2 backbone inside Def. 3.1's gated mixture).
 *
 * TEST INFRASTRUCTURE, like mot_oracle.c: only the tests, the smoke check and
 * the CPU-baseline leg of the benchmark may load or call it. It shares no code
 * with the CUDA path.
 *
 * What it computes, per token u (Def. 3.1 writes the translators as functions
 * of the token's source input z_u), per X in {K, V} (translated independently):
 *
 *   Channel window (App. C.3): N consecutive target layers t_r = q + r,
 *   r = 0..N-1, each paired with its mapped source layer pi(t_r). Slot r of
 *   the window is the source cache entry X_r = src_X[pi(t_r)][b][:, s, :],
 *   a P x d_s matrix (P = H_s source KV heads, one row per head).
 *
 *   Gate (Def. 3.1; linear + softmax as in the MLP variant) on the whole
 *   window: logit = Wg concat_r(flatten_headmajor(X_r)) + bg, g = softmax,
 *   Top-K renormalised.
 *
 *   Backbone translator m (App. C.2), all rows of a slot treated alike:
 *     z_r[p]  = GELU(W_in LN_in(X_r[p]) + b_in)              (P x d)
 *     h_0     = z_1   (the first slot of the window)
 *     for r = 1..N (block CAB_r, its own weights):
 *       Q[p]  = W_Q LN_Q(h_{r-1}[p]) + b_Q
 *       K[p]  = W_K LN_C(z_r[p]) + b_K,  V[p] = W_V LN_C(z_r[p]) + b_V
 *       o     = multi-head attention of the P query rows over the P key/value
 *               rows (heads of width d / n_a, scores scaled by 1/sqrt(d/n_a),
 *               softmax over the P keys, no mask)
 *       a[p]  = W_O o[p] + b_O
 *       ht[p] = h_{r-1}[p] + a[p]
 *       h_r[p]= ht[p] + W_F2 GELU(W_F1 LN_F(ht[p]) + b_F1) + b_F2
 *     F_r     = flatten(h_r) (P*d values, row-major over p)
 *     Y_r     = GELU(W_out LN_out(F_r) + b_out)                (D_t)
 *   Concat(h_1..h_N) followed by the output projection is read as the
 *   projection applied slot by slot: slot r's output goes to target layer t_r.
 *
 *   Output: y_r = sum over kept m of gtilde_m * Y_{m,r}, stored head-major
 *   (c = h*d_t + i) into target layer t_r.
 *
 *   LN(x) = gamma * (x - mean) / sqrt(var + 1e-5) + beta over the vector's
 *   features (biased variance). GELU in its exact erf form.
 *
 * Weight blob (storage dtype), block for X = K, then the block for X = V:
 *   Wg[E][N*D_s], bg[E], then for each expert m:
 *     ln_in.g[d_s], ln_in.b[d_s], W_in[d][d_s], b_in[d],
 *     for each slot r: ln_q.g[d], ln_q.b[d], ln_c.g[d], ln_c.b[d],
 *       W_Q[d][d], b_Q[d], W_K[d][d], b_K[d], W_V[d][d], b_V[d], W_O[d][d], b_O[d],
 *       ln_f.g[d], ln_f.b[d], W_F1[d_f][d], b_F1[d_f], W_F2[d][d_f], b_F2[d],
 *     ln_out.g[P*d], ln_out.b[P*d], W_out[D_t][P*d], b_out[D_t].
 *
 * Pins (tests without a GPU): layer norm invariants (zero mean, unit variance,
 * shift/scale invariance, constant rows give beta); attention against
 * torch's multi-head attention routine, uniform weights when the key map is
 * zero, a single key giving the value row, row-permutation equivariance; the
 * backbone against a composition of torch library modules on tiny shapes;
 * source-head permutation with the matching output-weight permutation;
 * invariance to per-head shifts and scalings of the source rows (LN_in's
 * axis); a zero residual branch making every slot's output equal; the one-hot
 * gate selecting one backbone. No function here is unpinned.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
  int32_t L_s, H_s, d_s;
  int32_t L_t, H_t, d_t;
  int32_t E;
  int32_t top_k;
  int32_t H;
  int32_t B, S;
  int32_t dtype;
} oracle_dims;   /* identical to the struct in mot_oracle.c */

typedef struct {
  int32_t win_start;   /* first target layer of the channel window */
  int32_t win_len;     /* N: slots in the window */
  int32_t width;       /* d: translator width of one source-head row */
  int32_t heads;       /* n_a: attention heads (d % n_a == 0) */
  int32_t ffn;         /* d_f: FFN hidden width */
} oracle_bt_dims;

double oracle_bf16_to_double(uint16_t bits);
double oracle_gelu(double x);
void oracle_gate_from_logits(const double* logit, int E, int top_k, double* g);
int oracle_depth_ratio_map(int32_t L_s, int32_t L_t, int32_t* out);

static const double kLnEps = 1e-5;

static double bld(const void* p, int dtype, int64_t idx) {
  if (dtype == 0) return oracle_bf16_to_double(((const uint16_t*)p)[idx]);
  return (double)((const float*)p)[idx];
}

static void bld_row(const void* p, int dtype, int64_t idx, int64_t n, double* out) {
  for (int64_t k = 0; k < n; ++k) out[k] = bld(p, dtype, idx + k);
}

/* ---- building blocks ------------------------------------------------------ */

/* Layer normalisation over n features with affine (gamma, beta); either may be
 * NULL (then 1 and 0). */
void oracle_layernorm(const double* x, int64_t n, const double* gamma, const double* beta,
                      double* y) {
  double mean = 0.0;
  for (int64_t i = 0; i < n; ++i) mean += x[i];
  mean /= (double)n;
  double var = 0.0;
  for (int64_t i = 0; i < n; ++i) var += (x[i] - mean) * (x[i] - mean);
  var /= (double)n;
  const double inv = 1.0 / sqrt(var + kLnEps);
  for (int64_t i = 0; i < n; ++i)
    y[i] = (x[i] - mean) * inv * (gamma ? gamma[i] : 1.0) + (beta ? beta[i] : 0.0);
}

/* Multi-head scaled dot-product attention of P query rows over P key/value
 * rows, all of width d split into `heads` heads: for head a and query p,
 * o[p][a] = sum_j softmax_j(q[p][a] . k[j][a] / sqrt(d/heads)) v[j][a].
 * q, k, v, o: [P][d]. Returns 0, or -1 on invalid sizes. */
int oracle_bt_attention(int P, int d, int heads, const double* q, const double* k,
                        const double* v, double* o) {
  if (P <= 0 || d <= 0 || heads <= 0 || d % heads) return -1;
  const int dh = d / heads;
  const double scale = 1.0 / sqrt((double)dh);
  double* sc = (double*)malloc(sizeof(double) * (size_t)P);
  if (!sc) return -1;
  for (int a = 0; a < heads; ++a)
    for (int p = 0; p < P; ++p) {
      double mx = -INFINITY;
      for (int j = 0; j < P; ++j) {
        double s = 0.0;
        for (int i = 0; i < dh; ++i) s += q[p * d + a * dh + i] * k[j * d + a * dh + i];
        sc[j] = s * scale;
        if (sc[j] > mx) mx = sc[j];
      }
      double den = 0.0;
      for (int j = 0; j < P; ++j) { sc[j] = exp(sc[j] - mx); den += sc[j]; }
      for (int i = 0; i < dh; ++i) {
        double acc = 0.0;
        for (int j = 0; j < P; ++j) acc += sc[j] * v[j * d + a * dh + i];
        o[p * d + a * dh + i] = acc / den;
      }
    }
  free(sc);
  return 0;
}

/* ---- blob layout ---------------------------------------------------------- */

typedef struct {
  int64_t P, ds, Ds, Dt, d, df, N, E, na;
  int64_t slot;     /* elements of one CAB block */
  int64_t expert;   /* elements of one expert */
  int64_t group;    /* elements of one X block (gate + experts) */
} bt_layout;

static bt_layout layout_of(const oracle_dims* dd, const oracle_bt_dims* bt) {
  bt_layout L;
  L.P = dd->H_s;
  L.ds = dd->d_s;
  L.Ds = (int64_t)dd->H_s * dd->d_s;
  L.Dt = (int64_t)dd->H_t * dd->d_t;
  L.d = bt->width;
  L.df = bt->ffn;
  L.N = bt->win_len;
  L.E = dd->E;
  L.na = bt->heads;
  L.slot = 4 * L.d + 4 * (L.d * L.d + L.d) + 2 * L.d + (L.df * L.d + L.df) + (L.d * L.df + L.d);
  L.expert = 2 * L.ds + L.d * L.ds + L.d + L.N * L.slot + 2 * L.P * L.d + L.Dt * L.P * L.d + L.Dt;
  L.group = L.E * L.N * L.Ds + L.E + L.E * L.expert;
  return L;
}

int64_t oracle_bt_blob_elems(const oracle_dims* dd, const oracle_bt_dims* bt) {
  return 2 * layout_of(dd, bt).group;
}

static int check_bt(const oracle_dims* d, const oracle_bt_dims* bt) {
  if (!d || !bt) return -1;
  if (d->L_s <= 0 || d->H_s <= 0 || d->d_s <= 0 || d->L_t <= 0 || d->H_t <= 0 || d->d_t <= 0)
    return -1;
  if (d->E <= 0 || d->E > 64 || d->top_k < 0 || d->top_k > d->E) return -1;
  if (d->B <= 0 || d->S <= 0 || (d->dtype != 0 && d->dtype != 1)) return -1;
  if (bt->win_len <= 0 || bt->win_start < 0 || bt->win_start + bt->win_len > d->L_t) return -1;
  if (bt->width <= 0 || bt->heads <= 0 || bt->width % bt->heads || bt->ffn <= 0) return -1;
  return 0;
}

/* ---- one backbone translator on one token --------------------------------- */

typedef struct {
  double *z, *h, *ht, *nq, *nc, *q, *k, *v, *o, *a, *nf, *f, *row, *vec, *F, *nF, *g, *b;
} bt_scratch;

static int scratch_alloc(bt_scratch* s, const bt_layout* L) {
  const int64_t Pd = L->P * L->d;
  int64_t mx = L->ds;
  if (L->d > mx) mx = L->d;
  if (L->df > mx) mx = L->df;
  if (Pd > mx) mx = Pd;
  if (L->Dt > mx) mx = L->Dt;
  double** ptrs[] = {&s->z, &s->h, &s->ht, &s->nq, &s->nc, &s->q, &s->k, &s->v, &s->o, &s->a,
                     &s->nf, &s->F, &s->nF};
  const int64_t sizes[] = {L->N * Pd, Pd, Pd, Pd, Pd, Pd, Pd, Pd, Pd, Pd, Pd, Pd, Pd};
  int ok = 1;
  for (int i = 0; i < 13; ++i) {
    *ptrs[i] = (double*)malloc(sizeof(double) * (size_t)sizes[i]);
    ok &= *ptrs[i] != NULL;
  }
  s->f = (double*)malloc(sizeof(double) * (size_t)L->df);
  s->row = (double*)malloc(sizeof(double) * (size_t)mx);
  s->vec = (double*)malloc(sizeof(double) * (size_t)mx);
  s->g = (double*)malloc(sizeof(double) * (size_t)mx);
  s->b = (double*)malloc(sizeof(double) * (size_t)mx);
  ok &= s->f && s->row && s->vec && s->g && s->b;
  return ok ? 0 : -1;
}

static void scratch_free(bt_scratch* s) {
  free(s->z); free(s->h); free(s->ht); free(s->nq); free(s->nc); free(s->q); free(s->k);
  free(s->v); free(s->o); free(s->a); free(s->nf); free(s->F); free(s->nF); free(s->f);
  free(s->row); free(s->vec); free(s->g); free(s->b);
}

/* y[n_out] = W[n_out][n_in] x + b, W and b read from the blob at offsets ow, ob. */
static void linear(const void* w, int dt, int64_t ow, int64_t ob, int64_t n_out, int64_t n_in,
                   const double* x, double* y, double* row) {
  for (int64_t i = 0; i < n_out; ++i) {
    bld_row(w, dt, ow + i * n_in, n_in, row);
    double s = 0.0;
    for (int64_t k = 0; k < n_in; ++k) s += row[k] * x[k];
    y[i] = s + bld(w, dt, ob + i);
  }
}

/* Layer norm with (gamma, beta) read from the blob at og, og + n. */
static void ln_blob(const void* w, int dt, int64_t og, int64_t n, const double* x, double* y,
                    bt_scratch* s) {
  bld_row(w, dt, og, n, s->g);
  bld_row(w, dt, og + n, n, s->b);
  oracle_layernorm(x, n, s->g, s->b, y);
}

/* Backbone translator whose blob block starts at element `base` of `w`.
 * x: [N][P][d_s] source rows of the window; y: [N][D_t]; h_out (optional):
 * [N][P][d] running states h_1..h_N. */
static void backbone(const bt_layout* L, const void* w, int dt, int64_t base, const double* x,
                     double* y, double* h_out, bt_scratch* s) {
  const int64_t P = L->P, d = L->d, df = L->df, ds = L->ds, Pd = P * d;
  const int64_t o_lnin = base, o_win = o_lnin + 2 * ds, o_bin = o_win + d * ds;
  const int64_t o_slot0 = o_bin + d;
  const int64_t o_lnout = o_slot0 + L->N * L->slot, o_wout = o_lnout + 2 * Pd;
  const int64_t o_bout = o_wout + L->Dt * Pd;

  /* z_r[p] = GELU(W_in LN_in(X_r[p]) + b_in) */
  for (int64_t r = 0; r < L->N; ++r)
    for (int64_t p = 0; p < P; ++p) {
      ln_blob(w, dt, o_lnin, ds, x + (r * P + p) * ds, s->vec, s);
      double* zr = s->z + (r * P + p) * d;
      linear(w, dt, o_win, o_bin, d, ds, s->vec, zr, s->row);
      for (int64_t i = 0; i < d; ++i) zr[i] = oracle_gelu(zr[i]);
    }
  memcpy(s->h, s->z, sizeof(double) * (size_t)Pd);   /* h_0 = z_1 */

  for (int64_t r = 0; r < L->N; ++r) {
    const int64_t o = o_slot0 + r * L->slot;
    const int64_t o_lnq = o, o_lnc = o + 2 * d;
    const int64_t o_wq = o + 4 * d, o_bq = o_wq + d * d;
    const int64_t o_wk = o_bq + d, o_bk = o_wk + d * d;
    const int64_t o_wv = o_bk + d, o_bv = o_wv + d * d;
    const int64_t o_wo = o_bv + d, o_bo = o_wo + d * d;
    const int64_t o_lnf = o_bo + d;
    const int64_t o_wf1 = o_lnf + 2 * d, o_bf1 = o_wf1 + df * d;
    const int64_t o_wf2 = o_bf1 + df, o_bf2 = o_wf2 + d * df;
    const double* zr = s->z + r * Pd;
    for (int64_t p = 0; p < P; ++p) {
      ln_blob(w, dt, o_lnq, d, s->h + p * d, s->nq + p * d, s);
      ln_blob(w, dt, o_lnc, d, zr + p * d, s->nc + p * d, s);
      linear(w, dt, o_wq, o_bq, d, d, s->nq + p * d, s->q + p * d, s->row);
      linear(w, dt, o_wk, o_bk, d, d, s->nc + p * d, s->k + p * d, s->row);
      linear(w, dt, o_wv, o_bv, d, d, s->nc + p * d, s->v + p * d, s->row);
    }
    oracle_bt_attention((int)P, (int)d, (int)L->na, s->q, s->k, s->v, s->o);
    for (int64_t p = 0; p < P; ++p) {
      linear(w, dt, o_wo, o_bo, d, d, s->o + p * d, s->a + p * d, s->row);
      for (int64_t i = 0; i < d; ++i) s->ht[p * d + i] = s->h[p * d + i] + s->a[p * d + i];
      ln_blob(w, dt, o_lnf, d, s->ht + p * d, s->nf + p * d, s);
      linear(w, dt, o_wf1, o_bf1, df, d, s->nf + p * d, s->f, s->row);
      for (int64_t j = 0; j < df; ++j) s->f[j] = oracle_gelu(s->f[j]);
      linear(w, dt, o_wf2, o_bf2, d, df, s->f, s->vec, s->row);
      for (int64_t i = 0; i < d; ++i) s->h[p * d + i] = s->ht[p * d + i] + s->vec[i];
    }
    if (h_out) memcpy(h_out + r * Pd, s->h, sizeof(double) * (size_t)Pd);
    /* Y_r = GELU(W_out LN_out(flatten(h_r)) + b_out) */
    ln_blob(w, dt, o_lnout, Pd, s->h, s->nF, s);
    double* yr = y + r * L->Dt;
    linear(w, dt, o_wout, o_bout, L->Dt, Pd, s->nF, yr, s->row);
    for (int64_t i = 0; i < L->Dt; ++i) yr[i] = oracle_gelu(yr[i]);
  }
}

/* ---- entry points --------------------------------------------------------- */

static int32_t* bt_map(const oracle_dims* d, const int32_t* layer_map) {
  int32_t* map = (int32_t*)malloc(sizeof(int32_t) * d->L_t);
  if (!map) return NULL;
  if (layer_map) {
    for (int l = 0; l < d->L_t; ++l) {
      if (layer_map[l] < 0 || layer_map[l] >= d->L_s) { free(map); return NULL; }
      map[l] = layer_map[l];
    }
  } else {
    oracle_depth_ratio_map(d->L_s, d->L_t, map);
  }
  return map;
}

/* Gather the window's source rows for token (b, s): x[N][P][d_s]. */
static void gather_window(const oracle_dims* d, const oracle_bt_dims* bt, const int32_t* map,
                          const void* src, int b, int s, double* x) {
  for (int r = 0; r < bt->win_len; ++r) {
    const int64_t sl = map[bt->win_start + r];
    for (int p = 0; p < d->H_s; ++p) {
      const int64_t idx = (((sl * d->B + b) * d->H_s + p) * d->S + s) * d->d_s;
      bld_row(src, d->dtype, idx, d->d_s, x + ((int64_t)r * d->H_s + p) * d->d_s);
    }
  }
}

/*
 * One backbone translator (expert m of the X block) on one token's window.
 * x: [N][P][d_s]; y: [N][D_t]; h_out (optional): [N][P][d].
 */
int oracle_bt_backbone(const oracle_dims* d, const oracle_bt_dims* bt, const void* blob, int X,
                       int m, const double* x, double* y, double* h_out) {
  if (check_bt(d, bt) || !blob || !x || !y || X < 0 || X > 1 || m < 0 || m >= d->E) return -1;
  const bt_layout L = layout_of(d, bt);
  bt_scratch s;
  if (scratch_alloc(&s, &L)) { scratch_free(&s); return -1; }
  const int64_t base = X * L.group + L.E * L.N * L.Ds + L.E + m * L.expert;
  backbone(&L, blob, d->dtype, base, x, y, h_out, &s);
  scratch_free(&s);
  return 0;
}

/*
 * Translate a list of tokens (tok_b[t], tok_s[t]) through the window.
 * out: [N][2][n_tok][D_t] (slot r is target layer win_start + r; c = h*d_t + i).
 * gate_fixed (optional): [2][n_tok][E] used instead of the gate (all experts
 * with a nonzero weight contribute). gate_out (optional): [2][n_tok][E], the
 * kept renormalised gate. layer_map: [L_t] or NULL for the depth-ratio default;
 * every window layer must be mapped. Returns 0, or -1 on invalid arguments.
 */
int oracle_bt_tokens(const oracle_dims* d, const oracle_bt_dims* bt, const int32_t* layer_map,
                     const void* src_k, const void* src_v, const void* blob, int64_t n_tok,
                     const int32_t* tok_b, const int32_t* tok_s, const double* gate_fixed,
                     double* out, double* gate_out) {
  if (check_bt(d, bt) || !src_k || !src_v || !blob || !out || n_tok < 0) return -1;
  if (n_tok > 0 && (!tok_b || !tok_s)) return -1;
  for (int64_t t = 0; t < n_tok; ++t)
    if (tok_b[t] < 0 || tok_b[t] >= d->B || tok_s[t] < 0 || tok_s[t] >= d->S) return -1;
  int32_t* map = bt_map(d, layer_map);
  if (!map) return -1;
  const bt_layout L = layout_of(d, bt);
  const int64_t E = L.E, N = L.N, Dt = L.Dt, WD = N * L.Ds;
  int err = 0;
  for (int X = 0; X < 2; ++X) {
    const void* src = X == 0 ? src_k : src_v;
    const int64_t gbase = X * L.group;
#pragma omp parallel
    {
      bt_scratch s;
      double* x = (double*)malloc(sizeof(double) * (size_t)WD);
      double* yb = (double*)malloc(sizeof(double) * (size_t)(N * Dt));
      double* acc = (double*)malloc(sizeof(double) * (size_t)(N * Dt));
      double* wrow = (double*)malloc(sizeof(double) * (size_t)WD);
      int ok = scratch_alloc(&s, &L) == 0 && x && yb && acc && wrow;
      double g[64], logit[64];
#pragma omp for schedule(dynamic, 1)
      for (int64_t t = 0; t < n_tok; ++t) {
        if (!ok) continue;
        gather_window(d, bt, map, src, tok_b[t], tok_s[t], x);
        /* gate on the window, flattened slot-major then head-major (Def. 3.1) */
        if (gate_fixed) {
          for (int64_t m = 0; m < E; ++m) g[m] = gate_fixed[(X * n_tok + t) * E + m];
        } else {
          for (int64_t m = 0; m < E; ++m) {
            bld_row(blob, d->dtype, gbase + m * WD, WD, wrow);
            double sdot = 0.0;
            for (int64_t c = 0; c < WD; ++c) sdot += wrow[c] * x[c];
            logit[m] = sdot + bld(blob, d->dtype, gbase + E * WD + m);
          }
          oracle_gate_from_logits(logit, (int)E, d->top_k, g);
        }
        for (int64_t i = 0; i < N * Dt; ++i) acc[i] = 0.0;
        for (int64_t m = 0; m < E; ++m) {
          if (g[m] == 0.0) continue;   /* not kept (Top-K), or zero weight */
          backbone(&L, blob, d->dtype, gbase + E * WD + E + m * L.expert, x, yb, NULL, &s);
          for (int64_t i = 0; i < N * Dt; ++i) acc[i] += g[m] * yb[i];
        }
        for (int64_t r = 0; r < N; ++r) {
          double* o = out + ((r * 2 + X) * n_tok + t) * Dt;
          for (int64_t i = 0; i < Dt; ++i) o[i] = acc[r * Dt + i];
        }
        if (gate_out)
          for (int64_t m = 0; m < E; ++m) gate_out[(X * n_tok + t) * E + m] = g[m];
      }
      if (!ok) {
#pragma omp atomic write
        err = 1;
      }
      scratch_free(&s);
      free(x); free(yb); free(acc); free(wrow);
    }
  }
  free(map);
  return err ? -1 : 0;
}
