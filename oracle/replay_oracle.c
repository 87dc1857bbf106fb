/*
 * fp64 CPU oracle for the replay attention of the post-translation phase
 * (App. C.4: Top-S source-guided sparse attention, with L_Full bottom layers
 * on full causal attention).
 *
 * TEST INFRASTRUCTURE, like mot_oracle.c: only the tests, the smoke check and
 * the CPU legs of the benchmark may load or call it. It shares no code with
 * the CUDA path.
 *
 * One target layer l, batch entry b, context query position u (0-based), target
 * query head h (GQA: key/value head h / (Hq / Hkv)):
 *
 *   reference set  N_l(u) = {0, .., u}                                if l < L_Full
 *                  N_l(u) = Top-S(A[b][u][0..u], S)                    otherwise
 *     where A is the source guidance map of layer pi(l) (the source attention
 *     averaged over heads), Top-S keeps the S positions j <= u with the largest
 *     A[b][u][j], equal values ordered by the lower position first, and all of
 *     {0, .., u} when u + 1 <= S;
 *   attention      s_j = q . k_j / sqrt(d) for j in N_l(u),
 *                  o   = sum_j softmax(s)_j v_j   (max-subtracted, in double).
 *
 * Layouts (bf16 bit patterns, as the caches): q [B][Hq][N][d], k and v
 * [B][Hkv][N][d] (one layer of the replay cache), A [B][N][N] (row u, column j;
 * only j <= u is read).
 *
 * Pins (tests without a GPU): the selection against numpy's sort on (value
 * descending, position ascending); all positions when u + 1 <= S; ties to the
 * lower positions; never a position after u; full attention against torch's
 * causal scaled_dot_product_attention with the key/value heads repeated for
 * GQA; sparse attention against the same routine with a boolean mask of the
 * selected positions; layer L_Full as the first guided layer; S >= N equal to
 * full attention. No function here is unpinned.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
  int32_t B, N;            /* batch capacity, context capacity */
  int32_t Hq, Hkv, d;      /* target query heads, key/value heads, head dim */
  int32_t S;               /* S_sparse */
  int32_t n_full;          /* L_Full: layers below it use full attention */
} oracle_replay_dims;

double oracle_bf16_to_double(uint16_t bits);

static int check_rd(const oracle_replay_dims* d) {
  if (!d || d->B <= 0 || d->N <= 0 || d->Hq <= 0 || d->Hkv <= 0 || d->d <= 0 || d->S <= 0 ||
      d->n_full < 0 || d->Hq % d->Hkv)
    return -1;
  return 0;
}

/* Top-S positions of row u of batch entry b's guidance map, ascending.
 * Returns the count (min(S, u + 1)), or -1 on invalid arguments. */
int oracle_replay_select(const oracle_replay_dims* d, const uint16_t* guide, int b, int u,
                         int32_t* out) {
  if (check_rd(d) || !guide || !out || b < 0 || b >= d->B || u < 0 || u >= d->N) return -1;
  int n = u + 1;   /* candidates: positions 0..u (causal) */
  if (n <= d->S) {
    for (int j = 0; j < n; ++j) out[j] = j;
    return n;
  }
  const uint16_t* row = guide + ((int64_t)b * d->N + u) * d->N;
  /* S rounds of "take the largest remaining value, lowest position among equals" */
  char* taken = (char*)calloc((size_t)n, 1);
  if (!taken) return -1;
  for (int k = 0; k < d->S; ++k) {
    int best = -1;
    double bv = 0.0;
    for (int j = 0; j < n; ++j) {
      if (taken[j]) continue;
      const double v = oracle_bf16_to_double(row[j]);
      if (best < 0 || v > bv) { best = j; bv = v; }   /* strict: the lower position wins ties */
    }
    taken[best] = 1;
  }
  int c = 0;
  for (int j = 0; j < n; ++j)
    if (taken[j]) out[c++] = j;
  free(taken);
  return c;
}

/* Attention output (d values) of query (b, h, u) in target layer `layer`. */
int oracle_replay_query(const oracle_replay_dims* d, int layer, const uint16_t* q,
                        const uint16_t* k, const uint16_t* v, const uint16_t* guide, int b, int h,
                        int u, double* out) {
  if (check_rd(d) || !q || !k || !v || !out || layer < 0 || b < 0 || b >= d->B || h < 0 ||
      h >= d->Hq || u < 0 || u >= d->N)
    return -1;
  const int sparse = layer >= d->n_full;
  if (sparse && !guide) return -1;
  int32_t* set = (int32_t*)malloc(sizeof(int32_t) * (size_t)(u + 1));
  double* s = (double*)malloc(sizeof(double) * (size_t)(u + 1));
  double* qv = (double*)malloc(sizeof(double) * (size_t)d->d);
  if (!set || !s || !qv) { free(set); free(s); free(qv); return -1; }
  int n;
  if (sparse) {
    n = oracle_replay_select(d, guide, b, u, set);
  } else {
    n = u + 1;
    for (int j = 0; j < n; ++j) set[j] = j;
  }
  const int hk = h / (d->Hq / d->Hkv);
  const int64_t qi = (((int64_t)b * d->Hq + h) * d->N + u) * d->d;
  for (int i = 0; i < d->d; ++i) qv[i] = oracle_bf16_to_double(q[qi + i]);
  const double scale = 1.0 / sqrt((double)d->d);
  double mx = -INFINITY;
  for (int t = 0; t < n; ++t) {
    const int64_t ki = (((int64_t)b * d->Hkv + hk) * d->N + set[t]) * d->d;
    double acc = 0.0;
    for (int i = 0; i < d->d; ++i) acc += qv[i] * oracle_bf16_to_double(k[ki + i]);
    s[t] = acc * scale;
    if (s[t] > mx) mx = s[t];
  }
  double den = 0.0;
  for (int t = 0; t < n; ++t) { s[t] = exp(s[t] - mx); den += s[t]; }
  for (int i = 0; i < d->d; ++i) out[i] = 0.0;
  for (int t = 0; t < n; ++t) {
    const int64_t vi = (((int64_t)b * d->Hkv + hk) * d->N + set[t]) * d->d;
    const double w = s[t] / den;
    for (int i = 0; i < d->d; ++i) out[i] += w * oracle_bf16_to_double(v[vi + i]);
  }
  free(set); free(s); free(qv);
  return 0;
}

/* A list of queries (tb[t], th[t], tu[t]): out [n][d]. Returns 0, or -1. */
int oracle_replay_tokens(const oracle_replay_dims* d, int layer, const uint16_t* q,
                         const uint16_t* k, const uint16_t* v, const uint16_t* guide, int64_t n,
                         const int32_t* tb, const int32_t* th, const int32_t* tu, double* out) {
  if (check_rd(d) || n < 0 || (n > 0 && (!tb || !th || !tu || !out))) return -1;
  int err = 0;
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t t = 0; t < n; ++t) {
    if (oracle_replay_query(d, layer, q, k, v, guide, tb[t], th[t], tu[t], out + t * d->d)) {
#pragma omp atomic write
      err = 1;
    }
  }
  return err ? -1 : 0;
}
