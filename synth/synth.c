/*
 * Seeded synthetic inputs for the MoT KV-cache translation pass.
 *
 * This module holds NO arithmetic of the translation method. It only draws
 * random numbers and rounds them to the storage type. Both the fp64 oracle
 * and the CUDA path consume what it writes, which is why it lives in a module
 * of its own.
 *
 * Generator (published definitions, restated):
 *   - SplitMix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number
 *     generators", OOPSLA 2014): output n of a stream with state s0 is
 *     mix(s0 + (n+1)*GAMMA), GAMMA = 0x9E3779B97F4A7C15, where mix is the
 *     variant-13 finaliser (shifts 30/27/31, multipliers 0xBF58476D1CE4E5B9,
 *     0x94D049BB133111EB).
 *   - Stream key: s0 = mix(seed ^ mix(stream + GAMMA)).
 *   - Normal draws 2k and 2k+1 of a stream: Box-Muller (1958) on outputs 2k
 *     and 2k+1: u1 = ((o_{2k} >> 11) + 1) * 2^-53 in (0,1],
 *     u2 = (o_{2k+1} >> 11) * 2^-53, R = sqrt(-2 ln u1),
 *     n_{2k} = R cos(2 pi u2), n_{2k+1} = R sin(2 pi u2).
 *   - Storage rounding: fp64 -> fp32 (C cast, round-to-nearest-even), then for
 *     bf16 the fp32 bit pattern is rounded to its top 16 bits with
 *     round-to-nearest-even.
 *
 * Every element depends only on (seed, stream, index), so generation is
 * parallel (OpenMP) and reproducible.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define SYNTH_GAMMA 0x9E3779B97F4A7C15ULL

static inline uint64_t synth_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

uint64_t synth_stream_key(uint64_t seed, uint64_t stream) {
  return synth_mix(seed ^ synth_mix(stream + SYNTH_GAMMA));
}

uint64_t synth_splitmix64(uint64_t key, uint64_t n) {
  return synth_mix(key + (n + 1) * SYNTH_GAMMA);
}

static inline void normal_pair(uint64_t key, uint64_t k, double* n0, double* n1) {
  const double two_m53 = 1.0 / 9007199254740992.0;
  uint64_t o1 = synth_splitmix64(key, 2 * k);
  uint64_t o2 = synth_splitmix64(key, 2 * k + 1);
  double u1 = (double)((o1 >> 11) + 1) * two_m53;
  double u2 = (double)(o2 >> 11) * two_m53;
  double r = sqrt(-2.0 * log(u1));
  double th = 6.283185307179586476925 * u2;
  *n0 = r * cos(th);
  *n1 = r * sin(th);
}

double synth_normal_at(uint64_t key, uint64_t i) {
  double a, b;
  normal_pair(key, i >> 1, &a, &b);
  return (i & 1) ? b : a;
}

static inline uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  uint32_t lsb = (u >> 16) & 1u;
  u += 0x7FFFu + lsb;
  return (uint16_t)(u >> 16);
}

static inline void store_val(void* out, int64_t idx, double v, int dtype) {
  float f = (float)v;
  if (dtype == 0)
    ((uint16_t*)out)[idx] = f32_to_bf16_rne(f);
  else
    ((float*)out)[idx] = f;
}

/* out[i] = stddev * N_i for i in [0, n); dtype 0 = bf16 bits, 1 = fp32, 2 = fp64. */
void synth_fill_normal(uint64_t seed, uint64_t stream, int64_t n, double stddev,
                       int dtype, void* out) {
  uint64_t key = synth_stream_key(seed, stream);
  const int64_t np = (n + 1) / 2;
#pragma omp parallel for schedule(static)
  for (int64_t k = 0; k < np; ++k) {
    double v[2];
    normal_pair(key, (uint64_t)k, &v[0], &v[1]);
    for (int j = 0; j < 2; ++j) {
      const int64_t i = 2 * k + j;
      if (i >= n) break;
      if (dtype == 2)
        ((double*)out)[i] = stddev * v[j];
      else
        store_val(out, i, stddev * v[j], dtype);
    }
  }
}

/* out[i] = mean + stddev * N_i (as synth_fill_normal, shifted by `mean`). */
void synth_fill_normal_shifted(uint64_t seed, uint64_t stream, int64_t n, double mean,
                               double stddev, int dtype, void* out) {
  uint64_t key = synth_stream_key(seed, stream);
  const int64_t np = (n + 1) / 2;
#pragma omp parallel for schedule(static)
  for (int64_t k = 0; k < np; ++k) {
    double v[2];
    normal_pair(key, (uint64_t)k, &v[0], &v[1]);
    for (int j = 0; j < 2; ++j) {
      const int64_t i = 2 * k + j;
      if (i >= n) break;
      if (dtype == 2)
        ((double*)out)[i] = mean + stddev * v[j];
      else
        store_val(out, i, mean + stddev * v[j], dtype);
    }
  }
}

/*
 * One layer of a KV cache laid out [B][H][S][d]: value = s_c * N, where the
 * per-channel scale s_c = exp(0.5 * n_c) ~ LogNormal(0, 0.5) is drawn once per
 * (layer, K/V, channel c = h*d + i) from `scale_stream` (draw c) and the values
 * from `value_stream` (draw = flat index of the element).
 */
void synth_fill_cache_layer(uint64_t seed, uint64_t scale_stream, uint64_t value_stream,
                            int B, int H, int S, int d, int dtype, void* out) {
  uint64_t kscale = synth_stream_key(seed, scale_stream);
  uint64_t kval = synth_stream_key(seed, value_stream);
  const int64_t per_b = (int64_t)H * S * d;
  const int64_t n = (int64_t)B * per_b;
  double* sc = (double*)malloc(sizeof(double) * (size_t)H * d);
  if (!sc) return;
  for (int64_t c = 0; c < (int64_t)H * d; ++c) sc[c] = exp(0.5 * synth_normal_at(kscale, (uint64_t)c));
  const int64_t np = (n + 1) / 2;
#pragma omp parallel for schedule(static)
  for (int64_t k = 0; k < np; ++k) {
    double v[2];
    normal_pair(kval, (uint64_t)k, &v[0], &v[1]);
    for (int j = 0; j < 2; ++j) {
      const int64_t idx = 2 * k + j;
      if (idx >= n) break;
      const int64_t r = idx % per_b;
      const int64_t h = r / ((int64_t)S * d);
      const int64_t i = r % d;
      store_val(out, idx, sc[h * d + i] * v[j], dtype);
    }
  }
  free(sc);
}

/*
 * Source guidance maps for the replay (App. C.4 reads the source attention
 * averaged over heads): rows u of a [B][N][N] map, positive scores at j <= u
 * and zeros above the diagonal. Each score is a LogNormal(0, 0.5) draw times a
 * structure weight with the shapes attention maps show: a sink at position 0
 * (x5), recency 1 + 3 exp(-(u - j) / 32), and a fixed set of "heavy" columns
 * (about 1 in 64, x3), drawn from `stream`. Only the order within a row
 * matters to the selection; the rows are not normalised.
 */
void synth_fill_guide(uint64_t seed, uint64_t stream, int B, int N, int dtype, void* out) {
  uint64_t kval = synth_stream_key(seed, stream);
  uint64_t kcol = synth_stream_key(seed, stream ^ 0x5A5A5A5AULL);
  const int64_t rows = (int64_t)B * N;
#pragma omp parallel for schedule(dynamic, 16)
  for (int64_t r = 0; r < rows; ++r) {
    const int64_t u = r % N;
    for (int64_t j = 0; j < N; ++j) {
      const int64_t idx = r * N + j;
      if (j > u) {
        store_val(out, idx, 0.0, dtype);
        continue;
      }
      double w = 1.0 + 3.0 * exp(-(double)(u - j) / 32.0);
      if (j == 0) w *= 5.0;
      if ((synth_splitmix64(kcol, (uint64_t)j) & 63u) == 0) w *= 3.0;
      const double v = w * exp(0.5 * synth_normal_at(kval, (uint64_t)idx));
      store_val(out, idx, v, dtype);
    }
  }
}
