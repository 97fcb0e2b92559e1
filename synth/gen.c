/*
 * Seeded, counter-based generator for the synthetic workloads.
 *
 * This file holds no arithmetic of the visual-memory method. It only draws
 * numbers; the oracle and the CUDA path both receive what it draws as input.
 *
 * Definition (so that any other implementation can reproduce it bit for bit):
 *   mix64(z): the SplitMix64 finaliser (Steele, Lea and Flood, "Fast splittable
 *             pseudorandom number generators", OOPSLA 2014; constants as in
 *             Vigna's public-domain splitmix64.c):
 *               z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9
 *               z = (z ^ (z >> 27)) * 0x94D049BB133111EB
 *               z =  z ^ (z >> 31)
 *   key(seed, stream)  = mix64(mix64(seed) ^ (stream * 0xD1B54A32D192ED03))
 *   draw(key, j)       = mix64(key + (j + 1) * 0x9E3779B97F4A7C15)
 *   normal i (Box-Muller, cosine branch) uses draws a = draw(key, 2i) and
 *     b = draw(key, 2i + 1):
 *       u1 = ((a >> 11) + 0.5) / 2^53          in (0, 1)
 *       u2 =  (b >> 11)        / 2^53          in [0, 1)
 *       n  = sqrt(-2 ln u1) * cos(2 pi u2)      (double)
 *   value_i = mean + sigma * n
 *   bf16 output: value_i -> float (round to nearest even) -> bf16 (round to
 *   nearest even on the top 16 bits of the float).
 *
 * Compiled with -ffp-contract=off so that x86-64 and aarch64 hosts agree.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <string.h>

static inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

uint64_t dvgen_key(uint64_t seed, uint64_t stream) {
  return mix64(mix64(seed) ^ (stream * 0xD1B54A32D192ED03ULL));
}

static inline uint64_t draw(uint64_t key, uint64_t j) {
  return mix64(key + (j + 1) * 0x9E3779B97F4A7C15ULL);
}

static inline double std_normal(uint64_t key, uint64_t i) {
  const double two53 = 9007199254740992.0;
  uint64_t a = draw(key, 2 * i), b = draw(key, 2 * i + 1);
  double u1 = ((double)(a >> 11) + 0.5) / two53;
  double u2 = (double)(b >> 11) / two53;
  return sqrt(-2.0 * log(u1)) * cos(6.283185307179586476925286766559 * u2);
}

uint16_t dvgen_f32_to_bf16(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  if ((u & 0x7F800000u) == 0x7F800000u) { /* inf / nan: keep, quiet nan */
    return (uint16_t)((u >> 16) | ((u & 0xFFFFu) ? 0x40u : 0u));
  }
  uint32_t lsb = (u >> 16) & 1u;
  u += 0x7FFFu + lsb;
  return (uint16_t)(u >> 16);
}

uint16_t dvgen_f64_to_bf16(double v) { return dvgen_f32_to_bf16((float)v); }

/* out[i] = bf16(mean + sigma * normal(key(seed, stream), offset + i)), i < n */
void dvgen_normal_bf16(uint64_t seed, uint64_t stream, uint64_t offset, int64_t n,
                       double mean, double sigma, uint16_t* out) {
  const uint64_t key = dvgen_key(seed, stream);
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i)
    out[i] = dvgen_f64_to_bf16(mean + sigma * std_normal(key, offset + (uint64_t)i));
}

/* out[i] = mean + sigma * normal(key(seed, stream), offset + i), in double */
void dvgen_normal_f64(uint64_t seed, uint64_t stream, uint64_t offset, int64_t n,
                      double mean, double sigma, double* out) {
  const uint64_t key = dvgen_key(seed, stream);
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i)
    out[i] = mean + sigma * std_normal(key, offset + (uint64_t)i);
}

/* Frame-correlated normals for video-shaped embeddings: an AR(1) chain over
 * frames, applied independently at every (token-in-frame, channel) element.
 *   e_0 = n_0,   e_f = rho * e_{f-1} + sqrt(1 - rho^2) * n_f
 * where n_f are standard normals drawn at counter f * per_frame + k.
 * out[f * per_frame + k] = bf16(scale * e_f[k]).  Each e_f is still N(0, 1). */
void dvgen_ar1_frames_bf16(uint64_t seed, uint64_t stream, int64_t n_frames,
                           int64_t per_frame, double rho, double scale, uint16_t* out) {
  const uint64_t key = dvgen_key(seed, stream);
  const double c = sqrt(1.0 - rho * rho);
#pragma omp parallel for schedule(static)
  for (int64_t k = 0; k < per_frame; ++k) {
    double e = 0.0;
    for (int64_t f = 0; f < n_frames; ++f) {
      double nf = std_normal(key, (uint64_t)(f * per_frame + k));
      e = (f == 0) ? nf : rho * e + c * nf;
      out[f * per_frame + k] = dvgen_f64_to_bf16(scale * e);
    }
  }
}

/* bf16 -> float widening (exact), for callers without a bf16 type. */
void dvgen_bf16_to_f32(const uint16_t* in, int64_t n, float* out) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    uint32_t u = ((uint32_t)in[i]) << 16;
    float f;
    memcpy(&f, &u, 4);
    out[i] = f;
  }
}
