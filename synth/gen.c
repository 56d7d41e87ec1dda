/*
 * Counter-based generator for the synthetic workloads (weights, visual
 * embeddings, prompt ids).  It holds no arithmetic of the decoding method:
 * it only turns (seed, stream, index) into numbers.
 *
 *   draw(seed, stream, i) = splitmix64 output number i+1 of the sequence whose
 *                           state starts at key(seed, stream)
 *   normal(i)             = Box-Muller on draws 2i and 2i+1, cosine branch
 *   bf16                  = round-to-nearest-even of the fp32 rounding of
 *                           mean + std * normal(i)
 *
 * Every element depends only on its own index, so any chunking or thread
 * count gives the same array.  Compiled with -ffp-contract=off so that the
 * fp64 arithmetic is the same on x86-64 and aarch64 hosts.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#define GOLDEN 0x9E3779B97F4A7C15ULL

static inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

static inline uint64_t stream_key(uint64_t seed, uint64_t stream) {
  return mix64(mix64(seed + GOLDEN) ^ (stream * 0xD1B54A32D192ED03ULL + 0x8CB92BA72F3D8DD7ULL));
}

static inline uint64_t draw(uint64_t key, uint64_t i) { return mix64(key + (i + 1) * GOLDEN); }

static inline uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  if ((u & 0x7F800000u) == 0x7F800000u) return (uint16_t)((u >> 16) | ((u & 0xFFFFu) ? 0x40u : 0u));
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

static inline double normal_at(uint64_t key, uint64_t i) {
  const double two_pi = 6.283185307179586476925286766559;
  uint64_t h1 = draw(key, 2 * i), h2 = draw(key, 2 * i + 1);
  double u1 = ((double)(h1 >> 11) + 1.0) * 0x1.0p-53; /* (0, 1] */
  double u2 = (double)(h2 >> 11) * 0x1.0p-53;         /* [0, 1) */
  return sqrt(-2.0 * log(u1)) * cos(two_pi * u2);
}

void synth_normal_bf16(uint64_t seed, uint64_t stream, double mean, double std, int64_t n, uint16_t* out) {
  uint64_t key = stream_key(seed, stream);
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) out[i] = f32_to_bf16_rne((float)(mean + std * normal_at(key, (uint64_t)i)));
}

void synth_normal_f64(uint64_t seed, uint64_t stream, double mean, double std, int64_t n, double* out) {
  uint64_t key = stream_key(seed, stream);
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) out[i] = mean + std * normal_at(key, (uint64_t)i);
}

/* Uniform integers in [lo, hi): multiply-shift of the top 32 bits (bias < 2^-32 * range). */
void synth_uniform_i32(uint64_t seed, uint64_t stream, int64_t lo, int64_t hi, int64_t n, int32_t* out) {
  uint64_t key = stream_key(seed, stream);
  uint64_t range = (uint64_t)(hi - lo);
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    uint64_t h = draw(key, (uint64_t)i) >> 32;
    out[i] = (int32_t)(lo + (int64_t)((h * range) >> 32));
  }
}

void synth_raw_u64(uint64_t seed, uint64_t stream, int64_t n, uint64_t* out) {
  uint64_t key = stream_key(seed, stream);
  for (int64_t i = 0; i < n; ++i) out[i] = draw(key, (uint64_t)i);
}

/* bf16 bit patterns -> fp64 values (exact widening), multi-threaded for large tensors. */
void synth_bf16_to_f64(const uint16_t* in, int64_t n, double* out) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    uint32_t u = ((uint32_t)in[i]) << 16;
    float f;
    memcpy(&f, &u, 4);
    out[i] = (double)f;
  }
}
