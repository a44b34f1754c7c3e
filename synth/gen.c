/*
 * Seeded synthetic inputs: counter-based SplitMix64 streams.
 *
 * Test and benchmark infrastructure shared by the CUDA path and the oracle.
 * It draws inputs only (weights, KV contents, tokens) and holds none of the
 * verification arithmetic.
 *
 * SplitMix64 (Steele, Lea and Flood, "Fast splittable pseudorandom number
 * generators", OOPSLA 2014): state advances by the golden gamma
 * 0x9E3779B97F4A7C15 and each output is the state passed through the
 * "mix64variant13" finaliser.  The i-th output (0-based) of a stream keyed by
 * `key` is mix(key + (i + 1) * gamma), so any element is computable alone.
 *
 * Approximately normal values: the four 16-bit lanes of one output are summed
 * (an Irwin-Hall sum of four discrete uniforms on 0..65535), centred, and
 * scaled by one correctly rounded fp32 multiply so that the standard deviation
 * is sigma.  Integer arithmetic plus one IEEE multiply gives identical bits on
 * every host (x86_64 here, aarch64 on the GPU hosts).  bf16 values are the
 * fp32 values rounded to nearest-even.
 */
#include <stdint.h>
#include <string.h>

#define GAMMA 0x9E3779B97F4A7C15ULL

static inline uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

static inline uint64_t stream_at(uint64_t key, uint64_t i) {
  return mix64(key + (i + 1) * GAMMA);
}

static inline float ih4(uint64_t r, float mult) {
  int32_t s = (int32_t)(r & 0xFFFFu) + (int32_t)((r >> 16) & 0xFFFFu) +
              (int32_t)((r >> 32) & 0xFFFFu) + (int32_t)(r >> 48) - 131070;
  return (float)s * mult;
}

static inline uint16_t bf16_rne(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  u += 0x7FFFu + ((u >> 16) & 1u);
  return (uint16_t)(u >> 16);
}

static inline double bf16_to_f64(uint16_t h) {
  uint32_t u = (uint32_t)h << 16;
  float f;
  memcpy(&f, &u, 4);
  return (double)f;
}

uint64_t synth_stream_at(uint64_t key, uint64_t i) { return stream_at(key, i); }

/* out[j] = bf16 bits of element offset+j; mult = fp32(sigma*sqrt(3)/65536). */
void synth_normal_bf16(uint64_t key, uint64_t offset, int64_t n, float mult,
                       uint16_t *out) {
#pragma omp parallel for schedule(static) if (n >= (1 << 20))
  for (int64_t j = 0; j < n; ++j)
    out[j] = bf16_rne(ih4(stream_at(key, offset + (uint64_t)j), mult));
}

void synth_normal_f32(uint64_t key, uint64_t offset, int64_t n, float mult,
                      float *out) {
#pragma omp parallel for schedule(static) if (n >= (1 << 20))
  for (int64_t j = 0; j < n; ++j)
    out[j] = ih4(stream_at(key, offset + (uint64_t)j), mult);
}

/* The same values widened exactly to fp64 (for the fp64 checker). */
void synth_normal_bf16_f64(uint64_t key, uint64_t offset, int64_t n, float mult,
                           double *out) {
#pragma omp parallel for schedule(static) if (n >= (1 << 20))
  for (int64_t j = 0; j < n; ++j)
    out[j] = bf16_to_f64(bf16_rne(ih4(stream_at(key, offset + (uint64_t)j), mult)));
}

void synth_normal_f32_f64(uint64_t key, uint64_t offset, int64_t n, float mult,
                          double *out) {
#pragma omp parallel for schedule(static) if (n >= (1 << 20))
  for (int64_t j = 0; j < n; ++j)
    out[j] = (double)ih4(stream_at(key, offset + (uint64_t)j), mult);
}

/* Uniform integers in [0, bound): high 32 bits times bound, shifted (Lemire). */
void synth_uniform_int(uint64_t key, uint64_t offset, int64_t n, uint32_t bound,
                       int32_t *out) {
#pragma omp parallel for schedule(static) if (n >= (1 << 20))
  for (int64_t j = 0; j < n; ++j)
    out[j] = (int32_t)(((stream_at(key, offset + (uint64_t)j) >> 32) * (uint64_t)bound) >> 32);
}
