/*
 * Seeded synthetic inputs for the verifier hot path.
 *
 * This file holds no arithmetic of the method itself: it only turns a 64-bit
 * seed into reproducible random tensors.  Both the CUDA path's tests/bench and
 * the fp64 oracle receive the arrays it writes, so the two sides see
 * bit-identical inputs without sharing any code of the computation.
 *
 * Generator (counter-based, so any element can be produced independently):
 *   SplitMix64 (Steele, Lea & Flood, OOPSLA 2014): the n-th output of the
 *   generator seeded with s is  mix(s + (n + 1) * 0x9E3779B97F4A7C15)  where
 *   mix is the published 64-bit finaliser (xor-shift 30 / multiply /
 *   xor-shift 27 / multiply / xor-shift 31).
 *   Stream key for tensor `stream` under seed s:  key = output #stream of s.
 *   Element i of a stream uses outputs 2i and 2i+1 of the key:
 *     u1 = ((x0 >> 11) + 1) * 2^-53   in (0, 1]
 *     u2 =  (x1 >> 11)      * 2^-53   in [0, 1)
 *   Normal variate (Box & Muller 1958, cosine branch):
 *     n = sqrt(-2 ln u1) * cos(2 pi u2)
 *   Uniform real in [a, b): a + (b - a) * u2 computed from output 2i+1 only.
 *   Uniform integer in [lo, hi): lo + floor(((x0 >> 32) * (hi - lo)) / 2^32)
 *     (multiply-shift range reduction on the high word of output 2i).
 * Rounding: bf16 = round-to-nearest-even(fp32(round-to-nearest-even(x)));
 *           fp16 = round-to-nearest-even(x) in one step (_Float16 cast).
 *
 * Build: gcc -O2 -fopenmp -shared -fPIC synth.c -o libfvrag_synth.so -lm
 */
#include <math.h>
#include <stdint.h>
#include <string.h>
#include <stddef.h>

#define SM64_GAMMA 0x9E3779B97F4A7C15ULL

static inline uint64_t sm64_mix(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

static inline uint64_t sm64_at(uint64_t seed, uint64_t n) {
  return sm64_mix(seed + (n + 1ULL) * SM64_GAMMA);
}

uint64_t synth_stream_key(uint64_t seed, uint64_t stream) { return sm64_at(seed, stream); }

uint64_t synth_raw(uint64_t key, uint64_t n) { return sm64_at(key, n); }

static inline double synth_normal_at(uint64_t key, uint64_t i) {
  const double two_m53 = 1.0 / 9007199254740992.0; /* 2^-53 */
  uint64_t x0 = sm64_at(key, 2ULL * i);
  uint64_t x1 = sm64_at(key, 2ULL * i + 1ULL);
  double u1 = ((double)(x0 >> 11) + 1.0) * two_m53;
  double u2 = (double)(x1 >> 11) * two_m53;
  return sqrt(-2.0 * log(u1)) * cos(6.283185307179586 * u2);
}

double synth_normal(uint64_t key, uint64_t i) { return synth_normal_at(key, i); }

static inline uint16_t f32_to_bf16_rne(float f) {
  uint32_t b;
  memcpy(&b, &f, 4);
  if ((b & 0x7F800000u) == 0x7F800000u) return (uint16_t)(b >> 16); /* inf/nan: not produced */
  b += 0x7FFFu + ((b >> 16) & 1u);
  return (uint16_t)(b >> 16);
}

void synth_fill_normal_f64(double* out, int64_t n, uint64_t key, double mean, double std) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) out[i] = mean + std * synth_normal_at(key, (uint64_t)i);
}

void synth_fill_normal_bf16(uint16_t* out, int64_t n, uint64_t key, double mean, double std) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    double x = mean + std * synth_normal_at(key, (uint64_t)i);
    out[i] = f32_to_bf16_rne((float)x);
  }
}

void synth_fill_uniform_f64(double* out, int64_t n, uint64_t key, double a, double b) {
  const double two_m53 = 1.0 / 9007199254740992.0;
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    uint64_t x1 = sm64_at(key, 2ULL * (uint64_t)i + 1ULL);
    out[i] = a + (b - a) * ((double)(x1 >> 11) * two_m53);
  }
}

void synth_fill_uniform_i32(int32_t* out, int64_t n, uint64_t key, int64_t lo, int64_t hi) {
  uint64_t range = (uint64_t)(hi - lo);
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    uint64_t x0 = sm64_at(key, 2ULL * (uint64_t)i);
    out[i] = (int32_t)(lo + (int64_t)(((x0 >> 32) * range) >> 32));
  }
}

/* fp64 -> fp16 with a single round-to-nearest-even (the compiler's _Float16
 * conversion is IEEE-correct on x86-64 and AArch64). */
void synth_round_f16(const double* in, uint16_t* out, int64_t n) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    _Float16 h = (_Float16)in[i];
    memcpy(&out[i], &h, 2);
  }
}

void synth_round_bf16(const double* in, uint16_t* out, int64_t n) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) out[i] = f32_to_bf16_rne((float)in[i]);
}
