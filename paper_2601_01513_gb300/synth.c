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

/* Rows of unit-length vectors: element (r, i) starts as normal variate r*E+i of
 * the stream, each row is divided by its Euclidean length, then rounded to fp16
 * (round-to-nearest-even).  Used for CLIP-like text embeddings of a corpus. */
void synth_fill_unit_rows_f16(uint16_t* out, int64_t rows, int E, uint64_t key) {
#pragma omp parallel
  {
    double* buf = (double*)__builtin_alloca(sizeof(double) * (size_t)E);
#pragma omp for schedule(static)
    for (int64_t r = 0; r < rows; ++r) {
      double ss = 0.0;
      for (int i = 0; i < E; ++i) {
        buf[i] = synth_normal_at(key, (uint64_t)(r * E + i));
        ss += buf[i] * buf[i];
      }
      const double inv = ss > 0.0 ? 1.0 / sqrt(ss) : 0.0;
      for (int i = 0; i < E; ++i) {
        _Float16 h = (_Float16)(buf[i] * inv);
        memcpy(&out[r * E + i], &h, 2);
      }
    }
  }
}

/* Synthetic RGB video frames, out[T][H][W][3] uint8.
 * A scene is a smooth two-colour gradient (angle, drift per frame) with a disc of
 * a third colour moving across it; frame t shows scene fa[t] at time ftau[t]
 * (frames since the scene began), blended with scene fb[t] by weight fw[t]
 * (a fade), plus uniform noise of amplitude sigma (of scene fa[t]).  The noise of
 * pixel p of frame t comes from output t * H * W + p of the stream: its bits
 * 21c .. 21c+20 give channel c a uniform u in [0, 1) and the noise is
 * sigma * (2u - 1).
 * scene parameters, 17 doubles each:
 *   c0[3] c1[3] c2[3] angle drift cx cy vx vy radius sigma
 * (cx, cy, radius in fractions of the frame; vx, vy in fractions per frame). */
typedef struct {
  double ca, sa, ph, cx, cy, rr;
  const double* sp;
} scene_state;

static void scene_at(const double* sp, double tau, double H, scene_state* st) {
  st->sp = sp;
  st->ca = cos(sp[9]);
  st->sa = sin(sp[9]);
  st->ph = sp[10] * tau;
  st->cx = sp[11] + sp[13] * tau;
  st->cy = sp[12] + sp[14] * tau;
  st->cx -= floor(st->cx);
  st->cy -= floor(st->cy);
  st->rr = sp[15] * H;
}

static inline void scene_colour(const scene_state* st, double xn, double yn, double W, double H,
                                double col[3]) {
  const double u = xn * st->ca + yn * st->sa + st->ph;
  double g = u - floor(u);
  g = g < 0.5 ? 2.0 * g : 2.0 - 2.0 * g;
  const double dx = (xn - st->cx) * W, dy = (yn - st->cy) * H;
  const double* sp = st->sp;
  if (dx * dx + dy * dy < st->rr * st->rr) {
    col[0] = sp[6]; col[1] = sp[7]; col[2] = sp[8];
  } else {
    for (int c = 0; c < 3; ++c) col[c] = sp[c] + (sp[3 + c] - sp[c]) * g;
  }
}

void synth_video_frames(uint8_t* out, int T, int H, int W, uint64_t key, const int32_t* fa,
                        const int32_t* fb, const double* fw, const double* ftau,
                        const double* scenes) {
  const int64_t npix = (int64_t)H * W;
  const double two_m21 = 1.0 / 2097152.0;
#pragma omp parallel for collapse(2) schedule(static)
  for (int t = 0; t < T; ++t) {
    for (int y = 0; y < H; ++y) {
      scene_state A, B;
      scene_at(scenes + 17 * (int64_t)fa[t], ftau[t], H, &A);
      scene_at(scenes + 17 * (int64_t)fb[t], ftau[t], H, &B);
      const double w = fw[t], sigma = A.sp[16];
      const double yn = (y + 0.5) / H;
      for (int x = 0; x < W; ++x) {
        const double xn = (x + 0.5) / W;
        double ca[3], cb[3];
        scene_colour(&A, xn, yn, W, H, ca);
        if (w > 0.0) scene_colour(&B, xn, yn, W, H, cb);
        const int64_t p = (int64_t)y * W + x;
        const uint64_t r = sm64_at(key, (uint64_t)((int64_t)t * npix + p));
        for (int c = 0; c < 3; ++c) {
          const double base = w > 0.0 ? (1.0 - w) * ca[c] + w * cb[c] : ca[c];
          const double u = (double)((r >> (21 * c)) & 0x1FFFFFu) * two_m21;
          double v = floor(base + sigma * (2.0 * u - 1.0) + 0.5);
          v = v < 0.0 ? 0.0 : (v > 255.0 ? 255.0 : v);
          out[(t * npix + p) * 3 + c] = (uint8_t)v;
        }
      }
    }
  }
}
