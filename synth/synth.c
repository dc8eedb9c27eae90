/*
 * Seeded synthetic inputs shared by the oracle and the CUDA path's tests and
 * benchmark: weights and token ids.  This file holds no arithmetic of the
 * forecasting method itself; it only draws numbers.
 *
 * Generator: Philox4x64-10, the counter-based generator of Salmon, Moraes,
 * Dror and Shaw, "Parallel random numbers: as easy as 1, 2, 3" (SC'11).
 * Every value is a pure function of (seed, stream, index), so any slice of
 * any tensor regenerates independently and in any order.
 *
 * Weights: each value is an Irwin-Hall sum of eight 16-bit uniforms,
 * recentred and scaled so that its mean is 0 and its standard deviation is
 * sigma, then rounded once to bf16 (round to nearest, ties to even).  Only
 * integer arithmetic, one int->float conversion and one float multiply are
 * involved, so the bits are identical on every IEEE-754 host.
 *
 * Token ids: uniform over [0, V) (Lemire's multiply-shift) or Zipf(s) over
 * ranks 1..V with id = rank - 1 (inverse CDF on a double-precision table).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define PHILOX_M0 0xD2E7470EE14C6C93ULL
#define PHILOX_M1 0xCA5A826395121157ULL
#define PHILOX_W0 0x9E3779B97F4A7C15ULL
#define PHILOX_W1 0xBB67AE8584CAA73BULL

static inline void mulhilo64(uint64_t a, uint64_t b, uint64_t* hi, uint64_t* lo) {
  unsigned __int128 p = (unsigned __int128)a * (unsigned __int128)b;
  *hi = (uint64_t)(p >> 64);
  *lo = (uint64_t)p;
}

void synth_philox4x64_10(const uint64_t ctr_in[4], const uint64_t key_in[2], uint64_t out[4]) {
  uint64_t x0 = ctr_in[0], x1 = ctr_in[1], x2 = ctr_in[2], x3 = ctr_in[3];
  uint64_t k0 = key_in[0], k1 = key_in[1];
  for (int r = 0; r < 10; ++r) {
    uint64_t hi0, lo0, hi1, lo1;
    mulhilo64(PHILOX_M0, x0, &hi0, &lo0);
    mulhilo64(PHILOX_M1, x2, &hi1, &lo1);
    uint64_t y0 = hi1 ^ x1 ^ k0;
    uint64_t y1 = lo1;
    uint64_t y2 = hi0 ^ x3 ^ k1;
    uint64_t y3 = lo0;
    x0 = y0; x1 = y1; x2 = y2; x3 = y3;
    k0 += PHILOX_W0;
    k1 += PHILOX_W1;
  }
  out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/* One Philox block for (seed, stream, block index). */
static inline void block_of(uint64_t seed, uint64_t stream, uint64_t blk, uint64_t out[4]) {
  const uint64_t ctr[4] = {blk, stream, 0x5EED0000u, 0};
  const uint64_t key[2] = {seed, 0x9A9E5F0C3A57B1D2ULL};
  synth_philox4x64_10(ctr, key, out);
}

static inline uint16_t f32_to_bf16_rne(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  if ((u & 0x7F800000u) == 0x7F800000u) return (uint16_t)((u >> 16) | ((u & 0xFFFFu) ? 0x40u : 0u));
  uint32_t lsb = (u >> 16) & 1u;
  u += 0x7FFFu + lsb;
  return (uint16_t)(u >> 16);
}

/* The fp32 scale that maps an Irwin-Hall(8) sum of 16-bit uniforms (centred)
 * to standard deviation sigma: var(one u16) = (65536^2 - 1) / 12. */
float synth_irwin_hall_scale(float sigma) {
  double var8 = 8.0 * (65536.0 * 65536.0 - 1.0) / 12.0;
  return (float)((double)sigma / sqrt(var8));
}

/* Value of element `index` of tensor `stream`, as fp32 before bf16 rounding. */
static inline float normal_value(uint64_t seed, uint64_t stream, uint64_t index, float scale) {
  uint64_t b[4];
  block_of(seed, stream, index >> 1, b);
  const uint64_t w0 = b[(index & 1) * 2], w1 = b[(index & 1) * 2 + 1];
  int64_t s = 0;
  for (int j = 0; j < 4; ++j) {
    s += (int64_t)((w0 >> (16 * j)) & 0xFFFFu);
    s += (int64_t)((w1 >> (16 * j)) & 0xFFFFu);
  }
  /* 8 * 32767.5 = 262140: the exact mean of the sum. */
  const float centred = (float)(s - 262140);
  return centred * scale;
}

void synth_normal_f32(uint64_t seed, uint64_t stream, uint64_t start, uint64_t n, float sigma, float* out) {
  const float scale = synth_irwin_hall_scale(sigma);
#pragma omp parallel for schedule(static)
  for (long long i = 0; i < (long long)n; ++i) out[i] = normal_value(seed, stream, start + (uint64_t)i, scale);
}

void synth_normal_bf16(uint64_t seed, uint64_t stream, uint64_t start, uint64_t n, float sigma, uint16_t* out) {
  const float scale = synth_irwin_hall_scale(sigma);
#pragma omp parallel for schedule(static)
  for (long long i = 0; i < (long long)n; ++i)
    out[i] = f32_to_bf16_rne(normal_value(seed, stream, start + (uint64_t)i, scale));
}

/* 64 random bits for draw i of (seed, stream). */
static inline uint64_t bits_of(uint64_t seed, uint64_t stream, uint64_t i) {
  uint64_t b[4];
  block_of(seed, stream, i >> 2, b);
  return b[i & 3];
}

/* Uniform integers in [lo, hi] inclusive. */
void synth_uniform_int(uint64_t seed, uint64_t stream, uint64_t n, int64_t lo, int64_t hi, int32_t* out) {
  const uint64_t span = (uint64_t)(hi - lo + 1);
  for (uint64_t i = 0; i < n; ++i) {
    uint64_t r = bits_of(seed, stream, i) >> 32; /* 32 uniform bits */
    out[i] = (int32_t)(lo + (int64_t)((r * span) >> 32));
  }
}

/* Uniform doubles in [0, 1) with 53 random bits. */
void synth_uniform_f64(uint64_t seed, uint64_t stream, uint64_t n, double* out) {
  for (uint64_t i = 0; i < n; ++i) out[i] = (double)(bits_of(seed, stream, i) >> 11) * (1.0 / 9007199254740992.0);
}

/* Zipf(s) ids: P(rank k) proportional to k^-s for k = 1..V; id = k - 1. */
int synth_zipf_ids(uint64_t seed, uint64_t stream, uint64_t n, uint32_t vocab, double s, int32_t* out) {
  double* cdf = (double*)malloc(sizeof(double) * vocab);
  if (!cdf) return -1;
  double acc = 0.0;
  for (uint32_t k = 0; k < vocab; ++k) {
    acc += pow((double)(k + 1), -s);
    cdf[k] = acc;
  }
  for (uint32_t k = 0; k < vocab; ++k) cdf[k] /= acc;
  cdf[vocab - 1] = 1.0;
  for (uint64_t i = 0; i < n; ++i) {
    const double u = (double)(bits_of(seed, stream, i) >> 11) * (1.0 / 9007199254740992.0);
    /* smallest k with cdf[k] > u */
    uint32_t lo = 0, hi = vocab - 1;
    while (lo < hi) {
      uint32_t mid = lo + (hi - lo) / 2;
      if (cdf[mid] > u) hi = mid; else lo = mid + 1;
    }
    out[i] = (int32_t)lo;
  }
  free(cdf);
  return 0;
}
