// Temperature sampling by the Gumbel-max identity.
//
// Every row of a forecast is sampled at temperature T (Sec. 3.1 setup: three
// repeats per row at T = 1).  Token t of sampled row r is
//     argmax_v ( l_v / T + G_v ),   G_v = -ln(-ln U_v),
// an exact draw from softmax(l / T); the lowest id wins an exact tie.
// U_v is reproducible from (seed, t, r, v) alone: it is output word r mod 4 of
// Philox4x64-10 under key (seed, 0) at counter (v, t, r / 4, 0), mapped to
// (floor(w / 2^41) + 1/2) 2^-23, which float32 holds exactly.  Rows of one
// call are numbered r = item * repeats + repeat; t = 0 is drawn from the
// prompt's logits and t = s + 1 from decode step s.
//
// Philox4x64-10 is the counter-based generator of Salmon, Moraes, Dror and
// Shaw ("Parallel random numbers: as easy as 1, 2, 3", SC 2011): ten rounds of
// two 64x64->128-bit products on a 256-bit counter, the key advanced by the
// Weyl constants between rounds.
#pragma once

#include <cstdint>

namespace gf {

// Orders (value, index) pairs by value, then by lower index: larger key = better.  The greedy
// arg max and the sampled draw both keep the largest key of a row (zero = no candidate yet).
__device__ __forceinline__ unsigned long long argmax_key(float v, int idx) {
  const uint32_t u = __float_as_uint(v);
  const uint32_t ord = (u & 0x80000000u) ? ~u : (u | 0x80000000u);
  return ((unsigned long long)ord << 32) | (0xFFFFFFFFu - (uint32_t)idx);
}

struct SampleParams {
  unsigned long long seed;
  float inv_temp;  // 1 / T
  int32_t reserved;
};

__device__ __forceinline__ void philox4x64_10(uint64_t c0, uint64_t c1, uint64_t c2, uint64_t c3, uint64_t k0,
                                              uint64_t k1, uint64_t w[4]) {
  constexpr uint64_t kMul0 = 0xD2E7470EE14C6C93ull, kMul1 = 0xCA5A826395121157ull;
  constexpr uint64_t kWeyl0 = 0x9E3779B97F4A7C15ull, kWeyl1 = 0xBB67AE8584CAA73Bull;
#pragma unroll
  for (int round = 0; round < 10; ++round) {
    const uint64_t hi0 = __umul64hi(kMul0, c0), lo0 = kMul0 * c0;
    const uint64_t hi1 = __umul64hi(kMul1, c2), lo1 = kMul1 * c2;
    c0 = hi1 ^ c1 ^ k0;
    c1 = lo1;
    c2 = hi0 ^ c3 ^ k1;
    c3 = lo0;
    k0 += kWeyl0;
    k1 += kWeyl1;
  }
  w[0] = c0;
  w[1] = c1;
  w[2] = c2;
  w[3] = c3;
}

// G = -ln(-ln U) for the uniform carried by the top 23 bits of w.
__device__ __forceinline__ float gumbel_from_word(uint64_t w) {
  const float u = (__uint2float_rn((uint32_t)(w >> 41)) + 0.5f) * 1.1920928955078125e-07f;  // * 2^-23
  return -logf(-logf(u));
}

// The perturbed score of vocabulary id v for row r at token t.
__device__ __forceinline__ float sample_score(float logit, const SampleParams& sp, int t, int r, int v) {
  uint64_t w[4];
  philox4x64_10((uint64_t)v, (uint64_t)t, (uint64_t)(r >> 2), 0ull, sp.seed, 0ull, w);
  const int j = r & 3;
  const uint64_t wr = j == 0 ? w[0] : (j == 1 ? w[1] : (j == 2 ? w[2] : w[3]));
  return fmaf(logit, sp.inv_temp, gumbel_from_word(wr));
}

}  // namespace gf
