// Counter-based Gumbel noise for the LM-head sample (Eqs. 6-7 draw a token
// from each masked position's marginal; Gumbel-max does it with one noise
// value per vocabulary entry).
//
// Generator: Philox4x32 with 10 rounds (Salmon, Moraes, Dror, Shaw,
// "Parallel random numbers: as easy as 1, 2, 3", SC 2011).  Each round
// multiplies counter words 0 and 2 by fixed odd constants, splits the 64-bit
// products into high and low halves, and mixes them with words 1 and 3 and
// the key; the key grows by two Weyl increments between rounds.
//
// Noise of block position n (= b * k + i) and vocabulary id v: x is word
// v mod 4 of the call with counter (v div 4, n, offset low, offset high) and
// key (seed low, seed high); u = ((x >> 9) + 1/2) 2^-23, exact in fp32 (24
// significant bits) and strictly inside (0, 1); g = -ln(-ln u).
#pragma once

#include <cstdint>
#include <math.h>

namespace sbd_philox {

constexpr uint32_t kM0 = 0xD2511F53u, kM1 = 0xCD9E8D57u;   // round multipliers
constexpr uint32_t kW0 = 0x9E3779B9u, kW1 = 0xBB67AE85u;   // key increments

__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += kW0;
      k1 += kW1;
    }
    const uint32_t hi0 = __umulhi(kM0, c.x), lo0 = kM0 * c.x;
    const uint32_t hi1 = __umulhi(kM1, c.z), lo1 = kM1 * c.z;
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
  }
  return c;
}

// The noise value of one 32-bit word.  The inner logarithm is the
// full-precision library logf: near u = 1 it is tiny, g = -ln t depends on
// its relative error, and the large g it gives is the one most likely to
// win the argmax.  The outer one is the fast __logf (CUDA documents at most
// 2^-21.41 absolute error for t in [0.5, 2] and 3 ulp elsewhere, here
// t = -ln u in [6e-8, 16.7]): at most ~6e-6 on g.
__device__ __forceinline__ float gumbel_of_word(uint32_t x) {
  const float u = ((float)(x >> 9) + 0.5f) * 1.1920928955078125e-7f;   // 2^-23
  return -__logf(-logf(u));
}

__device__ __forceinline__ uint32_t word_of(const uint4& w, int i) {
  return i == 0 ? w.x : (i == 1 ? w.y : (i == 2 ? w.z : w.w));
}

}  // namespace sbd_philox
