// Philox4x32-10 counter-based generator (Salmon, Moraes, Dror and Shaw, "Parallel random
// numbers: as easy as 1, 2, 3", SC 2011), written from the published round function:
// each round multiplies counter words 0 and 2 by 0xD2511F53 and 0xCD9E8D57 (32x32->64),
// mixes the high halves with words 1 and 3 and the key, and the key is bumped by the Weyl
// constants 0x9E3779B9 and 0xBB67AE85 between rounds.
#pragma once

#include <stdint.h>

namespace mp {

struct Philox4 {
  uint32_t w[4];
};

__device__ __forceinline__ Philox4 philox4x32_10(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3, uint32_t k0,
                                                 uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t lo0 = 0xD2511F53u * c0, hi0 = __umulhi(0xD2511F53u, c0);
    const uint32_t lo1 = 0xCD9E8D57u * c2, hi1 = __umulhi(0xCD9E8D57u, c2);
    const uint32_t n0 = hi1 ^ c1 ^ k0;
    const uint32_t n2 = hi0 ^ c3 ^ k1;
    c0 = n0;
    c1 = lo1;
    c2 = n2;
    c3 = lo0;
  }
  return Philox4{{c0, c1, c2, c3}};
}

// DARE keep bits for the 8 consecutive elements 8g..8g+7 of expert i: bit e set iff the
// e-th 16-bit output word (word e is bits 16*(e%2).. of output e/2) is >= T
__device__ __forceinline__ uint32_t dare_keep8(uint64_t seed, uint32_t expert, uint64_t g, uint32_t T) {
  Philox4 r = philox4x32_10((uint32_t)g, (uint32_t)(g >> 32), expert, 0x44415245u, (uint32_t)seed,
                            (uint32_t)(seed >> 32));
  uint32_t bits = 0;
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    uint32_t word = (r.w[e >> 1] >> (16 * (e & 1))) & 0xFFFFu;
    bits |= (word >= T ? 1u : 0u) << e;
  }
  return bits;
}

}  // namespace mp

namespace mp {

// The same generator with its ten round keys supplied by the caller (k0 + r*0x9E3779B9,
// k1 + r*0xBB67AE85 for r = 0..9): the key schedule does not depend on the counter, so a
// kernel can take it precomputed from its launch parameters.
__device__ __forceinline__ Philox4 philox4x32_10_rk(uint32_t c0, uint32_t c1, uint32_t c2, uint32_t c3,
                                                    const uint32_t (&rk)[10][2]) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    const uint32_t lo0 = 0xD2511F53u * c0, hi0 = __umulhi(0xD2511F53u, c0);
    const uint32_t lo1 = 0xCD9E8D57u * c2, hi1 = __umulhi(0xCD9E8D57u, c2);
    const uint32_t n0 = hi1 ^ c1 ^ rk[r][0];
    const uint32_t n2 = hi0 ^ c3 ^ rk[r][1];
    c0 = n0;
    c1 = lo1;
    c2 = n2;
    c3 = lo0;
  }
  return Philox4{{c0, c1, c2, c3}};
}

// dare_keep8 with precomputed round keys
__device__ __forceinline__ uint32_t dare_keep8_rk(const uint32_t (&rk)[10][2], uint32_t expert, uint64_t g, uint32_t T) {
  Philox4 r = philox4x32_10_rk((uint32_t)g, (uint32_t)(g >> 32), expert, 0x44415245u, rk);
  uint32_t bits = 0;
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    uint32_t word = (r.w[e >> 1] >> (16 * (e & 1))) & 0xFFFFu;
    bits |= (word >= T ? 1u : 0u) << e;
  }
  return bits;
}

}  // namespace mp
