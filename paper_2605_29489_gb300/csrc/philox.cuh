// Philox4x32-10 counter-based generator (Salmon, Moraes, Dror and Shaw, "Parallel random
// numbers: as easy as 1, 2, 3", SC 2011), written from the published round function:
// each round multiplies counter words 0 and 2 by 0xD2511F53 and 0xCD9E8D57 (32x32->64),
// mixes the high halves with words 1 and 3 and the round key, and the key (k0, k1) is
// bumped by the Weyl constants 0x9E3779B9 and 0xBB67AE85 between rounds.
#pragma once

#include <stdint.h>

namespace mp {

struct Philox4 {
  uint32_t w[4];
};

// The generator with its ten round keys supplied by the caller: rk[r] = (k0 + r*0x9E3779B9,
// k1 + r*0xBB67AE85) for r = 0..9.  The key schedule does not depend on the counter, so a
// kernel takes it precomputed from its launch parameters.
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

}  // namespace mp
