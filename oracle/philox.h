// Oracle-private Philox4x32-10 (test infrastructure; never linked into the CUDA path).
//
// Written from the definition in Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy as
// 1, 2, 3" (SC'11), Sec. 3.2: a 4-word counter is mixed by 10 rounds; each round multiplies words 0
// and 2 by the two Philox multipliers, swaps the high halves into the other lanes xored with the
// round key, and the 2-word key is bumped by the two Weyl increments (golden ratio and sqrt(3)-1,
// in 32-bit fixed point) between rounds.  The method draws its mini-batch indices from this
// generator keyed by (seed, worker k, step), per the paper's Eq. 2 ("I^k sampled from the worker's
// local data").
#pragma once
#include <cstdint>

namespace oracle {

struct Philox4 {
  uint32_t v[4];
};

inline Philox4 philox4x32_10(Philox4 ctr, uint32_t k0, uint32_t k1) {
  const uint32_t M0 = 0xD2511F53u, M1 = 0xCD9E8D57u;  // SC'11 Table 2, Philox4x32
  const uint32_t W0 = 0x9E3779B9u, W1 = 0xBB67AE85u;  // Weyl key increments
  for (int round = 0; round < 10; ++round) {
    const uint64_t p0 = (uint64_t)M0 * (uint64_t)ctr.v[0];
    const uint64_t p1 = (uint64_t)M1 * (uint64_t)ctr.v[2];
    const uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    const uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    Philox4 n;
    n.v[0] = hi1 ^ ctr.v[1] ^ k0;
    n.v[1] = lo1;
    n.v[2] = hi0 ^ ctr.v[3] ^ k1;
    n.v[3] = lo0;
    ctr = n;
    k0 += W0;
    k1 += W1;
  }
  return ctr;
}

}  // namespace oracle
