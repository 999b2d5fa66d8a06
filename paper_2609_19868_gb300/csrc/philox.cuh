// Counter-based random numbers of the sampling kernels: Philox4x32-10
// (Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy as 1, 2, 3",
// SC'11) and the uniform variate made from one of its 32-bit words.
#pragma once

#include <stdint.h>

namespace zarya {

// Each round multiplies counter words 0 and 2 by the round constants into
// 64-bit products and forms (hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0); the key
// advances by the Weyl increments between rounds.
__device__ __forceinline__ uint4 philox4x32_10(uint4 c, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    const uint32_t lo0 = 0xD2511F53u * c.x, hi0 = __umulhi(0xD2511F53u, c.x);
    const uint32_t lo1 = 0xCD9E8D57u * c.z, hi1 = __umulhi(0xCD9E8D57u, c.z);
    c = make_uint4(hi1 ^ c.y ^ k0, lo1, hi0 ^ c.w ^ k1, lo0);
  }
  return c;
}

// u = fl32(fl32(w) 2^-32 + 2^-33) in (0, 1]: the product is exact, so the
// fused multiply-add rounds once, like the separate add.
__device__ __forceinline__ float uniform_from_word(uint32_t w) {
  return fmaf(__uint2float_rn(w), 0x1p-32f, 0x1p-33f);
}

}  // namespace zarya
