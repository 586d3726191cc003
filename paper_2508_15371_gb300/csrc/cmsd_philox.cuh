// Philox4x32-10 counter-based generator, host and device.
//
// Written from Salmon, Moraes, Dror, Shaw, "Parallel Random Numbers: As Easy
// as 1, 2, 3" (SC'11): ten rounds over a 4 x 32-bit counter; each round takes
// the 64-bit products of counter words 0 and 2 with two odd multipliers,
// reorders the halves and XORs the key in; the 2 x 32-bit key advances by two
// Weyl increments between rounds.
//
// The paper (arXiv 2508.15371) does not say how its random draws are made;
// the acceptance uniform and the residual (group and entry) uniforms use the
// counter layout documented in include/cmsd.h.
#pragma once
#include <stdint.h>

#if defined(__CUDACC__)
#define CMSD_HD __host__ __device__ __forceinline__
#else
#define CMSD_HD inline
#endif

namespace cmsd {

constexpr uint32_t kPhiloxM0 = 0xD2511F53u;
constexpr uint32_t kPhiloxM1 = 0xCD9E8D57u;
constexpr uint32_t kPhiloxW0 = 0x9E3779B9u;
constexpr uint32_t kPhiloxW1 = 0xBB67AE85u;

constexpr uint32_t kPurposeAccept = 0u;
constexpr uint32_t kPurposeResidual = 1u;
constexpr uint32_t kPurposeGroup = 2u;

struct U4 { uint32_t x, y, z, w; };

CMSD_HD void mul_hilo(uint32_t a, uint32_t b, uint32_t& hi, uint32_t& lo) {
#if defined(__CUDA_ARCH__)
  lo = a * b;
  hi = __umulhi(a, b);
#else
  const uint64_t p = (uint64_t)a * (uint64_t)b;
  lo = (uint32_t)p;
  hi = (uint32_t)(p >> 32);
#endif
}

CMSD_HD U4 philox4x32_10(U4 c, uint32_t k0, uint32_t k1) {
#if defined(__CUDA_ARCH__)
#pragma unroll
#endif
  for (int r = 0; r < 10; ++r) {
    if (r) { k0 += kPhiloxW0; k1 += kPhiloxW1; }
    uint32_t hi0, lo0, hi1, lo1;
    mul_hilo(kPhiloxM0, c.x, hi0, lo0);
    mul_hilo(kPhiloxM1, c.z, hi1, lo1);
    U4 n;
    n.x = hi1 ^ c.y ^ k0;
    n.y = lo1;
    n.z = hi0 ^ c.w ^ k1;
    n.w = lo0;
    c = n;
  }
  return c;
}

CMSD_HD uint32_t seed_lo(uint64_t s) { return (uint32_t)(s & 0xFFFFFFFFull); }
CMSD_HD uint32_t seed_hi(uint64_t s) { return (uint32_t)(s >> 32); }

// 24-bit uniform in [0, 1), exact in float.
CMSD_HD float word_to_unit(uint32_t w) { return (float)(w >> 8) * (1.0f / 16777216.0f); }

CMSD_HD uint32_t iter_word(uint32_t iteration, uint32_t purpose) {
  return (iteration << 2) | purpose;
}

}  // namespace cmsd
