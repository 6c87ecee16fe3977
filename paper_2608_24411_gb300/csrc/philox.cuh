// Counter-based uniforms on the device: Philox4x64-10 (Salmon, Moraes,
// Dror, Shaw, "Parallel random numbers: as easy as 1, 2, 3", SC 2011).
// Each round multiplies words 0 and 2 by the two round constants, keeps the
// 128-bit products' halves, xors the high halves with words 1 / 3 and the
// round key, and swaps positions; the key advances by the Weyl increments
// (golden ratio, sqrt(3) - 1) between rounds.
#pragma once
#include <stdint.h>

namespace rs {

struct U64x4 {
  uint64_t w[4];
};

__device__ __forceinline__ U64x4 philox4x64_10(uint64_t c0, uint64_t c1, uint64_t c2,
                                               uint64_t c3, uint64_t k0, uint64_t k1) {
  constexpr uint64_t kMulA = 0xD2E7470EE14C6C93ull;
  constexpr uint64_t kMulB = 0xCA5A826395121157ull;
  constexpr uint64_t kWeylA = 0x9E3779B97F4A7C15ull;
  constexpr uint64_t kWeylB = 0xBB67AE8584CAA73Bull;
#pragma unroll
  for (int round = 0; round < 10; ++round) {
    const uint64_t hiA = __umul64hi(kMulA, c0), loA = kMulA * c0;
    const uint64_t hiB = __umul64hi(kMulB, c2), loB = kMulB * c2;
    const uint64_t n0 = hiB ^ c1 ^ k0;
    const uint64_t n2 = hiA ^ c3 ^ k1;
    c0 = n0;
    c1 = loB;
    c2 = n2;
    c3 = loA;
    k0 += kWeylA;
    k1 += kWeylB;
  }
  U64x4 r;
  r.w[0] = c0;
  r.w[1] = c1;
  r.w[2] = c2;
  r.w[3] = c3;
  return r;
}

// Top 24 bits of a 64-bit word as a float in [0, 1): exact in fp32.
__device__ __forceinline__ float u24(uint64_t word) {
  return static_cast<float>(static_cast<uint32_t>(word >> 40)) * (1.0f / 16777216.0f);
}

// U(seed, seq, row, draw) of the library's randomness contract.
__device__ __forceinline__ float uniform_draw(uint64_t seed, uint32_t seq, uint32_t row,
                                              int draw) {
  const U64x4 r = philox4x64_10(row, seq, 0, 0, seed, 0);
  const uint64_t w = draw == 0 ? r.w[0] : draw == 1 ? r.w[1] : draw == 2 ? r.w[2] : r.w[3];
  return u24(w);
}

}  // namespace rs
