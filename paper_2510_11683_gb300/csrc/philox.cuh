// Philox4x64-10 counter-based generator (Salmon, Moraes, Dror, Shaw, "Parallel
// Random Numbers: As Easy as 1, 2, 3", SC'11): four 64-bit counter words, two
// key words, ten rounds. Each round multiplies counter words 0 and 2 by fixed
// odd constants into 128-bit products and mixes the halves with the other two
// words and the key; the key is bumped by two Weyl constants between rounds.
#pragma once

#include <stdint.h>

namespace bgpo {

struct PhiloxOut {
  uint64_t w[4];
};

__device__ __forceinline__ PhiloxOut philox4x64_10(uint64_t c0, uint64_t c1, uint64_t c2,
                                                   uint64_t c3, uint64_t k0, uint64_t k1) {
  constexpr uint64_t kMul0 = 0xD2E7470EE14C6C93ull;
  constexpr uint64_t kMul1 = 0xCA5A826395121157ull;
  constexpr uint64_t kWeyl0 = 0x9E3779B97F4A7C15ull;
  constexpr uint64_t kWeyl1 = 0xBB67AE8584CAA73Bull;
#pragma unroll
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += kWeyl0;
      k1 += kWeyl1;
    }
    const uint64_t hi_a = __umul64hi(kMul0, c0), lo_a = kMul0 * c0;
    const uint64_t hi_b = __umul64hi(kMul1, c2), lo_b = kMul1 * c2;
    const uint64_t n0 = hi_b ^ c1 ^ k0;
    const uint64_t n2 = hi_a ^ c3 ^ k1;
    c0 = n0;
    c1 = lo_b;
    c2 = n2;
    c3 = lo_a;
  }
  PhiloxOut o;
  o.w[0] = c0;
  o.w[1] = c1;
  o.w[2] = c2;
  o.w[3] = c3;
  return o;
}

// Counter layout of the masking process: (c0, b, j, stream), key (seed, 0).
constexpr uint64_t kStreamMask = 0;  // c0 = i / 4, output word i % 4 -> position i
constexpr uint64_t kStreamT = 1;     // c0 = 0, output word 0 -> t_{b,j}
constexpr int kU24Shift = 40;        // uniform 24-bit integer = word >> 40

}  // namespace bgpo
