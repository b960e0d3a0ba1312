// Device helpers of the quantizer shared by the translation units that quantize (the
// ShiftQuant quantizer and the fully-quantized L1 batch normalization).  Both compile with
// -fmad=false: every step below is one IEEE binary32 operation.
#pragma once

#include <cstdint>

namespace sq {

// SplitMix64 (Steele, Lea, Flood 2014): the (idx+1)-th output of the generator whose
// state starts at `seed` is the output function applied to the state
// seed + (idx+1) * gamma (mod 2^64).
constexpr uint64_t kSplitMixGamma = 0x9E3779B97F4A7C15ull;

__device__ __forceinline__ uint64_t splitmix64_at(uint64_t seed, uint64_t idx) {
  uint64_t z = seed + (idx + 1ull) * kSplitMixGamma;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// bits 40..63 of the output for the state z (= seed + (idx+1) gamma).  The final step
// z ^ (z >> 31) leaves those bits as they are ((z >> 31) is zero above bit 32), so it is
// skipped; the result equals splitmix64_at(seed, idx) >> 40.
__device__ __forceinline__ uint32_t splitmix64_top24(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return static_cast<uint32_t>(z >> 40);
}

__device__ __forceinline__ float pow2f(int k) { return __int_as_float((127 + k) << 23); }

// The grouping of Eq. 3 for one channel: max{e in [0, G-1] : r 2^e <= tau}; the product by
// 2^e is exact (no rounding) for every finite r <= tau, so the comparison is exact.
__device__ __forceinline__ int group_exponent(float r, float tau, int G) {
  if (r == 0.0f) return G - 1;
  int e = 0;
#pragma unroll 1
  for (int k = 1; k < G; ++k) {
    const float scaled = __fmul_rn(r, __int_as_float((127 + k) << 23));  // r 2^k
    if (scaled <= tau) e = k;
    else break;
  }
  return e;
}

// The ShiftQuant code of one element (App. D; stochastic rounding of App. B): the scaled
// value v = fl(fl(x 2^e) invS) with invS = fl(Q / tau_0), rounded to nearest even
// (stochastic == false) or up with probability frac(v) on the draw of element `idx`,
// clamped to [-Q, Q]; 0 when the tensor quantizes to zero (tau_0 == 0 or not finite).
__device__ __forceinline__ int shift_code(float x, int e, float invS, bool zero, float Qf,
                                          bool stochastic, uint64_t seed, uint64_t idx) {
  if (zero) return 0;
  const float v = __fmul_rn(__fmul_rn(x, pow2f(e)), invS);
  float q;
  if (!stochastic) {
    q = rintf(v);
  } else {
    const float l = floorf(v);
    const float frac = __fsub_rn(v, l);
    const uint64_t h = splitmix64_at(seed, idx);
    const float u = __fmul_rn(static_cast<float>(static_cast<uint32_t>(h >> 40)),
                              5.9604644775390625e-08f);  // * 2^-24, exact
    q = (u < frac) ? __fadd_rn(l, 1.0f) : l;
  }
  q = fminf(fmaxf(q, -Qf), Qf);
  return static_cast<int>(q);
}

}  // namespace sq
