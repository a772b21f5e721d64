// Counter-based Gaussian noise for the ES step, regenerated from the integer
// seed wherever it is needed (§3: only the seed of each perturbation is
// stored; App. D.6: the update "reconstructs the same direction from its
// integer seed").
//
// Definition (fixed by this library; the paper names no generator):
//   block j = floor(g / 4) of global parameter index g;
//   Philox4x32-10 (Salmon et al., SC'11), key = (seed_lo, seed_hi),
//   counter = (j_lo, j_hi, 0, 0) -> words x0..x3;
//   u(x) = (2 (x >> 9) + 1) / 2^24;
//   Box-Muller (Box & Muller, 1958): (x0, x1) -> eps[4j], eps[4j+1] and
//   (x2, x3) -> eps[4j+2], eps[4j+3], with radius sqrt(-2 ln u(x_even)) and
//   angle 2 pi u(x_odd), cos for the even element and sin for the odd one.
#pragma once

#include <cstdint>

namespace esopt {

// Philox-4x32 round multipliers and Weyl key increments (SC'11).
constexpr uint32_t kPhiloxMulA = 0xD2511F53u;
constexpr uint32_t kPhiloxMulB = 0xCD9E8D57u;
constexpr uint32_t kPhiloxWeylA = 0x9E3779B9u;
constexpr uint32_t kPhiloxWeylB = 0xBB67AE85u;

struct PhiloxKey {
  uint32_t k0, k1;
};

__host__ __device__ inline PhiloxKey philox_key(uint64_t seed) {
  return PhiloxKey{static_cast<uint32_t>(seed), static_cast<uint32_t>(seed >> 32)};
}

// Ten Philox-4x32 rounds on counter (j_lo, j_hi, 0, 0). Each round is two
// 32x32->64 multiplies (one IMAD.WIDE each) and two three-input XORs; the key
// schedule depends only on the seed, so it stays warp-uniform.
__device__ __forceinline__ uint4 philox_block(uint64_t j, PhiloxKey key) {
  uint32_t c0 = static_cast<uint32_t>(j);
  uint32_t c1 = static_cast<uint32_t>(j >> 32);
  uint32_t c2 = 0u, c3 = 0u;
  uint32_t k0 = key.k0, k1 = key.k1;
#pragma unroll
  for (int round = 0; round < 10; ++round) {
    const uint64_t pa = static_cast<uint64_t>(kPhiloxMulA) * c0;
    const uint64_t pb = static_cast<uint64_t>(kPhiloxMulB) * c2;
    const uint32_t n0 = static_cast<uint32_t>(pb >> 32) ^ c1 ^ k0;
    const uint32_t n2 = static_cast<uint32_t>(pa >> 32) ^ c3 ^ k1;
    c1 = static_cast<uint32_t>(pb);
    c3 = static_cast<uint32_t>(pa);
    c0 = n0;
    c2 = n2;
    k0 += kPhiloxWeylA;
    k1 += kPhiloxWeylB;
  }
  return make_uint4(c0, c1, c2, c3);
}

// u = (2m + 1) / 2^24 with m = x >> 9, computed exactly: the bit pattern
// 0x3F800000 | m is 1 + m 2^-23, and subtracting 1 - 2^-24 (0x3F7FFFFF) leaves
// (2m + 1) 2^-24, which has at most 24 significant bits.
__device__ __forceinline__ float uniform_open(uint32_t x) {
  return __uint_as_float(0x3F800000u | (x >> 9)) - __uint_as_float(0x3F7FFFFFu);
}

// Below this u the radius comes from the hardware log2; above it (u within
// 2^-10 of 1, where an absolute log2 error would be a large relative error of
// the small radius) from the series of ln(1 - t), t = 1 - u exact.
constexpr float kNearOne = 0.9990234375f;  // 1 - 2^-10
constexpr float kMinusTwoLn2 = -1.38629436111989061883f;
constexpr float kTwoPi = 6.28318530717958647692f;

__device__ __forceinline__ float sqrt_approx(float x) {
  float r;
  asm("sqrt.approx.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

// radius^2 = -2 ln u for u = uniform_open(x), fast path:
//   for u <= 1 - 2^-10: -2 ln 2 * log2(u) with the MUFU log2 (__log2f);
//   for u >  1 - 2^-10: 2t + t^2 + (2/3) t^3 with t = 1 - u (exact), whose
//     truncation error is below t^3/4 relative (an absolute log2 error there
//     would be a large relative error of the small radius).
// Both are evaluated and one is selected, which keeps the code free of
// divergent branches.
__device__ __forceinline__ float radius_sq(float u) {
  const float t = 1.0f - u;
  const float series = t * fmaf(t, fmaf(t, 2.0f / 3.0f, 1.0f), 2.0f);
  const float logged = __log2f(u) * kMinusTwoLn2;
  return u > kNearOne ? series : logged;
}

// One Box-Muller pair, fast path:
//   radius = sqrt.approx(radius_sq(u_a));
//   angle: 2 pi u_b = 2 pi s + pi with s = u_b - 1/2 formed exactly from the
//     bits, so cos/sin of 2 pi u_b are -cos/-sin of 2 pi s, an argument in
//     (-pi, pi) where __sincosf is accurate.
// The result is checked against the exact pair over the whole input domain
// (every 23-bit radius input and every 23-bit angle input) by the test suite;
// the error stays below 1e-5 * max(1, |eps|).
__device__ __forceinline__ float2 box_muller(uint32_t xa, uint32_t xb) {
  const float r = sqrt_approx(radius_sq(uniform_open(xa)));
  const float s = (__uint_as_float(0x3F800000u | (xb >> 9)) - 1.5f) + 0x1p-24f;
  float sn, cs;
  __sincosf(s * kTwoPi, &sn, &cs);
  return make_float2(-r * cs, -r * sn);
}

// eps[4j .. 4j+3] for one seed.
__device__ __forceinline__ float4 gaussian4(uint64_t j, PhiloxKey key) {
  const uint4 x = philox_block(j, key);
  const float2 p = box_muller(x.x, x.y);
  const float2 q = box_muller(x.z, x.w);
  return make_float4(p.x, p.y, q.x, q.y);
}

}  // namespace esopt
