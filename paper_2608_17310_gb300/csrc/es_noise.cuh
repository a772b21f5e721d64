// Counter-based Gaussian noise for the ES step, regenerated from the integer
// seed wherever it is needed (§3: only the seed of each perturbation is
// stored; App. D.6: the update rebuilds each member's direction from that
// seed alone).
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

// High and low words of the 32x32->64-bit product m * x. Two forms, with the
// same words: two 32-bit multiplies (mul.hi.u32, mul.lo.u32), or one multiply
// with a 64-bit result (mul.wide.u32). Measured on sm_103a in the library's
// kernels, the fastest mix is the 64-bit form in the eight full rounds of the
// per-tile path (philox_block_tile) and the 32-bit pair everywhere else (the
// first two rounds, the per-tile constants and the general path): 5-8 %
// faster than either form throughout, which cost registers and occupancy in
// the fused update.
__device__ __forceinline__ uint32_t mul_hi(uint32_t m, uint32_t x) { return __umulhi(m, x); }
__device__ __forceinline__ uint32_t mul_lo(uint32_t m, uint32_t x) { return m * x; }
__device__ __forceinline__ void mul_wide(uint32_t m, uint32_t x, uint32_t& hi, uint32_t& lo) {
  const uint64_t p = static_cast<uint64_t>(m) * x;
  hi = static_cast<uint32_t>(p >> 32);
  lo = static_cast<uint32_t>(p);
}

// Ten Philox-4x32 rounds on counter (j_lo, j_hi, 0, 0). Each round is two
// 32x32->64 products (high and low words) and two three-input XORs; the key
// schedule depends only on the seed, so it stays warp-uniform.
__device__ __forceinline__ uint4 philox_block(uint64_t j, PhiloxKey key) {
  uint32_t c0 = static_cast<uint32_t>(j);
  uint32_t c1 = static_cast<uint32_t>(j >> 32);
  uint32_t c2 = 0u, c3 = 0u;
  uint32_t k0 = key.k0, k1 = key.k1;
#pragma unroll
  for (int round = 0; round < 10; ++round) {
    const uint32_t n0 = mul_hi(kPhiloxMulB, c2) ^ c1 ^ k0;
    const uint32_t n2 = mul_hi(kPhiloxMulA, c0) ^ c3 ^ k1;
    c1 = mul_lo(kPhiloxMulB, c2);
    c3 = mul_lo(kPhiloxMulA, c0);
    c0 = n0;
    c2 = n2;
    k0 += kPhiloxWeylA;
    k1 += kPhiloxWeylB;
  }
  return make_uint4(c0, c1, c2, c3);
}

// The same ten rounds for the blocks of one tile that share the high counter
// word j_hi. With counter (j_lo, j_hi, 0, 0) the first round's second product
// is zero and its word 0 is j_hi ^ k0, so the second round's first product
// depends only on (key, j_hi): those parts are computed once per tile
// (philox_tile) instead of once per block, saving one multiply per block.
// Bit-identical to philox_block.
struct PhiloxTile {
  PhiloxKey key;
  uint32_t w0;     // word 0 after round 0: j_hi ^ k0
  uint32_t x2;     // high word of kPhiloxMulA * w0, xored with round 1's k1
  uint32_t lo2;    // low word of kPhiloxMulA * w0
};

__device__ __forceinline__ PhiloxTile philox_tile(uint32_t j_hi, PhiloxKey key) {
  const uint32_t w0 = j_hi ^ key.k0;
  return PhiloxTile{key, w0, mul_hi(kPhiloxMulA, w0) ^ (key.k1 + kPhiloxWeylB),
                    mul_lo(kPhiloxMulA, w0)};
}

__device__ __forceinline__ uint4 philox_block_tile(uint32_t j_lo, const PhiloxTile& t) {
  // round 0 (keys k0, k1): products kPhiloxMulA * j_lo and kPhiloxMulB * 0
  const uint32_t a2 = mul_hi(kPhiloxMulA, j_lo) ^ t.key.k1;   // word 2
  const uint32_t a3 = mul_lo(kPhiloxMulA, j_lo);              // word 3
  // round 1 (keys k0 + W_A, k1 + W_B): word 0 is t.w0, its product is per tile
  uint32_t c0 = mul_hi(kPhiloxMulB, a2) ^ (t.key.k0 + kPhiloxWeylA);  // word 1 was 0
  uint32_t c1 = mul_lo(kPhiloxMulB, a2);
  uint32_t c2 = t.x2 ^ a3;
  uint32_t c3 = t.lo2;
  uint32_t k0 = t.key.k0 + 2u * kPhiloxWeylA, k1 = t.key.k1 + 2u * kPhiloxWeylB;
#pragma unroll
  for (int round = 2; round < 10; ++round) {
    uint32_t ha, la, hb, lb;
    mul_wide(kPhiloxMulA, c0, ha, la);
    mul_wide(kPhiloxMulB, c2, hb, lb);
    const uint32_t n0 = hb ^ c1 ^ k0;
    const uint32_t n2 = ha ^ c3 ^ k1;
    c1 = lb;
    c3 = la;
    c0 = n0;
    c2 = n2;
    k0 += kPhiloxWeylA;
    k1 += kPhiloxWeylB;
  }
  return make_uint4(c0, c1, c2, c3);
}

// The key schedule of one seed, computed once on the host or per CTA:
// rk[2r] = k0 + r W_A and rk[2r + 1] = k1 + r W_B are the keys of round r
// (r = 0..9). A kernel that takes it reads every round key as an operand
// instead of deriving it, so the schedule costs no instruction per block.
struct PhiloxSched {
  uint32_t rk[20];
};

__host__ __device__ inline PhiloxSched philox_sched(uint64_t seed) {
  PhiloxSched s;
  uint32_t k0 = static_cast<uint32_t>(seed), k1 = static_cast<uint32_t>(seed >> 32);
  for (int r = 0; r < 10; ++r) {
    s.rk[2 * r] = k0;
    s.rk[2 * r + 1] = k1;
    k0 += kPhiloxWeylA;
    k1 += kPhiloxWeylB;
  }
  return s;
}

// Per-tile constants of philox_tile, from a schedule: word 0 after round 0
// is j_hi ^ k0, and round 1's product of it is shared by every block whose
// counter has high word j_hi.
struct TileConst {
  uint32_t x2;   // high word of kPhiloxMulA * (j_hi ^ k0), xored with round 1's k1
  uint32_t lo2;  // low word of kPhiloxMulA * (j_hi ^ k0)
};

__device__ __forceinline__ TileConst tile_const(uint32_t j_hi, uint32_t k0, uint32_t k1_round1) {
  const uint32_t w0 = j_hi ^ k0;
  return TileConst{mul_hi(kPhiloxMulA, w0) ^ k1_round1, mul_lo(kPhiloxMulA, w0)};
}

// philox_block_tile with the round keys taken from a schedule: `rk1` is round
// 0's k1, `rk2` round 1's k0, `rk` points at the keys of rounds 2..9 (rk[2r - 4],
// rk[2r - 3] for round r). kWideFirst: the first two rounds' products also as
// one 64-bit-result multiply each (a high/low pair costs the integer pipe more
// cycles, but one more instruction issue less; which is faster depends on the
// kernel). Bit-identical to philox_block.
template <bool kWideFirst, class Keys>
__device__ __forceinline__ uint4 philox_block_rk(uint32_t j_lo, TileConst t, uint32_t rk1,
                                                 uint32_t rk2, const Keys& rk);

// Round 0's product kPhiloxMulA * j_lo as (high, low) words. It depends on
// the counter alone, not on the key: every seed's block j shares it.
struct Round0 {
  uint32_t hi, lo;
};

template <bool kWide>
__device__ __forceinline__ Round0 philox_round0(uint32_t j_lo) {
  Round0 p;
  if constexpr (kWide) {
    mul_wide(kPhiloxMulA, j_lo, p.hi, p.lo);
  } else {
    p.hi = mul_hi(kPhiloxMulA, j_lo);
    p.lo = mul_lo(kPhiloxMulA, j_lo);
  }
  return p;
}

// The product of round 0 for counter word j_lo + d, from the one for j_lo:
// the 64-bit product grows by kPhiloxMulA * d. Exact while j_lo + d stays
// below 2^32 (the caller's blocks share their high counter word).
__device__ __forceinline__ Round0 round0_step(Round0 p, uint32_t d) {
  const uint64_t q = ((static_cast<uint64_t>(p.hi) << 32) | p.lo) +
                     static_cast<uint64_t>(kPhiloxMulA) * d;
  return Round0{static_cast<uint32_t>(q >> 32), static_cast<uint32_t>(q)};
}

// philox_block_rk from round 0's product (philox_round0 of the block's j_lo).
template <bool kWideFirst, class Keys>
__device__ __forceinline__ uint4 philox_block_r0(Round0 p0, TileConst t, uint32_t rk1,
                                                 uint32_t rk2, const Keys& rk) {
  const uint32_t a2 = p0.hi ^ rk1;  // round 0: word 2 (its word 3 is p0.lo)
  const uint32_t a3 = p0.lo;
  uint32_t c0, c1;
  if constexpr (kWideFirst) {
    uint32_t h1;
    mul_wide(kPhiloxMulB, a2, h1, c1);  // round 1 (its word 1 was 0)
    c0 = h1 ^ rk2;
  } else {
    c0 = mul_hi(kPhiloxMulB, a2) ^ rk2;  // round 1 (its word 1 was 0)
    c1 = mul_lo(kPhiloxMulB, a2);
  }
  uint32_t c2 = t.x2 ^ a3;
  uint32_t c3 = t.lo2;
#pragma unroll
  for (int round = 2; round < 10; ++round) {
    uint32_t ha, la, hb, lb;
    mul_wide(kPhiloxMulA, c0, ha, la);
    mul_wide(kPhiloxMulB, c2, hb, lb);
    const uint32_t n0 = hb ^ c1 ^ rk[2 * round - 4];
    const uint32_t n2 = ha ^ c3 ^ rk[2 * round - 3];
    c1 = lb;
    c3 = la;
    c0 = n0;
    c2 = n2;
  }
  return make_uint4(c0, c1, c2, c3);
}

template <bool kWideFirst, class Keys>
__device__ __forceinline__ uint4 philox_block_rk(uint32_t j_lo, TileConst t, uint32_t rk1,
                                                 uint32_t rk2, const Keys& rk) {
  return philox_block_r0<kWideFirst>(philox_round0<kWideFirst>(j_lo), t, rk1, rk2, rk);
}

// The float 1 + m 2^-23 for m = x >> 9 (the top 23 bits of x).
__device__ __forceinline__ float one_plus_top23(uint32_t x) {
  return __uint_as_float(0x3F800000u | (x >> 9));
}

// u = (2m + 1) / 2^24 with m = x >> 9, computed exactly: 1 + m 2^-23 minus
// 1 - 2^-24 (0x3F7FFFFF) leaves (2m + 1) 2^-24, which has at most 24
// significant bits.
__device__ __forceinline__ float uniform_open(uint32_t x) {
  return one_plus_top23(x) - __uint_as_float(0x3F7FFFFFu);
}

// Below this u the radius comes from the hardware log2; above it (u within
// 2^-10 of 1, where an absolute log2 error would be a large relative error of
// the small radius) from the series of -ln(1 - t), t = 1 - u exact.
constexpr float kNearOne = 0.9990234375f;  // 1 - 2^-10
constexpr float kMinusTwoLn2 = -1.38629436111989061883f;
constexpr float kTwoPi = 6.28318530717958647692f;
// -3 pi + 2 pi 2^-24 rounded to float: 2 pi (f - 3/2 + 2^-24) = fma(f, 2 pi, this)
constexpr float kAngleOffset = -9.42477798f;

// The hardware approximations of log2, sqrt, sin and cos, in their
// flush-to-zero forms. These differ from the default forms only for subnormal
// inputs (which the default forms first scale into the normal range at the cost
// of extra instructions), and no input here is subnormal: u >= 2^-24, the
// radius squared is at least 2t + t^2 with t >= 2^-24 or at least
// 2 ln 2 * 2^-10 from the log path, and the angle is at least 2 pi 2^-24 in
// magnitude. Measured: the generator's kernels run 6-10 % faster.
__device__ __forceinline__ float sqrt_approx(float x) {
  float r;
  asm("sqrt.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

__device__ __forceinline__ float log2_approx(float x) {
  float r;
  asm("lg2.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

__device__ __forceinline__ void sincos_approx(float a, float* s, float* c) {
  asm("sin.approx.ftz.f32 %0, %1;" : "=f"(*s) : "f"(a));
  asm("cos.approx.ftz.f32 %0, %1;" : "=f"(*c) : "f"(a));
}

// radius^2 = -2 ln u for u = uniform_open(x), fast path:
//   for u <= 1 - 2^-10: -2 ln 2 * log2(u) with the MUFU log2 (radius_sq_log);
//   for u >  1 - 2^-10: 2t + t^2 with t = 1 - u (exact); the dropped terms
//     (2/3 t^3 + ...) are below t^2/3 <= 3.2e-7 relative (radius_sq_series).
// radius_sq evaluates both and selects one, which keeps the code free of
// divergent branches. Since u = (2m + 1) 2^-24 with m = x >> 9, u > 1 - 2^-10
// exactly when m >= 2^23 - 2^13, i.e. when the raw word x >= kNearOneWord; the
// streaming kernels test that instead and compute the series only on a rare
// branch (one radius input in 1024), with the same values.
constexpr uint32_t kNearOneWord = 0xFFC00000u;

__device__ __forceinline__ float radius_sq_log(float u) { return log2_approx(u) * kMinusTwoLn2; }

__device__ __forceinline__ float radius_sq_series(float u) {
  const float t = 1.0f - u;
  return fmaf(t, t, t + t);
}

__device__ __forceinline__ float radius_sq(float u) {
  const float series = radius_sq_series(u);
  const float logged = radius_sq_log(u);
  return u > kNearOne ? series : logged;
}

// Polar form of one Box-Muller pair: eps_even = -r * c, eps_odd = -r * s.
//   r = sqrt.approx(radius_sq(u_a));
//   angle: with f = 1 + m_b 2^-23 (bits 0x3F800000 | m_b), 2 pi u_b =
//     2 pi (f - 3/2 + 2^-24) + pi, so cos/sin of 2 pi u_b are -c/-s with
//     (s, c) = sincos_approx(fma(f, 2 pi, kAngleOffset)), an argument in
//     (-pi, pi) where the hardware sine and cosine are accurate; the fma
//     rounds once (|error| < 1e-6).
// Kernels that add scale * eps fold the scale into r: theta + scale * eps_even
// = fma(-(scale * r), c, theta).
// Checked against the exact pair over the whole input domain (every 23-bit
// radius input and every 23-bit angle input) by the test suite; the error
// stays below 1e-5 * max(1, |eps|).
struct Polar {
  float r, c, s;
};

// The pair before the square root: .r holds radius^2, from radius_sq (kLogOnly
// false) or from the hardware log2 alone (kLogOnly true; the caller then
// replaces the near-one inputs' radius^2 by radius_sq_series).
template <bool kLogOnly>
__device__ __forceinline__ Polar polar_sq(uint32_t xa, uint32_t xb) {
  Polar p;
  const float u = uniform_open(xa);
  p.r = kLogOnly ? radius_sq_log(u) : radius_sq(u);
  const float f = one_plus_top23(xb);
  sincos_approx(fmaf(f, kTwoPi, kAngleOffset), &p.s, &p.c);
  return p;
}

__device__ __forceinline__ Polar polar(uint32_t xa, uint32_t xb) {
  Polar p = polar_sq<false>(xa, xb);
  p.r = sqrt_approx(p.r);
  return p;
}

// Both pairs of one Philox block at once: .x is the pair (x0, x1), .y the pair
// (x2, x3). The same operations as polar(), issued as packed two-wide FP32
// instructions (each half rounds exactly like the scalar instruction, so the
// values are bit-identical to two polar() calls); the MUFU work stays scalar.
// Halving the FP32 instruction count keeps more of the FMA pipe free for the
// generator's integer multiplies.
struct Polar2 {
  float2 r, c, s;
};

// Both pairs before their square roots (.r holds radius^2), as polar_sq.
template <bool kLogOnly>
__device__ __forceinline__ Polar2 polar2_sq(const uint4& x) {
  Polar2 p;
  const float2 fa = make_float2(one_plus_top23(x.x), one_plus_top23(x.z));
  const float kHalfUlpBelowOne = __uint_as_float(0x3F7FFFFFu);
  const float2 u = __fadd2_rn(fa, make_float2(-kHalfUlpBelowOne, -kHalfUlpBelowOne));
  const float2 logged =
      __fmul2_rn(make_float2(log2_approx(u.x), log2_approx(u.y)),
                 make_float2(kMinusTwoLn2, kMinusTwoLn2));
  if constexpr (kLogOnly) {
    p.r = logged;
  } else {
    const float2 t = __fadd2_rn(make_float2(1.0f, 1.0f), make_float2(-u.x, -u.y));
    const float2 series = __ffma2_rn(t, t, __fadd2_rn(t, t));
    p.r.x = u.x > kNearOne ? series.x : logged.x;
    p.r.y = u.y > kNearOne ? series.y : logged.y;
  }
  const float2 fb = make_float2(one_plus_top23(x.y), one_plus_top23(x.w));
  const float2 ang = __ffma2_rn(fb, make_float2(kTwoPi, kTwoPi),
                                make_float2(kAngleOffset, kAngleOffset));
  sincos_approx(ang.x, &p.s.x, &p.c.x);
  sincos_approx(ang.y, &p.s.y, &p.c.y);
  return p;
}

__device__ __forceinline__ Polar2 polar2(const uint4& x) {
  Polar2 p = polar2_sq<false>(x);
  p.r = make_float2(sqrt_approx(p.r.x), sqrt_approx(p.r.y));
  return p;
}

// Radius^2 of every pair of NB Philox blocks (p[b].r, from the hardware log2)
// corrected where the radius input lies within 2^-10 of 1: such a pair takes
// the series instead. The test is on the raw words (xa[b] = the blocks' words
// x0 and x2), and the series is computed only when some pair needs it (one
// radius input in 1024), so the common path costs one compare per pair. The
// values equal radius_sq's.
template <int NB>
__device__ __forceinline__ void fix_near_one(const uint2 (&xa)[NB], Polar2 (&p)[NB]) {
  bool near = false;
#pragma unroll
  for (int b = 0; b < NB; ++b) near |= (xa[b].x >= kNearOneWord) | (xa[b].y >= kNearOneWord);
  if (__builtin_expect(near, 0)) {
#pragma unroll
    for (int b = 0; b < NB; ++b) {
      if (xa[b].x >= kNearOneWord) p[b].r.x = radius_sq_series(uniform_open(xa[b].x));
      if (xa[b].y >= kNearOneWord) p[b].r.y = radius_sq_series(uniform_open(xa[b].y));
    }
  }
}

// One Box-Muller pair, materialised.
__device__ __forceinline__ float2 box_muller(uint32_t xa, uint32_t xb) {
  const Polar p = polar(xa, xb);
  return make_float2(-p.r * p.c, -p.r * p.s);
}

// eps[4j .. 4j+3] for one seed, materialised.
__device__ __forceinline__ float4 gaussian4(uint64_t j, PhiloxKey key) {
  const uint4 x = philox_block_tile(static_cast<uint32_t>(j),
                                    philox_tile(static_cast<uint32_t>(j >> 32), key));
  const float2 p = box_muller(x.x, x.y);
  const float2 q = box_muller(x.z, x.w);
  return make_float4(p.x, p.y, q.x, q.y);
}

}  // namespace esopt
