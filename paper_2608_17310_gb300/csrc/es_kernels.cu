// sm_103a kernels of the ES step: in-place perturb/restore (theta += s eps) and
// the fused N-seed update (theta += sum_i c_i eps_i), plus a noise fill.
//
// All three stream the parameter set once per launch. Work is cut into tiles
// of kBlockThreads threads x kVecsPerThread 16-byte vectors that never
// straddle a segment; persistent CTAs walk the tiles in grid-stride
// order, so consecutive CTAs touch consecutive memory and each CTA advances
// through the segment table monotonically (one table lookup per tile, no
// per-element search).
// Every element is owned by exactly one thread: no atomics, no shared state
// between threads except the staged seeds of the update.
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_fp8.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "es_internal.h"
#include "es_noise.cuh"

namespace esopt {
namespace {

// 16-byte vector <-> fp32 registers, and single-element access for tails.
struct Bf16Io {
  static constexpr int kVec = 8;
  static constexpr bool kScaled = false;
  using Scalar = uint16_t;
  __device__ static uint32_t pack2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);  // one cvt.rn.bf16x2.f32
    return *reinterpret_cast<uint32_t*>(&h);
  }
  __device__ static float lo(uint32_t w) { return __uint_as_float(w << 16); }
  __device__ static float hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
  __device__ static void unpack(const uint4& v, float (&f)[8]) {
    f[0] = lo(v.x); f[1] = hi(v.x);
    f[2] = lo(v.y); f[3] = hi(v.y);
    f[4] = lo(v.z); f[5] = hi(v.z);
    f[6] = lo(v.w); f[7] = hi(v.w);
  }
  __device__ static uint4 pack(const float (&f)[8]) {
    return make_uint4(pack2(f[0], f[1]), pack2(f[2], f[3]), pack2(f[4], f[5]), pack2(f[6], f[7]));
  }
  // f <- value of round_to_storage(f), element-wise (one rounding to bf16).
  template <int M>
  __device__ static void round_trip(float (&f)[M]) {
#pragma unroll
    for (int k = 0; k < M; k += 2) {
      const uint32_t w = pack2(f[k], f[k + 1]);
      f[k] = lo(w);
      f[k + 1] = hi(w);
    }
  }
  // The first `rem` (< 8) elements at base[e], the rest zero, as one vector.
  __device__ static uint4 load_partial(const uint16_t* base, uint64_t e, int rem) {
    uint32_t w[4] = {0u, 0u, 0u, 0u};
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (k < rem) w[k >> 1] |= static_cast<uint32_t>(base[e + k]) << (16 * (k & 1));
    return make_uint4(w[0], w[1], w[2], w[3]);
  }
  __device__ static void store_partial(uint16_t* base, uint64_t e, int rem, const uint4& v) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int k = 0; k < 8; ++k)
      if (k < rem) base[e + k] = static_cast<uint16_t>(w[k >> 1] >> (16 * (k & 1)));
  }
};

struct F32Io {
  static constexpr int kVec = 4;
  static constexpr bool kScaled = false;
  using Scalar = float;
  __device__ static void unpack(const uint4& v, float (&f)[4]) {
    f[0] = __uint_as_float(v.x); f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z); f[3] = __uint_as_float(v.w);
  }
  __device__ static uint4 pack(const float (&f)[4]) {
    return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]),
                      __float_as_uint(f[2]), __float_as_uint(f[3]));
  }
  template <int M>
  __device__ static void round_trip(float (&)[M]) {}
  __device__ static uint4 load_partial(const float* base, uint64_t e, int rem) {
    uint32_t w[4] = {0u, 0u, 0u, 0u};
#pragma unroll
    for (int k = 0; k < 4; ++k)
      if (k < rem) w[k] = __float_as_uint(base[e + k]);
    return make_uint4(w[0], w[1], w[2], w[3]);
  }
  __device__ static void store_partial(float* base, uint64_t e, int rem, const uint4& v) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int k = 0; k < 4; ++k)
      if (k < rem) base[e + k] = __uint_as_float(w[k]);
  }
};

// FP8 E4M3 storage: 16 elements per 16-byte vector, byte k of the vector is
// element k. Values stay in units of the segment's scale: the kernels multiply
// the noise by 1 / scale instead (kScaled). Decoding goes through half
// precision, which holds every E4M3 value exactly; encoding rounds fp32 to the
// nearest E4M3 value, ties to even, saturating at +-448 (cvt .satfinite).
struct Fp8Io {
  static constexpr int kVec = 16;
  static constexpr bool kScaled = true;
  using Scalar = uint8_t;
  __device__ static float2 dec2(uint32_t pair) {
    const __half2_raw h =
        __nv_cvt_fp8x2_to_halfraw2(static_cast<__nv_fp8x2_storage_t>(pair & 0xFFFFu), __NV_E4M3);
    return __half22float2(__half2(h));
  }
  __device__ static uint32_t enc2(float lo, float hi) {
    return static_cast<uint32_t>(__nv_cvt_float2_to_fp8x2(make_float2(lo, hi), __NV_SATFINITE,
                                                          __NV_E4M3));
  }
  __device__ static void unpack(const uint4& v, float (&f)[16]) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const float2 a = dec2(w[k]), b = dec2(w[k] >> 16);
      f[4 * k + 0] = a.x; f[4 * k + 1] = a.y; f[4 * k + 2] = b.x; f[4 * k + 3] = b.y;
    }
  }
  __device__ static uint4 pack(const float (&f)[16]) {
    uint32_t w[4];
#pragma unroll
    for (int k = 0; k < 4; ++k)
      w[k] = enc2(f[4 * k + 0], f[4 * k + 1]) | (enc2(f[4 * k + 2], f[4 * k + 3]) << 16);
    return make_uint4(w[0], w[1], w[2], w[3]);
  }
  template <int M>
  __device__ static void round_trip(float (&f)[M]) {
#pragma unroll
    for (int k = 0; k < M; k += 2) {
      const float2 r = dec2(enc2(f[k], f[k + 1]));
      f[k] = r.x;
      f[k + 1] = r.y;
    }
  }
  // The first `rem` (< 16) elements at base[e], the rest zero, as one vector.
  __device__ static uint4 load_partial(const uint8_t* base, uint64_t e, int rem) {
    uint32_t w[4] = {0u, 0u, 0u, 0u};
#pragma unroll
    for (int k = 0; k < 16; ++k)
      if (k < rem) w[k >> 2] |= static_cast<uint32_t>(base[e + k]) << (8 * (k & 3));
    return make_uint4(w[0], w[1], w[2], w[3]);
  }
  __device__ static void store_partial(uint8_t* base, uint64_t e, int rem, const uint4& v) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int k = 0; k < 16; ++k)
      if (k < rem) base[e + k] = static_cast<uint8_t>(w[k >> 2] >> (8 * (k & 3)));
  }
};

// Vectors a thread processes at once for a kernel kind's group g (g bf16
// vectors of 8 elements): the same number of elements, hence of Philox
// chains, for every storage type, within the kVecsPerThread vectors of a tile.
template <class Io>
__host__ __device__ constexpr int group_for(int g) {
  return Io::kVec > 8 ? (g > 1 ? g / 2 : 1) : Io::kVec < 8 ? (2 * g < kVecsPerThread ? 2 * g : kVecsPerThread) : g;
}

// theta + acc in storage units: acc is in parameter units, so a scaled
// segment takes acc / scale (one fused multiply-add with 1 / scale).
template <class Io>
__device__ __forceinline__ float add_acc(float theta, float acc, float inv_scale) {
  if constexpr (Io::kScaled) return fmaf(acc, inv_scale, theta);
  else return theta + acc;
}

// Philox words of block j for one seed. SchedGen serves the blocks of a tile
// that share the high counter word, with the round keys read from a
// precomputed schedule (kernel parameters or registers loaded from shared
// memory) and the tile's constants computed once; AnyGen serves any block. Both
// give the same words.
template <class Keys, bool kWideFirst = false>
struct SchedGen {
  TileConst t;
  uint32_t rk1, rk2;  // round 0's k1, round 1's k0
  Keys rk;            // rounds 2..9: rk[2r - 4], rk[2r - 3]
  __device__ uint4 block(uint64_t j) const {
    return philox_block_rk<kWideFirst>(static_cast<uint32_t>(j), t, rk1, rk2, rk);
  }
  // The same words from round 0's product (philox_round0 of the block's j_lo).
  __device__ uint4 block_r0(Round0 p0) const {
    return philox_block_r0<kWideFirst>(p0, t, rk1, rk2, rk);
  }
};
struct AnyGen {
  PhiloxKey key;
  __device__ uint4 block(uint64_t j) const { return philox_block(j, key); }
};

// Generator of one seed whose schedule is a kernel parameter.
template <bool kUniformHi, bool kWideFirst = false>
__device__ __forceinline__ auto sched_gen(const PhiloxSched& s, uint32_t j_hi) {
  if constexpr (kUniformHi)
    return SchedGen<const uint32_t*, kWideFirst>{tile_const(j_hi, s.rk[0], s.rk[3]), s.rk[1],
                                                 s.rk[2], s.rk + 4};
  else return AnyGen{PhiloxKey{s.rk[0], s.rk[1]}};
}

// How each Philox block becomes theta updates. The forms give bit-identical
// values: a packed two-wide FP32 instruction rounds each half exactly like the
// scalar one. They differ only in instruction mix, which moves work between the
// FMA pipe's halves. Each kernel uses the form measured fastest for it:
//   kScalar     scalar transform (polar) and scalar FMAs;
//   kPackedFma  scalar transform, packed FMAs into theta or the accumulator;
//   kPacked     packed transform (polar2) and packed FMAs.
enum class NoiseForm { kScalar, kPackedFma, kPacked };
constexpr NoiseForm kAxpy1Form = static_cast<NoiseForm>(ES_AXPY1_FORM);
constexpr NoiseForm kAxpy2Form = static_cast<NoiseForm>(ES_AXPY2_FORM);
constexpr NoiseForm kUpdateForm = static_cast<NoiseForm>(ES_UPDATE_FORM);
constexpr bool kUpdatePipelined = ES_UPDATE_PIPELINED != 0;
constexpr bool kUpdatePingPong = ES_UPDATE_PIPELINED >= 2;
constexpr int kRound0 = ES_ROUND0;
constexpr bool kFlipPacked = ES_FLIP_PACKED != 0;
// Near-one radius inputs: a rare branch (true) or a select per pair (false).
constexpr bool kNearOneBranch = ES_NEAR_ONE_BRANCH != 0;

// The radius of every pair, from its radius^2.
template <int NB>
__device__ __forceinline__ void polar_roots(Polar2 (&p)[NB]) {
#pragma unroll
  for (int b = 0; b < NB; ++b) p[b].r = make_float2(sqrt_approx(p[b].r.x), sqrt_approx(p[b].r.y));
}

// The pairs of NB Philox blocks in polar form (r, cos, sin) from their words.
template <NoiseForm kForm, int NB>
__device__ __forceinline__ void polar_from_words(const uint4 (&x)[NB], Polar2 (&p)[NB]) {
  constexpr bool kLogOnly = kNearOneBranch;
  uint2 xa[NB];
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    xa[b] = make_uint2(x[b].x, x[b].z);
    if constexpr (kForm == NoiseForm::kPacked) {
      p[b] = polar2_sq<kLogOnly>(x[b]);
    } else {
      const Polar a = polar_sq<kLogOnly>(x[b].x, x[b].y), c = polar_sq<kLogOnly>(x[b].z, x[b].w);
      p[b] = Polar2{make_float2(a.r, c.r), make_float2(a.c, c.c), make_float2(a.s, c.s)};
    }
  }
  if constexpr (kLogOnly) fix_near_one<NB>(xa, p);
  polar_roots<NB>(p);
}

// Words of Philox blocks j0 .. j0 + NB - 1.
template <int NB, class Gen>
__device__ __forceinline__ void philox_words(const Gen& gen, uint64_t j0, uint4 (&x)[NB]) {
#pragma unroll
  for (int b = 0; b < NB; ++b) x[b] = gen.block(j0 + b);
}

template <NoiseForm kForm, int NB, class Gen>
__device__ __forceinline__ void polar_blocks(const Gen& gen, uint64_t j0, Polar2 (&p)[NB]) {
  uint4 x[NB];
  philox_words<NB>(gen, j0, x);
  polar_from_words<kForm, NB>(x, p);
}

// f[k] += scale * eps[4 j0 + k] for the V elements of blocks whose polar
// forms are pp[0 .. V / 4), with scale folded into each pair's radius.
template <NoiseForm kForm, int V>
__device__ __forceinline__ void apply_noise(const Polar2* pp, float scale, float (&f)[V]) {
  constexpr int NB = V / 4;
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    const Polar2& p = pp[b];
    if constexpr (kForm == NoiseForm::kScalar) {
      const float sp = -(scale * p.r.x), sq = -(scale * p.r.y);
      f[4 * b + 0] = fmaf(sp, p.c.x, f[4 * b + 0]);
      f[4 * b + 1] = fmaf(sp, p.s.x, f[4 * b + 1]);
      f[4 * b + 2] = fmaf(sq, p.c.y, f[4 * b + 2]);
      f[4 * b + 3] = fmaf(sq, p.s.y, f[4 * b + 3]);
    } else {
      const float2 sr = __fmul2_rn(make_float2(-scale, -scale), p.r);   // -(scale * r)
      const float2 lo = __ffma2_rn(make_float2(sr.x, sr.x), make_float2(p.c.x, p.s.x),
                                   make_float2(f[4 * b + 0], f[4 * b + 1]));
      const float2 hi = __ffma2_rn(make_float2(sr.y, sr.y), make_float2(p.c.y, p.s.y),
                                   make_float2(f[4 * b + 2], f[4 * b + 3]));
      f[4 * b + 0] = lo.x;
      f[4 * b + 1] = lo.y;
      f[4 * b + 2] = hi.x;
      f[4 * b + 3] = hi.y;
    }
  }
}

// f[k] += scale * eps[4 j0 + k] for the V elements of Philox blocks j0,
// j0 + 1, ..., with scale folded into each pair's radius.
template <NoiseForm kForm, int V, class Gen>
__device__ __forceinline__ void add_scaled_noise(const Gen& gen, uint64_t j0, float scale,
                                                 float (&f)[V]) {
  Polar2 pp[V / 4];
  polar_blocks<kForm, V / 4>(gen, j0, pp);
  apply_noise<kForm, V>(pp, scale, f);
}

// f[k] += scale * eps for the V elements of the Philox blocks whose words
// are x.
template <NoiseForm kForm, int V>
__device__ __forceinline__ void add_scaled_noise_words(const uint4 (&x)[V / 4], float scale,
                                                       float (&f)[V]) {
  Polar2 pp[V / 4];
  polar_from_words<kForm, V / 4>(x, pp);
  apply_noise<kForm, V>(pp, scale, f);
}

// f <- round(round(f + s1 * eps) + s2 * eps) for one seed's noise, computed
// once: an antithetic restore (+eps out) followed by the perturb (-eps in).
template <class Io, int V, class Gen>
__device__ __forceinline__ void add_scaled_noise_twice(const Gen& gen, uint64_t j0, float s1,
                                                       float s2, float (&f)[V]) {
  constexpr int NB = V / 4;
  Polar2 pp[NB];
  polar_blocks<NoiseForm::kScalar, NB>(gen, j0, pp);
#pragma unroll
  for (int b = 0; b < NB; ++b) {
    const Polar2& p = pp[b];
    float h[4];
    h[0] = fmaf(-(s1 * p.r.x), p.c.x, f[4 * b + 0]);
    h[1] = fmaf(-(s1 * p.r.x), p.s.x, f[4 * b + 1]);
    h[2] = fmaf(-(s1 * p.r.y), p.c.y, f[4 * b + 2]);
    h[3] = fmaf(-(s1 * p.r.y), p.s.y, f[4 * b + 3]);
    Io::round_trip(h);
    f[4 * b + 0] = fmaf(-(s2 * p.r.x), p.c.x, h[0]);
    f[4 * b + 1] = fmaf(-(s2 * p.r.x), p.s.x, h[1]);
    f[4 * b + 2] = fmaf(-(s2 * p.r.y), p.c.y, h[2]);
    f[4 * b + 3] = fmaf(-(s2 * p.r.y), p.s.y, h[3]);
  }
}

// Segment of `tile`; `seg` is the CTA's cursor and only moves forward.
__device__ __forceinline__ const SegDesc* find_segment(const SegDesc* __restrict__ segs,
                                                       int& seg, uint64_t tile) {
  while (tile >= segs[seg + 1].tile_begin) ++seg;
  return segs + seg;
}

// Whether every global index of the tile's elements [t0, t0 + tile) (clipped
// to the segment) shares the high word of its Philox block counter, i.e. the
// tile does not cross a multiple of 2^34 in index space.
__device__ __forceinline__ bool uniform_hi(uint64_t index_base, uint64_t t0, uint64_t tile,
                                           uint64_t numel) {
  const uint64_t last = index_base + (t0 + tile < numel ? t0 + tile : numel) - 1;
  return ((index_base + t0) >> 34) == (last >> 34);
}

// Location of one tile: its segment's storage, the tile's first element and,
// for a scaled storage type, 1 / the segment's scale.
template <class Io>
struct TileRef {
  typename Io::Scalar* base;
  uint64_t numel;
  uint64_t index_base;
  uint64_t t0;
  float inv;
};

template <class Io>
__device__ __forceinline__ TileRef<Io> tile_ref(const SegDesc* __restrict__ segs,
                                                const float* __restrict__ inv_scale, int& seg,
                                                uint64_t tile) {
  constexpr uint64_t kTile = static_cast<uint64_t>(kBlockThreads) * kVecsPerThread * Io::kVec;
  const SegDesc* d = find_segment(segs, seg, tile);
  return TileRef<Io>{static_cast<typename Io::Scalar*>(d->data), d->numel, d->index_base,
                     (tile - d->tile_begin) * kTile, Io::kScaled ? inv_scale[seg] : 1.0f};
}

// First element of the calling thread's vector u of a tile. Vector u of a
// tile is 256 consecutive 16-byte vectors, one per thread: each load and
// store instruction of a warp covers 512 contiguous bytes.
template <class Io>
__device__ __forceinline__ uint64_t vec_elem(const TileRef<Io>& r, int u) {
  return r.t0 + static_cast<uint64_t>(u * kBlockThreads + threadIdx.x) * Io::kVec;
}

// Vectors u0 .. u0 + G - 1 of the calling thread: a 16-byte load each; the
// ragged end of a segment element by element, zeros past it.
template <class Io, int G>
__device__ __forceinline__ void load_group(const TileRef<Io>& r, int u0, uint4 (&v)[G]) {
#pragma unroll
  for (int q = 0; q < G; ++q) {
    const uint64_t e = vec_elem(r, u0 + q);
    v[q] = make_uint4(0u, 0u, 0u, 0u);
    if (e + Io::kVec <= r.numel)
      v[q] = *reinterpret_cast<const uint4*>(r.base + e);
    else if (e < r.numel)
      v[q] = Io::load_partial(r.base, e, static_cast<int>(r.numel - e));
  }
}

template <class Io>
__device__ __forceinline__ void store_vec(const TileRef<Io>& r, uint64_t e, const uint4& v) {
  if (e + Io::kVec <= r.numel)
    *reinterpret_cast<uint4*>(r.base + e) = v;
  else if (e < r.numel)
    Io::store_partial(r.base, e, static_cast<int>(r.numel - e), v);
}

// Arguments of a perturb/restore launch: the schedule and scale of each step
// (step 2 only with kTwo). A __grid_constant__ parameter, so every round key
// is read from the constant bank as an instruction operand.
struct AxpyArgs {
  PhiloxSched s1, s2;
  float scale1, scale2;
};

// One tile of the perturb/restore pass (kTwo: fused restore + perturb; kSame:
// both steps use one seed, whose noise is generated once), G vectors at a
// time. The loads of the next group (at the last group: the first group of
// the CTA's next tile, `next`) are issued before the current group is
// computed, so the memory latency hides behind the generator's work. kFull:
// the whole tile lies inside its segment (every tile but a segment's last),
// so its vectors are addressed from one per-thread pointer and block index
// without bounds checks.
template <class Io, bool kTwo, bool kSame, bool kUniformHi, bool kFull, int G>
__device__ __forceinline__ void axpy_tile(const TileRef<Io>& cur, uint4 (&v)[G],
                                          const AxpyArgs& a, const SegDesc* __restrict__ segs,
                                          const float* __restrict__ inv_scale, int& seg,
                                          uint64_t next, bool has_next, TileRef<Io>& nxt) {
  constexpr int V = Io::kVec;
  constexpr NoiseForm kAxpyForm = kTwo ? kAxpy2Form : kAxpy1Form;
  constexpr int kGroups = kVecsPerThread / G;
  constexpr int kStride = kBlockThreads * V;  // elements from one vector of a thread to the next
  const uint32_t j_hi = static_cast<uint32_t>((cur.index_base + cur.t0) >> 34);
  // the one-seed pass is fastest with every Philox product 64-bit wide (in
  // FP8 storage, with twice the blocks per vector, that spills)
  constexpr bool kWide1 = !kTwo && V <= 8;
  const auto gen = sched_gen<kUniformHi, kWide1>(a.s1, j_hi);
  const auto gen2 = sched_gen<kUniformHi && kTwo && !kSame>(a.s2, j_hi);
  const float s1 = a.scale1 * cur.inv, s2 = a.scale2 * cur.inv;
  // the thread's first element of the tile, and its Philox block (index_base
  // is a multiple of 8 and t0 of the tile size, so the division is exact)
  typename Io::Scalar* const p = cur.base + cur.t0 + threadIdx.x * V;
  const uint64_t j_thread = ((cur.index_base + cur.t0) >> 2) + threadIdx.x * (V / 4);
  // Round 0's product from the counter alone (kRound0): once per block for
  // both seeds of the fused pass, and in a tile inside its segment stepped
  // from the thread's first block (its blocks share the high counter word,
  // so j_lo + d never wraps).
  constexpr int NB = V / 4;
  constexpr bool kR0 = kUniformHi && (kSame ? kFlipPacked && kFull && kRound0 >= 2
                                            : (kRound0 >= 2 ? (kFull || kTwo)
                                                            : kRound0 >= 1 && kTwo));
  constexpr bool kR0Step = kR0 && kFull && kRound0 >= 2;
  Round0 p0_thread{0u, 0u};
  if constexpr (kR0Step) p0_thread = philox_round0<kWide1>(static_cast<uint32_t>(j_thread));
#pragma unroll
  for (int grp = 0; grp < kGroups; ++grp) {
    uint4 nv[G];
    if (grp + 1 < kGroups) {
      if constexpr (kFull) {
#pragma unroll
        for (int q = 0; q < G; ++q)
          nv[q] = *reinterpret_cast<const uint4*>(p + ((grp + 1) * G + q) * kStride);
      } else {
        load_group<Io, G>(cur, (grp + 1) * G, nv);
      }
    } else if (has_next) {
      nxt = tile_ref<Io>(segs, inv_scale, seg, next);
      load_group<Io, G>(nxt, 0, nv);
    }
#pragma unroll
    for (int q = 0; q < G; ++q) {
      const int u = grp * G + q;
      if constexpr (!kFull) {
        if (vec_elem(cur, u) >= cur.numel) continue;
      }
      const uint64_t j0 = j_thread + static_cast<uint64_t>(u) * (kStride / 4);
      float f[V];
      Io::unpack(v[q], f);
      if constexpr (kSame && kFlipPacked) {
        // one seed's noise for both steps, in the packed form
        uint4 x[NB];
        if constexpr (kR0) {
#pragma unroll
          for (int b = 0; b < NB; ++b)
            x[b] = gen.block_r0(
                round0_step(p0_thread, static_cast<uint32_t>(u * (kStride / 4) + b)));
        } else {
          philox_words<NB>(gen, j0, x);
        }
        Polar2 pp[NB];
        polar_from_words<kAxpyForm, NB>(x, pp);
        apply_noise<kAxpyForm, V>(pp, s1, f);
        Io::round_trip(f);
        apply_noise<kAxpyForm, V>(pp, s2, f);
      } else if constexpr (kSame) {
        add_scaled_noise_twice<Io, V>(gen, j0, s1, s2, f);
      } else if constexpr (kR0) {
        Round0 p0[NB];
#pragma unroll
        for (int b = 0; b < NB; ++b)
          p0[b] = kR0Step ? round0_step(p0_thread, static_cast<uint32_t>(u * (kStride / 4) + b))
                          : philox_round0<kWide1>(static_cast<uint32_t>(j0 + b));
        uint4 x[NB];
#pragma unroll
        for (int b = 0; b < NB; ++b) x[b] = gen.block_r0(p0[b]);
        add_scaled_noise_words<kAxpyForm, V>(x, s1, f);
        if constexpr (kTwo) {
          Io::round_trip(f);
#pragma unroll
          for (int b = 0; b < NB; ++b) x[b] = gen2.block_r0(p0[b]);
          add_scaled_noise_words<kAxpyForm, V>(x, s2, f);
        }
      } else {
        add_scaled_noise<kAxpyForm, V>(gen, j0, s1, f);
        if constexpr (kTwo) {
          Io::round_trip(f);
          add_scaled_noise<kAxpyForm, V>(gen2, j0, s2, f);
        }
      }
      if constexpr (kFull)
        *reinterpret_cast<uint4*>(p + u * kStride) = Io::pack(f);
      else
        store_vec(cur, vec_elem(cur, u), Io::pack(f));
    }
    if (grp + 1 < kGroups || has_next) {
#pragma unroll
      for (int q = 0; q < G; ++q) v[q] = nv[q];
    }
  }
}

// theta[g] <- round(theta[g] + scale * eps_seed[g]) over every segment; with
// kTwo, a second step round(. + scale2 * eps_seed2[g]) follows in registers,
// after the first result has been rounded to the storage type exactly as a
// separate launch would store it (restore of one member fused with the
// perturb of the next).
// For a scaled storage type (FP8) the noise is added in units of the
// segment's scale: scale * inv_scale[segment].
template <class Io, bool kTwo, bool kSame>
__global__ void __launch_bounds__(kBlockThreads, axpy_min_blocks(kTwo, Io::kVec, kSame))
axpy_noise_kernel(const SegDesc* __restrict__ segs, const float* __restrict__ inv_scale,
                  uint64_t total_tiles, const __grid_constant__ AxpyArgs a) {
  constexpr int G = group_for<Io>(kTwo ? kAxpy2Group : kAxpy1Group);
  uint64_t tile = blockIdx.x;
  if (tile >= total_tiles) return;
  int seg = 0;
  TileRef<Io> cur = tile_ref<Io>(segs, inv_scale, seg, tile);
  uint4 v[G];
  load_group<Io, G>(cur, 0, v);
  for (;;) {
    const uint64_t next = tile + gridDim.x;
    const bool has_next = next < total_tiles;
    TileRef<Io> nxt = cur;
    constexpr uint64_t kTile = static_cast<uint64_t>(kBlockThreads) * kVecsPerThread * Io::kVec;
    if (!uniform_hi(cur.index_base, cur.t0, kTile, cur.numel))
      axpy_tile<Io, kTwo, kSame, false, false, G>(cur, v, a, segs, inv_scale, seg, next, has_next,
                                                  nxt);
    else if (cur.t0 + kTile <= cur.numel)
      axpy_tile<Io, kTwo, kSame, true, true, G>(cur, v, a, segs, inv_scale, seg, next, has_next,
                                                nxt);
    else
      axpy_tile<Io, kTwo, kSame, true, false, G>(cur, v, a, segs, inv_scale, seg, next, has_next,
                                                 nxt);
    if (!has_next) break;
    tile = next;
    cur = nxt;
  }
}

// Seeds of an update launch are staged in shared memory kSchedRows at a time,
// one row of kRowVecs 16-byte words per seed, filled by the CTA for the
// high counter word j_hi of the tile at hand:
//   row[0] = (k0, k1, round 1's k0, tile constant x2)
//   row[1] = (tile constant lo2, coefficient bits, 0, 0)
//   row[2 .. 5] = round keys of rounds 2..9
// so a seed costs its thread six shared-memory loads instead of deriving its
// key schedule and tile constants. Row kSchedRows is the trailing perturb's.
constexpr int kSchedRows = 128;
constexpr int kRowVecs = 6;
using SchedRow = uint4[kRowVecs];

__device__ __forceinline__ void fill_row(SchedRow& row, uint32_t k0, uint32_t k1, float coeff,
                                         uint32_t j_hi) {
  const PhiloxSched s = philox_sched(static_cast<uint64_t>(k1) << 32 | k0);
  const TileConst t = tile_const(j_hi, s.rk[0], s.rk[3]);
  row[0] = make_uint4(s.rk[0], s.rk[1], s.rk[2], t.x2);
  row[1] = make_uint4(t.lo2, __float_as_uint(coeff), 0u, 0u);
#pragma unroll
  for (int k = 0; k < 4; ++k)
    row[2 + k] = make_uint4(s.rk[4 + 4 * k], s.rk[5 + 4 * k], s.rk[6 + 4 * k], s.rk[7 + 4 * k]);
}

// Round keys of rounds 2..9 held in registers.
struct KeyRegs {
  uint32_t k[16];
  __device__ uint32_t operator[](int i) const { return k[i]; }
};

// Generator and coefficient of one staged row.
template <bool kUniformHi>
__device__ __forceinline__ auto row_gen(const SchedRow& row) {
  const uint4 r0 = row[0], r1 = row[1];
  if constexpr (kUniformHi) {
    KeyRegs kr;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
      const uint4 w = row[2 + k];
      kr.k[4 * k] = w.x;
      kr.k[4 * k + 1] = w.y;
      kr.k[4 * k + 2] = w.z;
      kr.k[4 * k + 3] = w.w;
    }
    return SchedGen<KeyRegs>{TileConst{r0.w, r1.x}, r0.y, r0.z, kr};
  } else {
    return AnyGen{PhiloxKey{r0.x, r0.y}};
  }
}

__device__ __forceinline__ float row_coeff(const SchedRow& row) { return __uint_as_float(row[1].y); }

// Which seeds the CTA's rows hold, and for which j_hi.
struct RowState {
  int first;
  uint32_t j_hi;
};

// Makes the rows hold seeds [c0, c0 + kSchedRows) (and the perturb row) for
// j_hi. Called by every thread of the CTA with the same arguments.
template <bool kPerturb>
__device__ __forceinline__ void ensure_rows(SchedRow* s_rows, RowState& rs, const UpdateArgs& args,
                                            int c0, uint32_t j_hi) {
  if (rs.first == c0 && rs.j_hi == j_hi) return;
  __syncthreads();  // every thread is done with the rows held so far
  const int m = args.n - c0 < kSchedRows ? args.n - c0 : kSchedRows;
  for (int k = threadIdx.x; k < m; k += kBlockThreads)
    fill_row(s_rows[k], args.key[c0 + k][0], args.key[c0 + k][1], args.coeff[c0 + k], j_hi);
  if (kPerturb && threadIdx.x == kBlockThreads - 1)
    fill_row(s_rows[kSchedRows], args.pkey[0], args.pkey[1], args.pscale, j_hi);
  __syncthreads();
  rs.first = c0;
  rs.j_hi = j_hi;
}

// acc[q] += c_i eps_i over the seeds i of [c0, c1) held in the rows from c0,
// for the thread's vectors u0 .. u0 + G - 1 (ascending i).
template <class Io, bool kUniformHi, int G>
__device__ __forceinline__ void accumulate_seeds(const TileRef<Io>& r, int u0, const SchedRow* rows,
                                                 int count, float (&acc)[G][Io::kVec]) {
  constexpr int V = Io::kVec;
  constexpr int kUnroll = ES_SEED_UNROLL;
  if constexpr (kUpdatePipelined && G == 1 && V <= 8) {
    // Software-pipelined over the seeds: seed i + 1's Philox words are
    // computed in the same basic block as seed i's transform, so the
    // integer-multiply phase of one seed overlaps the MUFU/FP32 phase of the
    // other.
    constexpr int NB = V / 4;
    const uint64_t e = vec_elem(r, u0);
    if (e >= r.numel || count < 1) return;
    const uint64_t j0 = (r.index_base + e) >> 2;
    // round 0's products, shared by every seed (kRound0)
    constexpr bool kR0 = kUniformHi && kRound0 >= 1;
    Round0 p0[NB];
#pragma unroll
    for (int b = 0; b < NB; ++b)
      p0[b] = kR0 ? philox_round0<false>(static_cast<uint32_t>(j0 + b)) : Round0{0u, 0u};
    auto words = [&](const SchedRow& row, uint4 (&w)[NB]) {
      const auto gen = row_gen<kUniformHi>(row);
#pragma unroll
      for (int b = 0; b < NB; ++b) {
        if constexpr (kR0) w[b] = gen.block_r0(p0[b]);
        else w[b] = gen.block(j0 + b);
      }
    };
    auto transform = [&](const uint4 (&w)[NB], const SchedRow& row) {
      add_scaled_noise_words<kUpdateForm, V>(w, row_coeff(row), acc[0]);
    };
    uint4 x[NB];
    words(rows[0], x);
    if constexpr (kUpdatePingPong) {
      // two seeds per iteration, the word buffers alternating, so no copies
      uint4 y[NB];
      int i = 0;
#pragma unroll 1
      for (; i + 2 < count; i += 2) {
        words(rows[i + 1], y);
        transform(x, rows[i]);
        words(rows[i + 2], x);
        transform(y, rows[i + 1]);
      }
      if (i + 1 < count) {
        words(rows[i + 1], y);
        transform(x, rows[i]);
        transform(y, rows[i + 1]);
      } else {
        transform(x, rows[i]);
      }
    } else {
#pragma unroll 1
      for (int i = 0; i + 1 < count; ++i) {
        uint4 xn[NB];
        words(rows[i + 1], xn);
        transform(x, rows[i]);
#pragma unroll
        for (int b = 0; b < NB; ++b) x[b] = xn[b];
      }
      transform(x, rows[count - 1]);
    }
  } else {
#pragma unroll kUnroll
    for (int i = 0; i < count; ++i) {
      const auto gen = row_gen<kUniformHi>(rows[i]);
      const float c = row_coeff(rows[i]);
#pragma unroll
      for (int q = 0; q < G; ++q) {
        const uint64_t e = vec_elem(r, u0 + q);
        if (e >= r.numel) continue;
        add_scaled_noise<kUpdateForm, V>(gen, (r.index_base + e) >> 2, c, acc[q]);
      }
    }
  }
}

// v[q] <- round(v[q] + acc[q]) in storage form; acc <- 0.
template <class Io, int G>
__device__ __forceinline__ void apply_acc(uint4 (&v)[G], float (&acc)[G][Io::kVec], float inv) {
#pragma unroll
  for (int q = 0; q < G; ++q) {
    float f[Io::kVec];
    Io::unpack(v[q], f);
#pragma unroll
    for (int k = 0; k < Io::kVec; ++k) {
      f[k] = add_acc<Io>(f[k], acc[q][k], inv);
      acc[q][k] = 0.0f;
    }
    v[q] = Io::pack(f);
  }
}

// One tile of a fused update launch, G vectors at a time. Theta stays in
// registers in storage form; generation g adds acc_g = sum_{i in g} c_i eps_i
// (fp32, ascending i) and rounds once, exactly as a separate launch per
// generation would store it (kSingle: one generation, and with kPerturb the
// next generation's first perturb follows, rounded again). Theta is read and
// written once.
template <class Io, bool kUniformHi, bool kSingle, bool kPerturb, int G>
__device__ __forceinline__ void update_tile(const TileRef<Io>& r, const UpdateArgs& args,
                                            SchedRow* s_rows, RowState& rs) {
  constexpr int V = Io::kVec;
  const uint32_t j_hi = static_cast<uint32_t>((r.index_base + r.t0) >> 34);
  const int n = args.n;
#pragma unroll 1
  for (int u0 = 0; u0 < kVecsPerThread; u0 += G) {
    uint4 v[G];
    load_group<Io, G>(r, u0, v);
    float acc[G][V];
#pragma unroll
    for (int q = 0; q < G; ++q)
#pragma unroll
      for (int k = 0; k < V; ++k) acc[q][k] = 0.0f;
    int g = 0;
#pragma unroll 1
    for (int c0 = 0; c0 < n; c0 += kSchedRows) {
      ensure_rows<kPerturb>(s_rows, rs, args, c0, j_hi);
      const int c1 = n - c0 < kSchedRows ? n : c0 + kSchedRows;
      if constexpr (kSingle) {
        accumulate_seeds<Io, kUniformHi, G>(r, u0, s_rows, c1 - c0, acc);
      } else {
        // generation by generation within the chunk (generations are never empty)
        int i = c0;
        while (i < c1) {
          const int end = args.gen_end[g] < c1 ? args.gen_end[g] : c1;
          accumulate_seeds<Io, kUniformHi, G>(r, u0, s_rows + (i - c0), end - i, acc);
          i = end;
          if (i == args.gen_end[g]) {
            apply_acc<Io, G>(v, acc, r.inv);
            ++g;
          }
        }
      }
    }
    if constexpr (kSingle) apply_acc<Io, G>(v, acc, r.inv);
    if constexpr (kPerturb) {
      const auto pgen = row_gen<kUniformHi>(s_rows[kSchedRows]);
      const float ps = row_coeff(s_rows[kSchedRows]) * r.inv;
#pragma unroll
      for (int q = 0; q < G; ++q) {
        const uint64_t e = vec_elem(r, u0 + q);
        if (e >= r.numel) continue;
        float f[V];
        Io::unpack(v[q], f);
        add_scaled_noise<kUpdateForm, V>(pgen, (r.index_base + e) >> 2, ps, f);
        v[q] = Io::pack(f);
      }
    }
#pragma unroll
    for (int q = 0; q < G; ++q) store_vec(r, vec_elem(r, u0 + q), v[q]);
  }
}

// Fused update launch (es_update, es_replay, es_update_perturb): for each
// generation g, theta[g] <- round(theta[g] + sum_{i in g} c_i eps_{s_i}[g]),
// then with kPerturb theta <- round(theta + pscale * eps_pseed).
// kSingle: one generation; otherwise args.n_gen generations, never empty.
template <class Io, bool kSingle, bool kPerturb>
__global__ void __launch_bounds__(kBlockThreads, update_min_blocks())
update_kernel(const SegDesc* __restrict__ segs, const float* __restrict__ inv_scale,
              uint64_t total_tiles, const __grid_constant__ UpdateArgs args) {
  constexpr int G = group_for<Io>(kUpdateGroup);
  __shared__ SchedRow s_rows[kSchedRows + 1];
  RowState rs{-1, 0u};
  int seg = 0;
  for (uint64_t tile = blockIdx.x; tile < total_tiles; tile += gridDim.x) {
    const TileRef<Io> r = tile_ref<Io>(segs, inv_scale, seg, tile);
    if (uniform_hi(r.index_base, r.t0, static_cast<uint64_t>(kBlockThreads) * kVecsPerThread * Io::kVec, r.numel))
      update_tile<Io, true, kSingle, kPerturb, G>(r, args, s_rows, rs);
    else
      update_tile<Io, false, kSingle, kPerturb, G>(r, args, s_rows, rs);
  }
}

// out[g - index_base] = eps_seed[g] for g in [index_base, index_base + n);
// one thread per Philox block.
__global__ void __launch_bounds__(kBlockThreads)
noise_fill_kernel(uint64_t index_base, uint64_t n, PhiloxKey key, float* __restrict__ out) {
  const uint64_t j_first = index_base >> 2;
  const uint64_t nblocks = ((index_base + n - 1) >> 2) - j_first + 1;
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * blockDim.x;
  for (uint64_t t = static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < nblocks;
       t += stride) {
    const uint64_t j = j_first + t;
    const float4 e = gaussian4(j, key);
    const float vals[4] = {e.x, e.y, e.z, e.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const uint64_t g = (j << 2) + q;
      if (g >= index_base && g - index_base < n) out[g - index_base] = vals[q];
    }
  }
}

// es_noise_fill when `out` is 16-byte aligned and index_base % 4 == 0:
// out4[b] = eps[4 (j_first + b) .. 4 (j_first + b) + 3] for b < nblocks. Tiles
// of 256 threads x kVecsPerThread blocks, each 16-byte store coalesced across
// the warp. The generator is the streaming kernels': round keys from the
// launch's schedule, the Philox constants of the blocks' high word per tile
// (when the tile stays within one 2^32-block range), the packed transform with
// the near-one series on a rare branch (values equal to box_muller's).
template <bool kUniformHi>
__device__ __forceinline__ void noise_fill_tile(uint64_t j_first, uint64_t b0, uint64_t nblocks,
                                                const PhiloxSched& sched,
                                                float4* __restrict__ out) {
  const auto gen = sched_gen<kUniformHi>(sched, static_cast<uint32_t>((j_first + b0) >> 32));
#pragma unroll
  for (int q = 0; q < kVecsPerThread; ++q) {
    const uint64_t b = b0 + static_cast<uint64_t>(q * kBlockThreads + threadIdx.x);
    if (b < nblocks) {
      Polar2 pp[1];
      polar_blocks<NoiseForm::kPacked, 1>(gen, j_first + b, pp);
      const Polar2& p = pp[0];
      const float2 lo = __fmul2_rn(make_float2(-p.r.x, -p.r.x), make_float2(p.c.x, p.s.x));
      const float2 hi = __fmul2_rn(make_float2(-p.r.y, -p.r.y), make_float2(p.c.y, p.s.y));
      out[b] = make_float4(lo.x, lo.y, hi.x, hi.y);
    }
  }
}

__global__ void __launch_bounds__(kBlockThreads)
noise_fill_vec_kernel(uint64_t j_first, uint64_t nblocks, const __grid_constant__ PhiloxSched sched,
                      float4* __restrict__ out) {
  constexpr uint64_t kTileBlocks = static_cast<uint64_t>(kBlockThreads) * kVecsPerThread;
  const uint64_t tiles = (nblocks + kTileBlocks - 1) / kTileBlocks;
  for (uint64_t tile = blockIdx.x; tile < tiles; tile += gridDim.x) {
    const uint64_t b0 = tile * kTileBlocks;
    const uint64_t last = (b0 + kTileBlocks < nblocks ? b0 + kTileBlocks : nblocks) - 1;
    if (((j_first + b0) >> 32) == ((j_first + last) >> 32))
      noise_fill_tile<true>(j_first, b0, nblocks, sched, out);
    else
      noise_fill_tile<false>(j_first, b0, nblocks, sched, out);
  }
}

// out[4t .. 4t+3] = Philox words of block block_base + t. Block j goes
// through one of the four implementations of the rounds by j mod 4: the
// general one (philox_block), the one with per-tile constants (philox_tile),
// and the scheduled-key one the streaming kernels use, with high/low product
// pairs in the first two rounds (philox_block_rk), or with 64-bit-result
// products throughout and round 0's product stepped from that of a lower
// counter word by 64-bit additions (round0_step, philox_block_r0). They give
// identical words, and this lets a bit-exact check of this output cover all
// four.
__global__ void __launch_bounds__(kBlockThreads)
noise_bits_kernel(uint64_t block_base, uint64_t nblocks, const __grid_constant__ PhiloxSched sched,
                  uint4* __restrict__ out) {
  const PhiloxKey key{sched.rk[0], sched.rk[1]};
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * blockDim.x;
  for (uint64_t t = static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < nblocks;
       t += stride) {
    const uint64_t j = block_base + t;
    const uint32_t j_lo = static_cast<uint32_t>(j), j_hi = static_cast<uint32_t>(j >> 32);
    const TileConst tc = tile_const(j_hi, sched.rk[0], sched.rk[3]);
    switch (j & 3) {
      case 0: out[t] = philox_block(j, key); break;
      case 1: out[t] = philox_block_tile(j_lo, philox_tile(j_hi, key)); break;
      case 2: out[t] = philox_block_rk<false>(j_lo, tc, sched.rk[1], sched.rk[2], sched.rk + 4); break;
      default: {
        // from j_lo rounded down to a multiple of 2^11, d = j_lo mod 2^11 (no wrap)
        const Round0 p0 = round0_step(philox_round0<true>(j_lo & ~0x7FFu), j_lo & 0x7FFu);
        out[t] = philox_block_r0<true>(p0, tc, sched.rk[1], sched.rk[2], sched.rk + 4);
      }
    }
  }
}

// out[2k], out[2k+1] = Box-Muller pair of words[2k], words[2k+1].
__global__ void __launch_bounds__(kBlockThreads)
box_muller_kernel(const uint2* __restrict__ words, uint64_t npairs, float2* __restrict__ out) {
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * blockDim.x;
  for (uint64_t k = static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x; k < npairs;
       k += stride) {
    const uint2 w = words[k];
    out[k] = box_muller(w.x, w.y);
  }
}

// Resident CTAs of one kernel on one device (SMs x CTAs per SM), looked up
// with the occupancy calculator on the kernel's first launch on that device
// and kept, so later launches make no query beyond cudaGetDevice.
struct GridEntry {
  const void* kernel;
  int device;
  int ctas;
};
constexpr int kGridCacheSize = 128;
std::mutex g_grid_mutex;
GridEntry g_grid_cache[kGridCacheSize];
int g_grid_used = 0;

int resident_ctas(const void* kernel, int dev) {
  {
    std::lock_guard<std::mutex> lock(g_grid_mutex);
    for (int k = 0; k < g_grid_used; ++k)
      if (g_grid_cache[k].kernel == kernel && g_grid_cache[k].device == dev)
        return g_grid_cache[k].ctas;
  }
  int sms = 0, per_sm = 0;
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kBlockThreads, 0);
  if (sms < 1) sms = 1;
  if (per_sm < 1) per_sm = 1;
  const int ctas = sms * per_sm;
  std::lock_guard<std::mutex> lock(g_grid_mutex);
  if (g_grid_used < kGridCacheSize) g_grid_cache[g_grid_used++] = GridEntry{kernel, dev, ctas};
  return ctas;
}

// Persistent grid: every SM filled to the kernel's occupancy, never more
// CTAs than tiles.
template <class K>
int persistent_grid(K kernel, uint64_t work_items) {
  int dev = 0;
  cudaGetDevice(&dev);
  uint64_t grid = static_cast<uint64_t>(resident_ctas(reinterpret_cast<const void*>(kernel), dev));
  if (work_items < grid) grid = work_items;
  return grid < 1 ? 1 : static_cast<int>(grid);
}

template <class Io, bool kTwo, bool kSame>
cudaError_t launch_axpy_io(const PlanView& plan, const AxpyArgs& a, cudaStream_t stream) {
  auto k = axpy_noise_kernel<Io, kTwo, kSame>;
  k<<<persistent_grid(k, plan.total_tiles), kBlockThreads, 0, stream>>>(
      plan.segs, plan.inv_scale, plan.total_tiles, a);
  return cudaGetLastError();
}

template <bool kTwo, bool kSame>
cudaError_t launch_axpy(const PlanView& plan, uint64_t seed, float scale, uint64_t seed2,
                        float scale2, cudaStream_t stream) {
  AxpyArgs a;
  a.s1 = philox_sched(seed);
  a.s2 = philox_sched(seed2);
  a.scale1 = scale;
  a.scale2 = scale2;
  if (plan.dtype == ES_BF16) return launch_axpy_io<Bf16Io, kTwo, kSame>(plan, a, stream);
  if (plan.dtype == ES_FP8_E4M3) return launch_axpy_io<Fp8Io, kTwo, kSame>(plan, a, stream);
  return launch_axpy_io<F32Io, kTwo, kSame>(plan, a, stream);
}

}  // namespace

cudaError_t launch_axpy_noise(const PlanView& plan, uint64_t seed, float scale,
                              cudaStream_t stream) {
  return launch_axpy<false, false>(plan, seed, scale, 0u, 0.0f, stream);
}

cudaError_t launch_axpy_noise2(const PlanView& plan, uint64_t seed, float scale, uint64_t seed2,
                               float scale2, cudaStream_t stream) {
  if (seed == seed2) return launch_axpy<true, true>(plan, seed, scale, seed2, scale2, stream);
  return launch_axpy<true, false>(plan, seed, scale, seed2, scale2, stream);
}

template <class Io>
cudaError_t launch_update_io(const PlanView& plan, const UpdateArgs& args, cudaStream_t stream) {
  auto k = update_kernel<Io, false, false>;
  if (args.n_gen == 1) k = args.perturb ? update_kernel<Io, true, true> : update_kernel<Io, true, false>;
  k<<<persistent_grid(k, plan.total_tiles), kBlockThreads, 0, stream>>>(
      plan.segs, plan.inv_scale, plan.total_tiles, args);
  return cudaGetLastError();
}

cudaError_t launch_update(const PlanView& plan, const UpdateArgs& args, cudaStream_t stream) {
  if (plan.dtype == ES_BF16) return launch_update_io<Bf16Io>(plan, args, stream);
  if (plan.dtype == ES_FP8_E4M3) return launch_update_io<Fp8Io>(plan, args, stream);
  return launch_update_io<F32Io>(plan, args, stream);
}

cudaError_t launch_noise_bits(uint64_t seed, uint64_t block_base, uint64_t nblocks,
                              uint32_t* out, cudaStream_t stream) {
  const uint64_t ctas = (nblocks + kBlockThreads - 1) / kBlockThreads;
  const int grid = persistent_grid(noise_bits_kernel, ctas);
  noise_bits_kernel<<<grid, kBlockThreads, 0, stream>>>(block_base, nblocks, philox_sched(seed),
                                                        reinterpret_cast<uint4*>(out));
  return cudaGetLastError();
}

cudaError_t launch_box_muller(const uint32_t* words, uint64_t npairs, float* out,
                              cudaStream_t stream) {
  const uint64_t ctas = (npairs + kBlockThreads - 1) / kBlockThreads;
  const int grid = persistent_grid(box_muller_kernel, ctas);
  box_muller_kernel<<<grid, kBlockThreads, 0, stream>>>(reinterpret_cast<const uint2*>(words),
                                                        npairs, reinterpret_cast<float2*>(out));
  return cudaGetLastError();
}

cudaError_t launch_noise_fill(uint64_t seed, uint64_t index_base, uint64_t n, float* out,
                              cudaStream_t stream) {
  const PhiloxKey key = philox_key(seed);
  // Aligned case: whole Philox blocks as 16-byte stores; the n % 4 elements
  // left over go through the general kernel below.
  if (reinterpret_cast<uintptr_t>(out) % 16 == 0 && index_base % 4 == 0 && n >= 4) {
    const uint64_t full = n / 4;
    constexpr uint64_t kTileBlocks = static_cast<uint64_t>(kBlockThreads) * kVecsPerThread;
    const int grid = persistent_grid(noise_fill_vec_kernel, (full + kTileBlocks - 1) / kTileBlocks);
    noise_fill_vec_kernel<<<grid, kBlockThreads, 0, stream>>>(index_base / 4, full,
                                                              philox_sched(seed),
                                                              reinterpret_cast<float4*>(out));
    const cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess || n % 4 == 0) return err;
    index_base += 4 * full;
    out += 4 * full;
    n %= 4;
  }
  const uint64_t nblocks = ((index_base + n - 1) >> 2) - (index_base >> 2) + 1;
  const uint64_t ctas = (nblocks + kBlockThreads - 1) / kBlockThreads;
  const int grid = persistent_grid(noise_fill_kernel, ctas);
  noise_fill_kernel<<<grid, kBlockThreads, 0, stream>>>(index_base, n, key, out);
  return cudaGetLastError();
}

}  // namespace esopt
