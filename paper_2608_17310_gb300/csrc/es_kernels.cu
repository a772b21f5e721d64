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
  __device__ static float to_f32(uint16_t h) { return __uint_as_float(static_cast<uint32_t>(h) << 16); }
  __device__ static uint16_t from_f32(float f) { return __bfloat16_as_ushort(__float2bfloat16_rn(f)); }
  __device__ static uint32_t pack2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);  // one cvt.rn.bf16x2.f32
    return *reinterpret_cast<uint32_t*>(&h);
  }
  __device__ static void unpack(const uint4& v, float (&f)[8]) {
    f[0] = __uint_as_float(v.x << 16); f[1] = __uint_as_float(v.x & 0xFFFF0000u);
    f[2] = __uint_as_float(v.y << 16); f[3] = __uint_as_float(v.y & 0xFFFF0000u);
    f[4] = __uint_as_float(v.z << 16); f[5] = __uint_as_float(v.z & 0xFFFF0000u);
    f[6] = __uint_as_float(v.w << 16); f[7] = __uint_as_float(v.w & 0xFFFF0000u);
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
      f[k] = __uint_as_float(w << 16);
      f[k + 1] = __uint_as_float(w & 0xFFFF0000u);
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
  __device__ static float to_f32(float f) { return f; }
  __device__ static float from_f32(float f) { return f; }
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
  __device__ static float to_f32(uint8_t c) {
    return __half2float(__half(__nv_cvt_fp8_to_halfraw(static_cast<__nv_fp8_storage_t>(c),
                                                       __NV_E4M3)));
  }
  __device__ static uint8_t from_f32(float f) {
    return static_cast<uint8_t>(__nv_cvt_float_to_fp8(f, __NV_SATFINITE, __NV_E4M3));
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

// Vectors a thread processes at once for a kernel kind's group g: FP8 vectors
// hold twice the elements of bf16 ones, so they go half as many at a time.
template <class Io>
__host__ __device__ constexpr int group_for(int g) {
  return Io::kVec > 8 ? (g > 1 ? g / 2 : 1) : g;
}

// theta + acc in storage units: acc is in parameter units, so a scaled
// segment takes acc / scale (one fused multiply-add with 1 / scale).
template <class Io>
__device__ __forceinline__ float add_acc(float theta, float acc, float inv_scale) {
  if constexpr (Io::kScaled) return fmaf(acc, inv_scale, theta);
  else return theta + acc;
}

// Philox words of block j for one seed. TileGen serves the blocks of a tile
// that share the high counter word (per-tile constants, see philox_tile);
// AnyGen serves any block. Both give the same words.
struct TileGen {
  PhiloxTile t;
  __device__ uint4 block(uint64_t j) const { return philox_block_tile(static_cast<uint32_t>(j), t); }
};
struct AnyGen {
  PhiloxKey key;
  __device__ uint4 block(uint64_t j) const { return philox_block(j, key); }
};

template <bool kUniformHi>
__device__ __forceinline__ auto make_gen(PhiloxKey key, uint32_t j_hi) {
  if constexpr (kUniformHi) return TileGen{philox_tile(j_hi, key)};
  else return AnyGen{key};
}

// How each Philox block becomes theta updates. The forms give bit-identical
// values: a packed two-wide FP32 instruction rounds each half exactly like the
// scalar one. They differ only in instruction mix, which moves work between the
// FMA pipe's halves. Each kernel uses the form measured fastest for it:
//   kScalar     scalar transform (polar) and scalar FMAs;
//   kPackedFma  scalar transform, packed FMAs into theta or the accumulator;
//   kPacked     packed transform (polar2) and packed FMAs.
enum class NoiseForm { kScalar, kPackedFma, kPacked };

// f[k] += scale * eps[g0 + k] for the V elements from global index g0
// (g0 % 4 == 0), with scale folded into each pair's radius.
template <NoiseForm kForm, int V, class Gen>
__device__ __forceinline__ void add_scaled_noise(const Gen& gen, uint64_t g0, float scale,
                                                 float (&f)[V]) {
#pragma unroll
  for (int b = 0; b < V / 4; ++b) {
    const uint4 x = gen.block((g0 >> 2) + b);
    if constexpr (kForm == NoiseForm::kScalar) {
      const Polar p = polar(x.x, x.y);
      const Polar q = polar(x.z, x.w);
      const float sp = -(scale * p.r), sq = -(scale * q.r);
      f[4 * b + 0] = fmaf(sp, p.c, f[4 * b + 0]);
      f[4 * b + 1] = fmaf(sp, p.s, f[4 * b + 1]);
      f[4 * b + 2] = fmaf(sq, q.c, f[4 * b + 2]);
      f[4 * b + 3] = fmaf(sq, q.s, f[4 * b + 3]);
    } else {
      Polar2 p;
      if constexpr (kForm == NoiseForm::kPacked) {
        p = polar2(x);
      } else {
        const Polar a = polar(x.x, x.y), c = polar(x.z, x.w);
        p = Polar2{make_float2(a.r, c.r), make_float2(a.c, c.c), make_float2(a.s, c.s)};
      }
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

// f <- round(round(f + s1 * eps) + s2 * eps) for one seed's noise, computed
// once: an antithetic restore (+eps out) followed by the perturb (-eps in).
template <class Io, int V, class Gen>
__device__ __forceinline__ void add_scaled_noise_twice(const Gen& gen, uint64_t g0, float s1,
                                                       float s2, float (&f)[V]) {
#pragma unroll
  for (int b = 0; b < V / 4; ++b) {
    const uint4 x = gen.block((g0 >> 2) + b);
    const Polar p = polar(x.x, x.y);
    const Polar q = polar(x.z, x.w);
    float h[4];
    h[0] = fmaf(-(s1 * p.r), p.c, f[4 * b + 0]);
    h[1] = fmaf(-(s1 * p.r), p.s, f[4 * b + 1]);
    h[2] = fmaf(-(s1 * q.r), q.c, f[4 * b + 2]);
    h[3] = fmaf(-(s1 * q.r), q.s, f[4 * b + 3]);
    Io::round_trip(h);
    f[4 * b + 0] = fmaf(-(s2 * p.r), p.c, h[0]);
    f[4 * b + 1] = fmaf(-(s2 * p.r), p.s, h[1]);
    f[4 * b + 2] = fmaf(-(s2 * q.r), q.c, h[2]);
    f[4 * b + 3] = fmaf(-(s2 * q.r), q.s, h[3]);
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

// Location of one tile: its segment's storage and the tile's first element.
template <class Io>
struct TileRef {
  typename Io::Scalar* base;
  uint64_t numel;
  uint64_t index_base;
  uint64_t t0;
};

template <class Io>
__device__ __forceinline__ TileRef<Io> tile_ref(const SegDesc* __restrict__ segs, int& seg,
                                                uint64_t tile, uint64_t tile_elems) {
  const SegDesc* d = find_segment(segs, seg, tile);
  return TileRef<Io>{static_cast<typename Io::Scalar*>(d->data), d->numel, d->index_base,
                     (tile - d->tile_begin) * tile_elems};
}

// One tile of the perturb/restore pass (kTwo: fused restore + perturb; kSame:
// both steps use one seed, whose noise is generated once). Each thread takes
// its kVecsPerThread vectors G at a time: loads them, adds the noise and
// stores them.
template <class Io, bool kTwo, bool kSame, bool kUniformHi, int G>
__device__ __forceinline__ void axpy_tile(const TileRef<Io>& r, PhiloxKey key, float scale,
                                          PhiloxKey key2, float scale2) {
  constexpr int V = Io::kVec;
  // the two-seed pass is fastest fully packed, the one-seed pass scalar
  constexpr NoiseForm kAxpyForm = kTwo ? NoiseForm::kPacked : NoiseForm::kScalar;
  typename Io::Scalar* const base = r.base;
  const uint64_t numel = r.numel, index_base = r.index_base, t0 = r.t0;
  const uint32_t j_hi = static_cast<uint32_t>((index_base + t0) >> 34);
  const auto gen = make_gen<kUniformHi>(key, j_hi);
  const auto gen2 = make_gen<kUniformHi && kTwo && !kSame>(key2, j_hi);
#pragma unroll 1
  for (int u0 = 0; u0 < kVecsPerThread; u0 += G) {
    uint4 v[G];
#pragma unroll
    for (int u = 0; u < G; ++u) {
      const uint64_t e = t0 + static_cast<uint64_t>((u0 + u) * kBlockThreads + threadIdx.x) * V;
      v[u] = make_uint4(0u, 0u, 0u, 0u);
      if (e + V <= numel) v[u] = *reinterpret_cast<const uint4*>(base + e);
    }
#pragma unroll
    for (int u = 0; u < G; ++u) {
      const uint64_t e = t0 + static_cast<uint64_t>((u0 + u) * kBlockThreads + threadIdx.x) * V;
      if (e >= numel) continue;
      const bool full = e + V <= numel;
      const int rem = full ? V : static_cast<int>(numel - e);
      float f[V];
      if (full) {
        Io::unpack(v[u], f);
      } else {  // ragged end of a segment
#pragma unroll
        for (int k = 0; k < V; ++k) f[k] = k < rem ? Io::to_f32(base[e + k]) : 0.0f;
      }
      if (kSame) {
        add_scaled_noise_twice<Io, V>(gen, index_base + e, scale, scale2, f);
      } else {
        add_scaled_noise<kAxpyForm, V>(gen, index_base + e, scale, f);
        if (kTwo) {
          Io::round_trip(f);
          add_scaled_noise<kAxpyForm, V>(gen2, index_base + e, scale2, f);
        }
      }
      if (full) {
        *reinterpret_cast<uint4*>(base + e) = Io::pack(f);
      } else {
#pragma unroll
        for (int k = 0; k < V; ++k)
          if (k < rem) base[e + k] = Io::from_f32(f[k]);
      }
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
__global__ void __launch_bounds__(kBlockThreads, axpy_min_blocks(kTwo))
axpy_noise_kernel(const SegDesc* __restrict__ segs, const float* __restrict__ inv_scale,
                  uint64_t total_tiles, PhiloxKey key, float scale, PhiloxKey key2,
                  float scale2) {
  constexpr uint64_t kTile = static_cast<uint64_t>(kBlockThreads) * kVecsPerThread * Io::kVec;
  constexpr int G = group_for<Io>(kTwo ? kAxpy2Group : kAxpy1Group);
  int seg = 0;
  for (uint64_t tile = blockIdx.x; tile < total_tiles; tile += gridDim.x) {
    const TileRef<Io> cur = tile_ref<Io>(segs, seg, tile, kTile);
    float s1 = scale, s2 = scale2;
    if constexpr (Io::kScaled) {
      const float inv = inv_scale[seg];
      s1 *= inv;
      s2 *= inv;
    }
    if (uniform_hi(cur.index_base, cur.t0, kTile, cur.numel))
      axpy_tile<Io, kTwo, kSame, true, G>(cur, key, s1, key2, s2);
    else
      axpy_tile<Io, kTwo, kSame, false, G>(cur, key, s1, key2, s2);
  }
}

// One tile of a single-generation update (es_update; with kPerturb also the
// trailing perturb of es_update_perturb): acc = sum_i c_i eps_i (fp32,
// ascending i), then theta + acc rounded once (then + pscale * eps_pseed,
// rounded again); theta read and written once. Vectors G at a time.
template <class Io, bool kUniformHi, bool kPerturb, int G>
__device__ __forceinline__ void update_tile_single(typename Io::Scalar* base, uint64_t numel,
                                                   uint64_t index_base, uint64_t t0,
                                                   const UpdateArgs& args, const PhiloxKey* s_key,
                                                   const float* s_coeff, float inv) {
  constexpr int V = Io::kVec;
  constexpr int kUnroll = ES_SEED_UNROLL;
  const uint32_t j_hi = static_cast<uint32_t>((index_base + t0) >> 34);
  const int n = args.n;
  const float pscale = Io::kScaled ? args.pscale * inv : args.pscale;
  const auto pgen = make_gen<kUniformHi && kPerturb>(PhiloxKey{args.pkey[0], args.pkey[1]}, j_hi);
#pragma unroll 1
  for (int u0 = 0; u0 < kVecsPerThread; u0 += G) {
    uint4 v[G];
#pragma unroll
    for (int q = 0; q < G; ++q) {
      const uint64_t e = t0 + static_cast<uint64_t>((u0 + q) * kBlockThreads + threadIdx.x) * V;
      v[q] = make_uint4(0u, 0u, 0u, 0u);
      if (e + V <= numel) v[q] = *reinterpret_cast<const uint4*>(base + e);
    }
    float acc[G][V];
#pragma unroll
    for (int q = 0; q < G; ++q)
#pragma unroll
      for (int k = 0; k < V; ++k) acc[q][k] = 0.0f;
#pragma unroll kUnroll
    for (int i = 0; i < n; ++i) {
      const auto gen = make_gen<kUniformHi>(s_key[i], j_hi);
      const float c = s_coeff[i];
#pragma unroll
      for (int q = 0; q < G; ++q) {
        const uint64_t e = t0 + static_cast<uint64_t>((u0 + q) * kBlockThreads + threadIdx.x) * V;
        if (e >= numel) continue;
        add_scaled_noise<NoiseForm::kPackedFma, V>(gen, index_base + e, c, acc[q]);
      }
    }
#pragma unroll
    for (int q = 0; q < G; ++q) {
      const uint64_t e = t0 + static_cast<uint64_t>((u0 + q) * kBlockThreads + threadIdx.x) * V;
      if (e >= numel) continue;
      const bool full = e + V <= numel;
      const int rem = full ? V : static_cast<int>(numel - e);
      float f[V];
      if (full) {
        Io::unpack(v[q], f);
      } else {
#pragma unroll
        for (int k = 0; k < V; ++k) f[k] = k < rem ? Io::to_f32(base[e + k]) : 0.0f;
      }
#pragma unroll
      for (int k = 0; k < V; ++k) f[k] = add_acc<Io>(f[k], acc[q][k], inv);
      if (kPerturb) {
        Io::round_trip(f);
        add_scaled_noise<NoiseForm::kPackedFma, V>(pgen, index_base + e, pscale, f);
      }
      if (full) {
        *reinterpret_cast<uint4*>(base + e) = Io::pack(f);
      } else {
#pragma unroll
        for (int k = 0; k < V; ++k)
          if (k < rem) base[e + k] = Io::from_f32(f[k]);
      }
    }
  }
}

// One tile of a fused update launch. Theta stays in registers in storage
// form; generation g adds acc_g = sum_{i in g} c_i eps_i (fp32, ascending i)
// and rounds once, exactly as a separate launch per generation would store it;
// an optional trailing perturb step follows. Theta is read and written once.
// Vectors G at a time; lanes past the segment's end hold zeros and are never
// stored.
template <class Io, bool kUniformHi, int G>
__device__ __forceinline__ void update_tile(typename Io::Scalar* base, uint64_t numel,
                                            uint64_t index_base, uint64_t t0,
                                            const UpdateArgs& args, const PhiloxKey* s_key,
                                            const float* s_coeff, const uint16_t* s_gen_end,
                                            float inv) {
  constexpr int V = Io::kVec;
  const uint32_t j_hi = static_cast<uint32_t>((index_base + t0) >> 34);
#pragma unroll 1
  for (int u0 = 0; u0 < kVecsPerThread; u0 += G) {
    uint4 v[G];
#pragma unroll
    for (int q = 0; q < G; ++q) {
      const uint64_t e = t0 + static_cast<uint64_t>((u0 + q) * kBlockThreads + threadIdx.x) * V;
      v[q] = make_uint4(0u, 0u, 0u, 0u);
      if (e + V <= numel)
        v[q] = *reinterpret_cast<const uint4*>(base + e);
      else if (e < numel)
        v[q] = Io::load_partial(base, e, static_cast<int>(numel - e));
    }
    int i = 0;
#pragma unroll 1
    for (int g = 0; g < args.n_gen; ++g) {
      float acc[G][V];
#pragma unroll
      for (int q = 0; q < G; ++q)
#pragma unroll
        for (int k = 0; k < V; ++k) acc[q][k] = 0.0f;
      const int end = s_gen_end[g];
#pragma unroll 1
      for (; i < end; ++i) {
        const auto gen = make_gen<kUniformHi>(s_key[i], j_hi);
        const float c = s_coeff[i];
#pragma unroll
        for (int q = 0; q < G; ++q) {
          const uint64_t e = t0 + static_cast<uint64_t>((u0 + q) * kBlockThreads + threadIdx.x) * V;
          if (e >= numel) continue;
          add_scaled_noise<NoiseForm::kPackedFma, V>(gen, index_base + e, c, acc[q]);
        }
      }
#pragma unroll
      for (int q = 0; q < G; ++q) {
        float f[V];
        Io::unpack(v[q], f);
#pragma unroll
        for (int k = 0; k < V; ++k) f[k] = add_acc<Io>(f[k], acc[q][k], inv);
        v[q] = Io::pack(f);
      }
    }
    if (args.perturb) {
      const auto gen = make_gen<kUniformHi>(PhiloxKey{args.pkey[0], args.pkey[1]}, j_hi);
#pragma unroll
      for (int q = 0; q < G; ++q) {
        const uint64_t e = t0 + static_cast<uint64_t>((u0 + q) * kBlockThreads + threadIdx.x) * V;
        if (e >= numel) continue;
        float f[V];
        Io::unpack(v[q], f);
        add_scaled_noise<NoiseForm::kPackedFma, V>(gen, index_base + e,
                                                   Io::kScaled ? args.pscale * inv : args.pscale, f);
        v[q] = Io::pack(f);
      }
    }
#pragma unroll
    for (int q = 0; q < G; ++q) {
      const uint64_t e = t0 + static_cast<uint64_t>((u0 + q) * kBlockThreads + threadIdx.x) * V;
      if (e + V <= numel)
        *reinterpret_cast<uint4*>(base + e) = v[q];
      else if (e < numel)
        Io::store_partial(base, e, static_cast<int>(numel - e), v[q]);
    }
  }
}

// Fused update launch (es_update, es_replay, es_update_perturb): for each
// generation g, theta[g] <- round(theta[g] + sum_{i in g} c_i eps_{s_i}[g]),
// then optionally theta <- round(theta + pscale * eps_pseed).
// kSingle: one generation (update_tile_single, with a trailing perturb when
// kPerturb); otherwise the general form (update_tile).
template <class Io, bool kSingle, bool kPerturb>
__global__ void __launch_bounds__(kBlockThreads, update_min_blocks())
update_kernel(const SegDesc* __restrict__ segs, const float* __restrict__ inv_scale,
              uint64_t total_tiles, const __grid_constant__ UpdateArgs args) {
  constexpr uint64_t kTile = static_cast<uint64_t>(kBlockThreads) * kVecsPerThread * Io::kVec;
  constexpr int G = group_for<Io>(kUpdateGroup);
  using S = typename Io::Scalar;
  __shared__ PhiloxKey s_key[ES_MAX_SEEDS];
  __shared__ float s_coeff[ES_MAX_SEEDS];
  __shared__ uint16_t s_gen_end[kMaxGenerations];
  for (int i = threadIdx.x; i < args.n; i += blockDim.x) {
    s_key[i] = PhiloxKey{args.key[i][0], args.key[i][1]};
    s_coeff[i] = args.coeff[i];
  }
  for (int g = threadIdx.x; g < args.n_gen; g += blockDim.x) s_gen_end[g] = args.gen_end[g];
  __syncthreads();

  int seg = 0;
  for (uint64_t tile = blockIdx.x; tile < total_tiles; tile += gridDim.x) {
    const SegDesc* d = find_segment(segs, seg, tile);
    S* const base = static_cast<S*>(d->data);
    const uint64_t numel = d->numel;
    const uint64_t index_base = d->index_base;
    const uint64_t t0 = (tile - d->tile_begin) * kTile;
    const bool uhi = uniform_hi(index_base, t0, kTile, numel);
    const float inv = Io::kScaled ? inv_scale[seg] : 1.0f;
    if constexpr (kSingle) {
      if (uhi)
        update_tile_single<Io, true, kPerturb, G>(base, numel, index_base, t0, args, s_key,
                                                  s_coeff, inv);
      else
        update_tile_single<Io, false, kPerturb, G>(base, numel, index_base, t0, args, s_key,
                                                   s_coeff, inv);
    } else {
      if (uhi)
        update_tile<Io, true, G>(base, numel, index_base, t0, args, s_key, s_coeff, s_gen_end,
                                 inv);
      else
        update_tile<Io, false, G>(base, numel, index_base, t0, args, s_key, s_coeff, s_gen_end,
                                  inv);
    }
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
// the warp; the Philox constants of the blocks' high word are hoisted per tile
// when the tile stays within one 2^32-block range. The pair transform is the
// packed form (bit-identical to box_muller).
template <bool kUniformHi>
__device__ __forceinline__ void noise_fill_tile(uint64_t j_first, uint64_t b0, uint64_t nblocks,
                                                PhiloxKey key, float4* __restrict__ out) {
  const auto gen = make_gen<kUniformHi>(key, static_cast<uint32_t>((j_first + b0) >> 32));
#pragma unroll
  for (int q = 0; q < kVecsPerThread; ++q) {
    const uint64_t b = b0 + static_cast<uint64_t>(q * kBlockThreads + threadIdx.x);
    if (b < nblocks) {
      const Polar2 p = polar2(gen.block(j_first + b));
      const float2 lo = __fmul2_rn(make_float2(-p.r.x, -p.r.x), make_float2(p.c.x, p.s.x));
      const float2 hi = __fmul2_rn(make_float2(-p.r.y, -p.r.y), make_float2(p.c.y, p.s.y));
      out[b] = make_float4(lo.x, lo.y, hi.x, hi.y);
    }
  }
}

__global__ void __launch_bounds__(kBlockThreads)
noise_fill_vec_kernel(uint64_t j_first, uint64_t nblocks, PhiloxKey key, float4* __restrict__ out) {
  constexpr uint64_t kTileBlocks = static_cast<uint64_t>(kBlockThreads) * kVecsPerThread;
  const uint64_t tiles = (nblocks + kTileBlocks - 1) / kTileBlocks;
  for (uint64_t tile = blockIdx.x; tile < tiles; tile += gridDim.x) {
    const uint64_t b0 = tile * kTileBlocks;
    const uint64_t last = (b0 + kTileBlocks < nblocks ? b0 + kTileBlocks : nblocks) - 1;
    if (((j_first + b0) >> 32) == ((j_first + last) >> 32))
      noise_fill_tile<true>(j_first, b0, nblocks, key, out);
    else
      noise_fill_tile<false>(j_first, b0, nblocks, key, out);
  }
}

// out[4t .. 4t+3] = Philox words of block block_base + t. Even and odd blocks
// go through the two implementations of the rounds (general, and with the
// per-tile constants of philox_tile); they give identical words, and this lets
// a bit-exact check of this output cover both.
__global__ void __launch_bounds__(kBlockThreads)
noise_bits_kernel(uint64_t block_base, uint64_t nblocks, PhiloxKey key, uint4* __restrict__ out) {
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * blockDim.x;
  for (uint64_t t = static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < nblocks;
       t += stride) {
    const uint64_t j = block_base + t;
    out[t] = (j & 1) ? philox_block_tile(static_cast<uint32_t>(j),
                                         philox_tile(static_cast<uint32_t>(j >> 32), key))
                     : philox_block(j, key);
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
cudaError_t launch_axpy_io(const PlanView& plan, PhiloxKey key, float scale, PhiloxKey key2,
                           float scale2, cudaStream_t stream) {
  auto k = axpy_noise_kernel<Io, kTwo, kSame>;
  k<<<persistent_grid(k, plan.total_tiles), kBlockThreads, 0, stream>>>(
      plan.segs, plan.inv_scale, plan.total_tiles, key, scale, key2, scale2);
  return cudaGetLastError();
}

template <bool kTwo, bool kSame>
cudaError_t launch_axpy(const PlanView& plan, PhiloxKey key, float scale, PhiloxKey key2,
                        float scale2, cudaStream_t stream) {
  if (plan.dtype == ES_BF16)
    return launch_axpy_io<Bf16Io, kTwo, kSame>(plan, key, scale, key2, scale2, stream);
  if (plan.dtype == ES_FP8_E4M3)
    return launch_axpy_io<Fp8Io, kTwo, kSame>(plan, key, scale, key2, scale2, stream);
  return launch_axpy_io<F32Io, kTwo, kSame>(plan, key, scale, key2, scale2, stream);
}

}  // namespace

cudaError_t launch_axpy_noise(const PlanView& plan, uint64_t seed, float scale,
                              cudaStream_t stream) {
  return launch_axpy<false, false>(plan, philox_key(seed), scale, PhiloxKey{0u, 0u}, 0.0f,
                                   stream);
}

cudaError_t launch_axpy_noise2(const PlanView& plan, uint64_t seed, float scale, uint64_t seed2,
                               float scale2, cudaStream_t stream) {
  if (seed == seed2)
    return launch_axpy<true, true>(plan, philox_key(seed), scale, philox_key(seed2), scale2,
                                   stream);
  return launch_axpy<true, false>(plan, philox_key(seed), scale, philox_key(seed2), scale2,
                                  stream);
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
  noise_bits_kernel<<<grid, kBlockThreads, 0, stream>>>(block_base, nblocks, philox_key(seed),
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
    noise_fill_vec_kernel<<<grid, kBlockThreads, 0, stream>>>(index_base / 4, full, key,
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
