// sm_103a kernels of the ES step: in-place perturb/restore (theta += s eps) and
// the fused N-seed update (theta += sum_i c_i eps_i), plus a noise fill.
//
// All three stream the parameter set once per launch. Work is cut into tiles
// of kBlockThreads * kVecsPerThread 16-byte vectors that never straddle a
// segment; persistent CTAs walk the tiles in grid-stride order, so consecutive
// CTAs touch consecutive memory and each CTA advances through the segment table
// monotonically (one table lookup per tile, no per-element search).
// Every element is owned by exactly one thread: no atomics, no shared state
// between threads except the staged seeds of the update.
#include <cuda_bf16.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "es_internal.h"
#include "es_noise.cuh"

namespace esopt {
namespace {

// 16-byte vector <-> fp32 registers, and single-element access for tails.
struct Bf16Io {
  static constexpr int kVec = 8;
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
  __device__ static void round_trip(float (&f)[8]) {
#pragma unroll
    for (int k = 0; k < 8; k += 2) {
      const uint32_t w = pack2(f[k], f[k + 1]);
      f[k] = __uint_as_float(w << 16);
      f[k + 1] = __uint_as_float(w & 0xFFFF0000u);
    }
  }
  __device__ static float round_trip1(float f) { return to_f32(from_f32(f)); }
  // Gaussians of the 8 elements starting at global index g0 (g0 % 8 == 0).
  __device__ static void noise(uint64_t g0, PhiloxKey key, float (&e)[8]) {
    const uint64_t j = g0 >> 2;
    const float4 a = gaussian4(j, key);
    const float4 b = gaussian4(j + 1, key);
    e[0] = a.x; e[1] = a.y; e[2] = a.z; e[3] = a.w;
    e[4] = b.x; e[5] = b.y; e[6] = b.z; e[7] = b.w;
  }
};

struct F32Io {
  static constexpr int kVec = 4;
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
  __device__ static void round_trip(float (&)[4]) {}
  __device__ static float round_trip1(float f) { return f; }
  __device__ static void noise(uint64_t g0, PhiloxKey key, float (&e)[4]) {
    const float4 a = gaussian4(g0 >> 2, key);
    e[0] = a.x; e[1] = a.y; e[2] = a.z; e[3] = a.w;
  }
};

// Segment of `tile`; `seg` is the CTA's cursor and only moves forward.
__device__ __forceinline__ const SegDesc* find_segment(const SegDesc* __restrict__ segs,
                                                       int& seg, uint64_t tile) {
  while (tile >= segs[seg + 1].tile_begin) ++seg;
  return segs + seg;
}

// theta[g] <- round(theta[g] + scale * eps_seed[g]) over every segment; with
// kTwo, a second step round(. + scale2 * eps_seed2[g]) follows in registers,
// after the first result has been rounded to the storage type exactly as a
// separate launch would store it (restore of one member fused with the
// perturb of the next).
template <class Io, bool kTwo>
__global__ void __launch_bounds__(kBlockThreads)
axpy_noise_kernel(const SegDesc* __restrict__ segs, uint64_t total_tiles, PhiloxKey key,
                  float scale, PhiloxKey key2, float scale2) {
  constexpr int V = Io::kVec;
  constexpr uint64_t kTile = static_cast<uint64_t>(kBlockThreads) * kVecsPerThread * V;
  using S = typename Io::Scalar;
  int seg = 0;
  for (uint64_t tile = blockIdx.x; tile < total_tiles; tile += gridDim.x) {
    const SegDesc* d = find_segment(segs, seg, tile);
    S* const base = static_cast<S*>(d->data);
    const uint64_t numel = d->numel;
    const uint64_t index_base = d->index_base;
    const uint64_t t0 = (tile - d->tile_begin) * kTile;

    uint4 v[kVecsPerThread];
#pragma unroll
    for (int u = 0; u < kVecsPerThread; ++u) {
      const uint64_t e = t0 + static_cast<uint64_t>(u * kBlockThreads + threadIdx.x) * V;
      if (e + V <= numel) v[u] = *reinterpret_cast<const uint4*>(base + e);
    }
#pragma unroll
    for (int u = 0; u < kVecsPerThread; ++u) {
      const uint64_t e = t0 + static_cast<uint64_t>(u * kBlockThreads + threadIdx.x) * V;
      if (e >= numel) continue;
      float eps[V];
      Io::noise(index_base + e, key, eps);
      if (e + V <= numel) {
        float f[V];
        Io::unpack(v[u], f);
#pragma unroll
        for (int k = 0; k < V; ++k) f[k] = fmaf(scale, eps[k], f[k]);
        if (kTwo) {
          Io::round_trip(f);
          Io::noise(index_base + e, key2, eps);
#pragma unroll
          for (int k = 0; k < V; ++k) f[k] = fmaf(scale2, eps[k], f[k]);
        }
        *reinterpret_cast<uint4*>(base + e) = Io::pack(f);
      } else {  // ragged end of a segment
        const int rem = static_cast<int>(numel - e);
        float f[V];
#pragma unroll
        for (int k = 0; k < V; ++k)
          f[k] = k < rem ? fmaf(scale, eps[k], Io::to_f32(base[e + k])) : 0.0f;
        if (kTwo) {
          Io::noise(index_base + e, key2, eps);
#pragma unroll
          for (int k = 0; k < V; ++k) f[k] = fmaf(scale2, eps[k], Io::round_trip1(f[k]));
        }
#pragma unroll
        for (int k = 0; k < V; ++k)
          if (k < rem) base[e + k] = Io::from_f32(f[k]);
      }
    }
  }
}

// theta[g] <- round(theta[g] + sum_i c_i eps_{s_i}[g]): fp32 accumulation in
// ascending i, one rounding; theta read and written once.
template <class Io>
__global__ void __launch_bounds__(kBlockThreads)
update_kernel(const SegDesc* __restrict__ segs, uint64_t total_tiles,
              const __grid_constant__ UpdateArgs args) {
  constexpr int V = Io::kVec;
  constexpr uint64_t kTile = static_cast<uint64_t>(kBlockThreads) * kVecsPerThread * V;
  using S = typename Io::Scalar;
  __shared__ PhiloxKey s_key[ES_MAX_SEEDS];
  __shared__ float s_coeff[ES_MAX_SEEDS];
  const int n = args.n;
  for (int i = threadIdx.x; i < n; i += blockDim.x) {
    s_key[i] = PhiloxKey{args.key[i][0], args.key[i][1]};
    s_coeff[i] = args.coeff[i];
  }
  __syncthreads();

  int seg = 0;
  for (uint64_t tile = blockIdx.x; tile < total_tiles; tile += gridDim.x) {
    const SegDesc* d = find_segment(segs, seg, tile);
    S* const base = static_cast<S*>(d->data);
    const uint64_t numel = d->numel;
    const uint64_t index_base = d->index_base;
    const uint64_t t0 = (tile - d->tile_begin) * kTile;

    uint4 v[kVecsPerThread];
#pragma unroll
    for (int u = 0; u < kVecsPerThread; ++u) {
      const uint64_t e = t0 + static_cast<uint64_t>(u * kBlockThreads + threadIdx.x) * V;
      if (e + V <= numel) v[u] = *reinterpret_cast<const uint4*>(base + e);
    }
    float acc[kVecsPerThread][V];
#pragma unroll
    for (int u = 0; u < kVecsPerThread; ++u)
#pragma unroll
      for (int k = 0; k < V; ++k) acc[u][k] = 0.0f;

#pragma unroll 1
    for (int i = 0; i < n; ++i) {
      const PhiloxKey key = s_key[i];
      const float c = s_coeff[i];
#pragma unroll
      for (int u = 0; u < kVecsPerThread; ++u) {
        const uint64_t e = t0 + static_cast<uint64_t>(u * kBlockThreads + threadIdx.x) * V;
        if (e >= numel) continue;
        float eps[V];
        Io::noise(index_base + e, key, eps);
#pragma unroll
        for (int k = 0; k < V; ++k) acc[u][k] = fmaf(c, eps[k], acc[u][k]);
      }
    }

#pragma unroll
    for (int u = 0; u < kVecsPerThread; ++u) {
      const uint64_t e = t0 + static_cast<uint64_t>(u * kBlockThreads + threadIdx.x) * V;
      if (e >= numel) continue;
      if (e + V <= numel) {
        float f[V];
        Io::unpack(v[u], f);
#pragma unroll
        for (int k = 0; k < V; ++k) f[k] = f[k] + acc[u][k];
        *reinterpret_cast<uint4*>(base + e) = Io::pack(f);
      } else {
        const int rem = static_cast<int>(numel - e);
#pragma unroll
        for (int k = 0; k < V; ++k)
          if (k < rem) base[e + k] = Io::from_f32(Io::to_f32(base[e + k]) + acc[u][k]);
      }
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

// out[4t .. 4t+3] = Philox words of block block_base + t.
__global__ void __launch_bounds__(kBlockThreads)
noise_bits_kernel(uint64_t block_base, uint64_t nblocks, PhiloxKey key, uint4* __restrict__ out) {
  const uint64_t stride = static_cast<uint64_t>(gridDim.x) * blockDim.x;
  for (uint64_t t = static_cast<uint64_t>(blockIdx.x) * blockDim.x + threadIdx.x; t < nblocks;
       t += stride)
    out[t] = philox_block(block_base + t, key);
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

// Persistent grid: every SM filled to the kernel's occupancy, never more
// CTAs than tiles.
template <class K>
int persistent_grid(K kernel, uint64_t work_items) {
  int dev = 0, sms = 0, per_sm = 0;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kBlockThreads, 0);
  if (sms < 1) sms = 1;
  if (per_sm < 1) per_sm = 1;
  uint64_t grid = static_cast<uint64_t>(sms) * per_sm;
  if (work_items < grid) grid = work_items;
  return grid < 1 ? 1 : static_cast<int>(grid);
}

template <bool kTwo>
cudaError_t launch_axpy(const PlanView& plan, PhiloxKey key, float scale, PhiloxKey key2,
                        float scale2, cudaStream_t stream) {
  if (plan.dtype == ES_BF16) {
    auto k = axpy_noise_kernel<Bf16Io, kTwo>;
    k<<<persistent_grid(k, plan.total_tiles), kBlockThreads, 0, stream>>>(
        plan.segs, plan.total_tiles, key, scale, key2, scale2);
  } else {
    auto k = axpy_noise_kernel<F32Io, kTwo>;
    k<<<persistent_grid(k, plan.total_tiles), kBlockThreads, 0, stream>>>(
        plan.segs, plan.total_tiles, key, scale, key2, scale2);
  }
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_axpy_noise(const PlanView& plan, uint64_t seed, float scale,
                              cudaStream_t stream) {
  return launch_axpy<false>(plan, philox_key(seed), scale, PhiloxKey{0u, 0u}, 0.0f, stream);
}

cudaError_t launch_axpy_noise2(const PlanView& plan, uint64_t seed, float scale, uint64_t seed2,
                               float scale2, cudaStream_t stream) {
  return launch_axpy<true>(plan, philox_key(seed), scale, philox_key(seed2), scale2, stream);
}

cudaError_t launch_update(const PlanView& plan, const UpdateArgs& args, cudaStream_t stream) {
  if (plan.dtype == ES_BF16) {
    auto k = update_kernel<Bf16Io>;
    k<<<persistent_grid(k, plan.total_tiles), kBlockThreads, 0, stream>>>(
        plan.segs, plan.total_tiles, args);
  } else {
    auto k = update_kernel<F32Io>;
    k<<<persistent_grid(k, plan.total_tiles), kBlockThreads, 0, stream>>>(
        plan.segs, plan.total_tiles, args);
  }
  return cudaGetLastError();
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
  const uint64_t nblocks = ((index_base + n - 1) >> 2) - (index_base >> 2) + 1;
  const uint64_t ctas = (nblocks + kBlockThreads - 1) / kBlockThreads;
  const int grid = persistent_grid(noise_fill_kernel, ctas);
  noise_fill_kernel<<<grid, kBlockThreads, 0, stream>>>(index_base, n, philox_key(seed), out);
  return cudaGetLastError();
}

}  // namespace esopt
