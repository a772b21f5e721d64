// Register-only throughput probes of the SM pipes that bound the noise
// generator (a measurement tool behind `bench.py --pipe-peaks`; not part of the
// ES-step library and not linked into it).
//
// Every probe runs `iters` iterations of a fixed instruction pattern on
// independent dependency chains held in registers: no memory traffic besides
// one timing record per CTA. Each CTA times itself in SM clock cycles
// (clock64) and in nanoseconds (globaltimer), so a rate comes out per SM per
// clock, independent of the clock the GPU happened to run at.
//
// Probes:
//   single pipes   mad.wide.u32 (the 32x32->64-bit product of each Philox
//                  round), mad.hi.u32, mad.lo.u32, lop3 (the round's
//                  three-input XOR), fma.rn.f32, packed fma.rn.f32x2, and MUFU
//                  lg2/ex2 pairs (the transcendental unit Box-Muller uses);
//   mixes          two pipes interleaved in one thread, in fixed ratios; the
//                  ratio 9 products : 4 MUFU is the generator's (18 products
//                  and 8 transcendentals per Philox block of 4 Gaussians), with
//                  each product as one mad.wide.u32 or as a mad.hi.u32 +
//                  mad.lo.u32 pair (the form the library uses);
//   warp split     even warps run mad.wide chains and odd warps MUFU chains
//                  (or only one half runs): whether the two pipes overlap at
//                  all when their instructions come from different warps;
//   generator      the library's own Philox4x32-10 (es_noise.cuh) in blocks,
//                  and the full generator in Gaussians in the form the
//                  streaming kernels use (scheduled round keys, packed
//                  transform, near-one series on a rare branch).
#include <cuda_runtime.h>

#include <cstdint>

#include "es_noise.cuh"

namespace {

constexpr int kThreads = 256;
constexpr uint32_t kMul = 0xD2511F53u;

enum Probe : int {
  kImadWide = 0,
  kImadHi,
  kImadLo,
  kLop3,
  kFfma,
  kFfma2,
  kMufu,
  kMixImadMufu,
  kMixImadFfma,
  kMixImadLop3,
  kMixMufuFfma,
  kMixHiLo,
  kMixHiLoMufu,
  kSplitImad,
  kSplitMufu,
  kSplitBoth,
  kPhilox,
  kGenerator,
  kImadWideMul,
  kGeneratorPipelined,
  kGeneratorSplit,
  kProbeCount
};

// Name, unit of one op, ops per active thread per iteration, and the share of
// threads that run (the split probes use half of the warps).
struct ProbeInfo {
  const char* name;
  const char* unit;
  double ops_per_iter;
  double active;
};

// The MUFU half of a split probe runs iters / kSplitMufuDiv iterations, which
// makes both halves take about as long when run alone.
constexpr int kSplitMufuDiv = 4;

const ProbeInfo kInfo[kProbeCount] = {
    {"imad_wide", "mad.wide.u32", 8, 1},
    {"imad_hi", "mad.hi.u32", 8, 1},
    {"imad_lo", "mad.lo.u32", 8, 1},
    {"lop3", "lop3.b32", 8, 1},
    {"ffma", "fma.rn.f32", 8, 1},
    {"ffma2", "fma.rn.f32x2 (2 lanes)", 8, 1},
    {"mufu", "MUFU lg2 or ex2", 16, 1},
    {"mix_imad_wide_mufu_9_4", "mad.wide.u32 (with 4 MUFU per 9)", 9, 1},
    {"mix_imad_wide_ffma_1_2", "mad.wide.u32 (with 2 fma.rn.f32 each)", 8, 1},
    {"mix_imad_wide_lop3_1_1", "mad.wide.u32 (with 1 lop3.b32 each)", 8, 1},
    {"mix_mufu_ffma_1_4", "MUFU (with 4 fma.rn.f32 each)", 8, 1},
    {"mix_imad_hi_lo_1_1", "mad.hi.u32 + mad.lo.u32 pair", 8, 1},
    {"mix_imad_hi_lo_mufu_9_4", "mad.hi.u32 + mad.lo.u32 pair (with 4 MUFU per 9)", 9, 1},
    {"split_imad_wide_only", "mad.wide.u32 (even warps; odd warps idle)", 8, 0.5},
    {"split_mufu_only", "MUFU (odd warps; even warps idle)", 16.0 / kSplitMufuDiv, 0.5},
    {"split_both", "warp-iterations (even warps mad.wide, odd warps MUFU)", 1, 1},
    {"philox", "Philox4x32-10 block (round keys from the launch's parameters)", 2, 1},
    {"generator", "Gaussian (Philox4x32-10 + Box-Muller)", 8, 1},
    {"imad_wide_mul", "mul.wide.u32 by a constant (no addend), with one add each", 8, 1},
    {"generator_pipelined",
     "Gaussian (two seeds alternating, the next one's Philox beside the current transform)", 16,
     1},
    {"generator_split",
     "Gaussian (Philox on warps 0-3, Box-Muller on warps 4-7, warp pairs through shared memory)",
     8, 0.5},
};

// Shared-memory slots of the split generator probe, and the most polls of an
// mbarrier before a wait gives up (the probe then stops and reports it).
constexpr int kSplitStages = 8;
constexpr int kWaitPolls = 1 << 20;

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint64_t* bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(bar)), "r"(count)
               : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint64_t* bar) {
  uint64_t state;
  asm volatile("mbarrier.arrive.shared::cta.b64 %0, [%1];"
               : "=l"(state)
               : "r"(smem_u32(bar))
               : "memory");
}
// Waits for the completion of the barrier's phase of the given parity; false
// if it has not completed after kWaitPolls polls.
__device__ __forceinline__ bool mbar_wait(uint64_t* bar, uint32_t parity) {
  for (int n = 0; n < kWaitPolls; ++n) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(smem_u32(bar)), "r"(parity)
        : "memory");
    if (done) return true;
  }
  return false;
}

__device__ __forceinline__ uint64_t mad_wide(uint32_t a, uint64_t c) {
  uint64_t d;
  asm volatile("mad.wide.u32 %0, %1, %2, %3;" : "=l"(d) : "r"(a), "r"(kMul), "l"(c));
  return d;
}
__device__ __forceinline__ uint32_t mad_hi(uint32_t a, uint32_t c) {
  uint32_t d;
  asm volatile("mad.hi.u32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(kMul), "r"(c));
  return d;
}
__device__ __forceinline__ uint32_t mad_lo(uint32_t a, uint32_t c) {
  uint32_t d;
  asm volatile("mad.lo.u32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(kMul), "r"(c));
  return d;
}
__device__ __forceinline__ uint32_t xor3(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t d;
  asm volatile("lop3.b32 %0, %1, %2, %3, 0x96;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}
__device__ __forceinline__ float ffma(float a, float b, float c) {
  float d;
  asm volatile("fma.rn.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}
// ex2(lg2(a)): two MUFU operations that return (about) a, so the chain stays
// finite and positive for any number of iterations.
__device__ __forceinline__ float mufu2(float a) {
  float l, e;
  asm volatile("lg2.approx.ftz.f32 %0, %1;" : "=f"(l) : "f"(a));
  asm volatile("ex2.approx.ftz.f32 %0, %1;" : "=f"(e) : "f"(l));
  return e;
}

// Round-key schedules of two seeds, passed as a __grid_constant__ parameter as
// the perturb/restore kernels pass theirs: every round key is a constant-bank
// operand, so the generator probes run the kernels' instruction stream.
struct ProbeKeys {
  esopt::PhiloxSched s[2];
};

template <int P>
__global__ void __launch_bounds__(kThreads)
probe_kernel(int iters, uint32_t seed, unsigned long long* __restrict__ rec,
             uint32_t* __restrict__ sink, const __grid_constant__ ProbeKeys keys) {
  const uint32_t t = seed + threadIdx.x * 0x9E3779B9u + blockIdx.x;
  uint64_t w[9];
  uint32_t x[8], y[8];
  float f[8], m[4];
  float2 f2[8];
#pragma unroll
  for (int k = 0; k < 9; ++k) w[k] = t * (2u * k + 1u);
#pragma unroll
  for (int k = 0; k < 8; ++k) {
    x[k] = t + 977u * k;
    y[k] = t ^ (0x85EBCA6Bu * k);
    f[k] = 1.0f + (t & 0xFFu) * 1e-4f + k * 1e-3f;
    f2[k] = make_float2(f[k], f[k] + 0.5f);
  }
#pragma unroll
  for (int k = 0; k < 4; ++k) m[k] = 1.5f + (t & 0xFFu) * 1e-3f + k * 0.25f;
  const float fb = 0.999f + (seed & 1) * 1e-7f, fc = 1e-3f * (seed & 3);
  const int warp = threadIdx.x >> 5;

  __syncthreads();
  unsigned long long c0 = 0, n0 = 0;
  if (threadIdx.x == 0) {
    c0 = clock64();
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(n0));
  }

  if constexpr (P == kImadWide || P == kSplitImad) {
    if (P == kImadWide || (warp & 1) == 0) {
#pragma unroll 1
      for (int i = 0; i < iters; ++i)
#pragma unroll
        for (int k = 0; k < 8; ++k) w[k] = mad_wide(static_cast<uint32_t>(w[k]), w[k]);
    }
  } else if constexpr (P == kImadHi) {
#pragma unroll 1
    for (int i = 0; i < iters; ++i)
#pragma unroll
      for (int k = 0; k < 8; ++k) x[k] = mad_hi(x[k], y[k]);
  } else if constexpr (P == kImadLo) {
#pragma unroll 1
    for (int i = 0; i < iters; ++i)
#pragma unroll
      for (int k = 0; k < 8; ++k) x[k] = mad_lo(x[k], y[k]);
  } else if constexpr (P == kLop3) {
#pragma unroll 1
    for (int i = 0; i < iters; ++i)
#pragma unroll
      for (int k = 0; k < 8; ++k) x[k] = xor3(x[k], y[k], x[(k + 1) & 7]);
  } else if constexpr (P == kFfma) {
#pragma unroll 1
    for (int i = 0; i < iters; ++i)
#pragma unroll
      for (int k = 0; k < 8; ++k) f[k] = ffma(f[k], fb, fc);
  } else if constexpr (P == kFfma2) {
    const float2 b2 = make_float2(fb, fb), c2 = make_float2(fc, fc);
#pragma unroll 1
    for (int i = 0; i < iters; ++i)
#pragma unroll
      for (int k = 0; k < 8; ++k) f2[k] = __ffma2_rn(f2[k], b2, c2);
  } else if constexpr (P == kMufu || P == kSplitMufu) {
    if (P == kMufu || (warp & 1) == 1) {
      const int n = P == kMufu ? iters : iters / kSplitMufuDiv;
#pragma unroll 1
      for (int i = 0; i < n; ++i)
#pragma unroll
        for (int k = 0; k < 8; ++k) f[k] = mufu2(f[k]);
    }
  } else if constexpr (P == kSplitBoth) {
    if ((warp & 1) == 0) {
#pragma unroll 1
      for (int i = 0; i < iters; ++i)
#pragma unroll
        for (int k = 0; k < 8; ++k) w[k] = mad_wide(static_cast<uint32_t>(w[k]), w[k]);
    } else {
#pragma unroll 1
      for (int i = 0; i < iters / kSplitMufuDiv; ++i)
#pragma unroll
        for (int k = 0; k < 8; ++k) f[k] = mufu2(f[k]);
    }
  } else if constexpr (P == kMixImadMufu) {
#pragma unroll 1
    for (int i = 0; i < iters; ++i) {
#pragma unroll
      for (int k = 0; k < 9; ++k) w[k] = mad_wide(static_cast<uint32_t>(w[k]), w[k]);
      m[0] = mufu2(m[0]);
      m[1] = mufu2(m[1]);
    }
  } else if constexpr (P == kMixImadFfma) {
#pragma unroll 1
    for (int i = 0; i < iters; ++i) {
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        w[k] = mad_wide(static_cast<uint32_t>(w[k]), w[k]);
        f[k] = ffma(ffma(f[k], fb, fc), fb, fc);
      }
    }
  } else if constexpr (P == kMixImadLop3) {
#pragma unroll 1
    for (int i = 0; i < iters; ++i) {
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        w[k] = mad_wide(static_cast<uint32_t>(w[k]), w[k]);
        x[k] = xor3(x[k], y[k], x[(k + 1) & 7]);
      }
    }
  } else if constexpr (P == kMixMufuFfma) {
#pragma unroll 1
    for (int i = 0; i < iters; ++i) {
#pragma unroll
      for (int k = 0; k < 4; ++k) m[k] = mufu2(m[k]);
#pragma unroll
      for (int k = 0; k < 8; ++k) f[k] = ffma(ffma(ffma(ffma(f[k], fb, fc), fb, fc), fb, fc), fb, fc);
    }
  } else if constexpr (P == kMixHiLo) {
#pragma unroll 1
    for (int i = 0; i < iters; ++i) {
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        x[k] = mad_hi(x[k], y[(k + 3) & 7]);
        y[k] = mad_lo(y[k], x[(k + 5) & 7]);
      }
    }
  } else if constexpr (P == kMixHiLoMufu) {
#pragma unroll 1
    for (int i = 0; i < iters; ++i) {
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        x[k] = mad_hi(x[k], y[(k + 3) & 7]);
        y[k] = mad_lo(y[k], x[(k + 5) & 7]);
      }
      w[8] = (static_cast<uint64_t>(mad_hi(static_cast<uint32_t>(w[8]), x[0])) << 32) |
             mad_lo(static_cast<uint32_t>(w[8] >> 32), y[0]);
      m[0] = mufu2(m[0]);
      m[1] = mufu2(m[1]);
    }
  } else if constexpr (P == kPhilox) {
    // the kernels' Philox alone: round keys from the launch's parameters
    const esopt::PhiloxSched& ps = keys.s[0];
    const esopt::TileConst tc = esopt::tile_const(0u, ps.rk[0], ps.rk[3]);
    uint32_t j = t * 2u;
#pragma unroll 1
    for (int i = 0; i < iters; ++i) {
      const uint4 a = esopt::philox_block_rk<false>(j, tc, ps.rk[1], ps.rk[2], ps.rk + 4);
      const uint4 b = esopt::philox_block_rk<false>(j + 1u, tc, ps.rk[1], ps.rk[2], ps.rk + 4);
      x[0] ^= a.x ^ b.x;
      x[1] ^= a.y ^ b.y;
      x[2] ^= a.z ^ b.z;
      x[3] ^= a.w ^ b.w;
      j += 0x20000u;
    }
  } else if constexpr (P == kImadWideMul) {
    // Philox's form: the product by a constant without an addend; the high
    // word feeds the chain, the low word an accumulator (one add on the ALU)
#pragma unroll 1
    for (int i = 0; i < iters; ++i)
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        uint32_t hi, lo;
        asm volatile("{\n\t.reg .u64 p;\n\tmul.wide.u32 p, %2, %3;\n\tmov.b64 {%1, %0}, p;\n\t}"
                     : "=r"(hi), "=r"(lo) : "r"(x[k]), "n"(kMul));
        x[k] = hi;
        y[k] += lo;
      }
  } else if constexpr (P == kGenerator) {
    // the kernels' generator: round keys from the launch's parameters, the
    // packed transform from the hardware log2, the near-one series on a rare
    // branch, then the square roots
    const esopt::PhiloxSched& ps = keys.s[0];
    const esopt::TileConst tc = esopt::tile_const(0u, ps.rk[0], ps.rk[3]);
    uint32_t j = t * 2u;
    float2 s0 = make_float2(0.f, 0.f), s1 = s0;
#pragma unroll 1
    for (int i = 0; i < iters; ++i) {
      uint2 xa[2];
      esopt::Polar2 p[2];
#pragma unroll
      for (int b = 0; b < 2; ++b) {
        const uint4 x = esopt::philox_block_rk<false>(j + b, tc, ps.rk[1], ps.rk[2], ps.rk + 4);
        xa[b] = make_uint2(x.x, x.z);
        p[b] = esopt::polar2_sq<true>(x);
      }
      esopt::fix_near_one<2>(xa, p);
#pragma unroll
      for (int b = 0; b < 2; ++b) {
        const float2 r = make_float2(esopt::sqrt_approx(p[b].r.x), esopt::sqrt_approx(p[b].r.y));
        s0 = __ffma2_rn(make_float2(r.x, r.x), make_float2(p[b].c.x, p[b].s.x), s0);
        s1 = __ffma2_rn(make_float2(r.y, r.y), make_float2(p[b].c.y, p[b].s.y), s1);
      }
      j += 0x20000u;
    }
    f[0] = s0.x + s0.y + s1.x + s1.y;
  } else if constexpr (P == kGeneratorPipelined) {
    // the update's seed loop in registers: the blocks of two seeds alternate,
    // and the next seed's Philox words are computed in the same basic block
    // as the current seed's transform, on alternating word buffers
    const esopt::PhiloxSched& ps0 = keys.s[0];
    const esopt::PhiloxSched& ps1 = keys.s[1];
    const esopt::TileConst tc0 = esopt::tile_const(0u, ps0.rk[0], ps0.rk[3]);
    const esopt::TileConst tc1 = esopt::tile_const(0u, ps1.rk[0], ps1.rk[3]);
    uint32_t j = t * 2u;
    float2 s0 = make_float2(0.f, 0.f), s1 = s0;
    auto words = [&](const esopt::PhiloxSched& ps, const esopt::TileConst& tc, uint32_t jj,
                     uint4 (&x)[2]) {
#pragma unroll
      for (int b = 0; b < 2; ++b)
        x[b] = esopt::philox_block_rk<false>(jj + b, tc, ps.rk[1], ps.rk[2], ps.rk + 4);
    };
    auto transform = [&](const uint4 (&x)[2]) {
      uint2 xa[2];
      esopt::Polar2 p[2];
#pragma unroll
      for (int b = 0; b < 2; ++b) {
        xa[b] = make_uint2(x[b].x, x[b].z);
        p[b] = esopt::polar2_sq<true>(x[b]);
      }
      esopt::fix_near_one<2>(xa, p);
#pragma unroll
      for (int b = 0; b < 2; ++b) {
        const float2 r = make_float2(esopt::sqrt_approx(p[b].r.x), esopt::sqrt_approx(p[b].r.y));
        s0 = __ffma2_rn(make_float2(r.x, r.x), make_float2(p[b].c.x, p[b].s.x), s0);
        s1 = __ffma2_rn(make_float2(r.y, r.y), make_float2(p[b].c.y, p[b].s.y), s1);
      }
    };
    uint4 xa0[2], xb0[2];
    words(ps0, tc0, j, xa0);
#pragma unroll 1
    for (int i = 0; i < iters; ++i) {
      words(ps1, tc1, j, xb0);
      transform(xa0);
      j += 0x20000u;
      words(ps0, tc0, j, xa0);
      transform(xb0);
    }
    f[0] = s0.x + s0.y + s1.x + s1.y + __uint_as_float(xa0[0].x & 0x3F000000u);
  } else if constexpr (P == kGeneratorSplit) {
    // Philox and Box-Muller on separate warps: producer warp w (0-3) writes
    // the words of two blocks per thread and iteration into its own ring of
    // kSplitStages shared slots, consumer warp w + 4 transforms them. Each
    // slot of a pair is handed over by mbarriers of 32 arrivals: full when
    // the producer warp has written it, empty when the consumer warp has read
    // it. Both warps of a pair run the same iterations in the same slot
    // order; every wait is bounded, and a thread whose wait gives up stops
    // (its partner's waits then give up too) and flags it in sink[1].
    __shared__ uint4 ring[kSplitStages][4][32][2];
    __shared__ uint64_t full_bar[kSplitStages][4], empty_bar[kSplitStages][4];
    if (threadIdx.x < 4 * kSplitStages) {
      mbar_init(&full_bar[threadIdx.x / 4][threadIdx.x % 4], 32);
      mbar_init(&empty_bar[threadIdx.x / 4][threadIdx.x % 4], 32);
    }
    __syncthreads();
    const int pair = (threadIdx.x >> 5) & 3, lane = threadIdx.x & 31;
    bool ok = true;
    if (threadIdx.x < 128) {
      const esopt::PhiloxSched& ps = keys.s[0];
      const esopt::TileConst tc = esopt::tile_const(0u, ps.rk[0], ps.rk[3]);
      uint32_t j = t * 2u;
#pragma unroll 1
      for (int i = 0; i < iters; ++i) {
        const int st = i % kSplitStages;
        const uint32_t use = static_cast<uint32_t>(i / kSplitStages);
        if (use > 0 && !mbar_wait(&empty_bar[st][pair], (use - 1) & 1u)) {
          ok = false;
          break;
        }
        ring[st][pair][lane][0] =
            esopt::philox_block_rk<false>(j, tc, ps.rk[1], ps.rk[2], ps.rk + 4);
        ring[st][pair][lane][1] =
            esopt::philox_block_rk<false>(j + 1u, tc, ps.rk[1], ps.rk[2], ps.rk + 4);
        mbar_arrive(&full_bar[st][pair]);
        j += 0x20000u;
      }
    } else {
      float2 s0 = make_float2(0.f, 0.f), s1 = s0;
#pragma unroll 1
      for (int i = 0; i < iters; ++i) {
        const int st = i % kSplitStages;
        const uint32_t use = static_cast<uint32_t>(i / kSplitStages);
        if (!mbar_wait(&full_bar[st][pair], use & 1u)) {
          ok = false;
          break;
        }
        const uint4 x0 = ring[st][pair][lane][0], x1 = ring[st][pair][lane][1];
        // the slot is free again; its last use needs no release
        if (i + kSplitStages < iters) mbar_arrive(&empty_bar[st][pair]);
        uint2 xa[2] = {make_uint2(x0.x, x0.z), make_uint2(x1.x, x1.z)};
        esopt::Polar2 p[2] = {esopt::polar2_sq<true>(x0), esopt::polar2_sq<true>(x1)};
        esopt::fix_near_one<2>(xa, p);
#pragma unroll
        for (int b = 0; b < 2; ++b) {
          const float2 r =
              make_float2(esopt::sqrt_approx(p[b].r.x), esopt::sqrt_approx(p[b].r.y));
          s0 = __ffma2_rn(make_float2(r.x, r.x), make_float2(p[b].c.x, p[b].s.x), s0);
          s1 = __ffma2_rn(make_float2(r.y, r.y), make_float2(p[b].c.y, p[b].s.y), s1);
        }
      }
      f[0] = s0.x + s0.y + s1.x + s1.y;
    }
    if (!ok) sink[1] = 1u;
  }

  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned long long n1;
    const unsigned long long c1 = clock64();
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(n1));
    unsigned int smid;
    asm volatile("mov.u32 %0, %%smid;" : "=r"(smid));
    rec[4 * blockIdx.x] = c0;
    rec[4 * blockIdx.x + 1] = c1;
    rec[4 * blockIdx.x + 2] = n1 - n0;
    rec[4 * blockIdx.x + 3] = smid;
  }
  // Fold every chain into one word so that no chain is dead code; the store
  // happens only for a value that depends on all of them and the seed.
  uint32_t s = 0;
#pragma unroll
  for (int k = 0; k < 9; ++k) s ^= static_cast<uint32_t>(w[k] ^ (w[k] >> 32));
#pragma unroll
  for (int k = 0; k < 8; ++k)
    s ^= x[k] ^ y[k] ^ __float_as_uint(f[k]) ^ __float_as_uint(f2[k].x) ^ __float_as_uint(f2[k].y);
#pragma unroll
  for (int k = 0; k < 4; ++k) s ^= __float_as_uint(m[k]);
  if (s == seed * 0x2545F491u + 0x1234567u) sink[0] = s;
}

template <int P>
void* kernel_of() {
  return reinterpret_cast<void*>(probe_kernel<P>);
}

void* const kKernels[kProbeCount] = {
    kernel_of<0>(),  kernel_of<1>(),  kernel_of<2>(),  kernel_of<3>(),
    kernel_of<4>(),  kernel_of<5>(),  kernel_of<6>(),  kernel_of<7>(),
    kernel_of<8>(),  kernel_of<9>(),  kernel_of<10>(), kernel_of<11>(),
    kernel_of<12>(), kernel_of<13>(), kernel_of<14>(), kernel_of<15>(),
    kernel_of<16>(), kernel_of<17>(), kernel_of<18>(), kernel_of<19>(),
    kernel_of<20>(),
};

}  // namespace

extern "C" {

int esprobe_count(void) { return kProbeCount; }

const char* esprobe_name(int probe) {
  return probe >= 0 && probe < kProbeCount ? kInfo[probe].name : "";
}

const char* esprobe_unit(int probe) {
  return probe >= 0 && probe < kProbeCount ? kInfo[probe].unit : "";
}

// Runs probe `probe` on the current device with ctas_per_sm CTAs of 256
// threads on every SM (all resident at once; fewer if the probe's registers
// allow fewer) for `iters` iterations, after one untimed launch.
// An SM's time is the span of its own SM clock (clock64) from the first of its
// CTAs to start to the last to finish: the CTAs of one SM neither start nor end
// together, so a CTA's own duration would overstate the SM's rate.
// out[0..6] = milliseconds (CUDA events), mean SM cycles per SM (that span),
// SM clock in MHz (CTA cycles / globaltimer ns), ops per clock per SM, ops in
// total, active threads per SM, CTAs per SM used. Returns 0, -1 for a bad
// argument, -2 if a bounded wait of the split probe gave up, else the
// cudaError_t.
int esprobe_run(int probe, int ctas_per_sm, int iters, double* out) {
  if (probe < 0 || probe >= kProbeCount || ctas_per_sm < 1 || iters < 1 || out == nullptr)
    return -1;
  int dev = 0, sms = 0, fit = 0;
  cudaError_t err = cudaGetDevice(&dev);
  if (err == cudaSuccess) err = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (err == cudaSuccess)
    err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&fit, kKernels[probe], kThreads, 0);
  if (err != cudaSuccess) return static_cast<int>(err);
  if (fit < 1) return -1;
  if (fit < ctas_per_sm) ctas_per_sm = fit;
  const int grid = sms * ctas_per_sm;
  unsigned long long* rec = nullptr;
  uint32_t* sink = nullptr;
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  err = cudaMalloc(&rec, sizeof(unsigned long long) * 4 * grid);
  if (err == cudaSuccess) err = cudaMalloc(&sink, 2 * sizeof(uint32_t));
  if (err == cudaSuccess) err = cudaMemset(sink, 0, 2 * sizeof(uint32_t));
  if (err == cudaSuccess) err = cudaEventCreate(&e0);
  if (err == cudaSuccess) err = cudaEventCreate(&e1);
  unsigned long long* host = new unsigned long long[4 * grid];
  float ms = 0.0f;
  bool waits_gave_up = false;
  if (err == cudaSuccess) {
    uint32_t seed = 0x51ED270Bu;
    ProbeKeys keys;
    keys.s[0] = esopt::philox_sched(seed);
    keys.s[1] = esopt::philox_sched(seed + 1u);
    int warm_iters = iters / 8 > 0 ? iters / 8 : 1;
    void* warm[] = {&warm_iters, &seed, &rec, &sink, &keys};
    err = cudaLaunchKernel(kKernels[probe], dim3(grid), dim3(kThreads), warm, 0, 0);
    if (err == cudaSuccess) err = cudaEventRecord(e0, 0);
    void* args[] = {&iters, &seed, &rec, &sink, &keys};
    if (err == cudaSuccess)
      err = cudaLaunchKernel(kKernels[probe], dim3(grid), dim3(kThreads), args, 0, 0);
    if (err == cudaSuccess) err = cudaEventRecord(e1, 0);
    if (err == cudaSuccess) err = cudaEventSynchronize(e1);
    if (err == cudaSuccess) err = cudaEventElapsedTime(&ms, e0, e1);
    if (err == cudaSuccess)
      err = cudaMemcpy(host, rec, sizeof(unsigned long long) * 4 * grid, cudaMemcpyDeviceToHost);
    uint32_t gave_up = 0;
    if (err == cudaSuccess)
      err = cudaMemcpy(&gave_up, sink + 1, sizeof(uint32_t), cudaMemcpyDeviceToHost);
    if (err == cudaSuccess && gave_up != 0) waits_gave_up = true;
  }
  if (err == cudaSuccess) {
    // per SM: [first start, last end] on its own clock (%smid may exceed the
    // SM count: ids need not be contiguous)
    constexpr int kMaxSmId = 4096;
    unsigned long long* first = new unsigned long long[kMaxSmId];
    unsigned long long* last = new unsigned long long[kMaxSmId];
    for (int k = 0; k < kMaxSmId; ++k) {
      first[k] = ~0ull;
      last[k] = 0ull;
    }
    double cta_cyc = 0.0, ns = 0.0;
    for (int b = 0; b < grid; ++b) {
      const unsigned long long c0 = host[4 * b], c1 = host[4 * b + 1];
      const int sm = static_cast<int>(host[4 * b + 3]);
      cta_cyc += static_cast<double>(c1 - c0);
      ns += static_cast<double>(host[4 * b + 2]);
      if (sm >= 0 && sm < kMaxSmId) {
        if (c0 < first[sm]) first[sm] = c0;
        if (c1 > last[sm]) last[sm] = c1;
      }
    }
    double cyc = 0.0;
    int used = 0;
    for (int k = 0; k < kMaxSmId; ++k)
      if (last[k] > first[k]) {
        cyc += static_cast<double>(last[k] - first[k]);
        ++used;
      }
    const double sum_spans = cyc > 0.0 ? cyc : 1.0;
    cyc = used > 0 ? cyc / used : 1.0;
    delete[] first;
    delete[] last;
    const double threads_per_sm = static_cast<double>(ctas_per_sm) * kThreads;
    const double ops = kInfo[probe].ops_per_iter * iters * threads_per_sm * kInfo[probe].active;
    out[0] = ms;
    out[1] = cyc;
    out[2] = ns > 0.0 ? cta_cyc / ns * 1e3 : 0.0;
    out[3] = ops * sms / sum_spans;  // every CTA's ops over every SM's span
    out[4] = ops * sms;
    out[5] = threads_per_sm * kInfo[probe].active;
    out[6] = ctas_per_sm;
  }
  delete[] host;
  if (e0) cudaEventDestroy(e0);
  if (e1) cudaEventDestroy(e1);
  cudaFree(rec);
  cudaFree(sink);
  if (err == cudaSuccess && waits_gave_up) return -2;
  return static_cast<int>(err);
}

}  // extern "C"
