// Internal interface between the C-ABI host layer (es_host.cpp) and the CUDA
// kernels (es_kernels.cu). Not part of the public ABI.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "../../include/esopt.h"

namespace esopt {

// Threads per CTA of the streaming kernels.
constexpr int kBlockThreads = 256;
// Minimum resident CTAs per SM requested from the compiler (a register cap)
// for the perturb/restore kernels and for the update kernel; 0 leaves the
// choice to the compiler.
#ifndef ES_AXPY_MIN_BLOCKS
#define ES_AXPY_MIN_BLOCKS 1
#endif
#ifndef ES_UPDATE_MIN_BLOCKS
#define ES_UPDATE_MIN_BLOCKS 0
#endif
#if ES_AXPY_MIN_BLOCKS > 0
#define ES_AXPY_BOUNDS __launch_bounds__(esopt::kBlockThreads, ES_AXPY_MIN_BLOCKS)
#else
#define ES_AXPY_BOUNDS __launch_bounds__(esopt::kBlockThreads)
#endif
#if ES_UPDATE_MIN_BLOCKS > 0
#define ES_UPDATE_BOUNDS __launch_bounds__(esopt::kBlockThreads, ES_UPDATE_MIN_BLOCKS)
#else
#define ES_UPDATE_BOUNDS __launch_bounds__(esopt::kBlockThreads)
#endif
// 16-byte vectors each thread owns per tile. All of them are processed in one
// pass: the independent Philox chains (ILP) matter more than occupancy here
// (measured: splitting into passes of 1 or 2 vectors, or 8 vectors per
// thread, were slower).
constexpr int kVecsPerThread = 4;
// Elements per 16-byte vector, per dtype.
constexpr int vec_elems(es_dtype_t dt) { return dt == ES_BF16 ? 8 : 4; }
// Elements per tile: a tile is the unit one CTA processes at a time; tiles
// never straddle segments.
constexpr uint64_t tile_elems(es_dtype_t dt) {
  return static_cast<uint64_t>(kBlockThreads) * kVecsPerThread * vec_elems(dt);
}

// Device-side segment descriptor. A plan's table has nseg + 1 entries; the
// last is a sentinel whose tile_begin is the total number of tiles.
struct SegDesc {
  void* data;           // 16-byte aligned storage of the segment
  uint64_t numel;       // elements in the segment
  uint64_t index_base;  // global index of element 0 (multiple of 8)
  uint64_t tile_begin;  // first tile of the segment in the plan's tile space
};
static_assert(sizeof(SegDesc) == 32, "SegDesc layout");

// Largest number of generations one fused update launch applies.
constexpr int kMaxGenerations = 256;

// One fused update launch: `n_gen` generations of updates, generation g
// using seeds [gen_end[g-1], gen_end[g]) (gen_end[-1] = 0), each generation
// rounded to the storage type in turn; then, if `perturb`, one perturb step
// with (pkey, pscale). Passed by value as a kernel parameter (about 13 KB) and
// staged in shared memory by each CTA.
struct UpdateArgs {
  int n;          // seeds in all generations, 1..ES_MAX_SEEDS
  int n_gen;      // generations, 1..kMaxGenerations
  int perturb;    // 1: trailing perturb step
  float pscale;
  uint32_t pkey[2];
  uint16_t gen_end[kMaxGenerations];
  uint32_t key[ES_MAX_SEEDS][2];
  float coeff[ES_MAX_SEEDS];
};
static_assert(sizeof(UpdateArgs) < 32000, "kernel parameter limit");

struct PlanView {
  const SegDesc* segs;  // device table (nseg + 1 entries)
  uint64_t total_tiles;
  es_dtype_t dtype;
};

// Kernel launchers (es_kernels.cu). Each returns the launch's cudaError_t.
cudaError_t launch_axpy_noise(const PlanView& plan, uint64_t seed, float scale,
                              cudaStream_t stream);
cudaError_t launch_axpy_noise2(const PlanView& plan, uint64_t seed, float scale, uint64_t seed2,
                               float scale2, cudaStream_t stream);  // seed2 may equal seed
cudaError_t launch_update(const PlanView& plan, const UpdateArgs& args,
                          cudaStream_t stream);
cudaError_t launch_noise_bits(uint64_t seed, uint64_t block_base, uint64_t nblocks,
                              uint32_t* out, cudaStream_t stream);
cudaError_t launch_box_muller(const uint32_t* words, uint64_t npairs, float* out,
                              cudaStream_t stream);
cudaError_t launch_noise_fill(uint64_t seed, uint64_t index_base, uint64_t n,
                              float* out, cudaStream_t stream);

// Sets the calling thread's es_last_error() text (es_host.cu).
es_status_t record_status(es_status_t status, const char* message);

}  // namespace esopt
