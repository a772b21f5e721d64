// Internal interface between the C-ABI host layer (es_host.cpp) and the CUDA
// kernels (es_kernels.cu). Not part of the public ABI.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "../../include/esopt.h"

namespace esopt {

// Threads per CTA of the streaming kernels.
constexpr int kBlockThreads = 256;
// 16-byte vectors per thread in one tile. A tile (kBlockThreads x
// kVecsPerThread vectors) is the unit a CTA takes from a plan; tiles never
// straddle segments.
#ifndef ES_VECS_PER_THREAD
#define ES_VECS_PER_THREAD 4
#endif
constexpr int kVecsPerThread = ES_VECS_PER_THREAD;

// Per kernel kind (one-seed pass, two-seed pass, update): how many 16-byte
// vectors of its tile a thread processes at once (the group; each bf16 vector
// is two independent Philox chains per seed), the resident CTAs per SM asked
// of the compiler (a register cap), and the instruction form of the noise step
// (0 scalar FP32, 1 scalar transform with packed FMAs, 2 packed; the values
// are bit-identical). Measured on sm_103a over the 4B-shaped set: one vector
// at a time is fastest for every kernel, at 2 CTAs per SM (128 registers) for
// the two-seed pass and 3 for the others; more CTAs per SM or larger groups
// gain nothing, since the generator is bound by the FMA-heavy pipe (its
// integer products and packed FP32), not by latency. What does gain is
// interleaving the phases of independent work in one basic block: the
// update's seed loop computes the next seed's Philox words beside the current
// seed's transform (ES_UPDATE_PIPELINED).
#ifndef ES_AXPY1_GROUP
#define ES_AXPY1_GROUP 1
#endif
#ifndef ES_AXPY1_MIN_BLOCKS
#define ES_AXPY1_MIN_BLOCKS 3
#endif
#ifndef ES_AXPY1_FORM
#define ES_AXPY1_FORM 2
#endif
#ifndef ES_AXPY2_GROUP
#define ES_AXPY2_GROUP 1
#endif
#ifndef ES_AXPY2_MIN_BLOCKS
#define ES_AXPY2_MIN_BLOCKS 2
#endif
#ifndef ES_AXPY2_FORM
#define ES_AXPY2_FORM 2
#endif
#ifndef ES_UPDATE_GROUP
#define ES_UPDATE_GROUP 1
#endif
#ifndef ES_UPDATE_MIN_BLOCKS
#define ES_UPDATE_MIN_BLOCKS 3
#endif
#ifndef ES_UPDATE_FORM
#define ES_UPDATE_FORM 2
#endif
// Radius inputs within 2^-10 of 1 (one in 1024), which take the series of
// -2 ln u instead of the hardware log2: found by a compare on the raw Philox
// word and fixed on a rarely taken branch (1), or by evaluating both forms
// for every pair and selecting (0). The values are identical.
#ifndef ES_NEAR_ONE_BRANCH
#define ES_NEAR_ONE_BRANCH 1
#endif
// Software pipelining of the update's seed loop: seed i + 1's Philox words
// are computed beside seed i's transform (1: one seed per iteration, the
// words copied to the next iteration's buffer; 2: two seeds per iteration
// on alternating buffers). The values are identical.
// (The same schedule in the perturb/restore passes, over (vector, seed)
// items, measured 2-4 % slower there and is not built.)
#ifndef ES_UPDATE_PIPELINED
#define ES_UPDATE_PIPELINED 2
#endif
// The antithetic flip (es_restore_perturb with one seed) in the scalar form
// per block (0) or in the packed form of the other passes, with round 0's
// product stepped in tiles inside their segment (1); values identical. Its
// resident CTAs per SM (a register cap), like the other passes'.
#ifndef ES_FLIP_PACKED
#define ES_FLIP_PACKED 1
#endif
#ifndef ES_FLIP_MIN_BLOCKS
#define ES_FLIP_MIN_BLOCKS 3
#endif
// Round 0's Philox product (kPhiloxMulA times the low counter word) depends
// on the counter alone: 0 computes it per block and seed; 1 once per block,
// shared by the seeds of a pass (both seeds of the fused restore + perturb,
// every seed of the update's loop); 2 as 1, and in the perturb/restore passes'
// tiles that lie inside their segment stepped from the thread's first block by
// 64-bit additions of constants instead of multiplied. The words are
// identical. Measured: 1 runs as fast as 0 (the compiler already shares the
// product), 2 is 0.8-1.3 % faster.
#ifndef ES_ROUND0
#define ES_ROUND0 2
#endif
// Seeds of the update's seed loop issued together (independent generator
// work per element across seeds; the accumulation stays in ascending order).
#ifndef ES_SEED_UNROLL
#define ES_SEED_UNROLL 1
#endif
constexpr int kAxpy1Group = ES_AXPY1_GROUP;
constexpr int kAxpy2Group = ES_AXPY2_GROUP;
constexpr int kUpdateGroup = ES_UPDATE_GROUP;
static_assert(kVecsPerThread % kAxpy1Group == 0 && kVecsPerThread % kAxpy2Group == 0 &&
                  kVecsPerThread % kUpdateGroup == 0,
              "groups divide the vectors of a tile");
constexpr int axpy_min_blocks(bool two, int vec_elems = 8, bool same = false) {
  const int want = same ? ES_FLIP_MIN_BLOCKS : two ? ES_AXPY2_MIN_BLOCKS : ES_AXPY1_MIN_BLOCKS;
  const int m = want > 0 ? want : 1;
  // FP8 vectors hold twice the elements (twice the Philox blocks per vector):
  // at most 2 CTAs per SM, so their registers do not spill
  return vec_elems > 8 && m > 2 ? 2 : m;
}
constexpr int update_min_blocks() { return ES_UPDATE_MIN_BLOCKS > 0 ? ES_UPDATE_MIN_BLOCKS : 1; }
// Elements per 16-byte vector, per dtype.
constexpr int vec_elems(es_dtype_t dt) { return dt == ES_FP8_E4M3 ? 16 : dt == ES_BF16 ? 8 : 4; }
// Bytes per element, per dtype.
constexpr size_t dtype_bytes(es_dtype_t dt) { return dt == ES_FP8_E4M3 ? 1u : dt == ES_BF16 ? 2u : 4u; }
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
  // ES_FP8_E4M3: device array of 1 / scale per segment; NULL otherwise
  const float* inv_scale;
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
