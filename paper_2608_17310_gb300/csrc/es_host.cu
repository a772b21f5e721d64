// C-ABI host layer: plan creation and validation, argument checks, the
// host-side generation control of the paper (population z-score, cosine sigma
// schedule, update coefficients) and dispatch to the kernels.
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <new>
#include <vector>

#include "../../include/esopt.h"
#include "es_internal.h"
#include "es_memcheck.h"
#include "es_noise.cuh"

struct es_plan {
  int device;
  es_dtype_t dtype;
  int nseg;
  uint64_t numel;
  uint64_t total_tiles;
  esopt::SegDesc* d_segs;    // one allocation: the table, then (FP8) the
  float* d_inv_scale;        // reciprocal scales, or NULL
};

namespace {

thread_local char g_last_error[512] = "";

es_status_t fail(es_status_t st, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  std::vsnprintf(g_last_error, sizeof g_last_error, fmt, ap);
  va_end(ap);
  return st;
}

es_status_t ok() {
  g_last_error[0] = '\0';
  return ES_OK;
}

es_status_t cuda_fail(cudaError_t err, const char* what) {
  return fail(ES_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(err), cudaGetErrorString(err));
}

size_t dtype_size(es_dtype_t dt) { return esopt::dtype_bytes(dt); }

es_status_t check_plan_device(const es_plan* plan) {
  int cur = -1;
  cudaError_t err = cudaGetDevice(&cur);
  if (err != cudaSuccess) return cuda_fail(err, "cudaGetDevice");
  if (cur != plan->device)
    return fail(ES_ERR_WRONG_DEVICE, "plan lives on device %d but device %d is current",
                plan->device, cur);
  return ES_OK;
}

es_status_t check_device_buffer(const void* p, const char* what) {
  int device = -1;
  cudaError_t err = cudaGetDevice(&device);
  if (err != cudaSuccess) return cuda_fail(err, "cudaGetDevice");
  if (!esopt::is_device_memory(p, device))
    return fail(ES_ERR_INVALID_ARG, "%s: buffer is not device memory of the current device %d",
                what, device);
  return ES_OK;
}

esopt::PlanView view(const es_plan* plan) {
  return esopt::PlanView{plan->d_segs, plan->total_tiles, plan->dtype, plan->d_inv_scale};
}

es_status_t check_update_inputs(es_plan_t plan, const uint64_t* seeds, const float* coeffs, int n,
                                const char* what) {
  if (plan == nullptr) return fail(ES_ERR_INVALID_ARG, "%s: plan is NULL", what);
  if (seeds == nullptr || coeffs == nullptr || n < 1)
    return fail(ES_ERR_INVALID_ARG, "%s: need n >= 1 seeds and coefficients", what);
  if (n > ES_MAX_SEEDS)
    return fail(ES_ERR_TOO_MANY_SEEDS, "%s: n = %d > ES_MAX_SEEDS = %d", what, n, ES_MAX_SEEDS);
  for (int i = 0; i < n; ++i)
    if (!std::isfinite(coeffs[i]))
      return fail(ES_ERR_NONFINITE, "%s: coefficient %d is not finite", what, i);
  return check_plan_device(plan);
}

void start_update(esopt::UpdateArgs& a) {
  a.n = 0;
  a.n_gen = 0;
  a.perturb = 0;
  a.pscale = 0.0f;
  a.pkey[0] = a.pkey[1] = 0u;
}

// Appends one generation, skipping seeds whose coefficient is 0 (they add
// exactly zero); a generation left empty is dropped, since theta + 0 rounds to
// theta. The caller guarantees the space.
void append_generation(esopt::UpdateArgs& a, const uint64_t* seeds, const float* coeffs,
                       int count) {
  const int before = a.n;
  for (int i = 0; i < count; ++i) {
    if (coeffs[i] == 0.0f) continue;
    const esopt::PhiloxKey key = esopt::philox_key(seeds[i]);
    a.key[a.n][0] = key.k0;
    a.key[a.n][1] = key.k1;
    a.coeff[a.n] = coeffs[i];
    ++a.n;
  }
  if (a.n > before) a.gen_end[a.n_gen++] = static_cast<uint16_t>(a.n);
}

es_status_t launch_update_args(es_plan_t plan, const esopt::UpdateArgs& args, void* stream,
                               const char* what) {
  cudaError_t err = esopt::launch_update(view(plan), args, static_cast<cudaStream_t>(stream));
  if (err != cudaSuccess) return cuda_fail(err, what);
  return ok();
}

es_status_t axpy(es_plan_t plan, uint64_t seed, float scale, void* stream, const char* what) {
  if (plan == nullptr) return fail(ES_ERR_INVALID_ARG, "%s: plan is NULL", what);
  if (!std::isfinite(scale)) return fail(ES_ERR_NONFINITE, "%s: sigma is not finite", what);
  es_status_t st = check_plan_device(plan);
  if (st != ES_OK) return st;
  cudaError_t err = esopt::launch_axpy_noise(view(plan), seed, scale,
                                             static_cast<cudaStream_t>(stream));
  if (err != cudaSuccess) return cuda_fail(err, what);
  return ok();
}

}  // namespace

namespace esopt {
// Records `message` as the calling thread's es_last_error() text and returns
// `status` (ES_OK clears the text). For entry points defined in other files.
es_status_t record_status(es_status_t status, const char* message) {
  if (status == ES_OK) return ok();
  return fail(status, "%s", message);
}
}  // namespace esopt

namespace {

// es_plan_create and es_plan_create_scaled: `scales` is NULL (scale 1 for
// every segment) or nseg checked positive scales, FP8 only.
es_status_t create_plan(const es_segment_t* segs, const float* scales, int nseg,
                        es_dtype_t dtype, es_plan_t* out) {
  if (out == nullptr) return fail(ES_ERR_INVALID_ARG, "es_plan_create: out is NULL");
  *out = nullptr;
  if (segs == nullptr || nseg < 1)
    return fail(ES_ERR_INVALID_ARG, "es_plan_create: need at least one segment");
  if (dtype != ES_BF16 && dtype != ES_FP32 && dtype != ES_FP8_E4M3)
    return fail(ES_ERR_INVALID_ARG, "es_plan_create: unknown dtype %d", static_cast<int>(dtype));
  const size_t esize = dtype_size(dtype);
  uint64_t total = 0;
  for (int k = 0; k < nseg; ++k) {
    const es_segment_t& s = segs[k];
    if (s.data == nullptr || s.numel == 0)
      return fail(ES_ERR_INVALID_ARG, "segment %d: NULL data or zero numel", k);
    if (reinterpret_cast<uintptr_t>(s.data) % 16 != 0)
      return fail(ES_ERR_ALIGNMENT, "segment %d: data is not 16-byte aligned", k);
    if (s.index_base % 8 != 0)
      return fail(ES_ERR_ALIGNMENT, "segment %d: index_base is not a multiple of 8", k);
    if (s.index_base > UINT64_MAX - s.numel)
      return fail(ES_ERR_INVALID_ARG, "segment %d: index range passes 2^64", k);
    if (s.numel > UINT64_MAX / esize ||
        reinterpret_cast<uintptr_t>(s.data) > UINTPTR_MAX - s.numel * esize)
      return fail(ES_ERR_INVALID_ARG, "segment %d: byte range overflows", k);
    if (total > UINT64_MAX - s.numel)
      return fail(ES_ERR_INVALID_ARG, "total element count overflows");
    total += s.numel;
  }
  // No two segments may share memory or global indices: each element must have
  // one owner and one noise stream.
  std::vector<int> order;
  std::vector<esopt::SegDesc> table;
  try {
    order.resize(static_cast<size_t>(nseg));
    table.resize(static_cast<size_t>(nseg) + 1);
  } catch (const std::bad_alloc&) {
    return fail(ES_ERR_NO_MEMORY, "es_plan_create: host allocation failed");
  }
  for (int k = 0; k < nseg; ++k) order[k] = k;
  std::sort(order.begin(), order.end(),
            [&](int a, int b) { return segs[a].index_base < segs[b].index_base; });
  for (int k = 0; k + 1 < nseg; ++k) {
    const es_segment_t& a = segs[order[k]];
    const es_segment_t& b = segs[order[k + 1]];
    if (a.index_base + a.numel > b.index_base)
      return fail(ES_ERR_OVERLAP, "segments %d and %d overlap in index space", order[k],
                  order[k + 1]);
  }
  std::sort(order.begin(), order.end(), [&](int a, int b) {
    return reinterpret_cast<uintptr_t>(segs[a].data) < reinterpret_cast<uintptr_t>(segs[b].data);
  });
  for (int k = 0; k + 1 < nseg; ++k) {
    const es_segment_t& a = segs[order[k]];
    const es_segment_t& b = segs[order[k + 1]];
    if (reinterpret_cast<uintptr_t>(a.data) + a.numel * esize > reinterpret_cast<uintptr_t>(b.data))
      return fail(ES_ERR_OVERLAP, "segments %d and %d overlap in memory", order[k], order[k + 1]);
  }

  const uint64_t tile = esopt::tile_elems(dtype);
  uint64_t tiles = 0;
  for (int k = 0; k < nseg; ++k) {
    table[k] = esopt::SegDesc{segs[k].data, segs[k].numel, segs[k].index_base, tiles};
    tiles += (segs[k].numel + tile - 1) / tile;
  }
  table[nseg] = esopt::SegDesc{nullptr, 0, 0, tiles};

  int device = -1;
  cudaError_t err = cudaGetDevice(&device);
  if (err != cudaSuccess) return cuda_fail(err, "cudaGetDevice");
  for (int k = 0; k < nseg; ++k)
    if (!esopt::is_device_memory(segs[k].data, device))
      return fail(ES_ERR_INVALID_ARG, "segment %d: not device memory of the current device %d",
                  k, device);
  // FP8 segments: the kernels take 1 / scale per segment (1 without scales).
  std::vector<float> inv;
  if (dtype == ES_FP8_E4M3) {
    try {
      inv.resize(static_cast<size_t>(nseg));
    } catch (const std::bad_alloc&) {
      return fail(ES_ERR_NO_MEMORY, "es_plan_create: host allocation failed");
    }
    for (int k = 0; k < nseg; ++k) inv[k] = scales ? 1.0f / scales[k] : 1.0f;
  }
  es_plan* plan = new (std::nothrow) es_plan{};
  if (plan == nullptr) return fail(ES_ERR_NO_MEMORY, "es_plan_create: host allocation failed");
  plan->device = device;
  const size_t table_bytes = table.size() * sizeof(esopt::SegDesc);
  const size_t bytes = table_bytes + inv.size() * sizeof(float);
  err = cudaMalloc(reinterpret_cast<void**>(&plan->d_segs), bytes);
  if (err != cudaSuccess) {
    delete plan;
    cudaGetLastError();
    return fail(err == cudaErrorMemoryAllocation ? ES_ERR_NO_MEMORY : ES_ERR_CUDA,
                "cudaMalloc(segment table): %s", cudaGetErrorString(err));
  }
  err = cudaMemcpy(plan->d_segs, table.data(), table_bytes, cudaMemcpyHostToDevice);
  if (err == cudaSuccess && !inv.empty()) {
    plan->d_inv_scale = reinterpret_cast<float*>(reinterpret_cast<char*>(plan->d_segs) + table_bytes);
    err = cudaMemcpy(plan->d_inv_scale, inv.data(), inv.size() * sizeof(float),
                     cudaMemcpyHostToDevice);
  }
  if (err != cudaSuccess) {
    cudaFree(plan->d_segs);
    delete plan;
    return cuda_fail(err, "cudaMemcpy(segment table)");
  }
  plan->dtype = dtype;
  plan->nseg = nseg;
  plan->numel = total;
  plan->total_tiles = tiles;
  *out = plan;
  return ok();
}

}  // namespace

extern "C" {

es_status_t es_plan_create(const es_segment_t* segs, int nseg, es_dtype_t dtype,
                           es_plan_t* out) {
  return create_plan(segs, nullptr, nseg, dtype, out);
}

es_status_t es_plan_create_scaled(const es_segment_t* segs, const float* scales, int nseg,
                                  es_dtype_t dtype, es_plan_t* out) {
  if (out != nullptr) *out = nullptr;
  if (dtype != ES_FP8_E4M3)
    return fail(ES_ERR_INVALID_ARG, "es_plan_create_scaled: only ES_FP8_E4M3 takes scales");
  if (scales == nullptr || nseg < 1)
    return fail(ES_ERR_INVALID_ARG, "es_plan_create_scaled: need one scale per segment");
  for (int k = 0; k < nseg; ++k)
    if (!std::isfinite(scales[k]) || !(scales[k] > 0.0f) || !std::isfinite(1.0f / scales[k]))
      return fail(ES_ERR_INVALID_ARG,
                  "es_plan_create_scaled: scale %d must be finite and > 0 with a finite "
                  "reciprocal", k);
  return create_plan(segs, scales, nseg, dtype, out);
}

es_status_t es_plan_destroy(es_plan_t plan) {
  if (plan == nullptr) return ok();
  int prev = -1;
  cudaGetDevice(&prev);
  if (prev != plan->device) cudaSetDevice(plan->device);
  cudaError_t err = cudaFree(plan->d_segs);
  if (prev != plan->device && prev >= 0) cudaSetDevice(prev);
  delete plan;
  if (err != cudaSuccess) return cuda_fail(err, "cudaFree(segment table)");
  return ok();
}

uint64_t es_plan_numel(es_plan_t plan) { return plan == nullptr ? 0 : plan->numel; }

uint64_t es_assign_index_bases(es_segment_t* segs, int nseg) {
  if (segs == nullptr || nseg < 1) return 0;
  uint64_t base = 0, end = 0;
  for (int k = 0; k < nseg; ++k) {
    if (segs[k].numel > UINT64_MAX - 7 - base) return 0;  // the range would pass 2^64
    segs[k].index_base = base;
    end = base + segs[k].numel;
    base = (end + 7) & ~static_cast<uint64_t>(7);
  }
  return end;
}

es_status_t es_noise_fill(uint64_t seed, uint64_t index_base, uint64_t n, float* out,
                          void* stream) {
  if (n == 0) return ok();
  if (out == nullptr) return fail(ES_ERR_INVALID_ARG, "es_noise_fill: out is NULL");
  if (reinterpret_cast<uintptr_t>(out) % 4 != 0)
    return fail(ES_ERR_ALIGNMENT, "es_noise_fill: out is not 4-byte aligned");
  if (index_base > UINT64_MAX - n)
    return fail(ES_ERR_INVALID_ARG, "es_noise_fill: index range passes 2^64");
  es_status_t st = check_device_buffer(out, "es_noise_fill");
  if (st != ES_OK) return st;
  cudaError_t err = esopt::launch_noise_fill(seed, index_base, n, out,
                                             static_cast<cudaStream_t>(stream));
  if (err != cudaSuccess) return cuda_fail(err, "es_noise_fill");
  return ok();
}

es_status_t es_noise_bits(uint64_t seed, uint64_t block_base, uint64_t nblocks, uint32_t* out,
                          void* stream) {
  if (nblocks == 0) return ok();
  if (out == nullptr) return fail(ES_ERR_INVALID_ARG, "es_noise_bits: out is NULL");
  if (reinterpret_cast<uintptr_t>(out) % 16 != 0)
    return fail(ES_ERR_ALIGNMENT, "es_noise_bits: out is not 16-byte aligned");
  const uint64_t kMaxBlock = uint64_t{1} << 62;
  if (block_base > kMaxBlock || nblocks > kMaxBlock - block_base)
    return fail(ES_ERR_INVALID_ARG, "es_noise_bits: block range passes 2^62");
  es_status_t st = check_device_buffer(out, "es_noise_bits");
  if (st != ES_OK) return st;
  cudaError_t err = esopt::launch_noise_bits(seed, block_base, nblocks, out,
                                             static_cast<cudaStream_t>(stream));
  if (err != cudaSuccess) return cuda_fail(err, "es_noise_bits");
  return ok();
}

es_status_t es_box_muller(const uint32_t* words, uint64_t npairs, float* out, void* stream) {
  if (npairs == 0) return ok();
  if (words == nullptr || out == nullptr)
    return fail(ES_ERR_INVALID_ARG, "es_box_muller: NULL buffer");
  if (reinterpret_cast<uintptr_t>(words) % 8 != 0 || reinterpret_cast<uintptr_t>(out) % 8 != 0)
    return fail(ES_ERR_ALIGNMENT, "es_box_muller: buffers must be 8-byte aligned");
  if (npairs > (UINT64_MAX >> 4))
    return fail(ES_ERR_INVALID_ARG, "es_box_muller: npairs too large");
  es_status_t st = check_device_buffer(words, "es_box_muller");
  if (st == ES_OK) st = check_device_buffer(out, "es_box_muller");
  if (st != ES_OK) return st;
  cudaError_t err = esopt::launch_box_muller(words, npairs, out, static_cast<cudaStream_t>(stream));
  if (err != cudaSuccess) return cuda_fail(err, "es_box_muller");
  return ok();
}

es_status_t es_perturb(es_plan_t plan, uint64_t seed, float sigma, void* stream) {
  return axpy(plan, seed, sigma, stream, "es_perturb");
}

es_status_t es_restore(es_plan_t plan, uint64_t seed, float sigma, void* stream) {
  return axpy(plan, seed, -sigma, stream, "es_restore");
}

es_status_t es_restore_perturb(es_plan_t plan, uint64_t restore_seed, float sigma_restore,
                               uint64_t perturb_seed, float sigma_perturb, void* stream) {
  if (plan == nullptr) return fail(ES_ERR_INVALID_ARG, "es_restore_perturb: plan is NULL");
  if (!std::isfinite(sigma_restore) || !std::isfinite(sigma_perturb))
    return fail(ES_ERR_NONFINITE, "es_restore_perturb: sigma is not finite");
  es_status_t st = check_plan_device(plan);
  if (st != ES_OK) return st;
  cudaError_t err = esopt::launch_axpy_noise2(view(plan), restore_seed, -sigma_restore,
                                              perturb_seed, sigma_perturb,
                                              static_cast<cudaStream_t>(stream));
  if (err != cudaSuccess) return cuda_fail(err, "es_restore_perturb");
  return ok();
}

es_status_t es_update(es_plan_t plan, const uint64_t* seeds, const float* coeffs, int n,
                      void* stream) {
  es_status_t st = check_update_inputs(plan, seeds, coeffs, n, "es_update");
  if (st != ES_OK) return st;
  esopt::UpdateArgs args;
  start_update(args);
  append_generation(args, seeds, coeffs, n);
  if (args.n_gen == 0) return ok();  // every coefficient 0: no update, theta bit-identical
  return launch_update_args(plan, args, stream, "es_update");
}

es_status_t es_update_perturb(es_plan_t plan, const uint64_t* seeds, const float* coeffs, int n,
                              uint64_t next_seed, float sigma_next, void* stream) {
  es_status_t st = check_update_inputs(plan, seeds, coeffs, n, "es_update_perturb");
  if (st != ES_OK) return st;
  if (!std::isfinite(sigma_next))
    return fail(ES_ERR_NONFINITE, "es_update_perturb: sigma_next is not finite");
  esopt::UpdateArgs args;
  start_update(args);
  append_generation(args, seeds, coeffs, n);
  if (args.n_gen == 0) return axpy(plan, next_seed, sigma_next, stream, "es_update_perturb");
  const esopt::PhiloxKey key = esopt::philox_key(next_seed);
  args.perturb = 1;
  args.pkey[0] = key.k0;
  args.pkey[1] = key.k1;
  args.pscale = sigma_next;
  return launch_update_args(plan, args, stream, "es_update_perturb");
}

es_status_t es_replay(es_plan_t plan, const uint64_t* seeds, const float* coeffs,
                      const int* counts, int generations, void* stream) {
  if (plan == nullptr) return fail(ES_ERR_INVALID_ARG, "es_replay: plan is NULL");
  if (counts == nullptr || generations < 1)
    return fail(ES_ERR_INVALID_ARG, "es_replay: need at least one generation");
  uint64_t total = 0;
  for (int g = 0; g < generations; ++g) {
    if (counts[g] < 1) return fail(ES_ERR_INVALID_ARG, "es_replay: generation %d is empty", g);
    if (counts[g] > ES_MAX_SEEDS)
      return fail(ES_ERR_TOO_MANY_SEEDS, "es_replay: generation %d has %d > ES_MAX_SEEDS = %d seeds",
                  g, counts[g], ES_MAX_SEEDS);
    total += static_cast<uint64_t>(counts[g]);
  }
  if (seeds == nullptr || coeffs == nullptr)
    return fail(ES_ERR_INVALID_ARG, "es_replay: NULL seeds or coefficients");
  for (uint64_t i = 0; i < total; ++i)
    if (!std::isfinite(coeffs[i]))
      return fail(ES_ERR_NONFINITE, "es_replay: coefficient %llu is not finite",
                  static_cast<unsigned long long>(i));
  es_status_t st = check_plan_device(plan);
  if (st != ES_OK) return st;
  // Launches break only between generations, so the roundings are those of
  // one es_update per generation. Small generations share a pass over theta
  // (fewer passes: measured 5 % faster at 2 seeds per generation, 15 % at 1);
  // a generation of kOwnLaunch or more non-zero seeds gets a launch of its own
  // through the single-generation kernel, which runs such generations faster
  // (measured 2-3 % at 6 to 16 seeds). Both orders give the same bits.
  constexpr int kOwnLaunch = 4;
  esopt::UpdateArgs args;
  start_update(args);
  uint64_t off = 0;
  for (int g = 0; g < generations; ++g) {
    int nonzero = 0;
    for (int i = 0; i < counts[g]; ++i) nonzero += coeffs[off + i] != 0.0f;
    const bool own = nonzero >= kOwnLaunch;
    if (nonzero > 0 && args.n_gen > 0 &&
        (own || args.n + nonzero > ES_MAX_SEEDS || args.n_gen == esopt::kMaxGenerations)) {
      st = launch_update_args(plan, args, stream, "es_replay");
      if (st != ES_OK) return st;
      start_update(args);
    }
    append_generation(args, seeds + off, coeffs + off, counts[g]);
    off += static_cast<uint64_t>(counts[g]);
    if (own) {
      st = launch_update_args(plan, args, stream, "es_replay");
      if (st != ES_OK) return st;
      start_update(args);
    }
  }
  if (args.n_gen > 0) return launch_update_args(plan, args, stream, "es_replay");
  return ok();
}

es_status_t es_normalize_rewards(const double* rewards, int n, double eps_z, double* rhat) {
  if (rewards == nullptr || rhat == nullptr || n < 1)
    return fail(ES_ERR_INVALID_ARG, "es_normalize_rewards: need n >= 1 rewards");
  if (!(eps_z >= 0.0) || !std::isfinite(eps_z))
    return fail(ES_ERR_INVALID_ARG, "es_normalize_rewards: eps_z must be finite and >= 0");
  // Invalid (non-finite) rewards take the smallest finite reward of the batch.
  int n_finite = 0;
  double lo = 0.0, hi = 0.0;
  for (int i = 0; i < n; ++i) {
    if (!std::isfinite(rewards[i])) continue;
    if (n_finite == 0 || rewards[i] < lo) lo = rewards[i];
    if (n_finite == 0 || rewards[i] > hi) hi = rewards[i];
    ++n_finite;
  }
  if (n_finite == 0 || lo == hi) {  // all invalid or all equal: no update
    for (int i = 0; i < n; ++i) rhat[i] = 0.0;
    return ok();
  }
  // rewards and rhat may alias: every rhat[i] is written after the last read
  // of rewards[i].
  auto value = [&](int i) { return std::isfinite(rewards[i]) ? rewards[i] : lo; };
  double mu = 0.0;
  for (int i = 0; i < n; ++i) mu += value(i);
  mu /= n;
  double var = 0.0;
  for (int i = 0; i < n; ++i) var += (value(i) - mu) * (value(i) - mu);
  var /= n;
  const double denom = std::sqrt(var) + eps_z;
  for (int i = 0; i < n; ++i) rhat[i] = (value(i) - mu) / denom;
  return ok();
}

double es_sigma_cosine(double sigma0, double sigmaT, int t, int T) {
  if (T <= 0) return sigma0;
  t = std::min(std::max(t, 0), T);
  return sigmaT + (sigma0 - sigmaT) * (1.0 + std::cos(M_PI * t / T)) / 2.0;
}

static es_status_t coeffs_common(int n, double alpha, double sigma, es_scale_t mode,
                                 double* denom_scale, const char* what) {
  if (n < 1) return fail(ES_ERR_INVALID_ARG, "%s: n must be >= 1", what);
  if (mode != ES_SCALE_PAPER && mode != ES_SCALE_CANONICAL)
    return fail(ES_ERR_INVALID_ARG, "%s: unknown scale mode %d", what, static_cast<int>(mode));
  if (!std::isfinite(alpha) || !std::isfinite(sigma))
    return fail(ES_ERR_NONFINITE, "%s: alpha and sigma must be finite", what);
  if (mode == ES_SCALE_CANONICAL && !(sigma > 0.0))
    return fail(ES_ERR_INVALID_ARG, "%s: canonical scale needs sigma > 0", what);
  *denom_scale = mode == ES_SCALE_CANONICAL ? sigma : 1.0;
  return ES_OK;
}

es_status_t es_update_coeffs(const double* rhat, int n, double alpha, double sigma,
                             es_scale_t mode, float* coeffs) {
  if (rhat == nullptr || coeffs == nullptr)
    return fail(ES_ERR_INVALID_ARG, "es_update_coeffs: NULL array");
  double s = 1.0;
  es_status_t st = coeffs_common(n, alpha, sigma, mode, &s, "es_update_coeffs");
  if (st != ES_OK) return st;
  const double denom = static_cast<double>(n) * s;
  for (int i = 0; i < n; ++i) {
    const double c = alpha * rhat[i] / denom;
    if (!std::isfinite(c) || !std::isfinite(static_cast<float>(c)))
      return fail(ES_ERR_NONFINITE, "es_update_coeffs: coefficient %d is not finite", i);
    coeffs[i] = static_cast<float>(c);
  }
  return ok();
}

es_status_t es_fold_antithetic(const double* rhat_pos, const double* rhat_neg, int npairs,
                               double alpha, double sigma, es_scale_t mode, float* coeffs) {
  if (rhat_pos == nullptr || rhat_neg == nullptr || coeffs == nullptr)
    return fail(ES_ERR_INVALID_ARG, "es_fold_antithetic: NULL array");
  double s = 1.0;
  es_status_t st = coeffs_common(npairs, alpha, sigma, mode, &s, "es_fold_antithetic");
  if (st != ES_OK) return st;
  const double denom = 2.0 * static_cast<double>(npairs) * s;
  for (int i = 0; i < npairs; ++i) {
    const double c = alpha * (rhat_pos[i] - rhat_neg[i]) / denom;
    if (!std::isfinite(c) || !std::isfinite(static_cast<float>(c)))
      return fail(ES_ERR_NONFINITE, "es_fold_antithetic: coefficient %d is not finite", i);
    coeffs[i] = static_cast<float>(c);
  }
  return ok();
}

const char* es_status_string(es_status_t status) {
  switch (status) {
    case ES_OK: return "ES_OK";
    case ES_ERR_INVALID_ARG: return "ES_ERR_INVALID_ARG: invalid argument";
    case ES_ERR_ALIGNMENT: return "ES_ERR_ALIGNMENT: misaligned pointer or index base";
    case ES_ERR_OVERLAP: return "ES_ERR_OVERLAP: segments overlap";
    case ES_ERR_NONFINITE: return "ES_ERR_NONFINITE: non-finite scalar";
    case ES_ERR_TOO_MANY_SEEDS: return "ES_ERR_TOO_MANY_SEEDS: more seeds than ES_MAX_SEEDS";
    case ES_ERR_CUDA: return "ES_ERR_CUDA: CUDA error";
    case ES_ERR_NO_MEMORY: return "ES_ERR_NO_MEMORY: allocation failed";
    case ES_ERR_WRONG_DEVICE: return "ES_ERR_WRONG_DEVICE: plan belongs to another device";
  }
  return "unknown es_status_t";
}

const char* es_last_error(void) { return g_last_error; }

}  // extern "C"
