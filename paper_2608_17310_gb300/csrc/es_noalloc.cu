// es_perturb_noalloc: the perturb/restore pass for callers that must not
// allocate device memory. Instead of a plan (whose segment table lives in
// memory es_plan_create obtains with cudaMalloc), the segment table is copied
// on every call into a fixed array of static device memory that belongs to
// this library module.
#include <cuda.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstdio>
#include <mutex>

#include "../../include/esopt.h"
#include "es_internal.h"
#include "es_memcheck.h"

namespace esopt {
namespace {

// Segment table of es_perturb_noalloc: nseg descriptors plus the end
// sentinel. Static device memory (about 32 KB), held by every device that
// loads the library until the process exits; shared by all calls.
__device__ __align__(256) SegDesc g_noalloc_table[ES_STATIC_MAX_SEGMENTS + 1];

constexpr int kMaxDevices = 64;
std::mutex g_setup_mutex;
SegDesc* g_table_address[kMaxDevices] = {};
// Id of the context the cached address belongs to (0: unknown). A device
// reset destroys the context and the module loaded into it; the next context
// gets a new id, and the address is looked up again.
unsigned long long g_table_context[kMaxDevices] = {};

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

// Id of the calling thread's current context, or 0 if the driver does not
// provide one. The driver functions are found at run time, so the library does
// not link against the driver library.
unsigned long long current_context_id() {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static bool looked_up = false;
  if (!looked_up) {
    looked_up = true;
    void* fn = nullptr;
    cudaDriverEntryPointQueryResult q{};
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(fn);
    fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &fn, 12000, cudaEnableDefault, &q) ==
            cudaSuccess && q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(fn);
    cudaGetLastError();
  }
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (get_current == nullptr || get_id == nullptr || get_current(&ctx) != CUDA_SUCCESS ||
      ctx == nullptr || get_id(ctx, &id) != CUDA_SUCCESS)
    return 0;
  return id;
}

// Device address of g_noalloc_table on `device`, which is current. In host
// code the name g_noalloc_table is only a host-side stand-in, so the address
// is looked up with cudaGetSymbolAddress once per device (the set-up done by
// the first call on each device) and cached; it is looked up again when the
// device's context has changed since (after a device reset), or on every call
// if the context cannot be identified.
es_status_t table_address(int device, SegDesc** out) {
  std::lock_guard<std::mutex> lock(g_setup_mutex);
  const unsigned long long ctx = current_context_id();
  if (g_table_address[device] == nullptr || ctx == 0 || ctx != g_table_context[device]) {
    void* p = nullptr;
    cudaError_t err = cudaGetSymbolAddress(&p, g_noalloc_table);
    if (err != cudaSuccess || p == nullptr) {
      char msg[256];
      std::snprintf(msg, sizeof msg, "es_perturb_noalloc: cudaGetSymbolAddress: %s",
                    cudaGetErrorString(err));
      return record_status(ES_ERR_CUDA, msg);
    }
    g_table_address[device] = static_cast<SegDesc*>(p);
    g_table_context[device] = ctx;
  }
  *out = g_table_address[device];
  return ES_OK;
}

es_status_t reject(es_status_t st, const char* fmt, int a = 0, int b = 0) {
  char msg[256];
  std::snprintf(msg, sizeof msg, fmt, a, b);
  return record_status(st, msg);
}

}  // namespace
}  // namespace esopt

extern "C" es_status_t es_perturb_noalloc(const es_segment_t* segs, int nseg, es_dtype_t dtype,
                                          uint64_t seed, float sigma, void* stream) {
  using esopt::reject;
  using esopt::SegDesc;
  if (segs == nullptr || nseg < 1)
    return reject(ES_ERR_INVALID_ARG, "es_perturb_noalloc: need at least one segment");
  if (nseg > ES_STATIC_MAX_SEGMENTS)
    return reject(ES_ERR_INVALID_ARG,
                  "es_perturb_noalloc: %d segments exceed ES_STATIC_MAX_SEGMENTS = %d", nseg,
                  ES_STATIC_MAX_SEGMENTS);
  if (dtype != ES_BF16 && dtype != ES_FP32)
    return reject(ES_ERR_INVALID_ARG, "es_perturb_noalloc: unknown dtype %d", dtype);
  if (!std::isfinite(sigma))
    return reject(ES_ERR_NONFINITE, "es_perturb_noalloc: sigma is not finite");
  const uint64_t esize = dtype == ES_BF16 ? 2u : 4u;
  for (int k = 0; k < nseg; ++k) {
    const es_segment_t& s = segs[k];
    if (s.data == nullptr || s.numel == 0)
      return reject(ES_ERR_INVALID_ARG, "es_perturb_noalloc: segment %d: NULL data or zero numel", k);
    if (reinterpret_cast<uintptr_t>(s.data) % 16 != 0)
      return reject(ES_ERR_ALIGNMENT, "es_perturb_noalloc: segment %d: data not 16-byte aligned", k);
    if (s.index_base % 8 != 0)
      return reject(ES_ERR_ALIGNMENT, "es_perturb_noalloc: segment %d: index_base not a multiple of 8", k);
    if (s.index_base > UINT64_MAX - s.numel || s.numel > UINT64_MAX / esize ||
        reinterpret_cast<uintptr_t>(s.data) > UINTPTR_MAX - s.numel * esize)
      return reject(ES_ERR_INVALID_ARG, "es_perturb_noalloc: segment %d: range overflows", k);
  }
  // Overlap checks on index and byte ranges, sorting indices on the stack.
  int order[ES_STATIC_MAX_SEGMENTS];
  for (int k = 0; k < nseg; ++k) order[k] = k;
  std::sort(order, order + nseg,
            [&](int a, int b) { return segs[a].index_base < segs[b].index_base; });
  for (int k = 0; k + 1 < nseg; ++k)
    if (segs[order[k]].index_base + segs[order[k]].numel > segs[order[k + 1]].index_base)
      return reject(ES_ERR_OVERLAP, "es_perturb_noalloc: segments %d and %d overlap in index space",
                    order[k], order[k + 1]);
  std::sort(order, order + nseg, [&](int a, int b) {
    return reinterpret_cast<uintptr_t>(segs[a].data) < reinterpret_cast<uintptr_t>(segs[b].data);
  });
  for (int k = 0; k + 1 < nseg; ++k)
    if (reinterpret_cast<uintptr_t>(segs[order[k]].data) + segs[order[k]].numel * esize >
        reinterpret_cast<uintptr_t>(segs[order[k + 1]].data))
      return reject(ES_ERR_OVERLAP, "es_perturb_noalloc: segments %d and %d overlap in memory",
                    order[k], order[k + 1]);

  SegDesc table[ES_STATIC_MAX_SEGMENTS + 1];
  const uint64_t tile = esopt::tile_elems(dtype);
  uint64_t tiles = 0;
  for (int k = 0; k < nseg; ++k) {
    table[k] = SegDesc{segs[k].data, segs[k].numel, segs[k].index_base, tiles};
    tiles += (segs[k].numel + tile - 1) / tile;
  }
  table[nseg] = SegDesc{nullptr, 0, 0, tiles};

  // The table is copied from this call's stack; a copy recorded into a graph
  // would read that memory again at every replay, long after it is gone. So a
  // stream that is being captured is refused before anything is done.
  const cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaStreamCaptureStatus capture = cudaStreamCaptureStatusNone;
  cudaError_t err = cudaStreamIsCapturing(s, &capture);
  if (err != cudaSuccess) {
    cudaGetLastError();
    return reject(ES_ERR_CUDA, "es_perturb_noalloc: cudaStreamIsCapturing failed");
  }
  if (capture != cudaStreamCaptureStatusNone)
    return reject(ES_ERR_INVALID_ARG,
                  "es_perturb_noalloc: the stream is being captured into a CUDA graph; this "
                  "entry point copies its segment table from host stack memory and is refused "
                  "on a capturing stream");

  int device = -1;
  err = cudaGetDevice(&device);
  if (err != cudaSuccess) return reject(ES_ERR_CUDA, "es_perturb_noalloc: cudaGetDevice failed");
  if (device < 0 || device >= esopt::kMaxDevices)
    return reject(ES_ERR_INVALID_ARG, "es_perturb_noalloc: device ordinal %d >= %d", device,
                  esopt::kMaxDevices);
  for (int k = 0; k < nseg; ++k)
    if (!esopt::is_device_memory(segs[k].data, device))
      return reject(ES_ERR_INVALID_ARG,
                    "es_perturb_noalloc: segment %d is not device memory of device %d", k, device);
  SegDesc* d_table = nullptr;
  es_status_t st = esopt::table_address(device, &d_table);
  if (st != ES_OK) return st;
  // The whole table (nseg entries and the sentinel) is rewritten by every
  // call, so nothing in it has to start at zero. From pageable host memory
  // the source is staged before cudaMemcpyAsync returns, so `table` may go
  // out of scope; the kernel below is ordered after the copy on `stream`.
  err = cudaMemcpyAsync(d_table, table, (static_cast<size_t>(nseg) + 1) * sizeof(SegDesc),
                        cudaMemcpyHostToDevice, s);
  if (err != cudaSuccess) return reject(ES_ERR_CUDA, "es_perturb_noalloc: copy of the segment table failed");
  err = esopt::launch_axpy_noise(esopt::PlanView{d_table, tiles, dtype, nullptr}, seed, sigma, s);
  if (err != cudaSuccess) return reject(ES_ERR_CUDA, "es_perturb_noalloc: kernel launch failed");
  return esopt::record_status(ES_OK, "");
}
