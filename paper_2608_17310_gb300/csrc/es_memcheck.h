// Host-side check that a buffer handed to the C ABI is device memory. Used by
// the entry points before any launch: a kernel given a host pointer would
// fault the GPU and lose the context, so such a call is refused with
// ES_ERR_INVALID_ARG instead.
#pragma once

#include <cuda_runtime.h>

namespace esopt {

// Whether `p` points into device memory of `device`, or into managed memory.
// Pageable host memory, page-locked host memory and unregistered addresses
// are all refused; a failed query leaves no sticky error behind.
inline bool is_device_memory(const void* p, int device) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    cudaGetLastError();
    return false;
  }
  if (a.type == cudaMemoryTypeManaged) return true;
  return a.type == cudaMemoryTypeDevice && a.device == device;
}

}  // namespace esopt
