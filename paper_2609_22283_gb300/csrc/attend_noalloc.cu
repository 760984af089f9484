// Split scratch for sva_attend_nodes_noalloc: a fixed array in device memory
// that the library itself owns, so callers that must not allocate device
// memory can still get key-range splits.  The array is part of the loaded
// module: every GPU that loads the library holds kStaticScratchBytes of it
// until the process exits, and all calls on a device share it.
#include <mutex>

#include <cuda_runtime.h>

#include "internal.h"

namespace sva {

static __device__ __align__(256) unsigned char g_split_scratch[kStaticScratchBytes];

// Device address of g_split_scratch on `device`, which must be the current
// device.  In host code the array's name only stands for the symbol; its
// device address is looked up once per device and kept.
cudaError_t static_split_scratch(int device, void** ptr) {
  static std::mutex mu;
  static void* addr[64] = {};
  if (device < 0 || device >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(mu);
  if (addr[device] == nullptr) {
    void* a = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&a, g_split_scratch);
    if (e != cudaSuccess) return e;
    addr[device] = a;
  }
  *ptr = addr[device];
  return cudaSuccess;
}

}  // namespace sva
