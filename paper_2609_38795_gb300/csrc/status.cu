// Per-device status word shared by all kernels of the library.  A kernel that gives up a
// bounded pipeline wait stores ALR_ERR_TIMEOUT here; alr_device_status() reads and clears it.
#include "kernels.h"

namespace alr {

__device__ int g_status_word;

int* device_status_ptr() {
  // The symbol's device address differs per device; look it up for the current one.
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return nullptr;
  static int* cache[64] = {nullptr};
  if (dev < 0 || dev >= 64) return nullptr;
  if (cache[dev] == nullptr) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return nullptr;
    cache[dev] = static_cast<int*>(p);
  }
  return cache[dev];
}

}  // namespace alr
