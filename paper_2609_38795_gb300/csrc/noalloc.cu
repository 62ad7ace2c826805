// Forward pass of the slot loss for callers that cannot allocate device memory.
//
// alr_slot_loss_fwd needs a caller-provided workspace.  Some callers cannot get one: code
// that runs inside a host that has handed all device memory to its own pool allocator at
// start-up and forbids any further allocation, and code on a latency-critical path where a
// cudaMalloc (which may synchronise the whole device) is not acceptable.  This entry point
// runs the very same forward kernels with their scratch placed in a fixed array in device
// global memory that is part of this library image, so it calls no allocator at all.
#include <cstdio>
#include <cuda.h>
#include <mutex>

#include "alr.h"
#include "kernels.h"

namespace {

// The scratch array.  It is reserved on every device that loads this library and stays
// there until the process exits.  In host code its name only stands in for the symbol; the
// device address comes from cudaGetSymbolAddress below.
static __device__ __align__(256) unsigned char g_fwd_scratch[ALR_NOALLOC_SCRATCH_BYTES];

// The array's device address per device, with the context it was looked up in: a device
// reset or a new primary context loads the module again at another address, so a cached
// address is used only while the current context is the one it came from.
std::mutex g_scratch_mu;
void* g_scratch_ptr[64] = {nullptr};
CUcontext g_scratch_ctx[64] = {nullptr};

// The current context of the calling thread (nullptr when it cannot be read: the address is
// then looked up on every call).
CUcontext current_context() {
  using Fn = CUresult (*)(CUcontext*);
  static Fn fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    return (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault,
                                             &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
               ? reinterpret_cast<Fn>(p)
               : nullptr;
  }();
  CUcontext c = nullptr;
  if (fn == nullptr || fn(&c) != CUDA_SUCCESS) return nullptr;
  return c;
}

}  // namespace

extern "C" int alr_slot_loss_fwd_noalloc(const alr_params* p, const void* Hd, const void* Ht,
                                         const void* W, const float* row_mask,
                                         const int32_t* corpus_tok, const alr_fwd_outputs* out,
                                         void* stream) {
  // Size check first, so that an oversized problem is rejected before anything is launched.
  const size_t need = alr_fwd_workspace_size(p);
  if (need == 0) {
    // invalid params, or no usable device: alr_fwd_workspace_size set no message of its own,
    // so let the regular entry point validate and describe the problem.
    return alr_slot_loss_fwd(p, Hd, Ht, W, row_mask, corpus_tok, out, nullptr, 0, stream);
  }
  if (need > size_t(ALR_NOALLOC_SCRATCH_BYTES)) {
    char msg[320];
    snprintf(msg, sizeof(msg),
             "alr_slot_loss_fwd_noalloc: this problem needs %zu bytes of scratch, more than the "
             "library's fixed %zu bytes; use alr_slot_loss_fwd with a workspace instead",
             need, size_t(ALR_NOALLOC_SCRATCH_BYTES));
    return alr::set_last_error(ALR_ERR_INVALID_ARG, msg);
  }
  // Set-up, once per device and context, with that device current: look up the array's
  // device address (cudaGetSymbolAddress also makes sure the module is loaded there).
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess || dev < 0 || dev >= 64) {
    char msg[320];
    snprintf(msg, sizeof(msg), "alr_slot_loss_fwd_noalloc: no usable current device (%s)",
             cudaGetErrorString(e));
    return alr::set_last_error(ALR_ERR_CUDA, msg);
  }
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lk(g_scratch_mu);
    const CUcontext ctx = current_context();
    if (g_scratch_ptr[dev] == nullptr || ctx == nullptr || ctx != g_scratch_ctx[dev]) {
      void* ptr = nullptr;
      e = cudaGetSymbolAddress(&ptr, g_fwd_scratch);
      if (e != cudaSuccess || ptr == nullptr) {
        char msg[320];
        snprintf(msg, sizeof(msg),
                 "alr_slot_loss_fwd_noalloc: cudaGetSymbolAddress failed on device %d: %s", dev,
                 cudaGetErrorString(e));
        return alr::set_last_error(ALR_ERR_CUDA, msg);
      }
      g_scratch_ptr[dev] = ptr;
      g_scratch_ctx[dev] = current_context();   // current now, after the runtime call
    }
    scratch = g_scratch_ptr[dev];
  }
  // The forward kernels overwrite every scratch element before reading it, so nothing has to
  // be cleared between calls.
  return alr_slot_loss_fwd(p, Hd, Ht, W, row_mask, corpus_tok, out, scratch,
                           size_t(ALR_NOALLOC_SCRATCH_BYTES), stream);
}
