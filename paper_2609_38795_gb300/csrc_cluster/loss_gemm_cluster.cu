// The fused loss kernel's cluster form (loss_gemm_kernel.cuh with Cl = ClusterOf<2>): bf16
// inputs, 256-column tiles, the dual modes.  Built into libalr_cluster.so only.
#include <atomic>

#include "cluster_forms.h"
#include "cluster_ptx.cuh"
#include "loss_gemm_kernel.cuh"

namespace alr {
namespace {

template <int kMode>
cudaError_t launch_cluster(const CUtensorMap& a0, const CUtensorMap& a1, const CUtensorMap& w,
                           const CUtensorMap& g, const CUtensorMap& g2, const LossArgs& args,
                           cudaStream_t s) {
  using Elem = __nv_bfloat16;
  using S = Shape<kMode, 256, is_staged(kMode, sizeof(Elem))>;
  auto kern = loss_gemm_kernel<Elem, kMode, true, 256, ClusterOf<2>>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(S::kSmem));
  if (e != cudaSuccess) return e;
  // as many clusters as fit at once (one CTA per SM), at most one per unit; per-device,
  // per-kernel occupancy, computed once (concurrent first calls agree)
  static std::atomic<int> max_clusters[64];
  int dev = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  cudaLaunchAttribute attr[1];
  int known = max_clusters[dev].load(std::memory_order_relaxed);
  if (known == 0) {
    cudaLaunchConfig_t q = cluster_config(attr, 2, 2, S::kThreads, S::kSmem, s);
    int n = 0;
    if ((e = cudaOccupancyMaxActiveClusters(&n, kern, &q)) != cudaSuccess) return e;
    if (n < 1) return cudaErrorInvalidConfiguration;
    max_clusters[dev].store(n, std::memory_order_relaxed);
    known = n;
  }
  const int clusters = known < args.plan.n_units ? known : args.plan.n_units;
  cudaLaunchConfig_t cfg = cluster_config(attr, 2, unsigned(2 * clusters), S::kThreads, S::kSmem, s);
  return cudaLaunchKernelEx(&cfg, kern, a0, a1, w, g, g2, args);
}

}  // namespace
}  // namespace alr

extern "C" {

size_t alr_cluster_args_size(int which) {
  return which == 0 ? sizeof(alr::LossArgs) : sizeof(alr::GemmArgs);
}

cudaError_t alr_cluster_launch_loss(int mode, const CUtensorMap* a0, const CUtensorMap* a1,
                                    const CUtensorMap* w, const CUtensorMap* g,
                                    const CUtensorMap* g2, const alr::LossArgs* args,
                                    cudaStream_t s) {
  using namespace alr;
  if (a0 == nullptr || a1 == nullptr || w == nullptr || g == nullptr || g2 == nullptr ||
      args == nullptr || args->plan.bn != 256 || !args->plan.mc)
    return cudaErrorInvalidValue;
  switch (mode) {
    case kModeFwd: return launch_cluster<kModeFwd>(*a0, *a1, *w, *g, *g2, *args, s);
    case kModeFwdKeep: return launch_cluster<kModeFwdKeep>(*a0, *a1, *w, *g, *g2, *args, s);
    case kModeBwd: return launch_cluster<kModeBwd>(*a0, *a1, *w, *g, *g2, *args, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // extern "C"
