// The plain GEMM's multicast cluster forms (plain_gemm_kernel.cuh with Cl = ClusterOf<2> or
// ClusterOf<4>, bf16 operands).  Built into libalr_cluster.so only.
#include <atomic>

#include "cluster_forms.h"
#include "cluster_ptx.cuh"
#include "plain_gemm_kernel.cuh"

namespace alr {
namespace {

template <bool kAMN, bool kBMN, bool kAcc, int kMc>
cudaError_t launch_t(const CUtensorMap& a, const CUtensorMap& b, const GemmArgs& args,
                     cudaStream_t s) {
  auto kern = plain_gemm_kernel<__nv_bfloat16, kAMN, kBMN, kAcc, ClusterOf<kMc>>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(kSmemBytes));
  if (e != cudaSuccess) return e;
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = cluster_config(attr, kMc, unsigned(args.grid), kThreads, kSmemBytes, s);
  return cudaLaunchKernelEx(&cfg, kern, a, b, args);
}

template <int kMc>
int max_clusters() {
  // per-device occupancy, computed once (concurrent first calls compute the same value)
  static std::atomic<int> cached[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  const int known = cached[dev].load(std::memory_order_relaxed);
  if (known > 0) return known;
  auto kern = plain_gemm_kernel<__nv_bfloat16, false, false, false, ClusterOf<kMc>>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           int(kSmemBytes)) != cudaSuccess)
    return 0;
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = cluster_config(attr, kMc, unsigned(kMc), kThreads, kSmemBytes, nullptr);
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) return 0;
  cached[dev].store(n, std::memory_order_relaxed);
  return n;
}

template <int kMc>
cudaError_t launch_mc(bool a_mn, bool b_mn, bool acc, const CUtensorMap& a, const CUtensorMap& b,
                      const GemmArgs& args, cudaStream_t s) {
  const int key = (a_mn ? 4 : 0) | (b_mn ? 2 : 0) | (acc ? 1 : 0);
  switch (key) {
    case 0: return launch_t<false, false, false, kMc>(a, b, args, s);
    case 1: return launch_t<false, false, true, kMc>(a, b, args, s);
    case 2: return launch_t<false, true, false, kMc>(a, b, args, s);
    case 3: return launch_t<false, true, true, kMc>(a, b, args, s);
    case 4: return launch_t<true, false, false, kMc>(a, b, args, s);
    case 5: return launch_t<true, false, true, kMc>(a, b, args, s);
    case 6: return launch_t<true, true, false, kMc>(a, b, args, s);
    default: return launch_t<true, true, true, kMc>(a, b, args, s);
  }
}

}  // namespace
}  // namespace alr

extern "C" {

int alr_cluster_gemm_max_clusters(int cluster) {
  return cluster == 4 ? alr::max_clusters<4>() : alr::max_clusters<2>();
}

cudaError_t alr_cluster_launch_gemm(int cluster, int a_mn, int b_mn, int accumulate,
                                    const CUtensorMap* a, const CUtensorMap* b,
                                    const alr::GemmArgs* args, cudaStream_t s) {
  if (a == nullptr || b == nullptr || args == nullptr || (cluster != 2 && cluster != 4))
    return cudaErrorInvalidValue;
  if (cluster == 4) return alr::launch_mc<4>(a_mn != 0, b_mn != 0, accumulate != 0, *a, *b, *args, s);
  return alr::launch_mc<2>(a_mn != 0, b_mn != 0, accumulate != 0, *a, *b, *args, s);
}

}  // extern "C"
