// Launchers of the fused head-GEMM kernels of the slot loss (loss_gemm_kernel.cuh): the
// single-CTA forms, built here; the cluster form of the dual modes is launched through
// libalr_cluster.so (cluster_forms.h).
#include "cluster_forms.h"
#include "loss_gemm_kernel.cuh"

namespace alr {
namespace {

template <typename Elem, int kMode, int kBN>
cudaError_t launch_impl(const CUtensorMap& a0, const CUtensorMap& a1, const CUtensorMap& w,
                        const CUtensorMap& g, const CUtensorMap& g2, const LossArgs& args,
                        cudaStream_t s) {
  using S = Shape<kMode, kBN, is_staged(kMode, sizeof(Elem))>;
  auto kern = loss_gemm_kernel<Elem, kMode, sizeof(Elem) == 2, kBN, NoCluster>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(S::kSmem));
  if (e != cudaSuccess) return e;
  kern<<<args.plan.grid, S::kThreads, S::kSmem, s>>>(a0, a1, w, g, g2, args);
  return cudaGetLastError();
}

template <typename Elem, int kMode>
cudaError_t by_width(const CUtensorMap& a0, const CUtensorMap& a1, const CUtensorMap& w,
                     const CUtensorMap& g, const CUtensorMap& g2, const LossArgs& args,
                     cudaStream_t s) {
  if (args.plan.bn == 128) return launch_impl<Elem, kMode, 128>(a0, a1, w, g, g2, args, s);
  return launch_impl<Elem, kMode, 256>(a0, a1, w, g, g2, args, s);
}

template <typename Elem>
cudaError_t by_mode(int mode, const CUtensorMap& a0, const CUtensorMap& a1, const CUtensorMap& w,
                    const CUtensorMap& g, const CUtensorMap& g2, const LossArgs& args,
                    cudaStream_t s) {
  switch (mode) {
    case kModeFwd: return by_width<Elem, kModeFwd>(a0, a1, w, g, g2, args, s);
    case kModeFwdKeep: return by_width<Elem, kModeFwdKeep>(a0, a1, w, g, g2, args, s);
    case kModeBwd: return by_width<Elem, kModeBwd>(a0, a1, w, g, g2, args, s);
    case kModeReadout: return by_width<Elem, kModeReadout>(a0, a1, w, g, g2, args, s);
    case kModeTopkFwd: return by_width<Elem, kModeTopkFwd>(a0, a1, w, g, g2, args, s);
    case kModeTopkBwd: return by_width<Elem, kModeTopkBwd>(a0, a1, w, g, g2, args, s);
    case kModeTopkFwdKeep: return by_width<Elem, kModeTopkFwdKeep>(a0, a1, w, g, g2, args, s);
    default: return cudaErrorInvalidValue;
  }
}

}  // namespace

cudaError_t launch_loss_kernel(int mode, int dtype, const CUtensorMap& a0, const CUtensorMap& a1,
                               const CUtensorMap& w, const CUtensorMap& g_store,
                               const CUtensorMap& g_store2, const LossArgs& args, cudaStream_t s) {
  if (args.plan.mc) {
    // the plan was made for the cluster form (bf16, 256-column tiles, dual modes only)
    const ClusterForms* cf = cluster_forms();
    if (cf == nullptr || dtype != 0 || args.plan.bn != 256 || !is_dual(mode))
      return cudaErrorNotSupported;
    return cf->launch_loss(mode, &a0, &a1, &w, &g_store, &g_store2, &args, s);
  }
  if (dtype == 0) return by_mode<__nv_bfloat16>(mode, a0, a1, w, g_store, g_store2, args, s);
  return by_mode<float>(mode, a0, a1, w, g_store, g_store2, args, s);
}

}  // namespace alr
