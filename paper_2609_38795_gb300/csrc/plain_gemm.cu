// Launchers of the tensor-core GEMM of the backward products (plain_gemm_kernel.cuh): the
// single-CTA form, built here; the cluster forms are launched through libalr_cluster.so
// (cluster_forms.h).
#include "plain_gemm_kernel.cuh"

namespace alr {
namespace {

template <typename Elem, bool kAMN, bool kBMN, bool kAcc>
cudaError_t launch_t(const CUtensorMap& a, const CUtensorMap& b, const GemmArgs& args,
                     cudaStream_t s) {
  auto kern = plain_gemm_kernel<Elem, kAMN, kBMN, kAcc, NoCluster>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(kSmemBytes));
  if (e != cudaSuccess) return e;
  kern<<<args.grid, kThreads, kSmemBytes, s>>>(a, b, args);
  return cudaGetLastError();
}

template <typename Elem>
cudaError_t dispatch(bool a_mn, bool b_mn, bool acc, const CUtensorMap& a, const CUtensorMap& b,
                     const GemmArgs& args, cudaStream_t s) {
  if constexpr (sizeof(Elem) == 4) {
    // tf32 products take K-major operands only
    if (a_mn || b_mn) return cudaErrorInvalidValue;
    return acc ? launch_t<Elem, false, false, true>(a, b, args, s)
               : launch_t<Elem, false, false, false>(a, b, args, s);
  } else {
    const int key = (a_mn ? 4 : 0) | (b_mn ? 2 : 0) | (acc ? 1 : 0);
    switch (key) {
      case 0: return launch_t<Elem, false, false, false>(a, b, args, s);
      case 1: return launch_t<Elem, false, false, true>(a, b, args, s);
      case 2: return launch_t<Elem, false, true, false>(a, b, args, s);
      case 3: return launch_t<Elem, false, true, true>(a, b, args, s);
      case 4: return launch_t<Elem, true, false, false>(a, b, args, s);
      case 5: return launch_t<Elem, true, false, true>(a, b, args, s);
      case 6: return launch_t<Elem, true, true, false>(a, b, args, s);
      default: return launch_t<Elem, true, true, true>(a, b, args, s);
    }
  }
}

}  // namespace

size_t plain_gemm_smem_bytes(int) { return kSmemBytes; }

cudaError_t launch_plain_gemm(int dtype, bool a_mn, bool b_mn, bool accumulate,
                              const CUtensorMap& a, const CUtensorMap& b, const GemmArgs& args,
                              cudaStream_t s) {
  if (dtype == 0) return dispatch<__nv_bfloat16>(a_mn, b_mn, accumulate, a, b, args, s);
  return dispatch<float>(a_mn, b_mn, accumulate, a, b, args, s);
}

}  // namespace alr
