// Interface between libalr.so and libalr_cluster.so, the library of the kernel forms that
// share operand tiles across the CTAs of a cluster: the fused loss kernel and the plain GEMM on
// clusters whose CTAs multicast their share of every head (B) tile into all of them, and the
// GEMM on CTA pairs issuing 2-SM (.cta_group::2) products.  Their sources sit in csrc_cluster/
// and are built into that library alone.  libalr.so loads it on first use, from its own
// directory, in a single-process run; a process that is one rank of several (WORLD_SIZE > 1)
// never loads it and runs the single-CTA forms, so multicast reads of device memory stay out of
// multi-rank processes.  Both libraries are built together from these headers; the argument
// structs' sizes are compared when the library is loaded.
//
// This is an internal interface (not part of include/alr.h): the structs are the kernels'
// own argument records, and every call returns the CUDA error of its launch.
#pragma once

#include <cstddef>
#include <cuda.h>
#include <cuda_runtime.h>

#include "kernels.h"

extern "C" {

// sizeof(LossArgs) for which = 0, sizeof(GemmArgs) for which = 1, as the cluster library was
// compiled.
size_t alr_cluster_args_size(int which);

// The fused loss kernel's cluster form (bf16 inputs, 256-column tiles, the dual modes
// kModeFwd, kModeFwdKeep and kModeBwd): args->plan as loss_plan builds it with mc = 1.
cudaError_t alr_cluster_launch_loss(int mode, const CUtensorMap* a0, const CUtensorMap* a1,
                                    const CUtensorMap* w, const CUtensorMap* g,
                                    const CUtensorMap* g2, const alr::LossArgs* args,
                                    cudaStream_t s);

// The plain GEMM's multicast form (bf16): clusters of `cluster` (2 or 4) CTAs over row blocks
// cluster i .. cluster i + cluster - 1 share each B tile (n_mb counts row-block groups, `grid` is
// `cluster` times the number of clusters; the K-major B map has 256 / cluster-row boxes).
cudaError_t alr_cluster_launch_gemm(int cluster, int a_mn, int b_mn, int accumulate,
                                    const CUtensorMap* a, const CUtensorMap* b,
                                    const alr::GemmArgs* args, cudaStream_t s);
// Clusters of `cluster` CTAs of the multicast GEMM that can be resident at once (0 on error).
int alr_cluster_gemm_max_clusters(int cluster);

// The same products on CTA pairs with M = 256 tcgen05 products: n_mb counts 256-row pair
// blocks, `grid` is twice the number of pairs, and the B tensor map has 128-row boxes (K-major)
// or 64 x 64 boxes (MN-major).
cudaError_t alr_cluster_launch_pair_gemm(int a_mn, int b_mn, int accumulate, const CUtensorMap* a,
                                         const CUtensorMap* b, const alr::GemmArgs* args,
                                         cudaStream_t s);
// CTA pairs of the pair GEMM that can be resident at once on the current device (0 on error).
int alr_cluster_pair_gemm_max_pairs(void);

}  // extern "C"

namespace alr {

struct ClusterForms {
  decltype(&alr_cluster_launch_loss) launch_loss;
  decltype(&alr_cluster_launch_gemm) launch_gemm;
  decltype(&alr_cluster_gemm_max_clusters) gemm_max_clusters;
  decltype(&alr_cluster_launch_pair_gemm) launch_pair_gemm;
  decltype(&alr_cluster_pair_gemm_max_pairs) pair_gemm_max_pairs;
};

// True in a process launched as one rank of several (WORLD_SIZE > 1, as torchrun and
// torch.distributed set it).
bool multi_rank_process();

// The cluster library's entry points, loaded once per process on first use; nullptr in a
// multi-rank process or when the library cannot be loaded, with the reason in
// cluster_forms_error().
const ClusterForms* cluster_forms();
const char* cluster_forms_error();

}  // namespace alr
