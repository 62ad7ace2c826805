// PTX of the kernel forms that share work across the CTAs of a cluster: TMA tile loads
// multicast into several CTAs' shared memory, tensor-core commits that arrive on several CTAs'
// mbarriers, and the 2-SM (.cta_group::2) products of CTA pairs.  Only the sources in this
// directory include it; they build libalr_cluster.so, which the main library loads in
// single-process runs only (a process that is one rank of several never loads it), so that
// multicast reads of device memory never happen in a multi-rank process.
#pragma once

#include "tc_common.cuh"

namespace alr {

// Shared::cluster address of the object at the same offset as `p` in CTA `rank`'s smem.
ALR_DEV uint32_t cluster_addr(const void* p, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(p)), "r"(rank));
  return r;
}

// Arrive on an mbarrier in any CTA of the cluster (release at cluster scope).
ALR_DEV void mbar_arrive_cluster(uint32_t cluster_bar) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_bar)
               : "memory");
}

// As mbar_try_wait, acquiring at cluster scope (arrivals come from the peer CTA too).
ALR_DEV bool mbar_try_wait_cl(uint64_t* bar, uint32_t parity) {
  uint32_t done;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(done)
      : "r"(smem_u32(bar)), "r"(parity), "r"(kSuspendHintNs)
      : "memory");
  return done != 0;
}

ALR_DEV bool mbar_wait_cl(uint64_t* bar, uint32_t parity, const AbortFlag& ab) {
  if (mbar_try_wait_cl(bar, parity)) return true;
  const uint64_t t0 = global_timer_ns();
  for (uint32_t i = 1;; ++i) {
    if (mbar_try_wait_cl(bar, parity)) return true;
    if (i % kWaitCheckEvery == 0) {
      if (*ab.smem) return false;
      if (global_timer_ns() - t0 > kWaitLimitNs) {
        *ab.smem = 1;
        atomicExch(ab.status, kStatusTimeout);
        return false;
      }
    }
  }
}

ALR_DEV void mbar_wait_drain_cl(uint64_t* bar, uint32_t parity) {
  const uint64_t t0 = global_timer_ns();
  while (!mbar_try_wait_cl(bar, parity)) {
    if (global_timer_ns() - t0 > kWaitLimitNs) return;
  }
}

// TMA tile load into this CTA's shared memory whose completion is counted on an mbarrier of
// either CTA of the pair (`cluster_bar`, a shared::cluster address).
ALR_DEV void tma_load_2d_pair(void* smem_dst, const CUtensorMap* map, uint32_t cluster_bar, int x,
                              int y) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(cluster_bar), "r"(x), "r"(y)
      : "memory");
}

// TMA tile load multicast to the CTAs of `cta_mask`: the tile lands at `smem_dst`'s offset in
// each of them and completes on the mbarrier at `bar`'s offset in each of them.
ALR_DEV void tma_load_2d_mc(void* smem_dst, const CUtensorMap* map, uint64_t* bar, int x, int y,
                            uint16_t cta_mask) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      ".multicast::cluster [%0], [%1, {%3, %4}], [%2], %5;" ::"r"(smem_u32(smem_dst)),
      "l"(reinterpret_cast<uint64_t>(map)), "r"(smem_u32(bar)), "r"(x), "r"(y), "h"(cta_mask)
      : "memory");
}

// mma_commit that arrives on the mbarrier at `bar`'s offset in every CTA of `cta_mask`.
ALR_DEV void mma_commit_mc(uint64_t* bar, uint16_t cta_mask) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_u32(bar)),
      "h"(cta_mask)
      : "memory");
}

// Collective tensor-memory allocation over the pair: one warp of each CTA executes it.
ALR_DEV void tmem_alloc_pair(uint32_t* smem_result, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                   smem_u32(smem_result)),
               "r"(ncols)
               : "memory");
}
ALR_DEV void tmem_relinquish_pair() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
ALR_DEV void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

// One M = 256 product for the pair (bf16 operands), issued by the even CTA.
ALR_DEV void mma_issue_pair(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                            uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(tmem_d),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrive once on the mbarrier at `bar`'s offset in every CTA of `cta_mask` when all pair
// products this thread issued so far have completed.
ALR_DEV void mma_commit_pair(uint64_t* bar, uint16_t cta_mask) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
      " [%0], %1;" ::"r"(smem_u32(bar)),
      "h"(cta_mask)
      : "memory");
}

// Host side: the launch configuration of a kernel on clusters of `ctas` CTAs along x (attr
// must outlive the launch).
inline cudaLaunchConfig_t cluster_config(cudaLaunchAttribute* attr, unsigned ctas, unsigned grid,
                                         unsigned threads, size_t smem, cudaStream_t s) {
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = ctas;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(threads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cfg;
}

// Cluster policies of the fused loss and plain GEMM kernels: clusters of kCtas CTAs in which
// each CTA loads a 1 / kCtas share of every head (B) tile, multicast into all of them, and each
// MMA issuer's commit releases the stage in all of them.
template <int kN>
struct ClusterOf {
  static constexpr int kCtas = kN;
  static ALR_DEV void load_mc(void* smem_dst, const CUtensorMap* map, uint64_t* bar, int x, int y,
                              uint16_t cta_mask) {
    tma_load_2d_mc(smem_dst, map, bar, x, y, cta_mask);
  }
  static ALR_DEV void commit_mc(uint64_t* bar, uint16_t cta_mask) { mma_commit_mc(bar, cta_mask); }
};

}  // namespace alr
