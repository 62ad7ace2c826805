// Tensor-core GEMM with fp32 output for the backward products of the slot loss:
//   dH_d = G W^T     (A = G [N, V] K-major, B = W [d, V] K-major, C stored)
//   dW  += H_d^T G   (A = H_d [N, d] read MN-major, B = G [N, V] MN-major, C accumulated)
// tf32 products (fp32 inputs) take K-major operands only; the caller transposes for them.
// 128 x 256 output tiles, tcgen05.mma (M=128, N=256) into two 256-column TMEM buffers,
// a 4-stage TMA pipeline with 128-byte swizzle, persistent CTAs over raster groups of
// `group_m` row blocks.  Warp roles as in loss_gemm_kernel.cuh.
//
// Cluster form (Cl = ClusterOf<2> or ClusterOf<4>, bf16; instantiated only in csrc_cluster/,
// whose policy supplies the multicast copy and commit): the kMc = Cl::kCtas CTAs of a cluster
// compute the 128-row tiles kMc i .. kMc i + kMc - 1 against the same 256 columns of B.  Each
// CTA loads its own A rows and a 1 / kMc share of the B tile, multicast into every CTA's
// stage, so every B byte leaves L2 once per cluster; a stage is refilled only after all the
// cluster's products have read it (every MMA issuer's commit arrives on every CTA's empty
// barrier).  Cl = NoCluster: one CTA per tile.
#pragma once

#include "kernels.h"
#include "tc_common.cuh"

namespace alr {
namespace {

constexpr int kBM = 128;
constexpr int kBN = 256;
constexpr int kThreads = 256;
constexpr int kEpiWarp0 = 4;
constexpr int kEpiWarps = 4;
constexpr int kEpiBarrier = 1;                    // named barrier of the epilogue warps
static_assert(kEpiWarp0 + kEpiWarps == kThreads / 32, "the epilogue warps end the block");
constexpr int kStages = 4;
constexpr int kABytes = kBM * 128;                // 16 KB
constexpr int kBBytes = kBN * 128;                // 32 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kCtrlBytes = 256;
constexpr size_t kSmemBytes = 1024 + size_t(kStages) * kStageBytes + kCtrlBytes;

template <typename Elem>
struct Geo {
  static constexpr int kElem = sizeof(Elem);
  static constexpr int kKE = 128 / kElem;
  static constexpr int kMmaK = 32 / kElem;
  static constexpr int kChunkMN = 128 / kElem;
  static constexpr uint32_t kChunkBytes = kKE * 128;
  static constexpr bool kTf32 = (kElem == 4);
};

ALR_DEV void decode_tile(const GemmArgs& a, int t, int& mb, int& nb) {
  const int per_group = a.group_m * a.n_nb;
  const int g = t / per_group;
  const int w = t - g * per_group;
  const int gm = min(a.group_m, a.n_mb - g * a.group_m);
  nb = w / gm;
  mb = g * a.group_m + (w - nb * gm);
}

ALR_DEV bool warp_wait(uint64_t* bar, uint32_t parity, const AbortFlag& ab) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, ab) ? 1 : 0;
  return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

// Operand tile descriptor for the kk-th MMA of a stage.
template <typename Elem, bool kMN>
ALR_DEV uint64_t operand_desc(uint32_t base, int kk) {
  using G = Geo<Elem>;
  if constexpr (kMN) return sdesc_sw128(base + kk * G::kMmaK * 128, G::kChunkBytes, 1024);
  else return sdesc_sw128(base + kk * 32, 16, 1024);
}

// Load one operand tile of `extent` rows (MN) over the stage's K range.
template <typename Elem, bool kMN, int kExtent>
ALR_DEV void load_operand(uint8_t* dst, const CUtensorMap* map, uint64_t* bar, int mn0, int kb) {
  using G = Geo<Elem>;
  if constexpr (kMN) {
#pragma unroll
    for (int c = 0; c < kExtent / G::kChunkMN; ++c)
      tma_load_2d(dst + c * G::kChunkBytes, map, bar, mn0 + c * G::kChunkMN, kb * G::kKE);
  } else {
    tma_load_2d(dst, map, bar, kb * G::kKE, mn0);
  }
}

// B share of the multicast form: `kExtent` / kParts MN rows starting at share `r`, into the same
// offsets of every CTA of the cluster.
template <class Cl, typename Elem, bool kMN, int kExtent, int kParts>
ALR_DEV void load_operand_share_mc(uint8_t* dst, const CUtensorMap* map, uint64_t* bar, int mn0,
                                   int kb, int r) {
  using G = Geo<Elem>;
  constexpr int kShare = kExtent / kParts;
  constexpr uint16_t kMask = uint16_t((1u << kParts) - 1u);
  if constexpr (kMN) {
    static_assert(kShare % G::kChunkMN == 0, "share of whole 128-byte chunks");
#pragma unroll
    for (int c = 0; c < kShare / G::kChunkMN; ++c) {
      const int cc = r * (kShare / G::kChunkMN) + c;
      Cl::load_mc(dst + cc * G::kChunkBytes, map, bar, mn0 + cc * G::kChunkMN, kb * G::kKE,
                     kMask);
    }
  } else {
    Cl::load_mc(dst + r * kShare * 128, map, bar, kb * G::kKE, mn0 + r * kShare, kMask);
  }
}

// Cl: NoCluster, or ClusterOf<kMc> (kMc CTAs per multicast cluster).
template <typename Elem, bool kAMN, bool kBMN, bool kAcc, class Cl>
__global__ void __launch_bounds__(kThreads, 1)
    plain_gemm_kernel(const __grid_constant__ CUtensorMap tm_a,
                      const __grid_constant__ CUtensorMap tm_b, const GemmArgs args) {
  constexpr int kMc = Cl::kCtas > 1 ? Cl::kCtas : 0;   // CTAs per cluster (0: none)
  using G = Geo<Elem>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align_1024(smem_raw);
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes);
  uint64_t* empty_bar = full_bar + kStages;
  uint64_t* tfull_bar = empty_bar + kStages;
  uint64_t* tempty_bar = tfull_bar + 2;
  uint64_t* drain_bar = tempty_bar + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile int* abort_word = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* tile_ready = abort_word + 1;   // [2], one per accumulator buffer

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const AbortFlag ab{abort_word, args.status};
  // kMc: tiles are handed out per cluster, and CTA `rank` takes row block kMc mb + rank
  const int rank = kMc ? int(cluster_ctarank()) : 0;
  const int t0 = kMc ? int(cluster_id_x()) : int(blockIdx.x);
  const int t_step = kMc ? int(n_clusters_x()) : int(gridDim.x);

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], kMc ? kMc : 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull_bar[i], 1);
      mbar_init(&tempty_bar[i], kEpiWarps);
    }
    mbar_init(drain_bar, 1);
    *abort_word = 0;
    fence_mbar_init();
  }
  if (threadIdx.x == 32) {
    tma_prefetch_desc(&tm_a);
    tma_prefetch_desc(&tm_b);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  if constexpr (kMc) cluster_sync();   // the peer's copies and commits find initialised barriers
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int n_kb = (args.K + G::kKE - 1) / G::kKE;

  if (warp == 0) {
    if (lane == 0) {
      // test hook: start filling at stage 1, so stage 0, the MMA issuer's first, stays empty;
      // its bounded wait runs out and every role of the CTA takes the timeout path
      int stage = args.withhold_first_stage ? 1 : 0;
      uint32_t phase = 0, armed = 0, armed_par = 0;
      bool ok = true;
      for (int t = t0; ok && t < args.n_tiles; t += t_step) {
        int mb, nb;
        decode_tile(args, t, mb, nb);
        if (kMc) mb = kMc * mb + rank;
        for (int kb = 0; kb < n_kb; ++kb) {
          if (!mbar_wait(&empty_bar[stage], phase ^ 1, ab)) {
            ok = false;
            break;
          }
          uint8_t* sb = smem + stage * kStageBytes;
          mbar_arrive_expect_tx(&full_bar[stage], kStageBytes);
          load_operand<Elem, kAMN, kBM>(sb, &tm_a, &full_bar[stage], mb * kBM, kb);
          if constexpr (kMc)
            load_operand_share_mc<Cl, Elem, kBMN, kBN, kMc>(sb + kABytes, &tm_b, &full_bar[stage],
                                                        nb * kBN, kb, rank);
          else
            load_operand<Elem, kBMN, kBN>(sb + kABytes, &tm_b, &full_bar[stage], nb * kBN, kb);
          armed |= 1u << stage;
          armed_par = (armed_par & ~(1u << stage)) | (phase << stage);
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (!ok) {
        for (int s = 0; s < kStages; ++s)
          if (armed & (1u << s)) mbar_wait_drain(&full_bar[s], (armed_par >> s) & 1u);
      }
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_make(G::kTf32, kBM, kBN, kAMN, kBMN);
      int stage = 0, abuf = 0;
      uint32_t phase = 0, aphase = 0;
      bool ok = true;
      for (int t = t0; ok && t < args.n_tiles; t += t_step) {
        if (!mbar_wait(&tempty_bar[abuf], aphase ^ 1, ab)) break;
        tc_fence_after();
        const uint32_t d_acc = tmem_base + uint32_t(abuf * kBN);
        for (int kb = 0; kb < n_kb; ++kb) {
          if (!mbar_wait(&full_bar[stage], phase, ab)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * kStageBytes);
#pragma unroll
          for (int kk = 0; kk < G::kKE / G::kMmaK; ++kk) {
            mma_issue<G::kTf32>(d_acc, operand_desc<Elem, kAMN>(sa, kk),
                                operand_desc<Elem, kBMN>(sa + kABytes, kk), idesc,
                                (kb > 0 || kk > 0) ? 1u : 0u);
          }
          if constexpr (kMc) Cl::commit_mc(&empty_bar[stage], uint16_t((1u << kMc) - 1u));
          else mma_commit(&empty_bar[stage]);
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        mma_commit(&tfull_bar[abuf]);
        if (++abuf == 2) {
          abuf = 0;
          aphase ^= 1;
        }
      }
      mma_commit(drain_bar);
      mbar_wait_drain(drain_bar, 0);
    }
  } else if (warp >= kEpiWarp0) {
    const int q = warp & 3;
    const uint32_t lane_addr = tmem_base + (uint32_t(q * 32) << 16);
    int abuf = 0;
    uint32_t aphase = 0;
    for (int t = t0; t < args.n_tiles; t += t_step) {
      int mb, nb;
      decode_tile(args, t, mb, nb);
      if (kMc) mb = kMc * mb + rank;
      // The first epilogue warp waits for the accumulator and posts the outcome in the
      // buffer's word; the others wait, descheduled, in a named barrier.  Every epilogue warp
      // passes the same barriers and follows the one outcome, so they leave together; a word
      // is rewritten only two barriers later, after every warp has read it.
      if (warp == kEpiWarp0) {
        const bool w = warp_wait(&tfull_bar[abuf], aphase, ab);
        if (lane == 0) tile_ready[abuf] = w ? 1 : 0;
        __syncwarp();
      }
      named_bar_sync(kEpiBarrier, kEpiWarps * 32);
      if (tile_ready[abuf] == 0) break;
      tc_fence_after();
      const int m = mb * kBM + q * 32 + lane;
      const bool m_ok = m < args.M;
      float* crow = args.C + size_t(m_ok ? m : 0) * size_t(args.ldc);
      const uint32_t tb = lane_addr + uint32_t(abuf * kBN);
#pragma unroll 1
      for (int c = 0; c < kBN / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(tb + c * 32, r);
        tmem_ld_wait();
        reg_fence(r);
        const int n0 = nb * kBN + c * 32;
        if (m_ok) {
#pragma unroll
          for (int j = 0; j < 32; j += 4) {
            const int n = n0 + j;
            if (n < args.Nc) {
              float4 v = make_float4(__uint_as_float(r[j]), __uint_as_float(r[j + 1]),
                                     __uint_as_float(r[j + 2]), __uint_as_float(r[j + 3]));
              float4* dst = reinterpret_cast<float4*>(crow + n);
              if (kAcc) {
                const float4 o = *dst;
                v.x += o.x;
                v.y += o.y;
                v.z += o.z;
                v.w += o.w;
              }
              *dst = v;
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&tempty_bar[abuf]);
      if (++abuf == 2) {
        abuf = 0;
        aphase ^= 1;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  if constexpr (kMc) cluster_sync();   // no CTA leaves while its peer may still write into it
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, 512);
  }
}

}  // namespace
}  // namespace alr
