// 2-SM tensor-core GEMM with fp32 output (bf16 operands) for the backward products of the
// slot loss:
//   dH_d = G W^T     (A = G [N, V] K-major, B = W [d, V] K-major, C stored)
//   dW  += H_d^T G   (A = H_d [N, d] read MN-major, B = G [N, V] MN-major, C accumulated)
// A cluster of two CTAs computes a 256 x 256 tile of C with tcgen05.mma.cta_group::2 (M = 256,
// N = 256): CTA r of the pair loads rows [128 r, 128 r + 128) of the A tile and columns
// [128 r, 128 r + 128) of the B tile into its own shared memory, the even CTA issues the
// products for both, and each CTA finds its 128 rows of the tile in its own tensor memory
// (two 256-column buffers).  Against the one-CTA kernel (plain_gemm_kernel.cuh) every CTA reads half
// the B bytes per product from shared memory and from L2.
//
// Pipeline: 6 stages of (A 16 KB + B half 16 KB) per CTA.  The even CTA's full barrier of a
// stage counts the bytes of both CTAs' loads (TMA .cta_group::2 completes on the peer's
// barrier); the products' commit releases the stage in both CTAs at once (multicast), and
// the epilogue warps of both CTAs release an accumulator buffer on the even CTA's barrier.
// Every wait is bounded (tc_common.cuh, cluster_ptx.cuh).  Built into libalr_cluster.so only.
#include <atomic>

#include "cluster_forms.h"
#include "cluster_ptx.cuh"
#include "kernels.h"

namespace alr {
namespace {

constexpr int kRows = 128;                  // rows of A and C per CTA (256 per pair)
constexpr int kCols = 256;                  // columns of C per pair tile
constexpr int kHalf = kCols / 2;            // columns of B loaded by each CTA
constexpr int kThreads = 256;
constexpr int kEpiWarp0 = 4;
constexpr int kEpiWarps = 4;
constexpr int kStages = 6;
constexpr int kABytes = kRows * 128;        // 16 KB: 128 rows x 64 bf16 of K
constexpr int kBBytes = kHalf * 128;        // 16 KB
constexpr int kStageBytes = kABytes + kBBytes;
constexpr int kKE = 64;                     // K elements per stage
constexpr int kMmaK = 16;                   // K per MMA
constexpr int kChunkMN = 64;                // MN elements per 128-byte chunk
constexpr uint32_t kChunkBytes = kKE * 128;
// Slack after the last stage: an operand tile read past its own extent still lands in this
// CTA's allocation.
constexpr int kGuardBytes = 16 * 1024;
constexpr int kCtrlBytes = 256;
constexpr size_t kSmemBytes =
    1024 + size_t(kStages) * kStageBytes + kGuardBytes + kCtrlBytes;
static_assert((2 * kStages + 2 * 2 + 1) * 8 + 8 <= kCtrlBytes, "control block");

ALR_DEV void decode_tile(const GemmArgs& a, int t, int& mb, int& nb) {
  const int per_group = a.group_m * a.n_nb;
  const int g = t / per_group;
  const int w = t - g * per_group;
  const int gm = min(a.group_m, a.n_mb - g * a.group_m);
  nb = w / gm;
  mb = g * a.group_m + (w - nb * gm);
}

ALR_DEV bool warp_wait_cl(uint64_t* bar, uint32_t parity, const AbortFlag& ab) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait_cl(bar, parity, ab) ? 1 : 0;
  return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

template <bool kMN>
ALR_DEV uint64_t operand_desc(uint32_t base, int kk) {
  if constexpr (kMN) return sdesc_sw128(base + kk * kMmaK * 128, kChunkBytes, 1024);
  else return sdesc_sw128(base + kk * 32, 16, 1024);
}

// Load `kExtent` MN rows of an operand over the stage's K range; completion counted on the
// even CTA's full barrier.
template <bool kMN, int kExtent>
ALR_DEV void load_operand(uint8_t* dst, const CUtensorMap* map, uint32_t bar, int mn0, int kb) {
  if constexpr (kMN) {
#pragma unroll
    for (int c = 0; c < kExtent / kChunkMN; ++c)
      tma_load_2d_pair(dst + c * kChunkBytes, map, bar, mn0 + c * kChunkMN, kb * kKE);
  } else {
    tma_load_2d_pair(dst, map, bar, kb * kKE, mn0);
  }
}

template <bool kAMN, bool kBMN, bool kAcc>
__global__ void __launch_bounds__(kThreads, 1)
    pair_gemm_kernel(const __grid_constant__ CUtensorMap tm_a,
                     const __grid_constant__ CUtensorMap tm_b, const GemmArgs args) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align_1024(smem_raw);
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(smem + kStages * kStageBytes + kGuardBytes);
  uint64_t* empty_bar = full_bar + kStages;
  uint64_t* tfull_bar = empty_bar + kStages;
  uint64_t* tempty_bar = tfull_bar + 2;
  uint64_t* drain_bar = tempty_bar + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile int* abort_word = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const uint32_t rank = cluster_ctarank();
  const bool leader = rank == 0;
  const int pair = int(cluster_id_x());
  const int n_pairs = int(n_clusters_x());
  const AbortFlag ab{abort_word, args.status};

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull_bar[i], 1);
      mbar_init(&tempty_bar[i], 2 * kEpiWarps);
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
    tmem_alloc_pair(tmem_slot, 512);
    tmem_relinquish_pair();
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync();   // both CTAs' barriers are initialised before any remote arrival
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int n_kb = (args.K + kKE - 1) / kKE;

  if (warp == 0) {
    // ------------------------------------------------------------- TMA producer ---
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, armed = 0, armed_par = 0;
      bool ok = true;
      for (int t = pair; ok && t < args.n_tiles; t += n_pairs) {
        int mb, nb;
        decode_tile(args, t, mb, nb);
        const int m0 = mb * 2 * kRows + int(rank) * kRows;
        const int n0 = nb * kCols + int(rank) * kHalf;
        for (int kb = 0; kb < n_kb; ++kb) {
          if (!mbar_wait_cl(&empty_bar[stage], phase ^ 1, ab)) {
            ok = false;
            break;
          }
          uint8_t* sb = smem + stage * kStageBytes;
          const uint32_t fb = cluster_addr(&full_bar[stage], 0);
          if (leader) mbar_arrive_expect_tx(&full_bar[stage], 2 * kStageBytes);
          load_operand<kAMN, kRows>(sb, &tm_a, fb, m0, kb);
          load_operand<kBMN, kHalf>(sb + kABytes, &tm_b, fb, n0, kb);
          armed |= 1u << stage;
          armed_par = (armed_par & ~(1u << stage)) | (phase << stage);
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
      }
      if (!ok && leader) {  // let every copy the even CTA armed land before the pair goes away
        for (int s = 0; s < kStages; ++s)
          if (armed & (1u << s)) mbar_wait_drain_cl(&full_bar[s], (armed_par >> s) & 1u);
      }
    }
  } else if (warp == 1) {
    // ---------------------------------------------- MMA issuer (even CTA of the pair) ---
    if (lane == 0 && leader) {
      constexpr uint32_t idesc = idesc_make(false, 2 * kRows, kCols, kAMN, kBMN);
      int stage = 0, abuf = 0;
      uint32_t phase = 0, aphase = 0;
      bool ok = true;
      for (int t = pair; ok && t < args.n_tiles; t += n_pairs) {
        if (!mbar_wait_cl(&tempty_bar[abuf], aphase ^ 1, ab)) break;
        tc_fence_after();
        const uint32_t d_acc = tmem_base + uint32_t(abuf * kCols);
        for (int kb = 0; kb < n_kb; ++kb) {
          if (!mbar_wait_cl(&full_bar[stage], phase, ab)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t sa = smem_u32(smem + stage * kStageBytes);
#pragma unroll
          for (int kk = 0; kk < kKE / kMmaK; ++kk)
            mma_issue_pair(d_acc, operand_desc<kAMN>(sa, kk), operand_desc<kBMN>(sa + kABytes, kk),
                           idesc, (kb > 0 || kk > 0) ? 1u : 0u);
          mma_commit_pair(&empty_bar[stage], 0x3);
          if (++stage == kStages) {
            stage = 0;
            phase ^= 1;
          }
        }
        if (!ok) break;
        mma_commit_pair(&tfull_bar[abuf], 0x3);
        if (++abuf == 2) {
          abuf = 0;
          aphase ^= 1;
        }
      }
      // all products complete before either CTA releases its tensor memory
      mma_commit_pair(drain_bar, 0x1);
      mbar_wait_drain_cl(drain_bar, 0);
    }
  } else if (warp >= kEpiWarp0) {
    // -------------------------------------------------------------------- epilogue ---
    const int q = warp & 3;
    const uint32_t lane_addr = tmem_base + (uint32_t(q * 32) << 16);
    const uint32_t tempty_cl0 = cluster_addr(&tempty_bar[0], 0);
    const uint32_t tempty_cl1 = cluster_addr(&tempty_bar[1], 0);
    int abuf = 0;
    uint32_t aphase = 0;
    for (int t = pair; t < args.n_tiles; t += n_pairs) {
      int mb, nb;
      decode_tile(args, t, mb, nb);
      if (!warp_wait_cl(&tfull_bar[abuf], aphase, ab)) break;
      tc_fence_after();
      const int m = mb * 2 * kRows + int(rank) * kRows + q * 32 + lane;
      const bool m_ok = m < args.M;
      float* crow = args.C + size_t(m_ok ? m : 0) * size_t(args.ldc);
      const uint32_t tb = lane_addr + uint32_t(abuf * kCols);
#pragma unroll 1
      for (int c = 0; c < kCols / 32; ++c) {
        uint32_t r[32];
        tmem_ld32(tb + c * 32, r);
        tmem_ld_wait();
        reg_fence(r);
        const int n0 = nb * kCols + c * 32;
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
      if (lane == 0) mbar_arrive_cluster(abuf ? tempty_cl1 : tempty_cl0);
      if (++abuf == 2) {
        abuf = 0;
        aphase ^= 1;
      }
    }
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync();   // the even CTA's products into both tensor memories are complete
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc_pair(tmem_base, 512);
  }
}

template <bool kAMN, bool kBMN, bool kAcc>
cudaError_t launch_t(const CUtensorMap& a, const CUtensorMap& b, const GemmArgs& args,
                     cudaStream_t s) {
  auto kern = pair_gemm_kernel<kAMN, kBMN, kAcc>;
  cudaError_t e =
      cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(kSmemBytes));
  if (e != cudaSuccess) return e;
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = cluster_config(attr, 2, unsigned(args.grid), kThreads, kSmemBytes, s);
  return cudaLaunchKernelEx(&cfg, kern, a, b, args);
}

}  // namespace

}  // namespace alr

extern "C" {

int alr_cluster_pair_gemm_max_pairs(void) {
  using namespace alr;
  // per-device occupancy, computed once (concurrent first calls compute the same value)
  static std::atomic<int> cached[64];
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
  const int known = cached[dev].load(std::memory_order_relaxed);
  if (known > 0) return known;
  auto kern = pair_gemm_kernel<false, false, false>;
  if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           int(kSmemBytes)) != cudaSuccess)
    return 0;
  cudaLaunchAttribute attr[1];
  cudaLaunchConfig_t cfg = cluster_config(attr, 2, 2, kThreads, kSmemBytes, nullptr);
  int n = 0;
  if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess) return 0;
  cached[dev].store(n, std::memory_order_relaxed);
  return n;
}

cudaError_t alr_cluster_launch_pair_gemm(int a_mn, int b_mn, int accumulate, const CUtensorMap* a,
                                         const CUtensorMap* b, const alr::GemmArgs* args,
                                         cudaStream_t s) {
  using namespace alr;
  if (a == nullptr || b == nullptr || args == nullptr) return cudaErrorInvalidValue;
  const int key = (a_mn ? 4 : 0) | (b_mn ? 2 : 0) | (accumulate ? 1 : 0);
  switch (key) {
    case 0: return launch_t<false, false, false>(*a, *b, *args, s);
    case 1: return launch_t<false, false, true>(*a, *b, *args, s);
    case 2: return launch_t<false, true, false>(*a, *b, *args, s);
    case 3: return launch_t<false, true, true>(*a, *b, *args, s);
    case 4: return launch_t<true, false, false>(*a, *b, *args, s);
    case 5: return launch_t<true, false, true>(*a, *b, *args, s);
    case 6: return launch_t<true, true, false>(*a, *b, *args, s);
    default: return launch_t<true, true, true>(*a, *b, *args, s);
  }
}

}  // extern "C"
