// Fused dual-GEMM kernels of the slot loss on the sm_103a tensor cores.
//
// Both kernels compute, for a 128-row block of H_d and H_t and a 128-column tile of the
// vocabulary head W, the two logit tiles z_d = H_d W and z_t = H_t W with tcgen05.mma into
// tensor memory (fp32 accumulators, 2 x 128 columns per tile, double-buffered so the epilogue
// of one tile overlaps the products of the next).  The logits never leave the SM:
//   forward  - the epilogue folds each tile into running per-row statistics (online max /
//              sum-exp for both sides, the label-weighted sums behind the soft cross-entropy
//              of Eq. 1, greedy top-2 with lowest-index ties, z_t at the corpus token) and
//              writes one partial record per row and vocabulary split;
//   backward - the epilogue forms G = lambda omega_r / sum omega (q - p) for the tile
//              (the gradient of Eq. 1 with respect to z_d) and streams it out with TMA.
//
// Warp roles (256 threads): warp 0 issues TMA loads, warp 1 owns tensor memory and issues
// the MMAs from one lane, warps 4-7 run the epilogue (warp w reads TMEM lanes 32(w%4)..+31,
// one row per thread).  Every pipeline wait is bounded (tc_common.cuh).
#include "kernels.h"
#include "tc_common.cuh"

namespace alr {
namespace {

constexpr int kBM = 128;                 // rows per tile = TMEM lanes
constexpr int kBN = 128;                 // vocabulary columns per tile (per GEMM)
constexpr int kThreads = 256;
constexpr int kEpiWarp0 = 4;
constexpr int kEpiThreads = 128;
constexpr int kTileBytes = kBM * 128;    // a 128-extent operand over 128 bytes of K
constexpr int kStageBytes = 3 * kTileBytes;  // H_d tile, H_t tile, W tile
constexpr int kCtrlBytes = 256;

template <typename Elem>
struct Geo {
  static constexpr int kElem = sizeof(Elem);
  static constexpr int kKE = 128 / kElem;          // K elements per pipeline stage
  static constexpr int kMmaK = 32 / kElem;         // K per MMA instruction
  static constexpr int kChunkMN = 128 / kElem;     // MN elements per 128-byte chunk
  static constexpr int kNChunks = kBN / kChunkMN;  // W chunks per tile
  static constexpr uint32_t kChunkBytes = kKE * 128;
  static constexpr bool kTf32 = (kElem == 4);
};

template <bool kBwd>
constexpr int stages() { return kBwd ? 3 : 4; }

template <typename Elem, bool kBwd>
constexpr size_t smem_bytes() {
  return 1024 + size_t(stages<kBwd>()) * kStageBytes + (kBwd ? size_t(kBM) * kBN * sizeof(Elem) : 0) +
         kCtrlBytes;
}

ALR_DEV void decode_unit(const LossPlan& p, int u, int& rb, int& vs) {
  const int per_group = p.group_rows * p.n_vs;
  const int full = p.n_rb / p.group_rows;
  int g, w, gr;
  if (u < full * per_group) {
    g = u / per_group;
    w = u - g * per_group;
    gr = p.group_rows;
  } else {
    g = full;
    w = u - full * per_group;
    gr = p.n_rb - full * p.group_rows;
  }
  vs = w / gr;
  rb = g * p.group_rows + (w - vs * gr);
}

ALR_DEV int split_begin(const LossPlan& p, int vs) {
  return static_cast<int>((static_cast<long long>(vs) * p.n_vt) / p.n_vs);
}

ALR_DEV float f32(uint32_t x) { return __uint_as_float(x); }

// Running statistics of one row (forward epilogue).
struct RowStats {
  float m_d, s_d, m_t, s_t, u, w;
  float b_d, sec_d, b_t, sec_t, zx;
  int i_d, i_t;
};

ALR_DEV void stats_init(RowStats& st) {
  st.m_d = st.m_t = -INFINITY;
  st.s_d = st.s_t = st.u = st.w = 0.f;
  st.b_d = st.sec_d = st.b_t = st.sec_t = -INFINITY;
  st.i_d = st.i_t = 0x7fffffff;
  st.zx = __int_as_float(0x7fc00000);
}

// Greedy top-2 over a chunk in increasing column order; a strictly larger value is needed to
// take the lead, so the lowest index wins exact ties.
ALR_DEV void top2_scan(float& best, float& sec, int& idx, const uint32_t (&z)[32], int v0, int nv) {
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    if (j < nv) {
      const float v = f32(z[j]);
      if (v > best) {
        sec = best;
        best = v;
        idx = v0 + j;
      } else if (v > sec) {
        sec = v;
      }
    }
  }
}

template <bool kFull>
ALR_DEV void stats_chunk(RowStats& st, const uint32_t (&rd)[32], const uint32_t (&rt)[32], int v0,
                         int nv, int x) {
  float cmd = -INFINITY, cmt = -INFINITY;
#pragma unroll
  for (int j = 0; j < 32; ++j) {
    if (kFull || j < nv) {
      cmd = fmaxf(cmd, f32(rd[j]));
      cmt = fmaxf(cmt, f32(rt[j]));
    }
  }
  if (cmd > st.sec_d) top2_scan(st.b_d, st.sec_d, st.i_d, rd, v0, kFull ? 32 : nv);
  if (cmt > st.sec_t) top2_scan(st.b_t, st.sec_t, st.i_t, rt, v0, kFull ? 32 : nv);
  const int xr = x - v0;
  if (xr >= 0 && xr < (kFull ? 32 : nv)) {
#pragma unroll
    for (int j = 0; j < 32; ++j)
      if (j == xr) st.zx = f32(rt[j]);
  }
  // target side: sum e, sum e z_d, sum e z_t with e = exp(z_t - m_t)
  const float nmt = fmaxf(st.m_t, cmt);
  const float sct = ex2((st.m_t - nmt) * kLog2e);
  const float bt = -nmt * kLog2e;
  float s0 = 0.f, s1 = 0.f, u0 = 0.f, u1 = 0.f, w0 = 0.f, w1 = 0.f;
#pragma unroll
  for (int j = 0; j < 32; j += 2) {
    if (kFull || j < nv) {
      const float zt = f32(rt[j]);
      const float e = ex2(fmaf(zt, kLog2e, bt));
      s0 += e;
      u0 = fmaf(e, f32(rd[j]), u0);
      w0 = fmaf(e, zt, w0);
    }
    if (kFull || j + 1 < nv) {
      const float zt = f32(rt[j + 1]);
      const float e = ex2(fmaf(zt, kLog2e, bt));
      s1 += e;
      u1 = fmaf(e, f32(rd[j + 1]), u1);
      w1 = fmaf(e, zt, w1);
    }
  }
  st.s_t = fmaf(st.s_t, sct, s0 + s1);
  st.u = fmaf(st.u, sct, u0 + u1);
  st.w = fmaf(st.w, sct, w0 + w1);
  st.m_t = nmt;
  // drafter side: sum exp(z_d - m_d)
  const float nmd = fmaxf(st.m_d, cmd);
  const float scd = ex2((st.m_d - nmd) * kLog2e);
  const float bd = -nmd * kLog2e;
  float r0 = 0.f, r1 = 0.f;
#pragma unroll
  for (int j = 0; j < 32; j += 2) {
    if (kFull || j < nv) r0 += ex2(fmaf(f32(rd[j]), kLog2e, bd));
    if (kFull || j + 1 < nv) r1 += ex2(fmaf(f32(rd[j + 1]), kLog2e, bd));
  }
  st.s_d = fmaf(st.s_d, scd, r0 + r1);
  st.m_d = nmd;
}

ALR_DEV uint32_t pack_bf16x2(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

// Warp-uniform bounded wait: lane 0 waits, the verdict is broadcast.
ALR_DEV bool warp_wait(uint64_t* bar, uint32_t parity, const AbortFlag& ab) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, ab) ? 1 : 0;
  return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

// kWMN: the head tile is read MN-major straight from W [d, V] (bf16), or K-major from a
// transposed copy W^T [V, d] (fp32 inputs, whose tf32 products take K-major operands only).
template <typename Elem, bool kBwd, bool kWMN>
__global__ void __launch_bounds__(kThreads, 1)
    loss_gemm_kernel(const __grid_constant__ CUtensorMap tm_hd,
                     const __grid_constant__ CUtensorMap tm_ht,
                     const __grid_constant__ CUtensorMap tm_w,
                     const __grid_constant__ CUtensorMap tm_g, const LossArgs args) {
  using G = Geo<Elem>;
  constexpr int kStages = stages<kBwd>();
  constexpr int kGStageBytes = kBwd ? kBM * kBN * int(sizeof(Elem)) : 0;

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align_1024(smem_raw);
  uint8_t* stage_mem = smem;
  uint8_t* gstage = smem + kStages * kStageBytes;
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(gstage + kGStageBytes);
  uint64_t* empty_bar = full_bar + kStages;
  uint64_t* tfull_bar = empty_bar + kStages;
  uint64_t* tempty_bar = tfull_bar + 2;
  uint64_t* drain_bar = tempty_bar + 2;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile int* abort_word = reinterpret_cast<volatile int*>(tmem_slot + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const LossPlan& P = args.plan;
  const AbortFlag ab{abort_word, args.status};

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&tfull_bar[i], 1);
      mbar_init(&tempty_bar[i], kEpiThreads / 32);
    }
    mbar_init(drain_bar, 1);
    *abort_word = 0;
    fence_mbar_init();
  }
  if (threadIdx.x == 32) {
    tma_prefetch_desc(&tm_hd);
    tma_prefetch_desc(&tm_ht);
    tma_prefetch_desc(&tm_w);
    if (kBwd) tma_prefetch_desc(&tm_g);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem_base = *tmem_slot;
  const int n_kb = (P.d + G::kKE - 1) / G::kKE;

  if (warp == 0) {
    // ------------------------------------------------------------- TMA producer ---
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, armed = 0, armed_par = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < P.n_units; u += gridDim.x) {
        int rb, vs;
        decode_unit(P, u, rb, vs);
        const int vt1 = split_begin(P, vs + 1);
        for (int vt = split_begin(P, vs); ok && vt < vt1; ++vt) {
          for (int kb = 0; kb < n_kb; ++kb) {
            if (!mbar_wait(&empty_bar[stage], phase ^ 1, ab)) {
              ok = false;
              break;
            }
            uint8_t* sb = stage_mem + stage * kStageBytes;
            mbar_arrive_expect_tx(&full_bar[stage], kStageBytes);
            tma_load_2d(sb, &tm_hd, &full_bar[stage], kb * G::kKE, rb * kBM);
            tma_load_2d(sb + kTileBytes, &tm_ht, &full_bar[stage], kb * G::kKE, rb * kBM);
            if constexpr (kWMN) {
#pragma unroll
              for (int c = 0; c < G::kNChunks; ++c)
                tma_load_2d(sb + 2 * kTileBytes + c * G::kChunkBytes, &tm_w, &full_bar[stage],
                            vt * kBN + c * G::kChunkMN, kb * G::kKE);
            } else {
              tma_load_2d(sb + 2 * kTileBytes, &tm_w, &full_bar[stage], kb * G::kKE, vt * kBN);
            }
            armed |= 1u << stage;
            armed_par = (armed_par & ~(1u << stage)) | (phase << stage);
            if (++stage == kStages) {
              stage = 0;
              phase ^= 1;
            }
          }
        }
      }
      if (!ok) {  // let every copy already issued land before the CTA goes away
        for (int s = 0; s < kStages; ++s)
          if (armed & (1u << s)) mbar_wait_drain(&full_bar[s], (armed_par >> s) & 1u);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------------ MMA issuer ---
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_make(G::kTf32, kBM, kBN, false, kWMN);
      int stage = 0, abuf = 0;
      uint32_t phase = 0, aphase = 0;
      bool ok = true;
      for (int u = blockIdx.x; ok && u < P.n_units; u += gridDim.x) {
        int rb, vs;
        decode_unit(P, u, rb, vs);
        const int vt1 = split_begin(P, vs + 1);
        for (int vt = split_begin(P, vs); ok && vt < vt1; ++vt) {
          if (!mbar_wait(&tempty_bar[abuf], aphase ^ 1, ab)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_acc = tmem_base + uint32_t(abuf * 2 * kBN);
          for (int kb = 0; kb < n_kb; ++kb) {
            if (!mbar_wait(&full_bar[stage], phase, ab)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sa = smem_u32(stage_mem + stage * kStageBytes);
#pragma unroll
            for (int kk = 0; kk < G::kKE / G::kMmaK; ++kk) {
              const uint64_t ad = sdesc_sw128(sa + kk * 32, 16, 1024);
              const uint64_t at = sdesc_sw128(sa + kTileBytes + kk * 32, 16, 1024);
              const uint64_t bd =
                  kWMN ? sdesc_sw128(sa + 2 * kTileBytes + kk * G::kMmaK * 128, G::kChunkBytes, 1024)
                       : sdesc_sw128(sa + 2 * kTileBytes + kk * 32, 16, 1024);
              const uint32_t acc = (kb > 0 || kk > 0) ? 1u : 0u;
              mma_issue<G::kTf32>(d_acc, ad, bd, idesc, acc);
              mma_issue<G::kTf32>(d_acc + kBN, at, bd, idesc, acc);
            }
            mma_commit(&empty_bar[stage]);
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
      }
      // all products issued by this thread complete before tensor memory is released
      mma_commit(drain_bar);
      mbar_wait_drain(drain_bar, 0);
    }
  } else if (warp >= kEpiWarp0) {
    // -------------------------------------------------------------------- epilogue ---
    const int q = warp & 3;
    const int row_in_tile = q * 32 + lane;
    const uint32_t lane_addr = tmem_base + (uint32_t(q * 32) << 16);
    int abuf = 0;
    uint32_t aphase = 0;
    bool ok = true;
    for (int u = blockIdx.x; ok && u < P.n_units; u += gridDim.x) {
      int rb, vs;
      decode_unit(P, u, rb, vs);
      const int vt1 = split_begin(P, vs + 1);
      const int row = rb * kBM + row_in_tile;
      const bool row_ok = row < P.N;
      if constexpr (!kBwd) {
        RowStats st;
        stats_init(st);
        const int x = (args.corpus_tok != nullptr && row_ok) ? args.corpus_tok[row] : -1;
        for (int vt = split_begin(P, vs); vt < vt1; ++vt) {
          if (!warp_wait(&tfull_bar[abuf], aphase, ab)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t tb = lane_addr + uint32_t(abuf * 2 * kBN);
          const int vbase = vt * kBN;
          const bool full_tile = vbase + kBN <= P.V;
#pragma unroll 1
          for (int c = 0; c < kBN / 32; ++c) {
            uint32_t rd[32], rt[32];
            tmem_ld32(tb + c * 32, rd);
            tmem_ld32(tb + kBN + c * 32, rt);
            tmem_ld_wait();
            reg_fence(rd);
            reg_fence(rt);
            const int v0 = vbase + c * 32;
            if (full_tile) {
              stats_chunk<true>(st, rd, rt, v0, 32, x);
            } else if (v0 < P.V) {
              stats_chunk<false>(st, rd, rt, v0, min(32, P.V - v0), x);
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
        if (ok && row_ok) {
          const size_t fs = size_t(P.n_vs) * P.N;
          float* o = args.part + size_t(vs) * P.N + row;
          o[kPMd * fs] = st.m_d;
          o[kPSd * fs] = st.s_d;
          o[kPMt * fs] = st.m_t;
          o[kPSt * fs] = st.s_t;
          o[kPU * fs] = st.u;
          o[kPW * fs] = st.w;
          o[kPBd * fs] = st.b_d;
          o[kPId * fs] = __int_as_float(st.i_d);
          o[kPSecd * fs] = st.sec_d;
          o[kPBt * fs] = st.b_t;
          o[kPIt * fs] = __int_as_float(st.i_t);
          o[kPSect * fs] = st.sec_t;
          o[kPZx * fs] = st.zx;
        }
      } else {
        float ad = 0.f, at = 0.f, cw = 0.f;
        if (row_ok) {
          ad = -args.lse_d[row] * kLog2e;
          at = -args.lse_t[row] * kLog2e;
          const float ws = *args.weight_sum;
          cw = ws > 0.f ? args.lam * args.weight[row] / ws : 0.f;
        }
        for (int vt = split_begin(P, vs); vt < vt1; ++vt) {
          if (!warp_wait(&tfull_bar[abuf], aphase, ab)) {
            ok = false;
            break;
          }
          tc_fence_after();
          // Each warp owns rows 32q..32q+31 of the staging tile and stores them itself, so
          // the epilogue warps never wait on one another.  The slab is free once this
          // warp's previous store has read it.
          if (lane == 0) tma_store_wait_read_all();
          __syncwarp();
          const uint32_t tb = lane_addr + uint32_t(abuf * 2 * kBN);
#pragma unroll 1
          for (int c = 0; c < kBN / 32; ++c) {
            uint32_t rd[32], rt[32];
            tmem_ld32(tb + c * 32, rd);
            tmem_ld32(tb + kBN + c * 32, rt);
            tmem_ld_wait();
            reg_fence(rd);
            reg_fence(rt);
            float g[32];
#pragma unroll
            for (int j = 0; j < 32; ++j)
              g[j] = cw * (ex2(fmaf(f32(rd[j]), kLog2e, ad)) - ex2(fmaf(f32(rt[j]), kLog2e, at)));
            if constexpr (sizeof(Elem) == 2) {
              uint8_t* rowp = gstage + (c >> 1) * (kBM * 128) + row_in_tile * 128;
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                const int unit = ((c & 1) * 4 + i) ^ (row_in_tile & 7);
                uint4 v;
                v.x = pack_bf16x2(g[8 * i + 0], g[8 * i + 1]);
                v.y = pack_bf16x2(g[8 * i + 2], g[8 * i + 3]);
                v.z = pack_bf16x2(g[8 * i + 4], g[8 * i + 5]);
                v.w = pack_bf16x2(g[8 * i + 6], g[8 * i + 7]);
                *reinterpret_cast<uint4*>(rowp + unit * 16) = v;
              }
            } else {
              uint8_t* rowp = gstage + c * (kBM * 128) + row_in_tile * 128;
#pragma unroll
              for (int i = 0; i < 8; ++i) {
                const int unit = i ^ (row_in_tile & 7);
                *reinterpret_cast<float4*>(rowp + unit * 16) =
                    make_float4(g[4 * i], g[4 * i + 1], g[4 * i + 2], g[4 * i + 3]);
              }
            }
          }
          tc_fence_before();
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            mbar_arrive(&tempty_bar[abuf]);
#pragma unroll
            for (int b = 0; b < G::kNChunks; ++b)
              tma_store_2d(&tm_g, gstage + b * (kBM * 128) + q * 32 * 128,
                           vt * kBN + b * G::kChunkMN, rb * kBM + q * 32);
            tma_store_commit();
          }
          if (++abuf == 2) {
            abuf = 0;
            aphase ^= 1;
          }
        }
        if (!ok) break;
      }
    }
    if constexpr (kBwd) {
      if (lane == 0) tma_store_wait_all();
    }
  }

  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem_base, 512);
  }
}

template <typename Elem, bool kBwd>
cudaError_t launch_impl(const CUtensorMap& hd, const CUtensorMap& ht, const CUtensorMap& w,
                        const CUtensorMap& g, const LossArgs& args, cudaStream_t s) {
  auto kern = loss_gemm_kernel<Elem, kBwd, sizeof(Elem) == 2>;
  const size_t smem = smem_bytes<Elem, kBwd>();
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
  if (e != cudaSuccess) return e;
  kern<<<args.plan.grid, kThreads, smem, s>>>(hd, ht, w, g, args);
  return cudaGetLastError();
}

}  // namespace

size_t loss_fwd_smem_bytes(int dtype) {
  return dtype == 0 ? smem_bytes<__nv_bfloat16, false>() : smem_bytes<float, false>();
}
size_t loss_bwd_smem_bytes(int dtype) {
  return dtype == 0 ? smem_bytes<__nv_bfloat16, true>() : smem_bytes<float, true>();
}

cudaError_t launch_loss_fwd(int dtype, const CUtensorMap& hd, const CUtensorMap& ht,
                            const CUtensorMap& w, const LossArgs& args, cudaStream_t s) {
  if (dtype == 0) return launch_impl<__nv_bfloat16, false>(hd, ht, w, w, args, s);
  return launch_impl<float, false>(hd, ht, w, w, args, s);
}

cudaError_t launch_loss_bwd(int dtype, const CUtensorMap& hd, const CUtensorMap& ht,
                            const CUtensorMap& w, const CUtensorMap& g_store,
                            const LossArgs& args, cudaStream_t s) {
  if (dtype == 0) return launch_impl<__nv_bfloat16, true>(hd, ht, w, g_store, args, s);
  return launch_impl<float, true>(hd, ht, w, g_store, args, s);
}

}  // namespace alr
