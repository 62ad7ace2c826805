// Logit gradient of the slot loss from the logits the forward kept (gradient of Eq. 1 with
// respect to z_d, and of the top-k + tail-bin form of Sec. 3.1): HBM-bound element-wise
// kernels over [N, V], which write G over the kept z_d.
#include <cuda_fp16.h>

#include "kernels.h"
#include "tc_common.cuh"

namespace alr {
namespace {
// ------------------------------------------------ logit gradient from kept logits ---
// G[r, v] = c_r (exp(z_d - lse_d) - exp(z_t - lse_t)) with c_r = lambda omega_r / sum omega:
// the gradient of Eq. 1 with respect to z_d, from the logits the forward wrote (fp16 values
// plus their 16-column group references for bf16 inputs: z = value + reference).
// A block takes 32 rows x 2048 columns: the rows' constants are staged in shared memory, then
// each pass of the 256 threads streams one row's 2048 columns (an 8-column vector per thread),
// with kLogitsUnroll rows' loads in flight.  (Blocks of 32 x 2048 measured 6.5 TB/s; staging
// the block's group references in shared memory first ran at 5.8 TB/s, whole rows per block
// with the same direct reference loads at 5.4, and tiles of 16 x 4096 or 8 x 8192 slower.)  G may be the z_d buffer itself: each element is read
// before the thread that read it overwrites it, and no other thread touches it.  Masked rows
// (c_r = 0) read nothing.
constexpr int kLogitsUnroll = 4;
constexpr int kGradRows = 32;
constexpr int kGradCols = 2048;
constexpr int kGradGroups = kGradCols / kKeepGroup;
constexpr int kGradThreads = kGradCols / 8;

// 8 kept logits as loaded: fp16 (bf16 inputs) or fp32 (fp32 inputs).
template <typename Z>
struct Raw8;

template <>
struct Raw8<__half> {
  uint4 u;
  __device__ __forceinline__ void load(const __half* p) {
    u = __ldcs(reinterpret_cast<const uint4*>(p));
  }
  __device__ __forceinline__ void to_float(float (&v)[8]) const {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const float2 f = __half22float2(*reinterpret_cast<const __half2*>(&w[i]));
      v[2 * i] = f.x;
      v[2 * i + 1] = f.y;
    }
  }
};

template <>
struct Raw8<float> {
  float4 a, b;
  __device__ __forceinline__ void load(const float* p) {
    a = __ldcs(reinterpret_cast<const float4*>(p));
    b = __ldcs(reinterpret_cast<const float4*>(p) + 1);
  }
  __device__ __forceinline__ void to_float(float (&v)[8]) const {
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
  }
};

__device__ __forceinline__ uint32_t bf16x2_bits(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

__device__ __forceinline__ void store8(__nv_bfloat16* p, const float (&g)[8]) {
  *reinterpret_cast<uint4*>(p) = make_uint4(bf16x2_bits(g[0], g[1]), bf16x2_bits(g[2], g[3]),
                                            bf16x2_bits(g[4], g[5]), bf16x2_bits(g[6], g[7]));
}

__device__ __forceinline__ void store8(float* p, const float (&g)[8]) {
  reinterpret_cast<float4*>(p)[0] = make_float4(g[0], g[1], g[2], g[3]);
  reinterpret_cast<float4*>(p)[1] = make_float4(g[4], g[5], g[6], g[7]);
}

__device__ __forceinline__ float load1(const __half* p) { return __half2float(*p); }
__device__ __forceinline__ float load1(const float* p) { return *p; }
__device__ __forceinline__ void store1(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }
__device__ __forceinline__ void store1(float* p, float v) { *p = v; }

// Reference of the group that holds vector i (8 columns; two vectors per 16-column group) of
// row r, from the group-major array, scaled by log2 e: a warp's 32 vectors of one row read 16
// groups, and the next rows of the block read the same sectors again (32 rows of a group are
// 64 contiguous bytes), so the loads go through the read-only cache.  fp32 logits have none.
template <typename Z>
__device__ __forceinline__ float ref_l2e(const uint16_t* ref, int N, int g, int r) {
  if constexpr (sizeof(Z) == 2)
    return __half2float(__ushort_as_half(__ldg(ref + size_t(g) * size_t(N) + r))) * kLog2e;
  else
    return 0.f;
}

// Row factor c_r = lambda omega_r / sum omega (0 when sum omega = 0).
__device__ __forceinline__ float row_factor(const float* weight, const float* weight_sum, float lam,
                                            int r) {
  const float ws = *weight_sum;
  return ws > 0.f ? lam * weight[r] / ws : 0.f;
}

template <typename Z, typename Gt>
__global__ void __launch_bounds__(kGradThreads) logits_grad_kernel(
    const Z* zd, const Z* zt, const uint16_t* __restrict__ zd_ref,
    const uint16_t* __restrict__ zt_ref, const float* __restrict__ lse_d,
    const float* __restrict__ lse_t, const float* __restrict__ weight,
    const float* __restrict__ weight_sum, float lam, int N, int V, Gt* G) {
  __shared__ float s_c[kGradRows], s_ad[kGradRows], s_at[kGradRows];
  const int r0 = blockIdx.x * kGradRows, c0 = blockIdx.y * kGradCols;
  const int nr = min(kGradRows, N - r0), nc = min(kGradCols, V - c0);
  if (threadIdx.x < nr) {
    const int r = r0 + threadIdx.x;
    s_c[threadIdx.x] = row_factor(weight, weight_sum, lam, r);
    s_ad[threadIdx.x] = -lse_d[r] * kLog2e;
    s_at[threadIdx.x] = -lse_t[r] * kLog2e;
  }
  __syncthreads();
  const int i = threadIdx.x;                   // this thread's 8-column vector of every row
  if (8 * i >= nc) return;
  const size_t col = size_t(c0) + 8 * size_t(i);
  const int g = c0 / kKeepGroup + (i >> 1);
  for (int rr0 = 0; rr0 < nr; rr0 += kLogitsUnroll) {
    Raw8<Z> a[kLogitsUnroll], b[kLogitsUnroll];
    float oa[kLogitsUnroll], ob[kLogitsUnroll];
#pragma unroll
    for (int u = 0; u < kLogitsUnroll; ++u) {
      const int rr = rr0 + u;
      if (rr < nr && s_c[rr] != 0.f) {
        const size_t e = size_t(r0 + rr) * size_t(V) + col;
        a[u].load(zd + e);
        b[u].load(zt + e);
        oa[u] = ref_l2e<Z>(zd_ref, N, g, r0 + rr) + s_ad[rr];
        ob[u] = ref_l2e<Z>(zt_ref, N, g, r0 + rr) + s_at[rr];
      }
    }
#pragma unroll
    for (int u = 0; u < kLogitsUnroll; ++u) {
      const int rr = rr0 + u;
      if (rr < nr) {
        const float c = s_c[rr];
        float gv[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
        if (c != 0.f) {
          float x[8], y[8];
          a[u].to_float(x);
          b[u].to_float(y);
#pragma unroll
          for (int j = 0; j < 8; ++j)
            gv[j] = c * (ex2(fmaf(x[j], kLog2e, oa[u])) - ex2(fmaf(y[j], kLog2e, ob[u])));
        }
        store8(G + size_t(r0 + rr) * size_t(V) + col, gv);
      }
    }
  }
}

// Gradient of the top-k + tail soft CE from the kept z_d, tiled like logits_grad_kernel:
// c beta q over the whole row, then c (q - prob_i) at the row's label tokens inside the block's
// columns, whose logits are read before the streaming pass overwrites them (G may be the z_d
// buffer).  The label tokens of a row are distinct.
template <typename Z, typename Gt>
__global__ void __launch_bounds__(kGradThreads) topk_logits_grad_kernel(
    const Z* zd, const uint16_t* __restrict__ zd_ref, const int32_t* __restrict__ top_idx,
    const float* __restrict__ top_prob, const float* __restrict__ tail,
    const float* __restrict__ tail_q, const float* __restrict__ lse_d,
    const float* __restrict__ weight, const float* __restrict__ weight_sum, float lam, int N,
    int V, Gt* G) {
  static_assert(kGradRows * kTopK <= kGradThreads, "one thread per label of the block's rows");
  __shared__ float s_c[kGradRows], s_cb[kGradRows], s_ad[kGradRows];
  __shared__ float lab_g[kGradRows * kTopK];
  __shared__ int lab_v[kGradRows * kTopK];
  const int r0 = blockIdx.x * kGradRows, c0 = blockIdx.y * kGradCols;
  const int nr = min(kGradRows, N - r0), nc = min(kGradCols, V - c0);
  if (threadIdx.x < nr) {
    const int r = r0 + threadIdx.x;
    const float c = row_factor(weight, weight_sum, lam, r);
    const float tl = tail[r];
    s_c[threadIdx.x] = c;
    s_cb[threadIdx.x] = c * (tl > 0.f ? 1.f - tl / tail_q[r] : 1.f);
    s_ad[threadIdx.x] = -lse_d[r] * kLog2e;
  }
  __syncthreads();
  {  // the label tokens of the block's rows that fall in its columns, before any overwrite
    const int rr = threadIdx.x / kTopK, k = threadIdx.x % kTopK;
    int v = -1;
    if (rr < nr) {
      const int r = r0 + rr;
      v = top_idx[size_t(r) * kTopK + k];
      if (v >= c0 && v < c0 + nc) {
        const float z = load1(zd + size_t(r) * size_t(V) + v);
        const float o = ref_l2e<Z>(zd_ref, N, v / kKeepGroup, r) + s_ad[rr];
        lab_g[threadIdx.x] = s_c[rr] * (ex2(fmaf(z, kLog2e, o)) - top_prob[size_t(r) * kTopK + k]);
      } else {
        v = -1;
      }
    }
    lab_v[threadIdx.x] = v;
  }
  __syncthreads();
  const int i = threadIdx.x;
  if (8 * i < nc) {
    const size_t col = size_t(c0) + 8 * size_t(i);
    const int g = c0 / kKeepGroup + (i >> 1);
    for (int rr0 = 0; rr0 < nr; rr0 += kLogitsUnroll) {
      Raw8<Z> a[kLogitsUnroll];
      float oa[kLogitsUnroll];
#pragma unroll
      for (int u = 0; u < kLogitsUnroll; ++u) {
        const int rr = rr0 + u;
        if (rr < nr && s_c[rr] != 0.f) {
          a[u].load(zd + size_t(r0 + rr) * size_t(V) + col);
          oa[u] = ref_l2e<Z>(zd_ref, N, g, r0 + rr) + s_ad[rr];
        }
      }
#pragma unroll
      for (int u = 0; u < kLogitsUnroll; ++u) {
        const int rr = rr0 + u;
        if (rr < nr) {
          const float cb = s_cb[rr];
          float gv[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
          if (s_c[rr] != 0.f) {
            float x[8];
            a[u].to_float(x);
#pragma unroll
            for (int j = 0; j < 8; ++j) gv[j] = cb * ex2(fmaf(x[j], kLog2e, oa[u]));
          }
          store8(G + size_t(r0 + rr) * size_t(V) + col, gv);
        }
      }
    }
  }
  __syncthreads();
  const int v = lab_v[threadIdx.x];
  if (v >= 0) store1(G + size_t(r0 + threadIdx.x / kTopK) * size_t(V) + v, lab_g[threadIdx.x]);
}

}  // namespace

cudaError_t launch_topk_logits_grad(int dtype, const void* zd, const uint16_t* zd_ref,
                                    const int32_t* top_idx, const float* top_prob,
                                    const float* tail, const float* tail_q, const float* lse_d,
                                    const float* weight, const float* weight_sum, float lam, int N,
                                    int V, void* G, cudaStream_t s) {
  const dim3 grid(unsigned((N + kGradRows - 1) / kGradRows), unsigned((V + kGradCols - 1) / kGradCols));
  if (dtype == 0)
    topk_logits_grad_kernel<__half, __nv_bfloat16><<<grid, kGradThreads, 0, s>>>(
        static_cast<const __half*>(zd), zd_ref, top_idx, top_prob, tail, tail_q, lse_d, weight,
        weight_sum, lam, N, V, static_cast<__nv_bfloat16*>(G));
  else
    topk_logits_grad_kernel<float, float><<<grid, kGradThreads, 0, s>>>(
        static_cast<const float*>(zd), nullptr, top_idx, top_prob, tail, tail_q, lse_d, weight,
        weight_sum, lam, N, V, static_cast<float*>(G));
  return cudaGetLastError();
}

cudaError_t launch_logits_grad(int dtype, const void* zd, const void* zt, const uint16_t* zd_ref,
                               const uint16_t* zt_ref, const float* lse_d, const float* lse_t,
                               const float* weight, const float* weight_sum, float lam, int N,
                               int V, void* G, cudaStream_t s) {
  const dim3 grid(unsigned((N + kGradRows - 1) / kGradRows), unsigned((V + kGradCols - 1) / kGradCols));
  if (dtype == 0)
    logits_grad_kernel<__half, __nv_bfloat16><<<grid, kGradThreads, 0, s>>>(
        static_cast<const __half*>(zd), static_cast<const __half*>(zt), zd_ref, zt_ref, lse_d,
        lse_t, weight, weight_sum, lam, N, V, static_cast<__nv_bfloat16*>(G));
  else
    logits_grad_kernel<float, float><<<grid, kGradThreads, 0, s>>>(
        static_cast<const float*>(zd), static_cast<const float*>(zt), nullptr, nullptr, lse_d,
        lse_t, weight, weight_sum, lam, N, V, static_cast<float*>(G));
  return cudaGetLastError();
}

}  // namespace alr
