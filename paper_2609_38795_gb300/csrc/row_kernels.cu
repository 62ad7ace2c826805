// Row-level kernels of the slot-loss path: the IRA gather, block plan, draws and context, the
// merge of per-split forward statistics into the per-row loss terms and slot weights, the
// batch reduction of Eq. 1, the accepted-length statistic and the erase-gate weights.  (The
// logit gradient from kept logits is in grad_kernels.cu.)
#include <cfloat>
#include <cuda_fp16.h>

#include "kernels.h"
#include "tc_common.cuh"

namespace alr {
namespace {

__device__ __forceinline__ float quiet_nan() { return __int_as_float(0x7fc00000); }

// ------------------------------------------------------------------ IRA gather ---
// One warp per output row; each lane moves 16-byte vectors, issuing a batch of loads before
// the matching stores so that many requests are in flight per SM.
constexpr int kGatherBatch = 16;

// Programmatic dependent launch of the gathers: each is launched so that it may be scheduled
// while the kernel before it in the stream is still running, waits (griddepcontrol.wait) until
// that kernel has completed and its writes are visible before touching global memory, and
// lets the kernel after it be scheduled early in turn.  A kernel launched without the
// attribute, or preceded by one that never triggers, behaves as under plain stream order.
ALR_DEV void pdl_wait_and_release() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), unsigned grid, unsigned block, cudaStream_t s,
                       Args... args) {
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg{};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, args...);
}

__global__ void __launch_bounds__(256) gather_kernel(const uint4* __restrict__ feat, int S, int L,
                                                     int vec_per_row,
                                                     const int32_t* __restrict__ seq,
                                                     const int32_t* __restrict__ pos,
                                                     const int32_t* __restrict__ valid_len,
                                                     int A, int B, uint4* __restrict__ out,
                                                     float* __restrict__ row_valid) {
  pdl_wait_and_release();
  const long long r = (long long)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (r >= (long long)A * B) return;
  const int a = int(r / B), s = int(r - (long long)a * B);
  const int sq = seq[a], p0 = pos[a];
  int lim = L;
  if (valid_len != nullptr) lim = min(lim, valid_len[a]);
  const bool ok = sq >= 0 && sq < S && p0 >= 0 && (long long)p0 + s < lim;   // no int overflow
  uint4* dst = out + r * vec_per_row;
  if (lane == 0 && row_valid != nullptr) row_valid[r] = ok ? 1.f : 0.f;
  if (!ok) {
    const uint4 z = make_uint4(0, 0, 0, 0);
    for (int i = lane; i < vec_per_row; i += 32) dst[i] = z;
    return;
  }
  const uint4* src = feat + ((long long)sq * L + p0 + s) * vec_per_row;
  for (int base = 0; base < vec_per_row; base += 32 * kGatherBatch) {
    uint4 v[kGatherBatch];
#pragma unroll
    for (int j = 0; j < kGatherBatch; ++j) {
      const int i = base + j * 32 + lane;
      if (i < vec_per_row) v[j] = __ldg(src + i);
    }
#pragma unroll
    for (int j = 0; j < kGatherBatch; ++j) {
      const int i = base + j * 32 + lane;
      if (i < vec_per_row) __stcs(dst + i, v[j]);
    }
  }
}

// ------------------------------------------------------------- gate (Eq. 2) ---
// Warp-level survival gate for one anchor: lane s holds row a*B+s (lanes >= B inactive).
// soft: g_s = exp(sum_{s'<s} logp_x[s']); hard: g_s = prod_{s'<s} 1[x == argmax_t].
__device__ __forceinline__ float gate_for_lane(bool active, int lane, bool hard, float logp,
                                               bool match) {
  if (hard) {
    const unsigned bad = __ballot_sync(0xffffffffu, active && !match);
    const unsigned below = (lane == 0) ? 0u : (0xffffffffu >> (32 - lane));
    return (bad & below) ? 0.f : 1.f;
  }
  float v = active ? logp : 0.f;
  float incl = v;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const float t = __shfl_up_sync(0xffffffffu, incl, off);
    if (lane >= off) incl += t;
  }
  return expf(incl - v);
}

// --------------------------------------------------------------- combine ---
// One warp per anchor.  Merges the per-split statistics of each row into the log-sum-exps,
// l_r = LSE_d - (sum_v e^{z_t - m_t} z_d) / (sum_v e^{z_t - m_t}), the label entropy,
// the greedy tokens with their top-1/top-2 gaps, log p_t(x), and the slot weight omega_r of
// Eq. 1 (envelope w_k, mask, optional gate of Eq. 2).  Writes the anchor's sum omega l and
// sum omega for the batch reduction.
__global__ void __launch_bounds__(256) combine_kernel(
    LossPlan P, const float* __restrict__ part, int mode, float gamma,
    const float* __restrict__ row_mask, const int32_t* __restrict__ corpus_tok,
    float* __restrict__ loss_row, float* __restrict__ ent_row, float* __restrict__ lse_d_out,
    float* __restrict__ lse_t_out, int32_t* __restrict__ argmax_d, int32_t* __restrict__ argmax_t,
    float* __restrict__ gap_d, float* __restrict__ gap_t, float* __restrict__ logp_x_out,
    float* __restrict__ weight, double* __restrict__ anchor_part) {
  const int A = P.N / P.B;
  const int a = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (a >= A) return;
  const bool active = lane < P.B;
  const int r = a * P.B + (active ? lane : 0);
  const size_t fs = size_t(P.n_parts) * P.N;

  // the sums of exponentials are merged in fp64: their logarithms are the near-zero parts of
  // the loss and the entropy when the softmax is sharp
  float Md = -INFINITY, Mt = -INFINITY, U = 0.f, Wt = 0.f;
  double Sd = 0.0, St = 0.0;
  float bd = -INFINITY, secd = -INFINITY, bt = -INFINITY, sect = -INFINITY, zx = quiet_nan();
  int id = 0x7fffffff, it = 0x7fffffff;
  if (active) {
    for (int k = 0; k < P.n_parts; ++k) {
      const float* p = part + size_t(k) * P.N + r;
      // a part's sums of exponentials, from their two-float parts
      const float md = p[kPMd * fs], mt = p[kPMt * fs];
      const double sd = double(p[kPSd * fs]) + double(p[kPSdLo * fs]);
      const double st = double(p[kPSt * fs]) + double(p[kPStLo * fs]);
      const float nmd = fmaxf(Md, md), nmt = fmaxf(Mt, mt);
      const float so = ex2((Mt - nmt) * kLog2e), sn = ex2((mt - nmt) * kLog2e);
      // U, Wt and the parts' u, w are measured from their own maxima (z_d - M_d, z_t - M_t):
      // move both to the merged references before adding.  A side with no columns yet (its
      // maximum still -inf: the merge's start, or a part past the vocabulary) adds nothing.
      const bool have = Mt > -INFINITY, part_has = mt > -INFINITY;
      const float Uo = have ? fmaf(Md - nmd, float(St), U) : 0.f;
      const float Wo = have ? fmaf(Mt - nmt, float(St), Wt) : 0.f;
      const float un = part_has ? fmaf(md - nmd, float(st), p[kPU * fs]) : 0.f;
      const float wn = part_has ? fmaf(mt - nmt, float(st), p[kPW * fs]) : 0.f;
      U = Uo * so + un * sn;
      Wt = Wo * so + wn * sn;
      Sd = (have ? Sd * double(ex2((Md - nmd) * kLog2e)) : 0.0) +
           (part_has ? sd * double(ex2((md - nmd) * kLog2e)) : 0.0);
      St = (have ? St * double(so) : 0.0) + (part_has ? st * double(sn) : 0.0);
      Md = nmd;
      Mt = nmt;
      // top-2 merge; equal leaders go to the lower token id
      const float b2 = p[kPBd * fs], s2 = p[kPSecd * fs];
      const int i2 = __float_as_int(p[kPId * fs]);
      if (b2 > bd || (b2 == bd && i2 < id)) {
        secd = fmaxf(bd, s2);
        bd = b2;
        id = i2;
      } else {
        secd = fmaxf(secd, b2);
      }
      const float b3 = p[kPBt * fs], s3 = p[kPSect * fs];
      const int i3 = __float_as_int(p[kPIt * fs]);
      if (b3 > bt || (b3 == bt && i3 < it)) {
        sect = fmaxf(bt, s3);
        bt = b3;
        it = i3;
      } else {
        sect = fmaxf(sect, b3);
      }
      const float z = p[kPZx * fs];
      if (z == z) zx = z;
    }
  }
  const double lsd = log(Sd), lst = log(St);
  const float lse_d = Md + float(lsd);
  const float lse_t = Mt + float(lst);
  // l = lse_d - E_p[z_d] = log S_d - E_p[z_d - M_d]: two non-negative terms, no cancellation
  const float loss = float(lsd - double(U) / St);
  const float logp = zx - lse_t;
  const bool erase = mode != 0;
  const int x = (erase && active) ? corpus_tok[r] : -1;
  const float gate = erase ? gate_for_lane(active, lane, mode == 2, logp, x == it) : 1.f;
  float w = 0.f;
  if (active) {
    w = expf(-float(lane) / gamma) * gate;
    if (row_mask != nullptr) w *= row_mask[r];
    loss_row[r] = loss;
    if (ent_row) ent_row[r] = float(lst - double(Wt) / St);
    lse_d_out[r] = lse_d;
    lse_t_out[r] = lse_t;
    argmax_d[r] = id;
    argmax_t[r] = it;
    if (gap_d) gap_d[r] = bd - secd;
    if (gap_t) gap_t[r] = bt - sect;
    if (erase && logp_x_out) logp_x_out[r] = logp;
    weight[r] = w;
  }
  double wl = active ? double(w) * double(loss) : 0.0;
  double ws = active ? double(w) : 0.0;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    wl += __shfl_xor_sync(0xffffffffu, wl, off);
    ws += __shfl_xor_sync(0xffffffffu, ws, off);
  }
  if (lane == 0) {
    anchor_part[2 * a] = wl;
    anchor_part[2 * a + 1] = ws;
  }
}

// Batch reduction of Eq. 1 in a fixed order (one block, deterministic).  wl_sum (nullable)
// receives the numerator sum omega l itself, for a sum across the shards of a batch.
__global__ void __launch_bounds__(1024) finalize_kernel(const double* __restrict__ anchor_part,
                                                        int A, float lam,
                                                        float* __restrict__ loss_total,
                                                        float* __restrict__ weight_sum,
                                                        float* __restrict__ wl_sum) {
  __shared__ double s_wl[32], s_ws[32];
  double wl = 0.0, ws = 0.0;
  for (int a = threadIdx.x; a < A; a += blockDim.x) {
    wl += anchor_part[2 * a];
    ws += anchor_part[2 * a + 1];
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    wl += __shfl_xor_sync(0xffffffffu, wl, off);
    ws += __shfl_xor_sync(0xffffffffu, ws, off);
  }
  const int warp = threadIdx.x / 32, lane = threadIdx.x & 31;
  if (lane == 0) {
    s_wl[warp] = wl;
    s_ws[warp] = ws;
  }
  __syncthreads();
  if (warp == 0) {
    wl = lane < int(blockDim.x / 32) ? s_wl[lane] : 0.0;
    ws = lane < int(blockDim.x / 32) ? s_ws[lane] : 0.0;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      wl += __shfl_xor_sync(0xffffffffu, wl, off);
      ws += __shfl_xor_sync(0xffffffffu, ws, off);
    }
    if (lane == 0) {
      *loss_total = ws > 0.0 ? float(double(lam) * wl / ws) : 0.f;
      *weight_sum = float(ws);
      if (wl_sum != nullptr) *wl_sum = float(wl);
    }
  }
}

// Eq. 1 from sums that the caller reduced over the shards of a batch: L = lambda * wl / ws,
// 0 when ws = 0 (no supervised slot anywhere in the batch).
__global__ void loss_from_sums_kernel(const float* __restrict__ wl_sum,
                                      const float* __restrict__ weight_sum, float lam,
                                      float* __restrict__ loss_total) {
  const double ws = *weight_sum;
  *loss_total = ws > 0.0 ? float(double(lam) * double(*wl_sum) / ws) : 0.f;
}

// ------------------------------------------------------------- accepted length ---
// One warp per anchor: the count of leading slots whose greedy drafter token equals the
// greedy target token (and whose row is active).
__global__ void __launch_bounds__(256) accept_len_kernel(const int32_t* __restrict__ am_d,
                                                         const int32_t* __restrict__ am_t,
                                                         const float* __restrict__ active_w,
                                                         int A, int B, int32_t* __restrict__ acc,
                                                         unsigned long long* __restrict__ hist) {
  const int a = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (a >= A) return;
  bool ok = false;
  if (lane < B) {
    const int r = a * B + lane;
    ok = am_d[r] == am_t[r];
    if (active_w != nullptr) ok = ok && active_w[r] > 0.f;
  }
  const unsigned bal = __ballot_sync(0xffffffffu, ok);
  const int n = (bal == 0xffffffffu) ? 32 : (__ffs(~bal) - 1);
  if (lane == 0) {
    acc[a] = n;
    if (hist != nullptr) atomicAdd(hist + n, 1ull);
  }
}

// ---------------------------------------------------------- erase weights ---
__global__ void __launch_bounds__(256) erase_weights_kernel(
    const float* __restrict__ logp_x, const int32_t* __restrict__ corpus_tok,
    const int32_t* __restrict__ argmax_t, const float* __restrict__ row_mask, int A, int B,
    float gamma, int hard, float* __restrict__ weight) {
  const int a = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (a >= A) return;
  const bool active = lane < B;
  const int r = a * B + (active ? lane : 0);
  float logp = 0.f;
  bool match = true;
  if (active) {
    if (hard) match = corpus_tok[r] == argmax_t[r];
    else logp = logp_x[r];
  }
  const float g = gate_for_lane(active, lane, hard != 0, logp, match);
  if (active) {
    float w = expf(-float(lane) / gamma) * g;
    if (row_mask != nullptr) w *= row_mask[r];
    weight[r] = w;
  }
}

// ---------------------------------------------------------- compact labels ---
// Insert (v, id) into a list sorted by value descending, equal values by id ascending.
__device__ __forceinline__ void insert_ranked(float (&t)[kTopK], int (&ti)[kTopK], float v,
                                              int id) {
  if (!(v > t[kTopK - 1] || (v == t[kTopK - 1] && id < ti[kTopK - 1]))) return;
  t[kTopK - 1] = v;
  ti[kTopK - 1] = id;
#pragma unroll
  for (int k = kTopK - 1; k > 0; --k) {
    const bool up = t[k] > t[k - 1] || (t[k] == t[k - 1] && ti[k] < ti[k - 1]);
    const float a = t[k], b = t[k - 1];
    const int ia = ti[k], ib = ti[k - 1];
    t[k - 1] = up ? a : b;
    t[k] = up ? b : a;
    ti[k - 1] = up ? ia : ib;
    ti[k] = up ? ib : ia;
  }
}

// 2^-r for the exponent residual r of a reference (|r| <= 4e-3 over the fp16 range of logits):
// 1 - x + x^2 / 2 with x = r ln 2, within 5e-9 relative (1e-15 for |r| <= 3e-5, |logit| < 1000).
__device__ __forceinline__ double inv_exp2_small(float r) {
  const double x = double(r) * 0.6931471805599453;
  return 1.0 - x + 0.5 * x * x;
}

// Label readout merge, one thread per row: log-sum-exp over all parts, the k best target
// logits (ties to the lower id), their probabilities and the tail mass
//   tail = (S - sum_k exp(t_k - M)) / S,
// the greedy token with its top-1 minus top-2 gap, and log p at the corpus token.
__global__ void __launch_bounds__(256) readout_combine_kernel(
    LossPlan P, const float* __restrict__ part, int has_corpus, int32_t* __restrict__ top_idx,
    float* __restrict__ top_prob, float* __restrict__ tail, float* __restrict__ lse_t,
    int32_t* __restrict__ argmax_t, float* __restrict__ gap_t, float* __restrict__ logp_x) {
  const int r = blockIdx.x * blockDim.x + threadIdx.x;
  if (r >= P.N) return;
  const size_t fs = size_t(P.n_parts) * P.N;
  float M = -INFINITY, zx = quiet_nan();
  double S = 0.0;   // merged in fp64 from the parts' two-float sums
  float t[kTopK];
  int ti[kTopK];
#pragma unroll
  for (int i = 0; i < kTopK; ++i) {
    t[i] = -INFINITY;
    ti[i] = 0x7fffffff;
  }
  for (int k = 0; k < P.n_parts; ++k) {
    const float* p = part + size_t(k) * P.N + r;
    const float m = p[kRM * fs];
    const float nm = fmaxf(M, m);
    const double sp = (double(p[kRS * fs]) + double(p[kRSLo * fs])) * inv_exp2_small(p[kRR * fs]);
    S = (M > -INFINITY ? S * double(ex2((M - nm) * kLog2e)) : 0.0) +
        (m > -INFINITY ? sp * double(ex2((m - nm) * kLog2e)) : 0.0);
    M = nm;
#pragma unroll
    for (int i = 0; i < kTopK; ++i) {
      const float v = p[(kRTop + i) * fs];
      if (v > -INFINITY) insert_ranked(t, ti, v, __float_as_int(p[(kRIdx + i) * fs]));
    }
    const float z = p[kRZx * fs];
    if (z == z) zx = z;
  }
  const double ls = log(S);
  const float lse = M + float(ls);
  double inside = 0.0;
#pragma unroll
  for (int i = 0; i < kTopK; ++i) {
    const double e = exp(double(t[i]) - double(M));
    top_idx[size_t(r) * kTopK + i] = ti[i];
    top_prob[size_t(r) * kTopK + i] = float(e / S);
    inside += e;
  }
  // with V <= k every token is in the list and the tail is empty by definition
  tail[r] = P.V <= kTopK ? 0.f : float(fmax(0.0, (S - inside) / S));
  if (lse_t) lse_t[r] = lse;
  if (argmax_t) argmax_t[r] = ti[0];
  if (gap_t) gap_t[r] = t[0] - t[1];
  if (has_corpus && logp_x) logp_x[r] = float((double(zx) - double(M)) - ls);
}

// Top-k loss merge, one warp per anchor: log-sum-exp and greedy top-2 of z_d, the label
// tokens' z_d, the drafter's mass outside them
//   tail_q = (S_d - sum_i exp(z_i - M_d)) / S_d,
// the loss l = -sum_i prob_i (z_i - LSE_d) - tail log tail_q (no tail term when tail = 0),
// the slot weight (given, or envelope times mask) and the anchor's sums for Eq. 1.
__global__ void __launch_bounds__(256) topk_combine_kernel(
    LossPlan P, const float* __restrict__ part, const float* __restrict__ top_prob,
    const float* __restrict__ tail, const float* __restrict__ row_mask,
    const float* __restrict__ weight_in, float gamma, float* __restrict__ loss_row,
    float* __restrict__ lse_d_out, float* __restrict__ tail_q_out, int32_t* __restrict__ argmax_d,
    float* __restrict__ gap_d, float* __restrict__ weight, double* __restrict__ anchor_part) {
  const int A = P.N / P.B;
  const int a = blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (a >= A) return;
  const bool active = lane < P.B;
  const int r = a * P.B + (active ? lane : 0);
  const size_t fs = size_t(P.n_parts) * P.N;
  // the sum of exponentials is merged in fp64 from its two-float parts: with a sharp drafter
  // its logarithm is the near-zero part of every log q
  float M = -INFINITY, bd = -INFINITY, secd = -INFINITY;
  double S = 0.0, Sout = 0.0;   // all columns; the columns outside the row's label tokens
  int id = 0x7fffffff;
  float zk[kTopK];
#pragma unroll
  for (int i = 0; i < kTopK; ++i) zk[i] = quiet_nan();
  if (active) {
    for (int k = 0; k < P.n_parts; ++k) {
      const float* p = part + size_t(k) * P.N + r;
      const float m = p[kKM * fs];
      const float nm = fmaxf(M, m);
      // the part's sums without the factor 2^r its exponentials carry
      const double unr = inv_exp2_small(p[kKR * fs]);
      const double sp = (double(p[kKS * fs]) + double(p[kKSLo * fs])) * unr;
      const double so =
          ((double(p[kKS * fs]) - double(p[kKSIn * fs])) + double(p[kKSLo * fs])) * unr;
      const double f_old = M > -INFINITY ? double(ex2((M - nm) * kLog2e)) : 0.0;
      const double f_new = m > -INFINITY ? double(ex2((m - nm) * kLog2e)) : 0.0;
      S = S * f_old + sp * f_new;
      Sout = Sout * f_old + so * f_new;
      M = nm;
      const float b2 = p[kKBest * fs], s2 = p[kKSec * fs];
      const int i2 = __float_as_int(p[kKIdx * fs]);
      if (b2 > bd || (b2 == bd && i2 < id)) {
        secd = fmaxf(bd, s2);
        bd = b2;
        id = i2;
      } else {
        secd = fmaxf(secd, b2);
      }
#pragma unroll
      for (int i = 0; i < kTopK; ++i) {
        const float z = p[(kKZ + i) * fs];
        if (z == z) zk[i] = z;
      }
    }
  }
  float loss = 0.f, w = 0.f;
  if (active) {
    const double ls = log(S);
    const float lse = M + float(ls);
    // log q_i = (z_i - M) - log S: the difference z_i - M is exact in fp64
    double ce = 0.0;
    for (int i = 0; i < kTopK; ++i)
      ce -= double(top_prob[size_t(r) * kTopK + i]) * ((double(zk[i]) - double(M)) - ls);
    const double tq = fmax(Sout / S, 1e-30);
    const float tl = tail[r];
    if (tl > 0.f) ce -= double(tl) * log(tq);
    loss = float(ce);
    w = weight_in != nullptr ? weight_in[r]
                             : expf(-float(lane) / gamma) * (row_mask ? row_mask[r] : 1.f);
    loss_row[r] = loss;
    lse_d_out[r] = lse;
    tail_q_out[r] = float(tq);
    argmax_d[r] = id;
    if (gap_d) gap_d[r] = bd - secd;
    weight[r] = w;
  }
  double wl = active ? double(w) * double(loss) : 0.0;
  double ws = active ? double(w) : 0.0;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    wl += __shfl_xor_sync(0xffffffffu, wl, off);
    ws += __shfl_xor_sync(0xffffffffu, ws, off);
  }
  if (lane == 0) {
    anchor_part[2 * a] = wl;
    anchor_part[2 * a + 1] = ws;
  }
}

// ------------------------------------------------------------- IRA block plan ---
// One thread per block slot (s, b): sample s keeps m = min(v_s, max_blocks) blocks, the
// first ceil(m/2) primary, the next floor(m/2) secondary (Sec. 3.2); secondary i sits in
// primary i's rollout at offset j.  Emits the label-row gather (seq, pos, valid_len) over
// the primary label buffer [S * P, K, d], the anchor token and the rollout context length.
__global__ void __launch_bounds__(256) ira_blocks_kernel(
    int S, int K, int max_blocks, const int32_t* __restrict__ valid_anchors,
    const int32_t* __restrict__ rollout_len, const int32_t* __restrict__ offsets,
    const int32_t* __restrict__ rollout_tok, const int32_t* __restrict__ corpus_anchor_tok,
    int32_t* __restrict__ seq, int32_t* __restrict__ pos, int32_t* __restrict__ vlen,
    int32_t* __restrict__ ctx_len, int32_t* __restrict__ anchor_tok) {
  const long long t = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= (long long)S * max_blocks) return;
  const int s = int(t / max_blocks), b = int(t - (long long)s * max_blocks);
  const int P = max_blocks - max_blocks / 2, Q = max_blocks / 2;
  const int m = max(0, min(valid_anchors[s], max_blocks));
  const int n_prim = (m + 1) / 2;
  int p = -1, j = 0;
  if (b < n_prim) {
    p = b;
  } else if (b < m) {
    p = b - n_prim;
    j = offsets[size_t(s) * Q + p];
    // an offset outside the rollout leaves the block unused: past K - 1, or past the end of
    // a primary rollout that terminated early (y*_j, the block's anchor token, never existed)
    if (j < 1 || j > K - 1 || j > rollout_len[size_t(s) * P + p]) p = -1;
  }
  if (p < 0) {
    seq[t] = -1;
    pos[t] = 0;
    vlen[t] = 0;
    if (ctx_len) ctx_len[t] = 0;
    if (anchor_tok) anchor_tok[t] = -1;
    return;
  }
  const size_t prim = size_t(s) * P + p;
  seq[t] = int(prim);
  pos[t] = j;
  vlen[t] = rollout_len[prim];
  if (ctx_len) ctx_len[t] = j > 0 ? j - 1 : 0;
  if (anchor_tok) {
    int tok = -1;
    if (j == 0 && corpus_anchor_tok) tok = corpus_anchor_tok[t];
    if (j > 0 && rollout_tok) tok = rollout_tok[prim * K + (j - 1)];   // y*_j
    anchor_tok[t] = tok;
  }
}

// ------------------------------------------------------------------ IRA draws ---
// One block per sample.  The anchor draw is the sample's valid positions in increasing
// (key, position) order; each valid position's rank in that order is the number of smaller
// (key, position) pairs, counted over the sample's pairs held in shared memory (invalid
// positions hold the largest value and are never counted or drawn).  Ranks below m =
// min(v, max_blocks) are the draw.  Offsets: j = 2 + floor(u (K - 2) / 2^32).
__global__ void __launch_bounds__(1024) ira_draw_kernel(int L, int K, int max_blocks,
                                                        const uint8_t* __restrict__ anchor_ok,
                                                        const uint32_t* __restrict__ keys,
                                                        const uint32_t* __restrict__ offset_u,
                                                        int32_t* __restrict__ n_valid,
                                                        int32_t* __restrict__ anchor_pos,
                                                        int32_t* __restrict__ offsets) {
  extern __shared__ unsigned long long pair[];   // [L] (key << 32 | position), or ~0
  __shared__ int s_count;
  const int s = blockIdx.x;
  const size_t row = size_t(s) * size_t(L);
  if (threadIdx.x == 0) s_count = 0;
  __syncthreads();
  int mine = 0;
  for (int a = threadIdx.x; a < L; a += blockDim.x) {
    const bool ok = anchor_ok[row + a] != 0;
    pair[a] = ok ? ((static_cast<unsigned long long>(keys[row + a]) << 32) | unsigned(a))
                 : ~0ull;
    mine += ok ? 1 : 0;
  }
  atomicAdd(&s_count, mine);
  __syncthreads();
  const int v = s_count, m = min(v, max_blocks);
  int32_t* out = anchor_pos + size_t(s) * size_t(max_blocks);
  for (int i = m + threadIdx.x; i < max_blocks; i += blockDim.x) out[i] = -1;
  for (int a = threadIdx.x; a < L; a += blockDim.x) {
    const unsigned long long c = pair[a];
    if (c == ~0ull) continue;
    int rank = 0;
    for (int q = 0; q < L; ++q) rank += pair[q] < c ? 1 : 0;
    if (rank < m) out[rank] = a;
  }
  const int H = max_blocks / 2;
  for (int i = threadIdx.x; i < H; i += blockDim.x) {
    const unsigned long long u = offset_u[size_t(s) * H + i];
    offsets[size_t(s) * H + i] = 2 + int((u * unsigned(K - 2)) >> 32);
  }
  if (threadIdx.x == 0) n_valid[s] = v;
}

// ------------------------------------------------------------------ IRA context ---
// Context rows of the secondary blocks: output row (s, i, r) of [S, H, C, F] is row r of
// primary i's stored rollout features when secondary i of sample s exists and r < j - 1,
// zero otherwise.  One warp per output row, 16-byte vectors in batches as in the gather.
__global__ void __launch_bounds__(256) ira_context_kernel(
    const uint4* __restrict__ store, int C, int vec_per_row, int S, int K, int max_blocks,
    const int32_t* __restrict__ n_valid, const int32_t* __restrict__ rollout_len,
    const int32_t* __restrict__ offsets, const int32_t* __restrict__ anchor_pos,
    uint4* __restrict__ ctx, int32_t* __restrict__ ctx_len, int32_t* __restrict__ prefix_end) {
  pdl_wait_and_release();
  const int H = max_blocks / 2, P = max_blocks - H;
  const long long t = (long long)blockIdx.x * (blockDim.x / 32) + threadIdx.x / 32;
  const int lane = threadIdx.x & 31;
  if (t >= (long long)S * H * C) return;
  const int r = int(t % C);
  const long long si = t / C;
  const int s = int(si / H), i = int(si - (long long)s * H);
  const int m = max(0, min(n_valid[s], max_blocks));
  const int j = offsets[si];
  const size_t prim = size_t(s) * P + i;
  const bool exists = i < m / 2 && j >= 1 && j <= K - 1 && j <= rollout_len[prim];
  const int n = exists ? j - 1 : 0;
  if (r == 0 && lane == 0) {
    if (ctx_len) ctx_len[si] = n;
    if (prefix_end) prefix_end[si] = exists ? anchor_pos[size_t(s) * max_blocks + i] : -1;
  }
  uint4* dst = ctx + t * vec_per_row;
  if (r >= n) {
    const uint4 z = make_uint4(0, 0, 0, 0);
    for (int k = lane; k < vec_per_row; k += 32) __stcs(dst + k, z);
    return;
  }
  const uint4* src = store + ((long long)prim * C + r) * vec_per_row;
  for (int base = 0; base < vec_per_row; base += 32 * kGatherBatch) {
    uint4 v[kGatherBatch];
#pragma unroll
    for (int k = 0; k < kGatherBatch; ++k) {
      const int e = base + k * 32 + lane;
      if (e < vec_per_row) v[k] = __ldg(src + e);
    }
#pragma unroll
    for (int k = 0; k < kGatherBatch; ++k) {
      const int e = base + k * 32 + lane;
      if (e < vec_per_row) __stcs(dst + e, v[k]);
    }
  }
}

// ------------------------------------------------------------------ transpose ---
// out[c * ld_out + r] = in[r * C + c] for 32-bit elements, 32 x 32 tiles through shared memory.
__global__ void __launch_bounds__(256) transpose32_kernel(const float* __restrict__ in,
                                                          float* __restrict__ out, int R, int C,
                                                          int ld_out) {
  __shared__ float tile[32][33];
  const int c0 = blockIdx.x * 32, r0 = blockIdx.y * 32;
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int r = r0 + i, c = c0 + threadIdx.x;
    if (r < R && c < C) tile[i][threadIdx.x] = in[(long long)r * C + c];
  }
  __syncthreads();
  for (int i = threadIdx.y; i < 32; i += 8) {
    const int c = c0 + i, r = r0 + threadIdx.x;
    if (r < R && c < C) out[(long long)c * ld_out + r] = tile[threadIdx.x][i];
  }
}

}  // namespace

cudaError_t launch_ira_blocks(int S, int K, int max_blocks, const int32_t* valid_anchors,
                              const int32_t* rollout_len, const int32_t* offsets,
                              const int32_t* rollout_tok, const int32_t* corpus_anchor_tok,
                              int32_t* seq, int32_t* pos, int32_t* vlen, int32_t* ctx_len,
                              int32_t* anchor_tok, cudaStream_t s) {
  const long long n = (long long)S * max_blocks;
  ira_blocks_kernel<<<unsigned((n + 255) / 256), 256, 0, s>>>(
      S, K, max_blocks, valid_anchors, rollout_len, offsets, rollout_tok, corpus_anchor_tok, seq,
      pos, vlen, ctx_len, anchor_tok);
  return cudaGetLastError();
}

cudaError_t launch_ira_draw(int S, int L, int K, int max_blocks, const uint8_t* anchor_ok,
                            const uint32_t* keys, const uint32_t* offset_u, int32_t* n_valid,
                            int32_t* anchor_pos, int32_t* offsets, cudaStream_t s) {
  const size_t smem = size_t(L) * sizeof(unsigned long long);
  cudaError_t e = cudaFuncSetAttribute(ira_draw_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       int(smem));
  if (e != cudaSuccess) return e;
  ira_draw_kernel<<<S, 1024, smem, s>>>(L, K, max_blocks, anchor_ok, keys, offset_u, n_valid,
                                        anchor_pos, offsets);
  return cudaGetLastError();
}

cudaError_t launch_ira_context(const void* store, int C, int F, int elem_bytes, int S, int K,
                               int max_blocks, const int32_t* n_valid, const int32_t* rollout_len,
                               const int32_t* offsets, const int32_t* anchor_pos, void* ctx,
                               int32_t* ctx_len, int32_t* prefix_end, cudaStream_t s) {
  const long long rows = (long long)S * (max_blocks / 2) * C;
  const int vec = int((long long)F * elem_bytes / 16);
  if (rows == 0) return cudaSuccess;
  return launch_pdl(ira_context_kernel, unsigned((rows + 7) / 8), 256, s,
                    static_cast<const uint4*>(store), C, vec, S, K, max_blocks, n_valid,
                    rollout_len, offsets, anchor_pos, static_cast<uint4*>(ctx), ctx_len,
                    prefix_end);
}

cudaError_t launch_transpose32(const float* in, float* out, int R, int C, int ld_out,
                               cudaStream_t s) {
  dim3 grid((C + 31) / 32, (R + 31) / 32);
  transpose32_kernel<<<grid, dim3(32, 8), 0, s>>>(in, out, R, C, ld_out);
  return cudaGetLastError();
}

cudaError_t launch_gather(const void* feat, int S, int L, int d, int elem_bytes,
                          const int32_t* seq, const int32_t* pos, const int32_t* valid_len,
                          int A, int B, void* out, float* row_valid, cudaStream_t s) {
  const long long rows = (long long)A * B;
  const int vec = int((long long)d * elem_bytes / 16);
  const long long blocks = (rows + 7) / 8;
  if (blocks == 0) return cudaSuccess;
  return launch_pdl(gather_kernel, unsigned(blocks), 256, s, static_cast<const uint4*>(feat), S,
                    L, vec, seq, pos, valid_len, A, B, static_cast<uint4*>(out), row_valid);
}

cudaError_t launch_combine(const LossPlan& plan, const float* part, int mode, float gamma,
                           const float* row_mask, const int32_t* corpus_tok, float* loss_row,
                           float* ent_row, float* lse_d, float* lse_t, int32_t* argmax_d,
                           int32_t* argmax_t, float* gap_d, float* gap_t, float* logp_x,
                           float* weight, double* anchor_part, cudaStream_t s) {
  const int A = plan.N / plan.B;
  combine_kernel<<<(A + 7) / 8, 256, 0, s>>>(plan, part, mode, gamma, row_mask, corpus_tok,
                                             loss_row, ent_row, lse_d, lse_t, argmax_d, argmax_t,
                                             gap_d, gap_t, logp_x, weight, anchor_part);
  return cudaGetLastError();
}

cudaError_t launch_readout_combine(const LossPlan& plan, const float* part, bool has_corpus,
                                   int32_t* top_idx, float* top_prob, float* tail, float* lse_t,
                                   int32_t* argmax_t, float* gap_t, float* logp_x,
                                   cudaStream_t s) {
  readout_combine_kernel<<<(plan.N + 255) / 256, 256, 0, s>>>(plan, part, has_corpus ? 1 : 0,
                                                              top_idx, top_prob, tail, lse_t,
                                                              argmax_t, gap_t, logp_x);
  return cudaGetLastError();
}

cudaError_t launch_topk_combine(const LossPlan& plan, const float* part, const float* top_prob,
                                const float* tail, const float* row_mask, const float* weight_in,
                                float gamma, float* loss_row, float* lse_d, float* tail_q,
                                int32_t* argmax_d, float* gap_d, float* weight,
                                double* anchor_part, cudaStream_t s) {
  const int A = plan.N / plan.B;
  topk_combine_kernel<<<(A + 7) / 8, 256, 0, s>>>(plan, part, top_prob, tail, row_mask, weight_in,
                                                  gamma, loss_row, lse_d, tail_q, argmax_d, gap_d,
                                                  weight, anchor_part);
  return cudaGetLastError();
}

cudaError_t launch_finalize(const double* anchor_part, int A, float lam, float* loss_total,
                            float* weight_sum, float* wl_sum, cudaStream_t s) {
  finalize_kernel<<<1, 1024, 0, s>>>(anchor_part, A, lam, loss_total, weight_sum, wl_sum);
  return cudaGetLastError();
}

cudaError_t launch_loss_from_sums(const float* wl_sum, const float* weight_sum, float lam,
                                  float* loss_total, cudaStream_t s) {
  loss_from_sums_kernel<<<1, 1, 0, s>>>(wl_sum, weight_sum, lam, loss_total);
  return cudaGetLastError();
}

cudaError_t launch_accept_len(const int32_t* am_d, const int32_t* am_t, const float* active,
                              int A, int B, int32_t* acc, int64_t* hist, cudaStream_t s) {
  if (hist != nullptr) {
    cudaError_t e = cudaMemsetAsync(hist, 0, sizeof(int64_t) * size_t(B + 1), s);
    if (e != cudaSuccess) return e;
  }
  accept_len_kernel<<<(A + 7) / 8, 256, 0, s>>>(am_d, am_t, active, A, B, acc,
                                                reinterpret_cast<unsigned long long*>(hist));
  return cudaGetLastError();
}

cudaError_t launch_erase_weights(const float* logp_x, const int32_t* corpus_tok,
                                 const int32_t* argmax_t, const float* row_mask, int A, int B,
                                 float gamma, int hard, float* weight, cudaStream_t s) {
  erase_weights_kernel<<<(A + 7) / 8, 256, 0, s>>>(logp_x, corpus_tok, argmax_t, row_mask, A, B,
                                                   gamma, hard, weight);
  return cudaGetLastError();
}

}  // namespace alr
