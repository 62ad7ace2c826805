// Internal launch interface between the C-ABI layer (api.cu) and the kernel translation units.
#pragma once

#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

namespace alr {

// Row-block x vocabulary-split work plan of the fused loss kernels.
//   A "unit" is one 128-row block times one contiguous range of 128-column vocabulary tiles.
//   Units are numbered group by group: a group holds `group_rows` consecutive row blocks,
//   and inside a group the row block varies fastest, so the CTAs running at the same time
//   share both their hidden-state tiles and their head tiles through L2.
struct LossPlan {
  int N, d, V, B;
  int bn;          // vocabulary columns per tile (128 or 256)
  int n_rb;        // ceil(N / 128)
  int n_vt;        // ceil(V / bn)
  int n_vs;        // vocabulary splits
  int n_parts;     // partial records per row: n_vs * (bn / 64), one per split and 64-column group
  int group_rows;  // row blocks per group
  int n_units;     // n_rb * n_vs
  int grid;        // persistent CTAs
  int mc;          // 1: clusters of two CTAs share each head tile by TMA multicast (bf16,
                   // 256-column tiles); n_rb and group_rows then count row-block pairs and
                   // the grid is sized from the clusters that fit
};

// Partial statistics of one row over the columns of one vocabulary split seen by one
// epilogue thread (structure of arrays, field-major: part[f * n_parts * N + part * N + row]).
enum PartField {
  kPMd = 0,   // running max of z_d
  kPSd,       // sum exp(z_d - m_d)
  kPMt,       // running max of z_t
  kPSt,       // sum exp(z_t - m_t)
  kPU,        // sum exp(z_t - m_t) * (z_d - m_d)
  kPW,        // sum exp(z_t - m_t) * (z_t - m_t)
  kPBd,       // best z_d
  kPId,       // its index (int bits)
  kPSecd,     // second-best z_d (any other index)
  kPBt,
  kPIt,
  kPSect,
  kPZx,       // z_t at the corpus token if it lies in the split, else NaN
  kPSdLo,     // rounding error of kPSd (the sum is kPSd + kPSdLo)
  kPStLo,     // rounding error of kPSt
  kPFields
};

// Compact labels (top-k target probabilities + tail bin): k tokens per row.
constexpr int kTopK = 8;

// Partial record of the label readout: log-sum-exp state, the k best target logits with their
// token ids, z_t at the corpus token.
// kRSLo: the rounding error of the sum kRS (the sum is kRS + kRSLo); kRR: the exponent
// residual r of the reference kRM (every summed exponential carries the factor 2^r).
enum ReadoutField {
  kRM = 0, kRS, kRTop, kRIdx = kRTop + kTopK, kRZx = kRIdx + kTopK, kRSLo, kRR, kRFields
};

// Partial record of the top-k loss forward: log-sum-exp state and greedy top-2 of z_d, and
// z_d at the row's k label tokens (NaN where the token is outside the part's columns).
// kKSLo: the rounding error of the sum kKS; kKSIn: the part of kKS that the row's label
// tokens contributed (the same rounded terms); kKR: the exponent residual of kKM.
enum TopkField {
  kKM = 0, kKS, kKBest, kKIdx, kKSec, kKZ, kKSLo = kKZ + kTopK, kKSIn, kKR, kKFields
};

// What one launch of the fused loss kernel computes.
enum LossMode {
  kModeFwd = 0,      // dual GEMM: full-vocabulary statistics of z_d and z_t
  kModeBwd = 1,      // dual GEMM: G = c (q - p)
  kModeReadout = 2,  // single GEMM on H_t: log-sum-exp, top-k, z_t at the corpus token
  kModeTopkFwd = 3,  // single GEMM on H_d: log-sum-exp, top-2, z_d at the label tokens
  kModeTopkBwd = 4,  // single GEMM on H_d: gradient of the top-k + tail soft CE
  kModeFwdKeep = 5,  // kModeFwd that also writes z_d and z_t to global memory
  kModeTopkFwdKeep = 6  // kModeTopkFwd that also writes z_d to global memory
};

struct LossArgs {
  LossPlan plan;
  float* part;                // forward: partial statistics
  const int32_t* corpus_tok;  // forward: nullable
  void* G;                    // backward: logit gradient [N, V] (element type of the inputs)
  const float* lse_d;         // backward
  const float* lse_t;
  const float* weight;
  const float* weight_sum;
  float lam;
  int* status;
  int withhold_first_stage;   // test hook: the producer never fills its first stage
  const int32_t* top_idx;     // top-k modes: label tokens [N, kTopK]
  const float* top_prob;      // top-k backward: label probabilities [N, kTopK]
  const float* tail;          // top-k backward: label tail mass [N]
  const float* tail_q;        // top-k backward: drafter mass outside the label tokens [N]
  void* zd_out;               // keep modes: z_d (and z_t) [N, V] (fp16 for bf16 inputs, else fp32)
  void* zt_out;
  uint16_t* zd_ref;           // keep modes, bf16 inputs: fp16 reference of each 16-column group
  uint16_t* zt_ref;           // of z_d / z_t, group-major [ceil(V / 16), N] (see kKeepGroup)
};

// Kept fp16 logits are stored relative to a per-group reference: the columns of a row go in
// groups of kKeepGroup, whose reference R is the group's maximum rounded up to fp16, and each
// logit is kept as fp16(z - R).  The rounding error then scales with R - z, which is small
// exactly where exp(z - lse) is large.  The references are stored group-major,
// R[v / 16, r] at (v / 16) * N + r, so that one warp's 32 rows of a group are contiguous.
constexpr int kKeepGroup = 16;

// Fused loss kernels (loss_gemm_kernel.cuh, launched from loss_gemm.cu).  dtype: 0 bf16, 1 fp32
// (tf32 products).
//   a0: the first hidden-state operand (H_d; H_t for the readout), a1: H_t (dual modes).
//   g_store: bf16 G [N, V] as 16-column x 32-row boxes without swizzle (gradient modes, bf16),
//            or fp16 z_d [N, V] in the same boxes (kModeFwdKeep, bf16);
//   g_store2: fp16 z_t [N, V] (kModeFwdKeep, bf16).  Unused maps may be any valid map.
cudaError_t launch_loss_kernel(int mode, int dtype, const CUtensorMap& a0, const CUtensorMap& a1,
                               const CUtensorMap& w, const CUtensorMap& g_store,
                               const CUtensorMap& g_store2, const LossArgs& args, cudaStream_t s);

// Plain GEMM C[M, Nc] (+)= A[M, K] B[K, Nc] with fp32 output (plain_gemm_kernel.cuh, single-CTA
// form launched from plain_gemm.cu).
struct GemmArgs {
  int M, Nc, K;
  float* C;
  int64_t ldc;
  int n_mb, n_nb;   // 128-row and 256-column tile counts
  int group_m;      // m-blocks per raster group
  int n_tiles;
  int grid;
  int* status;
  int withhold_first_stage;   // test hook: the producer never fills its first stage
};
// a_mn / b_mn: operand stored MN-major (A as [K, M], B as [K, Nc]) instead of K-major
// (A as [M, K], B as [Nc, K]).  accumulate: C += A B instead of C = A B.
cudaError_t launch_plain_gemm(int dtype, bool a_mn, bool b_mn, bool accumulate,
                              const CUtensorMap& a, const CUtensorMap& b, const GemmArgs& args,
                              cudaStream_t s);
size_t plain_gemm_smem_bytes(int dtype);
// The cluster forms of the same kernel (multicast clusters, CTA pairs) are in
// libalr_cluster.so (cluster_forms.h).

// Row-level kernels (row_kernels.cu).
cudaError_t launch_gather(const void* feat, int S, int L, int d, int elem_bytes,
                          const int32_t* seq, const int32_t* pos, const int32_t* valid_len,
                          int A, int B, void* out, float* row_valid, cudaStream_t s);
cudaError_t launch_combine(const LossPlan& plan, const float* part, int mode, float gamma,
                           const float* row_mask, const int32_t* corpus_tok, float* loss_row,
                           float* ent_row, float* lse_d, float* lse_t, int32_t* argmax_d,
                           int32_t* argmax_t, float* gap_d, float* gap_t, float* logp_x,
                           float* weight, double* anchor_part, cudaStream_t s);
cudaError_t launch_finalize(const double* anchor_part, int A, float lam, float* loss_total,
                            float* weight_sum, float* wl_sum, cudaStream_t s);
// loss_total = lambda * wl_sum / weight_sum (0 when weight_sum = 0), from reduced sums.
cudaError_t launch_loss_from_sums(const float* wl_sum, const float* weight_sum, float lam,
                                  float* loss_total, cudaStream_t s);
cudaError_t launch_readout_combine(const LossPlan& plan, const float* part, bool has_corpus,
                                   int32_t* top_idx, float* top_prob, float* tail, float* lse_t,
                                   int32_t* argmax_t, float* gap_t, float* logp_x,
                                   cudaStream_t s);
cudaError_t launch_topk_combine(const LossPlan& plan, const float* part, const float* top_prob,
                                const float* tail, const float* row_mask, const float* weight_in,
                                float gamma, float* loss_row, float* lse_d, float* tail_q,
                                int32_t* argmax_d, float* gap_d, float* weight,
                                double* anchor_part, cudaStream_t s);
// G = lambda omega_r / sum omega (exp(z_d - lse_d) - exp(z_t - lse_t)) from kept logits
// (dtype 0: fp16 values plus the group references zd_ref / zt_ref [ceil(V / 16), N];
// dtype 1: fp32, references unused) into G [N, V] (bf16 / fp32); G may be zd itself.
cudaError_t launch_logits_grad(int dtype, const void* zd, const void* zt, const uint16_t* zd_ref,
                               const uint16_t* zt_ref, const float* lse_d, const float* lse_t,
                               const float* weight, const float* weight_sum, float lam, int N,
                               int V, void* G, cudaStream_t s);
// Gradient of the top-k + tail soft CE from kept z_d (as in launch_logits_grad):
// G = c_r beta_r q outside the row's label tokens, c_r (q - prob_i) at label token i, with
// q = exp(z_d - lse_d), c_r = lambda omega_r / sum omega, beta_r = 1 - tail_r / tail_q_r (1 when
// tail_r = 0).  G (bf16 / fp32) may be zd itself.
cudaError_t launch_topk_logits_grad(int dtype, const void* zd, const uint16_t* zd_ref,
                                    const int32_t* top_idx,
                                    const float* top_prob, const float* tail, const float* tail_q,
                                    const float* lse_d, const float* weight,
                                    const float* weight_sum, float lam, int N, int V, void* G,
                                    cudaStream_t s);
cudaError_t launch_accept_len(const int32_t* am_d, const int32_t* am_t, const float* active,
                              int A, int B, int32_t* acc, int64_t* hist, cudaStream_t s);
cudaError_t launch_erase_weights(const float* logp_x, const int32_t* corpus_tok,
                                 const int32_t* argmax_t, const float* row_mask, int A, int B,
                                 float gamma, int hard, float* weight, cudaStream_t s);

cudaError_t launch_ira_blocks(int S, int K, int max_blocks, const int32_t* valid_anchors,
                              const int32_t* rollout_len, const int32_t* offsets,
                              const int32_t* rollout_tok, const int32_t* corpus_anchor_tok,
                              int32_t* seq, int32_t* pos, int32_t* vlen, int32_t* ctx_len,
                              int32_t* anchor_tok, cudaStream_t s);

// IRA draws (one block per sample, L * 8 bytes of shared memory): n_valid [S], anchor_pos
// [S, max_blocks] (draw order, -1 past m), offsets [S, max_blocks / 2].
cudaError_t launch_ira_draw(int S, int L, int K, int max_blocks, const uint8_t* anchor_ok,
                            const uint32_t* keys, const uint32_t* offset_u, int32_t* n_valid,
                            int32_t* anchor_pos, int32_t* offsets, cudaStream_t s);
// Context rows of the secondary blocks: ctx [S, max_blocks / 2, C, F] from the primaries'
// stored rollout features [S * P, C, F]; ctx_len, prefix_end [S, max_blocks / 2] (nullable).
cudaError_t launch_ira_context(const void* store, int C, int F, int elem_bytes, int S, int K,
                               int max_blocks, const int32_t* n_valid, const int32_t* rollout_len,
                               const int32_t* offsets, const int32_t* anchor_pos, void* ctx,
                               int32_t* ctx_len, int32_t* prefix_end, cudaStream_t s);

// out[c, r] = in[r, c] for an fp32 [R, C] matrix; out rows are ld_out elements apart.
cudaError_t launch_transpose32(const float* in, float* out, int R, int C, int ld_out,
                               cudaStream_t s);

// Record `msg` as this host thread's alr_last_error() text and return `code` (api.cu).
int set_last_error(int code, const char* msg);

// Per-device status word (status.cu).
int* device_status_ptr();

}  // namespace alr
