/*
 * libalr — GB300 (sm_103a) hot path of Anchor-Label Relabelling with In-Rollout Anchors.
 *
 * The operations follow "Recovering Off-Policy Supervision for Speculative Decoding":
 *   - the weighted, normalised soft cross-entropy of Eq. 1 with the slot envelope
 *     w_k = exp(-(k-1)/gamma), evaluated over the full vocabulary;
 *   - the ALR label distribution pi = p_T(. | ...) read through the vocabulary head (Eq. 3);
 *   - the erase comparator's survival gate (Eq. 2, soft and hard variants);
 *   - the IRA placement of blocks inside a rollout, with weights w_k 1[j+k <= K] (Eq. 4);
 *   - the greedy accepted length behind the MAT metric (Sec. 3.2, Sec. 4), ties to the
 *     lower token id (App. A, rollout implementation).
 *
 * Conventions shared by every entry point
 *   Rows.      A batch holds A anchors with B rows each, N = A*B; row r = a*B + s holds the
 *              paper's slot k = s+1 of anchor a.  1 <= B <= 32.
 *   Memory.    Every pointer is a DEVICE pointer owned by the caller, unless stated.  The
 *              library allocates no device memory; scratch comes from a caller workspace whose
 *              size the matching *_workspace_size function returns.  Matrices are row-major
 *              and dense; every base pointer must be 16-byte aligned.
 *   Streams.   `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *              Every call only enqueues work on it and returns without synchronising.
 *   Errors.    Every call returns an int status (ALR_OK = 0) and never throws.  Arguments
 *              are validated before anything is enqueued; on failure nothing is launched and
 *              alr_last_error() (per host thread) describes the problem.  Kernels that wait
 *              on on-chip pipelines give up after a bounded time and record ALR_ERR_TIMEOUT
 *              in a per-device status word that alr_device_status() reads.
 *   Inputs.    Outputs are unspecified when the inputs contain NaN or Inf.
 *   Kernel forms (environment, read at every call; results do not depend on them except for
 *              floating-point rounding of the GEMMs, and the loss kernels' outputs not at all):
 *              ALR_GEMM_FORM = mcast (default: clusters of two CTAs share each B tile by TMA
 *              multicast) | single | mcast4 | pair (CTA pairs with M = 256 tcgen05 products)
 *              selects the bf16 GEMM kernel; ALR_LOSS_FORM = single (default) | mcast selects
 *              the fused loss kernels' form.  fp32 (tf32) products always run on single CTAs.
 *              The cluster forms (mcast, mcast4, pair, and the loss kernels' mcast) are built
 *              into a second library, libalr_cluster.so, which this library loads from its own
 *              directory on first use.  A process launched as one rank of several (environment
 *              WORLD_SIZE > 1) never loads it, so TMA multicast loads stay out of multi-rank
 *              processes; there, or if it cannot be loaded, every form runs on single CTAs.
 *              alr_kernel_forms() reports the choice, alr_cluster_forms_error() the reason.
 */
#ifndef ALR_H
#define ALR_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Status codes. */
#define ALR_OK 0
#define ALR_ERR_INVALID_ARG 1   /* null pointer, bad size, misalignment, workspace too small */
#define ALR_ERR_UNSUPPORTED 2   /* dtype / mode not supported, or the device is not sm_103 */
#define ALR_ERR_CUDA 3          /* a CUDA runtime or driver call failed (launch, encode)   */
#define ALR_ERR_TIMEOUT 4       /* a device-side bounded wait expired (alr_device_status)  */

/* Element types of H_d, H_t, W (and the feature buffer of the gather). */
#define ALR_BF16 0              /* bfloat16 inputs, bf16 tensor-core products, fp32 accumulate */
#define ALR_F32 1               /* fp32 inputs, tf32 tensor-core products, fp32 accumulate     */

/* Slot-weight modes of the loss (omega_{a,k} of Eq. 1). */
#define ALR_MODE_ALR 0          /* omega = w_k * mask             (ALR / IRA, Sec. 3.2)        */
#define ALR_MODE_ERASE_SOFT 1   /* omega = w_k * mask * g_{a,k}   (soft survival gate, Eq. 2)  */
#define ALR_MODE_ERASE_HARD 2   /* omega = w_k * mask * prod 1[x == greedy target] (Eq. 2)     */

/* Problem description shared by the forward and backward calls. */
typedef struct {
    int64_t N;       /* rows, N = A*B, N >= 1                                                 */
    int32_t d;       /* hidden size (contraction length), d >= 8, d % 8 == 0                  */
    int32_t V;       /* vocabulary size, V >= 2, V % 8 == 0                                   */
    int32_t B;       /* rows per anchor, 1 <= B <= 32, N % B == 0                             */
    int32_t dtype;   /* ALR_BF16 or ALR_F32                                                   */
    int32_t mode;    /* ALR_MODE_*                                                            */
    float lambda;    /* KD loss scale lambda multiplying Eq. 1 (App. A: 1.013441 VL, 1.0 text) */
    float gamma;     /* envelope constant gamma of Eq. 1, > 0 (default 2)                     */
} alr_params;

/* Forward outputs, all device pointers, length N unless stated. */
typedef struct {
    float* loss_row;     /* l_r = -sum_v p log q (required)                                    */
    float* ent_row;      /* H(p_r), the label entropy (nullable)                               */
    float* lse_d;        /* log-sum-exp of the drafter logits z_d = H_d W (required)           */
    float* lse_t;        /* log-sum-exp of the target logits z_t = H_t W (required)            */
    int32_t* argmax_d;   /* greedy drafter token, lowest id on ties (required)                 */
    int32_t* argmax_t;   /* greedy target token, lowest id on ties (required)                  */
    float* gap_d;        /* top-1 minus top-2 drafter logit, 0 on an exact tie (nullable)      */
    float* gap_t;        /* same for the target logits (nullable)                              */
    float* logp_x;       /* erase modes: log p_t(corpus_tok_r); other modes untouched (nullable) */
    float* weight;       /* omega_r, the final slot weight (required)                          */
    float* loss_total;   /* [1] L = lambda * sum omega l / sum omega, 0 when sum omega = 0     */
    float* weight_sum;   /* [1] sum omega (the backward's normaliser)                          */
    float* wl_sum;       /* [1] sum omega l, the numerator of Eq. 1 (nullable; for sums across
                            the shards of a batch, see alr_loss_from_sums)                      */
} alr_fwd_outputs;

/* Library version string (static storage). */
const char* alr_version(void);

/* Description of the last failed call on this host thread (static thread-local storage). */
const char* alr_last_error(void);

/* ALR_OK when the current device is compute capability 10.3 (sm_103), else ALR_ERR_UNSUPPORTED. */
int alr_device_supported(void);

/*
 * Synchronises `stream`, then reads the current device's status word: ALR_OK, or
 * ALR_ERR_TIMEOUT if any kernel of this library gave up a bounded wait since the last clear.
 * clear != 0 resets the word to ALR_OK.
 */
int alr_device_status(void* stream, int clear);

/*
 * The kernel forms the next bf16 call will use in this process (no device needed):
 *   *gemm: 0 single CTAs, 1 clusters of two sharing B tiles by TMA multicast, 2 CTA pairs
 *          (cta_group::2), 3 clusters of four with multicast;
 *   *loss: 0 single CTAs, 1 clusters of two sharing head tiles by TMA multicast.
 */
int alr_kernel_forms(int32_t* gemm, int32_t* loss);

/*
 * "" when libalr_cluster.so (the cluster kernel forms) is loaded in this process, else why it
 * is not: the process is one rank of several, or the loader's message.  Loads it on first use
 * (no device needed).  The string is owned by the library and stays valid.
 */
const char* alr_cluster_forms_error(void);

/*
 * Test hook for the failure-detection path (the paper has no counterpart).  With enable != 0,
 * the next launch, on any thread, of the fused loss kernel by a forward (alr_slot_loss_fwd,
 * alr_slot_loss_fwd_keep_logits, alr_slot_loss_fwd_noalloc) or of a tensor-core GEMM in the
 * single or multicast form (alr_gemm, and the dH / dW products of the backward entry points)
 * withholds the first pipeline stage of each CTA: nothing ever fills it, so the MMA issuer's
 * bounded wait runs out after about 1.5 s, every role of the CTA leaves its loop (copies in
 * flight are waited for, tensor memory is released) and the kernel records ALR_ERR_TIMEOUT in
 * the device status word.  That call's outputs are meaningless; alr_device_status() then
 * returns ALR_ERR_TIMEOUT and the context stays usable.  Nothing faults, traps or hangs.  The
 * hook disarms itself after one launch.
 */
int alr_debug_withhold_next_stage(int enable);

/*
 * IRA gather (Eq. 4; App. A: rollout features stored for y*_1..y*_13).
 *   feat      [S, L, d] features of S rollout sequences of length L, element type `dtype`.
 *   seq, pos  [A] int32: anchor a reads sequence seq[a] from position pos[a].
 *   valid_len [A] int32 or NULL (= L): positions >= min(valid_len[a], L) are not supervised.
 *   out       [A*B, d] (same dtype): out[a*B+s] = feat[seq[a], pos[a]+s] for a valid row,
 *             zeros otherwise.
 *   row_valid [A*B] float or NULL: 1 for a valid row, 0 otherwise.  A row is invalid when
 *             seq[a] is outside [0, S), pos[a] < 0, or pos[a]+s >= min(valid_len[a], L).
 * A secondary IRA block at offset j inside a primary block's K stored rows is the gather
 * with L = K, pos = j and valid_len = K, whose row_valid is 1[j + k <= K].
 * Requires d * elemsize % 16 == 0.
 */
int alr_gather_ira_blocks(const void* feat, int32_t S, int32_t L, int32_t d, int32_t dtype,
                          const int32_t* seq, const int32_t* pos, const int32_t* valid_len,
                          int32_t A, int32_t B, void* out, float* row_valid, void* stream);

/*
 * IRA block plan (Sec. 3.2, In-rollout anchors; Eq. 4; App. A).  For S samples, sample s with
 * valid_anchors[s] = v valid anchor positions keeps m = min(v, max_blocks) blocks: the first
 * ceil(m/2) are primary (their rollouts produce labels), the next floor(m/2) secondary, the
 * rest unused.  Secondary block i sits in primary block i's rollout at offset
 * j = offsets[s * (max_blocks/2) + i] (the method draws j ~ U{2..K-1}; the caller passes the
 * draws; j outside [1, K-1] leaves the block unused).  Primary block p of sample s owns rows
 * [s*P + p] of a label buffer [S*P, K, ...] with P = max_blocks - max_blocks/2, of which
 * rollout_len[s*P + p] are valid (K, fewer after early termination); a secondary block whose
 * offset lies past them (j > rollout_len: y*_j was never generated) is unused.
 * Outputs per block slot t = s*max_blocks + b (int32 [S*max_blocks]):
 *   seq, pos, valid_len - the alr_gather_ira_blocks arguments that read the block's K label
 *             rows from that buffer: a secondary block's row k reads primary row j + k - 1 and
 *             is supervised iff j + k <= rollout_len (Eq. 4); unused blocks get seq = -1;
 *   ctx_len   (nullable) - rollout features in the block's context: j - 1 (0 for primary);
 *   anchor_tok (nullable) - corpus_anchor_tok[t] for a primary block, the rollout token y*_j
 *             = rollout_tok[(s*P + p)*K + j - 1] for a secondary one, -1 when not given.
 */
int alr_ira_blocks(int32_t S, int32_t K, int32_t max_blocks, const int32_t* valid_anchors,
                   const int32_t* rollout_len, const int32_t* offsets, const int32_t* rollout_tok,
                   const int32_t* corpus_anchor_tok, int32_t* seq, int32_t* pos,
                   int32_t* valid_len, int32_t* ctx_len, int32_t* anchor_tok, void* stream);

/*
 * IRA draws (Sec. 3.2, In-rollout anchors: m = min(v, max_blocks) blocks from the v valid
 * anchor positions of a sample, secondary offsets j ~ U{2, ..., K-1}; App. A: 128 anchors per
 * sample, j in {2..14}).  The random numbers are inputs, so that a run is reproducible from
 * the caller's generator:
 *   anchor_ok [S, L] uint8: nonzero where position a of sample s may anchor a block.
 *   keys      [S, L] uint32: independent uniform random integers, one per position.  The draw
 *             (uniform, without replacement) is the valid positions in increasing order of
 *             their keys, equal keys in position order, the first m taken.
 *   offset_u  [S, max_blocks/2] uint32 uniform: j = 2 + floor(u * (K - 2) / 2^32).
 * Outputs: n_valid [S] (v); anchor_pos [S, max_blocks] the drawn positions in draw order, -1
 * past m (the first ceil(m/2) anchor the primary blocks, see alr_ira_blocks); offsets
 * [S, max_blocks/2] (j, the offsets argument of alr_ira_blocks and alr_ira_context).
 * Requires 1 <= L <= ALR_IRA_MAX_LEN (L * 8 bytes of shared memory per sample) and K >= 3.
 */
#define ALR_IRA_MAX_LEN 16384
int alr_ira_draw(int32_t S, int32_t L, int32_t K, int32_t max_blocks, const uint8_t* anchor_ok,
                 const uint32_t* keys, const uint32_t* offset_u, int32_t* n_valid,
                 int32_t* anchor_pos, int32_t* offsets, void* stream);

/*
 * Context of the IRA secondary blocks (Sec. 3.2: the target representations of the corpus
 * prefix up to the anchor a, concatenated with those stored for y*_1..y*_{j-1}; App. A: the
 * rollout stores the outputs of the five target layers the drafter reads for y*_1..y*_13).
 *   store [S*P, C, F] (dtype), P = max_blocks - max_blocks/2: primary block p of sample s
 *         keeps C >= K-2 rows of F features (e.g. the five layers' d-vectors side by side,
 *         F = 5 d), row r for rollout token y*_{r+1}.
 *   n_valid [S], offsets [S, max_blocks/2], anchor_pos [S, max_blocks]: from alr_ira_draw;
 *   rollout_len [S*P]: label rows of each primary rollout (K, fewer after early termination).
 * Secondary i of sample s (i < floor(m/2)) sits in primary i at offset j; it exists when
 * 1 <= j <= K-1 and j <= rollout_len (as in alr_ira_blocks).  Outputs:
 *   ctx [S, max_blocks/2, C, F]: rows r < j-1 are store[s*P + i, r] (y*_1..y*_{j-1}), the
 *       other rows, and every row of a slot without a block, are zero;
 *   ctx_len [S, max_blocks/2] (nullable): j - 1, or 0;
 *   prefix_end [S, max_blocks/2] (nullable): the corpus position a whose prefix x_0..x_a the
 *       context starts with (primary i's anchor), -1 without a block.
 * Requires F * elemsize % 16 == 0, 16-byte aligned store and ctx.
 */
int alr_ira_context(const void* store, int32_t C, int32_t F, int32_t dtype, int32_t S, int32_t K,
                    int32_t max_blocks, const int32_t* n_valid, const int32_t* rollout_len,
                    const int32_t* offsets, const int32_t* anchor_pos, void* ctx,
                    int32_t* ctx_len, int32_t* prefix_end, void* stream);

/* Workspace bytes alr_slot_loss_fwd needs for `p` (0 on invalid params). */
size_t alr_fwd_workspace_size(const alr_params* p);

/*
 * Forward pass of the slot loss (Eq. 1 with labels from Eq. 3, gate from Eq. 2).
 *   Hd, Ht     [N, d] drafter and target hidden states (dtype p->dtype).
 *   W          [d, V] vocabulary head shared by both sides (row-major, V contiguous).
 *   row_mask   [N] float or NULL (= all ones): multiplies omega (termination, IRA validity).
 *   corpus_tok [N] int32, required in the erase modes: the corpus token x that row r's
 *              label predicts; must lie in [0, V).  Ignored in ALR mode.
 *   out        output pointers (see alr_fwd_outputs).
 * The logits are produced tile by tile in tensor memory and reduced on chip; they are never
 * written to global memory.
 */
int alr_slot_loss_fwd(const alr_params* p, const void* Hd, const void* Ht, const void* W,
                      const float* row_mask, const int32_t* corpus_tok,
                      const alr_fwd_outputs* out, void* workspace, size_t ws_bytes,
                      void* stream);

/*
 * Forward pass for callers that cannot allocate device memory.  The paper has no counterpart:
 * this is a deployment variant of alr_slot_loss_fwd.
 *
 * Who needs it: a caller whose host process has handed all device memory to its own pool at
 * start-up and allows no further allocation, or a caller on a latency-critical path where a
 * device allocation (which can synchronise the whole device) is not acceptable, cannot
 * provide the workspace alr_slot_loss_fwd asks for.  This call takes the same arguments minus
 * the workspace and runs the same kernels; their scratch lives in a fixed array of
 * ALR_NOALLOC_SCRATCH_BYTES bytes in device global memory that belongs to the library image.
 * It calls no cudaMalloc, cudaFree or other allocating routine.
 *
 *   - Limit: problems whose alr_fwd_workspace_size exceeds ALR_NOALLOC_SCRATCH_BYTES are
 *     rejected with ALR_ERR_INVALID_ARG and a message naming both sizes (bf16 at d=4096,
 *     V=151936, B=16 on a 152-SM GB300: about 14 700 rows).
 *   - Memory: every device that loads the library holds the array until the process exits.
 *   - Set-up: the first call on a device (with that device current) looks up the array's
 *     device address; make that first call before any stream capture.  The address is kept
 *     per device and context, so after a device reset or a new primary context the next call
 *     looks it up again (again, before any capture).
 *   - Sharing: all calls on a device share the one array and it keeps the last call's
 *     contents.  Nothing in it needs clearing (the kernels overwrite what they read), but
 *     calls whose work overlaps on the GPU (different streams, or different host threads
 *     without ordering) race on it and give undefined results: serialise them.
 */
#define ALR_NOALLOC_SCRATCH_BYTES (64u * 1024u * 1024u)
int alr_slot_loss_fwd_noalloc(const alr_params* p, const void* Hd, const void* Ht,
                              const void* W, const float* row_mask, const int32_t* corpus_tok,
                              const alr_fwd_outputs* out, void* stream);

/* Workspace bytes alr_slot_loss_bwd needs for `p` (includes the logit gradient, N*V*elem). */
size_t alr_bwd_workspace_size(const alr_params* p);

/*
 * Backward pass of the slot loss.  The label p, the weights and the gate are constants, so
 * the gradient reaches z_d only: G = lambda * omega_r / sum omega * (q - p), recomputed
 * tile by tile from Hd, Ht, W and the forward's lse_d, lse_t.
 *   weight, weight_sum, lse_d, lse_t   forward outputs (device).
 *   dHd  [N, d] float, overwritten with G W^T.
 *   dW   [d, V] float or NULL; when given, H_d^T G is ADDED to it (gradient accumulation).
 */
int alr_slot_loss_bwd(const alr_params* p, const void* Hd, const void* Ht, const void* W,
                      const float* weight, const float* weight_sum, const float* lse_d,
                      const float* lse_t, float* dHd, float* dW, void* workspace,
                      size_t ws_bytes, void* stream);

/* Workspace bytes alr_logit_grad needs for `p` (0 for bf16; W^T for fp32). */
size_t alr_logit_grad_workspace_size(const alr_params* p);

/*
 * The first step of alr_slot_loss_bwd on its own: the gradient of Eq. 1 with respect to the
 * drafter logits, G[r, v] = lambda * omega_r / sum omega * (q[r, v] - p[r, v]), recomputed
 * tile by tile from Hd, Ht, W and the forward's lse_d, lse_t, written to G [N, V] (element
 * type p->dtype, row-major).  dH_d = G W^T and dW += H_d^T G then follow with alr_gemm
 * (bf16: layouts (0, 0) and (1, 1)).
 */
int alr_logit_grad(const alr_params* p, const void* Hd, const void* Ht, const void* W,
                   const float* weight, const float* weight_sum, const float* lse_d,
                   const float* lse_t, void* G, void* workspace, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------------------
 * Kept logits: the same loss with the logits stored by the forward instead of recomputed by
 * the backward.  The forward's two head products are the path's dominant cost; keeping their
 * results costs 2 * N * V logit elements of device memory (fp16 for bf16 inputs: 2 x 9.96 GB
 * at N = 32768, V = 151936) and spares the backward those two products.  The gradient is the
 * one of Eq. 1 with respect to z_d, as in alr_slot_loss_bwd.
 *
 * Storage of a kept logit matrix Z of bf16 inputs: fp16 values relative to group references.
 * The columns of a row go in groups of ALR_KEEP_GROUP; group c of row r has the reference
 *     R[c, r] = the largest logit of the group, rounded up to fp16,
 * and each logit is kept as Z[r, v] = fp16(z[r, v] - R[v / 16, r]) (rounded to nearest), so
 *     z[r, v] = Z[r, v] + R[v / 16, r]   (both fp16, added in fp32).
 * Rounding then moves z by at most 2^-11 (R - z) instead of 2^-11 |z|: the error is small
 * exactly where the softmax weight exp(z - lse) is large (lse >= every z of the row), and the
 * relative error of q = exp(z - lse) stays near 2^-11 (1 + ln(1/q)) however large the logits
 * are (trained heads reach |z| of 30-40, where plain fp16 would move q by ~2 %).
 * R is stored group-major: [alr_kept_ref_groups(V), N] fp16 (uint16_t bits), R[c, r] at
 * c * N + r, so that the forward writes the references of 32 consecutive rows as one run.
 * fp32 inputs keep plain fp32 logits and no references (their *_ref arguments are ignored
 * and may be NULL).  |z| must stay below 65504.
 * ------------------------------------------------------------------------------------- */
#define ALR_KEEP_GROUP 16

/* Number of 16-column groups of a row of V logits, ceil(V / 16): the leading dimension of a
 * group-reference array [groups, N] (0 for V < 1). */
int32_t alr_kept_ref_groups(int32_t V);

/*
 * alr_slot_loss_fwd, which also writes the logits z_d = H_d W and z_t = H_t W:
 *   Zd, Zt          [N, V] row-major: fp16 relative to the group references for ALR_BF16
 *                   inputs, fp32 for ALR_F32 inputs;
 *   Zd_ref, Zt_ref  [alr_kept_ref_groups(V), N] fp16 group references (ALR_BF16 inputs);
 *   all caller-owned, 16-byte aligned, not overlapping any input or output.
 * Every other argument, output and error is that of alr_slot_loss_fwd (same workspace size),
 * and the forward outputs are bit-identical to it.
 */
int alr_slot_loss_fwd_keep_logits(const alr_params* p, const void* Hd, const void* Ht,
                                  const void* W, const float* row_mask, const int32_t* corpus_tok,
                                  void* Zd, void* Zt, uint16_t* Zd_ref, uint16_t* Zt_ref,
                                  const alr_fwd_outputs* out, void* workspace, size_t ws_bytes,
                                  void* stream);

/*
 * G[r, v] = lambda * omega_r / sum omega * (exp(z_d[r, v] - lse_d[r]) - exp(z_t[r, v] - lse_t[r]))
 * from kept logits (Zd, Zt and, for bf16 inputs, Zd_ref, Zt_ref as written by
 * alr_slot_loss_fwd_keep_logits) and the forward's weight, weight_sum, lse_d, lse_t; G [N, V]
 * has the element type of p->dtype (bf16 / fp32).  G may be Zd itself (the gradient then
 * overwrites z_d in place); it must not otherwise overlap Zd, Zt or the references.  Rows with
 * omega_r = 0 (or sum omega = 0) get G = 0.  No workspace.
 */
int alr_logit_grad_from_logits(const alr_params* p, const void* Zd, const void* Zt,
                               const uint16_t* Zd_ref, const uint16_t* Zt_ref,
                               const float* weight, const float* weight_sum, const float* lse_d,
                               const float* lse_t, void* G, void* stream);

/* Workspace bytes alr_slot_loss_bwd_from_logits needs (0 for bf16; G^T and H_d^T for fp32). */
size_t alr_bwd_from_logits_workspace_size(const alr_params* p);

/*
 * Backward pass from kept logits: alr_logit_grad_from_logits into G (caller-owned [N, V],
 * may be Zd), then dH_d = G W^T (overwrites dHd [N, d] fp32) and, when dW is given,
 * dW += H_d^T G (dW [d, V] fp32).  Errors as in alr_slot_loss_bwd.
 */
int alr_slot_loss_bwd_from_logits(const alr_params* p, const void* Hd, const void* W,
                                  const void* Zd, const void* Zt, const uint16_t* Zd_ref,
                                  const uint16_t* Zt_ref, const float* weight,
                                  const float* weight_sum, const float* lse_d, const float* lse_t,
                                  void* G, float* dHd, float* dW, void* workspace,
                                  size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------------------
 * Compact labels: the target's top-k probabilities plus a tail bin.
 *
 * The paper's loss l evaluates soft cross-entropy against the target distribution restricted
 * to its 8 most probable tokens, with the remaining mass in one tail bin (Sec. 3.1 under
 * Eq. 1; App. A, KD loss), and each rollout step keeps exactly that label (App. A, rollout
 * implementation: top 8 tokens and the remaining mass, greedy ties to the lower id).  These
 * entry points compute that label from the target hidden states (the readout) and the loss
 * against it, whose forward and backward need only the drafter's head product.
 * ------------------------------------------------------------------------------------- */
#define ALR_TOPK 8

/* Workspace bytes alr_label_readout needs for `p` (0 on invalid params). */
size_t alr_readout_workspace_size(const alr_params* p);

/*
 * Label readout: for each row, z_t = h_t W over the whole vocabulary (never stored), then
 *   top_idx  [N, ALR_TOPK] int32: the most probable tokens, probability descending, equal
 *            probabilities to the lower token id (top_idx[r*8] is the greedy token y*);
 *   top_prob [N, ALR_TOPK]: their probabilities p_T(v);   tail [N]: 1 - sum of top_prob,
 *            computed as the mass of the other tokens;
 *   lse_t, argmax_t, gap_t [N] (nullable): log-sum-exp, greedy token, top-1 minus top-2;
 *   logp_x [N] (nullable, needs corpus_tok): log p_T(corpus_tok), the erase gate's factor.
 * Uses p->N, d, V (>= ALR_TOPK), dtype; mode, lambda, gamma and B are ignored (B must still
 * divide N).
 */
int alr_label_readout(const alr_params* p, const void* Ht, const void* W,
                      const int32_t* corpus_tok, int32_t* top_idx, float* top_prob, float* tail,
                      float* lse_t, int32_t* argmax_t, float* gap_t, float* logp_x,
                      void* workspace, size_t ws_bytes, void* stream);

/* Outputs of alr_topk_loss_fwd, device pointers, length N unless stated. */
typedef struct {
    float* loss_row;     /* l_r (required)                                                     */
    float* lse_d;        /* log-sum-exp of z_d (required: the backward reads it)               */
    float* tail_q;       /* drafter mass outside the row's label tokens (required: backward)   */
    int32_t* argmax_d;   /* greedy drafter token, lowest id on ties (required)                 */
    float* gap_d;        /* top-1 minus top-2 drafter logit (nullable)                         */
    float* weight;       /* omega_r used (required)                                            */
    float* loss_total;   /* [1] L of Eq. 1 times lambda                                        */
    float* weight_sum;   /* [1] sum omega                                                      */
    float* wl_sum;       /* [1] sum omega l (nullable; as in alr_fwd_outputs)                  */
} alr_topk_fwd_outputs;

/* Workspace bytes alr_topk_loss_fwd needs for `p` (0 on invalid params). */
size_t alr_topk_fwd_workspace_size(const alr_params* p);

/*
 * Forward pass of Eq. 1 with the top-k + tail soft cross-entropy:
 *   l_r = -sum_i top_prob_i log q(top_idx_i) - tail_r log tail_q_r,
 *   tail_q_r = 1 - sum_i q(top_idx_i) (the drafter's mass outside the label tokens; a zero
 *   tail contributes nothing), q = softmax(h_d W) over the whole vocabulary.
 * omega_r = weight_in[r] when weight_in is given (e.g. erase weights from alr_erase_weights),
 * else w_k * row_mask[r] (row_mask nullable = ones).  Label tokens must lie in [0, V).
 * tail_q is the drafter's mass outside the label tokens, summed from the same exponentials as
 * the log-sum-exp (the label tokens' own terms taken out as they were added), so its relative
 * precision holds however little mass the drafter leaves outside the label.
 */
int alr_topk_loss_fwd(const alr_params* p, const void* Hd, const void* W, const int32_t* top_idx,
                      const float* top_prob, const float* tail, const float* row_mask,
                      const float* weight_in, const alr_topk_fwd_outputs* out, void* workspace,
                      size_t ws_bytes, void* stream);

/*
 * Gradient of that loss with respect to the drafter logits, recomputed tile by tile:
 *   G[r, v] = c_r (q_v - top_prob_i)            for v = top_idx_i,
 *   G[r, v] = c_r q_v (1 - tail_r / tail_q_r)   for the other tokens,
 * c_r = lambda omega_r / sum omega.  Workspace: alr_logit_grad_workspace_size.
 */
int alr_topk_logit_grad(const alr_params* p, const void* Hd, const void* W,
                        const int32_t* top_idx, const float* top_prob, const float* tail,
                        const float* weight, const float* weight_sum, const float* lse_d,
                        const float* tail_q, void* G, void* workspace, size_t ws_bytes,
                        void* stream);

/*
 * Backward pass of the top-k loss: G as above, dHd = G W^T (overwritten) and, when dW is
 * given, dW += H_d^T G.  Workspace: alr_bwd_workspace_size.
 */
int alr_topk_loss_bwd(const alr_params* p, const void* Hd, const void* W, const int32_t* top_idx,
                      const float* top_prob, const float* tail, const float* weight,
                      const float* weight_sum, const float* lse_d, const float* tail_q,
                      float* dHd, float* dW, void* workspace, size_t ws_bytes, void* stream);

/*
 * Kept logits for the top-k loss (as for the full-vocabulary loss above): the forward also
 * writes z_d = H_d W, and the gradient is then formed from it instead of recomputing the head
 * product.
 *
 * alr_topk_loss_fwd_keep_logits: alr_topk_loss_fwd (same arguments, outputs, workspace and
 * errors, bit-identical outputs) that also writes Zd [N, V] and, for ALR_BF16 inputs, its group
 * references Zd_ref [alr_kept_ref_groups(V), N] in the kept-logit storage described above;
 * caller-owned, 16-byte aligned, overlapping nothing else.
 */
int alr_topk_loss_fwd_keep_logits(const alr_params* p, const void* Hd, const void* W,
                                  const int32_t* top_idx, const float* top_prob, const float* tail,
                                  const float* row_mask, const float* weight_in, void* Zd,
                                  uint16_t* Zd_ref, const alr_topk_fwd_outputs* out,
                                  void* workspace, size_t ws_bytes, void* stream);

/*
 * G of the top-k + tail loss from kept z_d (Zd and, for bf16 inputs, Zd_ref) and the
 * forward's weight, weight_sum, lse_d, tail_q: G = c_r beta_r q outside the row's label tokens and
 * c_r (q - top_prob) at them, q = exp(z_d - lse_d), c_r = lambda omega_r / sum omega,
 * beta_r = 1 - tail_r / tail_q_r.  G [N, V] (bf16 / fp32) may be Zd itself (in place); it must
 * not otherwise overlap Zd.  A row's label tokens must be distinct.  No workspace.
 */
int alr_topk_logit_grad_from_logits(const alr_params* p, const void* Zd, const uint16_t* Zd_ref,
                                    const int32_t* top_idx, const float* top_prob,
                                    const float* tail, const float* weight,
                                    const float* weight_sum, const float* lse_d,
                                    const float* tail_q, void* G, void* stream);

/*
 * Backward of the top-k loss from kept z_d: alr_topk_logit_grad_from_logits into G (may be Zd),
 * dHd = G W^T (overwritten) and, when dW is given, dW += H_d^T G.
 * Workspace: alr_bwd_from_logits_workspace_size.
 */
int alr_topk_loss_bwd_from_logits(const alr_params* p, const void* Hd, const void* W,
                                  const void* Zd, const uint16_t* Zd_ref,
                                  const int32_t* top_idx, const float* top_prob,
                                  const float* tail, const float* weight, const float* weight_sum,
                                  const float* lse_d, const float* tail_q, void* G, float* dHd,
                                  float* dW, void* workspace, size_t ws_bytes, void* stream);

/* ---------------------------------------------------------------------------------------
 * Row-sharded (data-parallel) batches.  Eq. 1 normalises over the whole batch, so when the
 * anchors of one batch are spread over several ranks (App. A: FSDP data parallelism), each
 * rank:
 *   1. runs its forward on its own anchors, with out->wl_sum and out->weight_sum giving its
 *      partial sums (sum omega l, sum omega);
 *   2. sums both scalars over the ranks (an all-reduce of 2 floats, by the caller);
 *   3. calls alr_loss_from_sums on the reduced sums for the batch's L;
 *   4. runs its backward with weight_sum pointing at the REDUCED sum omega (every backward
 *      entry point takes it as a device pointer), so that its G = lambda omega_r / sum omega
 *      (q - p) is its rows' share of the batch gradient;
 *   5. sums dW over the ranks (dW = H_d^T G is a sum over rows: an all-reduce, or a
 *      reduce-scatter when the head is sharded), while each rank keeps its own rows of dH.
 * Accepted-length histograms add up over ranks the same way.
 * ------------------------------------------------------------------------------------- */

/*
 * L = lambda * wl_sum / weight_sum, or 0 when weight_sum = 0 (Eq. 1, from sums the caller
 * reduced over the shards of a batch).  All three are device pointers to one float.
 */
int alr_loss_from_sums(const float* wl_sum, const float* weight_sum, float lambda,
                       float* loss_total, void* stream);

/*
 * Greedy accepted length per anchor (Sec. 3.2: slot k counts only when slots 1..k-1 were
 * accepted; MAT tau = acc + 1, Sec. 4).
 *   argmax_d, argmax_t [A*B] int32; active [A*B] float or NULL (rows with active <= 0 stop
 *   the count).  acc_len [A] int32 output; hist [B+1] int64 or NULL, overwritten with
 *   hist[n] = #{a : acc_len[a] = n}.  A = 0 is allowed: hist is then all zero and no kernel
 *   is launched.
 */
int alr_accept_len(const int32_t* argmax_d, const int32_t* argmax_t, const float* active,
                   int32_t A, int32_t B, int32_t* acc_len, int64_t* hist, void* stream);

/*
 * Slot weights of the erase comparator (Eq. 2) from per-row target statistics.
 *   logp_x   [A*B] float: log p_T of the corpus token row r's label predicts (soft gate).
 *   corpus_tok, argmax_t [A*B] int32 (hard gate; may be NULL when hard == 0).
 *   row_mask [A*B] float or NULL.
 *   weight   [A*B] output: w_k * mask * g, g = prod over earlier rows of the anchor of
 *            exp(logp_x) (soft) or 1[corpus_tok == argmax_t] (hard); 1 for the first row.
 */
int alr_erase_weights(const float* logp_x, const int32_t* corpus_tok, const int32_t* argmax_t,
                      const float* row_mask, int32_t A, int32_t B, float gamma, int32_t hard,
                      float* weight, void* stream);

/*
 * The tensor-core GEMM the backward pass runs on, exposed on its own:
 *   C[M, Nc] = A B   (accumulate == 0)   or   C[M, Nc] += A B   (accumulate != 0)
 * with fp32 C (row-major, leading dimension Nc) and A, B of element type `dtype`:
 *   a_mn == 0: A stored [M, K] row-major;  a_mn != 0: A stored [K, M] row-major.
 *   b_mn == 0: B stored [Nc, K] row-major; b_mn != 0: B stored [K, Nc] row-major.
 * dH_d = G W^T is (a_mn, b_mn) = (0, 0) and dW += H_d^T G is (1, 1).  Row strides must be
 * multiples of 16 bytes and Nc % 4 == 0.
 */
int alr_gemm(int32_t dtype, int32_t a_mn, int32_t b_mn, int32_t accumulate, const void* A,
             const void* B, float* C, int32_t M, int32_t Nc, int32_t K, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* ALR_H */
