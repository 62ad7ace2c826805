// Fused head-GEMM kernels of the slot loss on the sm_103a tensor cores.
//
// Every mode computes logit tiles z = H W for a 128-row block of hidden states and a
// kBN-column tile of the vocabulary head W with tcgen05.mma into tensor memory (fp32
// accumulators) and consumes them on chip; only kModeFwdKeep writes logits to global memory.
//   kModeFwd     z_d = H_d W and z_t = H_t W (both share every W stage): running per-row
//                statistics (online max / sum-exp of both sides, the label-weighted sums behind
//                the soft cross-entropy of Eq. 1, greedy top-2 with lowest-index ties, z_t at
//                the corpus token), one partial record per row, vocabulary split and 64-column
//                group;
//   kModeFwdKeep the same, and both logit tiles are also written to global memory (fp16
//                relative to per-16-column-group references for bf16 inputs, fp32 for fp32
//                inputs) so that the backward need not recompute them;
//   kModeBwd     the same two tiles recomputed: G = lambda omega_r / sum omega (q - p), the
//                gradient of Eq. 1 with respect to z_d;
//   kModeReadout z_t only: log-sum-exp and the k most probable tokens (the label a rollout
//                step keeps, App. A) plus z_t at the corpus token;
//   kModeTopkFwd z_d only: log-sum-exp, greedy top-2 and z_d at the row's k label tokens (the
//                top-k + tail-bin soft CE of Sec. 3.1);
//   kModeTopkBwd z_d only, recomputed: the gradient of that loss;
//   kModeTopkFwdKeep  kModeTopkFwd that also writes z_d (as kModeFwdKeep).
//
// Accumulators: 2 x kBN TMEM columns per tile (single-buffered at kBN = 256).  The dual modes
// hold z_d and z_t of one 128-row block; the single-operand modes (readout, top-k) hold one
// logit tile of each of two row blocks (rows 256 i .. 256 i + 255), so that they too read every
// head tile from shared memory once for two products.
//
// Warp roles: warp 0 issues TMA loads, warp 1 owns tensor memory and issues the MMAs from one
// lane, warps 2.. run the epilogue: warp w reads TMEM lanes 32(w%4)..+31 (one row per thread)
// in 16-column sub-chunks; in the dual modes it takes columns [64 g, 64 g + 64) of both tiles,
// g = (w-2)/4; in the two-row modes columns [128 h, 128 h + 128) of row block b's tile,
// b = ((w-2)/4) % 2, h = (w-2)/8.
// Every pipeline wait is bounded (tc_common.cuh).
//
// Cluster form (Cl = ClusterOf<2>, bf16 inputs, 256-column tiles; instantiated only in
// csrc_cluster/, whose policy supplies the multicast copy and commit): clusters of two CTAs
// take row blocks 2i and 2i + 1 of the same vocabulary split and walk its tiles in lockstep.
// Each CTA loads its own hidden-state tiles and one 128-column half of every head tile,
// multicast into both CTAs' stage, so each W byte leaves L2 once per pair; a stage is refilled
// only after both CTAs' products have read it.  Cl = NoCluster: one CTA per unit.
#pragma once

#include <cuda_fp16.h>

#include "kernels.h"
#include "tc_common.cuh"

namespace alr {
namespace {

constexpr int kBM = 128;                 // rows per tile = TMEM lanes
constexpr int kEpiWarp0 = 2;
constexpr int kEpiBarrier = 1;           // named barrier of the epilogue warps (0 is __syncthreads)
constexpr int kColsPerWarp = 64;
constexpr int kSub = 16;                 // columns per TMEM load / processing step
constexpr int kATileBytes = kBM * 128;   // a 128-row operand over 128 bytes of K
constexpr int kCtrlBytes = 256;
constexpr int kSmemBudget = 227 * 1024;
constexpr int kGStageBytes = 32 * kSub * 2;   // one warp's bf16 G sub-chunk: 32 rows x 16 cols

template <typename Elem>
struct Geo {
  static constexpr int kElem = sizeof(Elem);
  static constexpr int kKE = 128 / kElem;          // K elements per pipeline stage
  static constexpr int kMmaK = 32 / kElem;         // K per MMA instruction
  static constexpr int kChunkMN = 128 / kElem;     // MN elements per 128-byte chunk
  static constexpr uint32_t kChunkBytes = kKE * 128;
  static constexpr bool kTf32 = (kElem == 4);
};

constexpr bool is_fwd(int mode) { return mode == kModeFwd || mode == kModeFwdKeep; }
constexpr bool is_dual(int mode) { return is_fwd(mode) || mode == kModeBwd; }
constexpr bool is_grad(int mode) { return mode == kModeBwd || mode == kModeTopkBwd; }
constexpr bool is_topk_fwd(int mode) { return mode == kModeTopkFwd || mode == kModeTopkFwdKeep; }
// Single-operand modes: one product per row block, two row blocks per unit.
constexpr bool is_two_rows(int mode) { return !is_dual(mode); }
// Modes whose epilogue writes 16-bit [N, V] tiles through shared staging and TMA stores: the
// bf16 gradient (two buffers per warp, double-buffered) and the kept fp16 logits (one buffer
// per logit matrix).  fp32 outputs are written directly.
constexpr bool is_staged(int mode, int elem_bytes) {
  return elem_bytes == 2 && (is_grad(mode) || mode == kModeFwdKeep || mode == kModeTopkFwdKeep);
}

template <int kMode, int kBN, bool kStaged>
struct Shape {
  static constexpr bool kTwoRows = is_two_rows(kMode);
  static constexpr int kATiles = 2;                    // (H_d, H_t) or two row blocks of H
  static constexpr int kBTileBytes = kBN * 128;
  static constexpr int kStageBytes = kATiles * kATileBytes + kBTileBytes;
  static constexpr int kAccCols = kATiles * kBN;       // first tile's columns, then the second's
  static constexpr int kAccBufs = 512 / kAccCols;
  static constexpr int kWarpCols = kTwoRows ? 2 * kColsPerWarp : kColsPerWarp;
  static constexpr int kColGroups = kBN / kWarpCols;   // partial records per row and split
  static constexpr int kEpiWarps = 4 * (kBN / kColsPerWarp);
  static constexpr int kThreads = 32 * (kEpiWarp0 + kEpiWarps);
  static constexpr int kStaging = kStaged ? kEpiWarps * 2 * kGStageBytes : 0;
  static constexpr int kFit = (kSmemBudget - 1024 - kCtrlBytes - kStaging) / kStageBytes;
  static constexpr int kStages = kFit < 4 ? kFit : 4;
  static constexpr size_t kSmem = 1024 + size_t(kStages) * kStageBytes + kStaging + kCtrlBytes;
  // control block: full / empty barrier per stage, full / empty per accumulator buffer, the
  // drain barrier, the TMEM address, the abort word and the epilogue's two tile-ready words
  static_assert((2 * kStages + 2 * kAccBufs + 1) * 8 + 16 <= kCtrlBytes, "control block");
};

// Unit u -> (row block, vocabulary split).  Units go group by group (group_rows row blocks);
// inside a group the row block varies fastest, and the split index is rotated by the group
// number so that every CTA of a static round-robin sees every split size in turn.
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
  const int k = w / gr;
  rb = g * p.group_rows + (w - k * gr);
  vs = (k + g) % p.n_vs;
}

ALR_DEV int split_begin(const LossPlan& p, int vs) {
  return static_cast<int>((static_cast<long long>(vs) * p.n_vt) / p.n_vs);
}

ALR_DEV float f32(uint32_t x) { return __uint_as_float(x); }
ALR_DEV float qnan() { return __int_as_float(0x7fc00000); }

// Load 16 consecutive 32-bit TMEM columns of this warp's 32 lanes (see tmem_ld32).
ALR_DEV void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
      "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15}, [%16];"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
        "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
        "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
      : "r"(taddr));
}

// Maximum of 16 values: seven three-input maxima, depth 3 (max is exact, so any order gives
// the same value).
ALR_DEV float max16(const float (&z)[16]) {
  const float a = max3(z[0], z[1], z[2]), b = max3(z[3], z[4], z[5]);
  const float c = max3(z[6], z[7], z[8]), d = max3(z[9], z[10], z[11]);
  const float e = max3(z[12], z[13], z[14]);
  return max3(max3(a, b, c), max3(d, e, z[15]), -INFINITY);
}

// The sub-chunk's values, with columns at or past nv set to -inf.
template <bool kFull>
ALR_DEV void load_masked(float (&z)[16], const uint32_t (&r)[16], int nv) {
#pragma unroll
  for (int j = 0; j < kSub; ++j) z[j] = (kFull || j < nv) ? f32(r[j]) : -INFINITY;
}

// (s, c) <- (s, c) * sc + x with the rounding error of the addition moved into c (Knuth's
// TwoSum, branch-free: s + c holds the sum to about twice fp32 precision).  The error of the
// product s * sc (sc < 1 only when the running maximum moves) is not kept.
ALR_DEV void sum2_scaled(float& s, float& c, float sc, float x) {
  const float t = s * sc;
  const float y = t + x;
  const float xb = y - t;
  const float e = (t - (y - xb)) + (x - xb);
  s = y;
  c = fmaf(c, sc, e);
}

// The exponent every column gets relative to the reference m is fma(z, log2 e, -m log2 e),
// which at z = m is not 0 but the rounding residual of m log2 e (exactly representable, up to
// ~4e-6 at |m| ~ 40): every exponential summed against m carries the factor 2^r.  The merge
// divides it out, so that log S and the log-probabilities taken from it keep their precision.
ALR_DEV float exp_residual(float m) { return fmaf(m, kLog2e, -m * kLog2e); }

// Online log-sum-exp: move the reference from m to max(m, cm) and add the sub-chunk's
// exp(z - ref) (masked -inf columns add 0) to the compensated sum (s, c).  Even and odd
// columns are summed in the two lanes of packed registers; each lane's exponential equals the
// scalar ex2(fmaf(z, kLog2e, -m * kLog2e)) of its column.  Returns the factor the old sums
// were rescaled by.
ALR_DEV float lse_update(float& m, float& s, float& c, const float (&z)[16], float cm) {
  const float nm = fmaxf(m, cm);
  const float sc = ex2((m - nm) * kLog2e);
  const float b = -nm * kLog2e;
  const uint64_t l2e = f2_pack(kLog2e, kLog2e), b2 = f2_pack(b, b);
  uint64_t r = f2_pack(0.f, 0.f);
#pragma unroll
  for (int j = 0; j < kSub; j += 2)
    r = f2_add(r, f2_ex2(f2_fma(f2_pack(z[j], z[j + 1]), l2e, b2)));
  float r0, r1;
  f2_unpack(r, r0, r1);
  sum2_scaled(s, c, sc, r0 + r1);
  m = nm;
  return sc;
}

// Greedy top-2 with lowest-index ties, given the sub-chunk maximum cm.  Columns reach a
// thread in increasing order, so an equal later value never takes the lead.
ALR_DEV int first_at(const float (&z)[16], float cm) {
  int jj = kSub - 1;
#pragma unroll
  for (int j = kSub - 1; j >= 0; --j) jj = (z[j] == cm) ? j : jj;
  return jj;
}

// top2_update for a sub-chunk whose new leader (cm > best) sits at column jj.
ALR_DEV void top2_lead(float& best, float& sec, int& idx, const float (&z)[16], float cm, int jj,
                       int v0) {
  float c2 = -INFINITY;
#pragma unroll
  for (int j = 0; j < kSub; ++j) c2 = fmaxf(c2, j == jj ? -INFINITY : z[j]);
  sec = fmaxf(best, c2);
  best = cm;
  idx = v0 + jj;
}

ALR_DEV void top2_update(float& best, float& sec, int& idx, const float (&z)[16], float cm,
                         int v0) {
  sec = fmaxf(sec, fminf(cm, best));
  if (cm > best) top2_lead(best, sec, idx, z, cm, first_at(z, cm), v0);  // a new leader
}

// Insert (v, i) into a list sorted by value descending; an equal value stays below the
// entries already there (they came from lower columns).
ALR_DEV void topk_insert(float (&t)[kTopK], int (&ti)[kTopK], float v, int i) {
  t[kTopK - 1] = v;
  ti[kTopK - 1] = i;
#pragma unroll
  for (int k = kTopK - 1; k > 0; --k) {
    const bool up = t[k] > t[k - 1];
    const float a = t[k], b = t[k - 1];
    const int ia = ti[k], ib = ti[k - 1];
    t[k - 1] = up ? a : b;
    t[k] = up ? b : a;
    ti[k - 1] = up ? ia : ib;
    ti[k] = up ? ib : ia;
  }
}

// Running statistics of one row over the columns one thread sees (full-vocabulary forward).
// best_x is both the greedy top-1 and the online-softmax reference of side x; s_x sums
// exp(z_x - best_x), with the rounding error of its additions kept in c_x: once the row's
// maximum is in, the sum sits at 1 + small and each added term would otherwise lose up to half
// a unit of 1, while the small part is what a near-zero loss or entropy is made of.
// u and w sum exp(z_t - best_t) * (z_d - best_d) and * (z_t - best_t): measured from the
// running maxima, the terms that carry weight are near zero, so these sums stay small and
// precise when the logits are large, and the soft CE comes out as log s_d - u / s_t, a sum of
// two non-negative terms, instead of a difference of two numbers of the logits' size.
struct RowStats {
  float best_d, sec_d, s_d, c_d, best_t, sec_t, s_t, c_t, u, w, zx;
  int i_d, i_t;
};

ALR_DEV void stats_init(RowStats& st) {
  st.best_d = st.sec_d = st.best_t = st.sec_t = -INFINITY;
  st.s_d = st.s_t = st.c_d = st.c_t = st.u = st.w = 0.f;
  st.i_d = st.i_t = 0x7fffffff;
  st.zx = qnan();
}

// Fold one 16-column sub-chunk (nv valid columns) into the full-vocabulary statistics.
// cd, ct: the sub-chunk's maxima of z_d and z_t (over its valid columns), returned.
template <bool kFull>
ALR_DEV void stats_sub(RowStats& st, const uint32_t (&rd)[16], const uint32_t (&rt)[16], int v0,
                       int nv, int x, float& cd, float& ct) {
  float zd[16], zt[16];
  load_masked<kFull>(zd, rd, nv);
  load_masked<kFull>(zt, rt, nv);
  cd = max16(zd);
  ct = max16(zt);
  const float nbt = fmaxf(st.best_t, ct), nbd = fmaxf(st.best_d, cd);
  const float bt = -nbt * kLog2e, bd = -nbd * kLog2e;
  // per column: T = (z_t - nbt) log2 e, D = (z_d - nbd) log2 e, E = 2^T; sums of E, 2^D,
  // E D and E T (the last two in log2 units, converted once below)
  float s0 = 0.f, s1 = 0.f, d0 = 0.f, d1 = 0.f, u0 = 0.f, u1 = 0.f, w0 = 0.f, w1 = 0.f;
  if constexpr (kFull) {
    // even / odd columns in the two lanes of packed registers
    const uint64_t l2e = f2_pack(kLog2e, kLog2e), bt2 = f2_pack(bt, bt), bd2 = f2_pack(bd, bd);
    uint64_t S = f2_pack(0.f, 0.f), SD = S, U = S, Wt = S;
#pragma unroll
    for (int j = 0; j < kSub; j += 2) {
      const uint64_t T = f2_fma(f2_pack(zt[j], zt[j + 1]), l2e, bt2);
      const uint64_t D = f2_fma(f2_pack(zd[j], zd[j + 1]), l2e, bd2);
      const uint64_t E = f2_ex2(T);
      S = f2_add(S, E);
      SD = f2_add(SD, f2_ex2(D));
      U = f2_fma(E, D, U);
      Wt = f2_fma(E, T, Wt);
    }
    f2_unpack(S, s0, s1);
    f2_unpack(SD, d0, d1);
    f2_unpack(U, u0, u1);
    f2_unpack(Wt, w0, w1);
  } else {
#pragma unroll
    for (int j = 0; j < kSub; ++j) {
      if (j < nv) {
        const float T = fmaf(zt[j], kLog2e, bt), D = fmaf(zd[j], kLog2e, bd);
        const float e = ex2(T);
        s0 += e;
        d0 += ex2(D);
        u0 = fmaf(e, D, u0);
        w0 = fmaf(e, T, w0);
      }
    }
  }
  // u, w: move to the new references (skipped while nothing has been summed: the old
  // reference is still -inf), rescale, add this sub-chunk
  const bool any = st.s_t > 0.f;
  const float u_sh = any ? fmaf(st.best_d - nbd, st.s_t + st.c_t, st.u) : 0.f;
  const float w_sh = any ? fmaf(st.best_t - nbt, st.s_t + st.c_t, st.w) : 0.f;
  const float sct = ex2((st.best_t - nbt) * kLog2e);
  const float scd = ex2((st.best_d - nbd) * kLog2e);
  st.u = fmaf(u_sh, sct, (u0 + u1) * kLn2);
  st.w = fmaf(w_sh, sct, (w0 + w1) * kLn2);
  sum2_scaled(st.s_t, st.c_t, sct, s0 + s1);
  sum2_scaled(st.s_d, st.c_d, scd, d0 + d1);
  // greedy top-2 of both sides (moves best_d / best_t to the new maxima nbd / nbt)
  top2_update(st.best_d, st.sec_d, st.i_d, zd, cd, v0);
  top2_update(st.best_t, st.sec_t, st.i_t, zt, ct, v0);
  const int xr = x - v0;
  if (xr >= 0 && xr < (kFull ? kSub : nv)) {
#pragma unroll
    for (int j = 0; j < kSub; ++j)
      if (j == xr) st.zx = zt[j];
  }
}

ALR_DEV uint32_t pack_bf16x2(float a, float b) {
  __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<uint32_t*>(&h);
}

// fp16 pair of (a - ref, b - ref), rounded to nearest (one packed subtraction for the pair).
ALR_DEV uint32_t pack_f16x2(uint32_t a, uint32_t b, uint64_t ref2) {
  float x, y;
  f2_unpack(f2_sub(f2_pack(f32(a), f32(b)), ref2), x, y);
  __half2 h = __floats2half2_rn(x, y);
  return *reinterpret_cast<uint32_t*>(&h);
}

// Reference of a kept 16-column group from its maximum cm: cm rounded up to fp16, so that every
// kept value z - ref is at most 0 and its fp16 rounding error, at most 2^-11 (ref - z), is small
// exactly for the logits that dominate the softmax.
ALR_DEV __half group_ref(float cm) { return __float2half_ru(cm); }

// Store the reference of the group at columns v0.. of `row`: references are group-major,
// [groups, N], so the 32 lanes of a warp (32 consecutive rows) write 64 contiguous bytes.
ALR_DEV void store_ref(uint16_t* ref, int n, int row, int v0, __half h) {
  ref[size_t(v0 / kSub) * size_t(n) + size_t(row)] = __half_as_ushort(h);
}

// One lane's 16 logits relative to `ref`, as two 16-byte fp16 vectors.
ALR_DEV void pack_rel(uint4* b, const uint32_t (&r)[16], float ref_value) {
  const uint64_t ref = f2_pack(ref_value, ref_value);
  b[0] = make_uint4(pack_f16x2(r[0], r[1], ref), pack_f16x2(r[2], r[3], ref),
                    pack_f16x2(r[4], r[5], ref), pack_f16x2(r[6], r[7], ref));
  b[1] = make_uint4(pack_f16x2(r[8], r[9], ref), pack_f16x2(r[10], r[11], ref),
                    pack_f16x2(r[12], r[13], ref), pack_f16x2(r[14], r[15], ref));
}

// Keep one warp's 32 x 16 sub-chunk of z_d and z_t, fp16 relative to each row's group
// references (bf16 inputs): each lane packs its row into the warp's two staging buffers, then
// one lane issues a TMA store per matrix (rows past N and columns past V are clipped by the
// tensor maps).  The stores of the previous sub-chunk must have finished reading the buffers.
ALR_DEV void keep_logits_staged(const uint32_t (&rd)[16], const uint32_t (&rt)[16], float ref_d,
                                float ref_t, uint8_t* my_stage, const CUtensorMap* tm_zd,
                                const CUtensorMap* tm_zt, int v0, int row0, int lane) {
  if (lane == 0) tma_store_wait_read_all();
  __syncwarp();
  pack_rel(reinterpret_cast<uint4*>(my_stage + lane * 32), rd, ref_d);
  pack_rel(reinterpret_cast<uint4*>(my_stage + kGStageBytes + lane * 32), rt, ref_t);
  fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0) {
    tma_store_2d(tm_zd, my_stage, v0, row0);
    tma_store_2d(tm_zt, my_stage + kGStageBytes, v0, row0);
    tma_store_commit();
  }
}

// Keep one warp's 32 x 16 sub-chunk of z_d alone, fp16 relative to the group references (bf16
// inputs), through the warp's two staging buffers in turn (the store issued from a buffer two
// sub-chunks ago must have read it).
ALR_DEV void keep_one_staged(const uint32_t (&r)[16], float ref, uint8_t* my_stage,
                             uint32_t& n_stores, const CUtensorMap* tm, int v0, int row0,
                             int lane) {
  uint8_t* buf = my_stage + (n_stores & 1u) * kGStageBytes;
  if (lane == 0) tma_store_wait_read_le1();
  __syncwarp();
  pack_rel(reinterpret_cast<uint4*>(buf + lane * 32), r, ref);
  fence_proxy_async_smem();
  __syncwarp();
  if (lane == 0) {
    tma_store_2d(tm, buf, v0, row0);
    tma_store_commit();
  }
  ++n_stores;
}

// Keep one thread's 16 fp32 logits (fp32 inputs) with direct streaming stores: columns v0..
// of its row, nv of them valid (8 or 16, as V is a multiple of 8); row * V + v0 is a multiple
// of 8, so every vector store is aligned.
ALR_DEV void keep_logits_f32(const uint32_t (&r)[16], void* base, size_t off, int nv) {
  uint4* p = reinterpret_cast<uint4*>(static_cast<float*>(base) + off);
#pragma unroll
  for (int i = 0; i < 4; ++i)
    if (4 * i < nv) __stcs(p + i, make_uint4(r[4 * i], r[4 * i + 1], r[4 * i + 2], r[4 * i + 3]));
}

// Warp-uniform bounded wait: lane 0 waits and broadcasts the outcome.
ALR_DEV bool warp_wait(uint64_t* bar, uint32_t parity, const AbortFlag& ab) {
  int ok = 1;
  if ((threadIdx.x & 31) == 0) ok = mbar_wait(bar, parity, ab) ? 1 : 0;
  return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

// Write one warp's 32 x 16 sub-chunk of G: bf16 through its shared staging buffer and a TMA
// store (the buffer used two stores ago must have been read first), fp32 directly.
template <typename Elem, bool kStaged>
ALR_DEV void store_g(const float (&g)[16], uint8_t* my_stage, uint32_t& n_stores,
                     const CUtensorMap* tm_g, Elem* grow, int v0, int row0, bool row_ok, int V,
                     int lane) {
  if constexpr (kStaged) {
    uint8_t* buf = my_stage + (n_stores & 1u) * kGStageBytes;
    if (lane == 0) tma_store_wait_read_le1();
    __syncwarp();
    uint4 a, b;
    a.x = pack_bf16x2(g[0], g[1]);
    a.y = pack_bf16x2(g[2], g[3]);
    a.z = pack_bf16x2(g[4], g[5]);
    a.w = pack_bf16x2(g[6], g[7]);
    b.x = pack_bf16x2(g[8], g[9]);
    b.y = pack_bf16x2(g[10], g[11]);
    b.z = pack_bf16x2(g[12], g[13]);
    b.w = pack_bf16x2(g[14], g[15]);
    *reinterpret_cast<uint4*>(buf + lane * 32) = a;
    *reinterpret_cast<uint4*>(buf + lane * 32 + 16) = b;
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
      tma_store_2d(tm_g, buf, v0, row0);
      tma_store_commit();
    }
    ++n_stores;
  } else if (row_ok) {
#pragma unroll
    for (int i = 0; i < kSub / 4; ++i) {
      if (v0 + 4 * i < V)
        *reinterpret_cast<float4*>(grow + v0 + 4 * i) =
            make_float4(g[4 * i], g[4 * i + 1], g[4 * i + 2], g[4 * i + 3]);
    }
  }
}

// kWMN: the head tile is read MN-major straight from W [d, V] (bf16), or K-major from a
// transposed copy W^T [V, d] (fp32 inputs, whose tf32 products take K-major operands only).
// tm_g: the bf16 G store map (gradient modes) or the z_d store map (kModeFwdKeep, bf16);
// tm_g2: the z_t store map (kModeFwdKeep, bf16).
// One block per SM.  With 18 warps (256-column tiles) two of the four SM sub-partitions hold
// five warps in their 16K-register files, which caps a thread at 96 registers.
template <typename Elem, int kMode, bool kWMN, int kBN, class Cl>
__global__ void __launch_bounds__(Shape<kMode, kBN, is_staged(kMode, sizeof(Elem))>::kThreads, 1)
    loss_gemm_kernel(const __grid_constant__ CUtensorMap tm_a0,
                     const __grid_constant__ CUtensorMap tm_a1,
                     const __grid_constant__ CUtensorMap tm_w,
                     const __grid_constant__ CUtensorMap tm_g,
                     const __grid_constant__ CUtensorMap tm_g2, const LossArgs args) {
  using G = Geo<Elem>;
  constexpr bool kDual = is_dual(kMode);
  constexpr bool kStaged = is_staged(kMode, sizeof(Elem));
  using S = Shape<kMode, kBN, kStaged>;
  constexpr int kStages = S::kStages;
  constexpr bool kMc = Cl::kCtas > 1;
  static_assert(Cl::kCtas == 1 || Cl::kCtas == 2, "single CTAs or pairs of CTAs");

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align_1024(smem_raw);
  uint8_t* stage_mem = smem;
  uint8_t* gstage = smem + kStages * S::kStageBytes;
  uint64_t* full_bar = reinterpret_cast<uint64_t*>(gstage + S::kStaging);
  uint64_t* empty_bar = full_bar + kStages;
  uint64_t* tfull_bar = empty_bar + kStages;
  uint64_t* tempty_bar = tfull_bar + S::kAccBufs;
  uint64_t* drain_bar = tempty_bar + S::kAccBufs;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(drain_bar + 1);
  volatile int* abort_word = reinterpret_cast<volatile int*>(tmem_slot + 1);
  volatile int* tile_ready = abort_word + 1;   // [2], alternating by accumulator tile

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const LossPlan& P = args.plan;
  const AbortFlag ab{abort_word, args.status};
  // kMc: units are handed out per cluster (P.n_rb counts row-block pairs) and CTA `rank`
  // takes row block 2 rb + rank
  static_assert(!kMc || (kWMN && kBN == 256), "multicast form: bf16 head, 256-column tiles");
  const int rank = kMc ? int(cluster_ctarank()) : 0;
  const int u0 = kMc ? int(cluster_id_x()) : int(blockIdx.x);
  const int u_step = kMc ? int(n_clusters_x()) : int(gridDim.x);

  if (threadIdx.x == 0) {
    for (int i = 0; i < kStages; ++i) {
      mbar_init(&full_bar[i], 1);
      mbar_init(&empty_bar[i], kMc ? 2 : 1);
    }
    for (int i = 0; i < S::kAccBufs; ++i) {
      mbar_init(&tfull_bar[i], 1);
      mbar_init(&tempty_bar[i], S::kEpiWarps);
    }
    mbar_init(drain_bar, 1);
    *abort_word = 0;
    fence_mbar_init();
  }
  if (threadIdx.x == 32) {
    tma_prefetch_desc(&tm_a0);
    if (kDual) tma_prefetch_desc(&tm_a1);  // the two-row modes read both tiles from tm_a0
    tma_prefetch_desc(&tm_w);
    if (kStaged) tma_prefetch_desc(&tm_g);
    if (kStaged && kMode == kModeFwdKeep) tma_prefetch_desc(&tm_g2);
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
  const int n_kb = (P.d + G::kKE - 1) / G::kKE;

  if (warp == 0) {
    // ------------------------------------------------------------- TMA producer ---
    if (lane == 0) {
      int stage = 0;
      uint32_t phase = 0, armed = 0, armed_par = 0;
      bool ok = true;
      for (int u = u0; ok && u < P.n_units; u += u_step) {
        int rb, vs;
        decode_unit(P, u, rb, vs);
        if (kMc) rb = 2 * rb + rank;
        const int vt1 = split_begin(P, vs + 1);
        for (int vt = split_begin(P, vs); ok && vt < vt1; ++vt) {
          for (int kb = 0; kb < n_kb; ++kb) {
            if (!mbar_wait(&empty_bar[stage], phase ^ 1, ab)) {
              ok = false;
              break;
            }
            if (args.withhold_first_stage && u == u0 && vt == split_begin(P, vs) &&
                kb == 0) {
              // test hook: leave this stage empty, so the MMA issuer's bounded wait on it runs
              // out and the whole CTA takes the timeout path
              if (++stage == kStages) {
                stage = 0;
                phase ^= 1;
              }
              continue;
            }
            uint8_t* sb = stage_mem + stage * S::kStageBytes;
            uint8_t* sw = sb + S::kATiles * kATileBytes;
            mbar_arrive_expect_tx(&full_bar[stage], S::kStageBytes);
            if constexpr (kDual) {
              tma_load_2d(sb, &tm_a0, &full_bar[stage], kb * G::kKE, rb * kBM);
              tma_load_2d(sb + kATileBytes, &tm_a1, &full_bar[stage], kb * G::kKE, rb * kBM);
            } else {  // row blocks 2 rb and 2 rb + 1
              tma_load_2d(sb, &tm_a0, &full_bar[stage], kb * G::kKE, 2 * rb * kBM);
              tma_load_2d(sb + kATileBytes, &tm_a0, &full_bar[stage], kb * G::kKE,
                          (2 * rb + 1) * kBM);
            }
            if constexpr (kMc) {
              // this CTA's half of the head tile, into both CTAs' stage
              constexpr int kHalfChunks = kBN / G::kChunkMN / 2;
#pragma unroll
              for (int c = 0; c < kHalfChunks; ++c) {
                const int cc = rank * kHalfChunks + c;
                Cl::load_mc(sw + cc * G::kChunkBytes, &tm_w, &full_bar[stage],
                               vt * kBN + cc * G::kChunkMN, kb * G::kKE, 0x3);
              }
            } else if constexpr (kWMN) {
#pragma unroll
              for (int c = 0; c < kBN / G::kChunkMN; ++c)
                tma_load_2d(sw + c * G::kChunkBytes, &tm_w, &full_bar[stage],
                            vt * kBN + c * G::kChunkMN, kb * G::kKE);
            } else {
              tma_load_2d(sw, &tm_w, &full_bar[stage], kb * G::kKE, vt * kBN);
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
      for (int u = u0; ok && u < P.n_units; u += u_step) {
        int rb, vs;
        decode_unit(P, u, rb, vs);
        if (kMc) rb = 2 * rb + rank;
        const int vt1 = split_begin(P, vs + 1);
        for (int vt = split_begin(P, vs); ok && vt < vt1; ++vt) {
          if (!mbar_wait(&tempty_bar[abuf], aphase ^ 1, ab)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d_acc = tmem_base + uint32_t(abuf * S::kAccCols);
          for (int kb = 0; kb < n_kb; ++kb) {
            if (!mbar_wait(&full_bar[stage], phase, ab)) {
              ok = false;
              break;
            }
            tc_fence_after();
            const uint32_t sa = smem_u32(stage_mem + stage * S::kStageBytes);
            const uint32_t swb = sa + S::kATiles * kATileBytes;
#pragma unroll
            for (int kk = 0; kk < G::kKE / G::kMmaK; ++kk) {
              const uint64_t bd =
                  kWMN ? sdesc_sw128(swb + kk * G::kMmaK * 128, G::kChunkBytes, 1024)
                       : sdesc_sw128(swb + kk * 32, 16, 1024);
              const uint32_t acc = (kb > 0 || kk > 0) ? 1u : 0u;
              mma_issue<G::kTf32>(d_acc, sdesc_sw128(sa + kk * 32, 16, 1024), bd, idesc, acc);
              mma_issue<G::kTf32>(d_acc + kBN, sdesc_sw128(sa + kATileBytes + kk * 32, 16, 1024),
                                  bd, idesc, acc);
            }
            if constexpr (kMc) Cl::commit_mc(&empty_bar[stage], 0x3);
            else mma_commit(&empty_bar[stage]);
            if (++stage == kStages) {
              stage = 0;
              phase ^= 1;
            }
          }
          if (!ok) break;
          mma_commit(&tfull_bar[abuf]);
          if (++abuf == S::kAccBufs) {
            abuf = 0;
            aphase ^= 1;
          }
        }
      }
      // all products issued by this thread complete before tensor memory is released
      mma_commit(drain_bar);
      mbar_wait_drain(drain_bar, 0);
    }
  } else {
    // -------------------------------------------------------------------- epilogue ---
    // a warp may only read the TMEM lane quarter warp % 4; each run of four consecutive
    // epilogue warps covers the four quarters
    const int q = warp & 3;
    const int e = (warp - kEpiWarp0) >> 2;                  // which run of four warps
    const int blk = S::kTwoRows ? (e & 1) : 0;              // row block of the unit's pair
    const int cg = S::kTwoRows ? (e >> 1) : e;              // column group of the tile
    const int row_in_tile = q * 32 + lane;
    const uint32_t lane_addr = tmem_base + (uint32_t(q * 32) << 16) + uint32_t(blk * kBN) +
                               uint32_t(cg * S::kWarpCols);
    uint8_t* my_stage = gstage + (warp - kEpiWarp0) * 2 * kGStageBytes;
    uint32_t n_stores = 0;
    int abuf = 0;
    uint32_t aphase = 0;
    bool ok = true;
    for (int u = u0; ok && u < P.n_units; u += u_step) {
      int rb, vs;
      decode_unit(P, u, rb, vs);
      if (kMc) rb = 2 * rb + rank;
      if (S::kTwoRows) rb = 2 * rb + blk;
      const int vt1 = split_begin(P, vs + 1);
      const int row = rb * kBM + row_in_tile;
      const bool row_ok = row < P.N;
      const size_t part = size_t(vs * S::kColGroups + cg);
      const size_t fs = size_t(P.n_parts) * P.N;

      // ---- per-row state for this unit ----
      RowStats st;                       // forward modes
      float m = -INFINITY, s = 0.f, sc = 0.f;   // single-operand log-sum-exp state (s + sc)
      float s_in = 0.f;                  // top-k forward: the label tokens' part of s
      float best = -INFINITY, sec = -INFINITY, zx = qnan();
      int bidx = 0x7fffffff, x = -1;
      float tk[kTopK];                   // readout: k best values / top-k forward: z_d at labels
      int ti[kTopK];                     // readout: their ids / top-k modes: label tokens
      float tp[kTopK];                   // top-k backward: label probabilities
      float ad = 0.f, at = 0.f, cw = 0.f, beta = 1.f;
#pragma unroll
      for (int i = 0; i < kTopK; ++i) {
        tk[i] = kMode == kModeReadout ? -INFINITY : qnan();
        ti[i] = kMode == kModeReadout ? 0x7fffffff : -1;
        tp[i] = 0.f;
      }
      if constexpr (is_fwd(kMode)) stats_init(st);
      if constexpr (is_fwd(kMode) || kMode == kModeReadout)
        x = (args.corpus_tok != nullptr && row_ok) ? args.corpus_tok[row] : -1;
      if constexpr (is_topk_fwd(kMode) || kMode == kModeTopkBwd) {
        if (row_ok) {
#pragma unroll
          for (int i = 0; i < kTopK; ++i) ti[i] = args.top_idx[size_t(row) * kTopK + i];
        }
      }
      if constexpr (is_grad(kMode)) {
        if (row_ok) {
          ad = -args.lse_d[row] * kLog2e;
          const float ws = *args.weight_sum;
          cw = ws > 0.f ? args.lam * args.weight[row] / ws : 0.f;
          if constexpr (kMode == kModeBwd) {
            at = -args.lse_t[row] * kLog2e;
          } else {
            const float tl = args.tail[row];
            beta = tl > 0.f ? 1.f - tl / args.tail_q[row] : 1.f;
#pragma unroll
            for (int i = 0; i < kTopK; ++i) tp[i] = args.top_prob[size_t(row) * kTopK + i];
          }
        }
      }
      Elem* grow = static_cast<Elem*>(args.G) + size_t(row_ok ? row : 0) * size_t(P.V);

      for (int vt = split_begin(P, vs); vt < vt1; ++vt) {
        // The first epilogue warp waits for the accumulator and posts the outcome; the other
        // warps wait in a named barrier, descheduled, instead of each polling the mbarrier.
        // All epilogue warps pass the same barriers in the same order and follow the one
        // posted outcome, so they leave the loop together.  The word alternates between two
        // slots (consecutive tiles differ in the buffer's parity, or in the phase when there
        // is one buffer): a slot is rewritten only two barriers later, after every warp has
        // read it.
        volatile int* ready = tile_ready + (S::kAccBufs == 1 ? int(aphase) : (abuf & 1));
        if (warp == kEpiWarp0) {
          const bool w = warp_wait(&tfull_bar[abuf], aphase, ab);
          if (lane == 0) *ready = w ? 1 : 0;
          __syncwarp();
        }
        named_bar_sync(kEpiBarrier, S::kEpiWarps * 32);
        if (*ready == 0) {
          ok = false;
          break;
        }
        tc_fence_after();
        const uint32_t tb = lane_addr + uint32_t(abuf * S::kAccCols);
        const int vbase = vt * kBN + cg * S::kWarpCols;
#pragma unroll 1
        for (int c = 0; c < S::kWarpCols / kSub; ++c) {
          uint32_t r0[16], r1[16];
          tmem_ld16(tb + c * kSub, r0);
          if constexpr (kDual) tmem_ld16(tb + kBN + c * kSub, r1);
          tmem_ld_wait();
          reg_fence(r0);
          if constexpr (kDual) reg_fence(r1);
          const int v0 = vbase + c * kSub;
          if (v0 >= P.V) continue;   // warp-uniform: the whole sub-chunk is past the vocabulary
          const int nv = min(kSub, P.V - v0);

          if constexpr (is_fwd(kMode)) {
            float cd, ct;   // the sub-chunk's maxima, which also give the kept references
            if (nv == kSub) stats_sub<true>(st, r0, r1, v0, kSub, x, cd, ct);
            else stats_sub<false>(st, r0, r1, v0, nv, x, cd, ct);
            if constexpr (kMode == kModeFwdKeep) {
              if constexpr (kStaged) {
                const __half hd = group_ref(cd), ht = group_ref(ct);
                if (row_ok) {
                  store_ref(args.zd_ref, P.N, row, v0, hd);
                  store_ref(args.zt_ref, P.N, row, v0, ht);
                }
                keep_logits_staged(r0, r1, __half2float(hd), __half2float(ht), my_stage, &tm_g,
                                   &tm_g2, v0, rb * kBM + q * 32, lane);
              } else if (row_ok) {
                const size_t off = size_t(row) * size_t(P.V) + size_t(v0);
                keep_logits_f32(r0, args.zd_out, off, nv);
                keep_logits_f32(r1, args.zt_out, off, nv);
              }
            }
          } else if constexpr (kMode == kModeReadout || is_topk_fwd(kMode)) {
            float z[16];
            if (nv == kSub) load_masked<true>(z, r0, nv);
            else load_masked<false>(z, r0, nv);
            const float cm = max16(z);
            if constexpr (kMode == kModeTopkFwdKeep) {
              if constexpr (kStaged) {
                const __half h = group_ref(cm);
                if (row_ok) store_ref(args.zd_ref, P.N, row, v0, h);
                keep_one_staged(r0, __half2float(h), my_stage, n_stores, &tm_g, v0,
                                rb * kBM + q * 32, lane);
              } else if (row_ok) {
                keep_logits_f32(r0, args.zd_out, size_t(row) * size_t(P.V) + size_t(v0), nv);
              }
            }
            const float resc = lse_update(m, s, sc, z, cm);
            if constexpr (kMode == kModeReadout) {
              const int xr = x - v0;
              if (xr >= 0 && xr < nv) {
#pragma unroll
                for (int j = 0; j < kSub; ++j)
                  if (j == xr) zx = z[j];
              }
              // the sub-chunk's entrants, largest first (equal values lowest column first, so
              // each goes below the equal ones already listed): one pass per entrant instead
              // of one per column
              float c = cm;
#pragma unroll 1
              while (c > tk[kTopK - 1]) {
                int jj = kSub - 1;
#pragma unroll
                for (int j = kSub - 1; j >= 0; --j) jj = (z[j] == c) ? j : jj;
                topk_insert(tk, ti, c, v0 + jj);
#pragma unroll
                for (int j = 0; j < kSub; ++j) z[j] = (j == jj) ? -INFINITY : z[j];
                c = max16(z);
              }
            } else {
              top2_update(best, sec, bidx, z, cm, v0);
              // the label tokens' exponentials, the very terms lse_update added to s, so that
              // s - s_in is the drafter's mass outside the label (the tail bin's q) without a
              // cancellation between separately rounded sums
              s_in *= resc;
              bool hit = false;
#pragma unroll
              for (int i = 0; i < kTopK; ++i) hit |= unsigned(ti[i] - v0) < unsigned(nv);
              if (hit) {
                const float b = -m * kLog2e;
#pragma unroll
                for (int i = 0; i < kTopK; ++i) {
                  const int rel = ti[i] - v0;
#pragma unroll
                  for (int j = 0; j < kSub; ++j)
                    if (j == rel) {
                      tk[i] = z[j];
                      s_in += ex2(fmaf(z[j], kLog2e, b));
                    }
                }
              }
            }
          } else {   // gradient modes
            float g[16];
            const uint64_t l2e = f2_pack(kLog2e, kLog2e), ad2 = f2_pack(ad, ad);
            if constexpr (kMode == kModeBwd) {
              const uint64_t at2 = f2_pack(at, at), cw2 = f2_pack(cw, cw);
#pragma unroll
              for (int j = 0; j < kSub; j += 2) {
                const uint64_t q2 = f2_ex2(f2_fma(f2_pack(f32(r0[j]), f32(r0[j + 1])), l2e, ad2));
                const uint64_t p2 = f2_ex2(f2_fma(f2_pack(f32(r1[j]), f32(r1[j + 1])), l2e, at2));
                f2_unpack(f2_mul(cw2, f2_sub(q2, p2)), g[j], g[j + 1]);
              }
            } else {
              float qv[16];
              const float cb = cw * beta;
              const uint64_t cb2 = f2_pack(cb, cb);
#pragma unroll
              for (int j = 0; j < kSub; j += 2) {
                const uint64_t q2 = f2_ex2(f2_fma(f2_pack(f32(r0[j]), f32(r0[j + 1])), l2e, ad2));
                f2_unpack(q2, qv[j], qv[j + 1]);
                f2_unpack(f2_mul(cb2, q2), g[j], g[j + 1]);
              }
              bool hit = false;
#pragma unroll
              for (int i = 0; i < kTopK; ++i) hit |= unsigned(ti[i] - v0) < unsigned(nv);
              if (hit) {   // the row's label tokens in this sub-chunk: c (q - prob)
#pragma unroll
                for (int i = 0; i < kTopK; ++i) {
                  const int rel = ti[i] - v0;
#pragma unroll
                  for (int j = 0; j < kSub; ++j)
                    if (j == rel) g[j] = cw * (qv[j] - tp[i]);
                }
              }
            }
            store_g<Elem, kStaged>(g, my_stage, n_stores, &tm_g, grow, v0, rb * kBM + q * 32,
                                   row_ok, P.V, lane);
          }
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&tempty_bar[abuf]);
        if (++abuf == S::kAccBufs) {
          abuf = 0;
          aphase ^= 1;
        }
      }

      // ---- per-row partial record at the end of the unit ----
      if (ok && row_ok) {
        float* o = args.part + part * P.N + row;
        if constexpr (is_fwd(kMode)) {
          o[kPMd * fs] = st.best_d;
          o[kPSd * fs] = st.s_d;
          o[kPSdLo * fs] = st.c_d;
          o[kPMt * fs] = st.best_t;
          o[kPSt * fs] = st.s_t;
          o[kPStLo * fs] = st.c_t;
          o[kPU * fs] = st.u;
          o[kPW * fs] = st.w;
          o[kPBd * fs] = st.best_d;
          o[kPId * fs] = __int_as_float(st.i_d);
          o[kPSecd * fs] = st.sec_d;
          o[kPBt * fs] = st.best_t;
          o[kPIt * fs] = __int_as_float(st.i_t);
          o[kPSect * fs] = st.sec_t;
          o[kPZx * fs] = st.zx;
        } else if constexpr (kMode == kModeReadout) {
          o[kRM * fs] = m;
          o[kRS * fs] = s;
          o[kRSLo * fs] = sc;
          o[kRR * fs] = exp_residual(m);
#pragma unroll
          for (int i = 0; i < kTopK; ++i) {
            o[(kRTop + i) * fs] = tk[i];
            o[(kRIdx + i) * fs] = __int_as_float(ti[i]);
          }
          o[kRZx * fs] = zx;
        } else if constexpr (is_topk_fwd(kMode)) {
          o[kKM * fs] = m;
          o[kKS * fs] = s;
          o[kKSLo * fs] = sc;
          o[kKSIn * fs] = s_in;
          o[kKR * fs] = exp_residual(m);
          o[kKBest * fs] = best;
          o[kKIdx * fs] = __int_as_float(bidx);
          o[kKSec * fs] = sec;
#pragma unroll
          for (int i = 0; i < kTopK; ++i) o[(kKZ + i) * fs] = tk[i];
        }
      }
    }
    if constexpr (kStaged) {
      if (lane == 0) tma_store_wait_all();   // staging must stay valid until read
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
