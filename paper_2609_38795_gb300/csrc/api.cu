// C ABI of libalr (declared in include/alr.h): argument validation, tensor-map encoding,
// work planning and kernel launches.  No entry point allocates device memory.
#include <cudaTypedefs.h>

#include <atomic>
#include <cstdarg>
#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <mutex>

#include <nvtx3/nvToolsExt.h>

#include "alr.h"
#include "cluster_forms.h"
#include "kernels.h"

namespace {

thread_local char g_err[1024] = "";

int fail(int code, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof(g_err), fmt, ap);
  va_end(ap);
  return code;
}

int cuda_fail(cudaError_t e, const char* what) {
  return fail(ALR_ERR_CUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

std::mutex g_mu;

// Every compute entry point opens an NVTX range named after itself, so a profiler attached to
// the process shows each call as a span on the host timeline (and ncu can filter launches by
// it).  With no tool attached, push and pop return after one branch each.
struct Range {
  explicit Range(const char* name) { nvtxRangePushA(name); }
  ~Range() { nvtxRangePop(); }
  Range(const Range&) = delete;
  Range& operator=(const Range&) = delete;
};
#define ALR_RANGE() const Range alr_nvtx_range_(__func__)

// Test hook state: when set, the next launch of the fused loss kernel by a forward, or of the
// plain GEMM (single or multicast form), withholds its first pipeline stage.
std::atomic<int> g_withhold_next{0};

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  std::lock_guard<std::mutex> lk(g_mu);
  if (fn == nullptr) {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  }
  return fn;
}

struct DevInfo {
  int sms = 0;
  int cc = 0;
};

int device_info(DevInfo* out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
  static DevInfo cache[64];
  if (dev < 0 || dev >= 64) return fail(ALR_ERR_UNSUPPORTED, "device ordinal %d out of range", dev);
  std::lock_guard<std::mutex> lk(g_mu);
  if (cache[dev].sms == 0) {
    int sms = 0, major = 0, minor = 0;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess ||
        (e = cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev)) !=
            cudaSuccess ||
        (e = cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev)) != cudaSuccess)
      return cuda_fail(e, "cudaDeviceGetAttribute");
    cache[dev].sms = sms;
    cache[dev].cc = major * 10 + minor;
  }
  *out = cache[dev];
  return ALR_OK;
}

int require_sm103(DevInfo* info) {
  int rc = device_info(info);
  if (rc != ALR_OK) return rc;
  if (info->cc != 103)
    return fail(ALR_ERR_UNSUPPORTED,
                "libalr kernels are built for sm_103a only; current device is sm_%d", info->cc);
  return ALR_OK;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

size_t elem_size(int dtype) { return dtype == ALR_BF16 ? 2 : 4; }

size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Element type of the kept logits for bf16 inputs (tensor maps only; not an ALR_* dtype).
constexpr int kMapF16 = 2;

// 2-D tiled tensor map (128-byte swizzle unless stated): `inner` contiguous elements per row,
// `outer` rows `row_bytes` apart; boxes of box_inner x box_outer elements.  dtype: ALR_BF16,
// ALR_F32 or kMapF16.
int make_map(CUtensorMap* m, const void* ptr, int dtype, uint64_t inner, uint64_t outer,
             uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer,
             CUtensorMapSwizzle swizzle = CU_TENSOR_MAP_SWIZZLE_128B) {
  auto enc = encode_fn();
  if (enc == nullptr) return fail(ALR_ERR_CUDA, "cuTensorMapEncodeTiled is not available");
  cuuint64_t dims[2] = {inner, outer};
  cuuint64_t strides[1] = {row_bytes};
  cuuint32_t box[2] = {box_inner, box_outer};
  cuuint32_t estr[2] = {1, 1};
  const CUtensorMapDataType ty = dtype == ALR_BF16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16
                                 : dtype == kMapF16 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT16
                                                    : CU_TENSOR_MAP_DATA_TYPE_FLOAT32;
  CUresult r = enc(m, ty,
                   2, const_cast<void*>(ptr), dims, strides, box, estr,
                   CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
                   CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (r != CUDA_SUCCESS)
    return fail(ALR_ERR_CUDA, "cuTensorMapEncodeTiled failed (%d) for %llu x %llu", int(r),
                (unsigned long long)inner, (unsigned long long)outer);
  return ALR_OK;
}

// K elements per 128-byte swizzle row, and MN elements per 128-byte chunk.
uint32_t k_per_row(int dtype) { return uint32_t(128 / elem_size(dtype)); }

int check_params(const alr_params* p) {
  if (p == nullptr) return fail(ALR_ERR_INVALID_ARG, "params is NULL");
  if (p->dtype != ALR_BF16 && p->dtype != ALR_F32)
    return fail(ALR_ERR_UNSUPPORTED, "dtype %d is not ALR_BF16 or ALR_F32", p->dtype);
  if (p->mode < ALR_MODE_ALR || p->mode > ALR_MODE_ERASE_HARD)
    return fail(ALR_ERR_UNSUPPORTED, "mode %d is not an ALR_MODE_* value", p->mode);
  if (p->B < 1 || p->B > 32) return fail(ALR_ERR_INVALID_ARG, "B = %d must lie in [1, 32]", p->B);
  if (p->N < 1 || p->N % p->B != 0)
    return fail(ALR_ERR_INVALID_ARG, "N = %lld must be a positive multiple of B = %d",
                (long long)p->N, p->B);
  if (p->N > (int64_t(1) << 30)) return fail(ALR_ERR_INVALID_ARG, "N = %lld too large", (long long)p->N);
  if (p->d < 8 || p->d % 8 != 0) return fail(ALR_ERR_INVALID_ARG, "d = %d must be a positive multiple of 8", p->d);
  if (p->V < 2 || p->V % 8 != 0) return fail(ALR_ERR_INVALID_ARG, "V = %d must be >= 2 and a multiple of 8", p->V);
  if (!(p->gamma > 0.f)) return fail(ALR_ERR_INVALID_ARG, "gamma must be > 0");
  if (!(p->lambda == p->lambda)) return fail(ALR_ERR_INVALID_ARG, "lambda is NaN");
  return ALR_OK;
}

// A kept logit matrix and its group references: both needed (and 16-byte aligned) for bf16
// inputs, whose logits are kept as fp16 relative to the references; fp32 inputs keep plain
// fp32 logits and ignore `ref`.
int check_kept(const alr_params* p, const void* Z, const void* ref, const char* name) {
  if (Z == nullptr || !aligned16(Z))
    return fail(ALR_ERR_INVALID_ARG, "%s must be non-NULL and 16-byte aligned", name);
  if (p->dtype == ALR_BF16 && (ref == nullptr || !aligned16(ref)))
    return fail(ALR_ERR_INVALID_ARG,
                "%s_ref (the fp16 group references of bf16 inputs) must be non-NULL and "
                "16-byte aligned", name);
  return ALR_OK;
}

// Vocabulary tile width of the fused loss kernels (columns of z_d and of z_t per tile).
#ifndef ALR_LOSS_BN
#define ALR_LOSS_BN 256
#endif

// The fused loss kernels run on single CTAs unless the environment variable ALR_LOSS_FORM is
// "mcast" (bf16 inputs): clusters of two CTAs sharing every head tile by TMA multicast, from
// libalr_cluster.so, which only a single-process run loads (alr::cluster_forms() is nullptr in
// a multi-rank process, and then the single form runs).  The dual-product modes already share
// each head tile between z_d and z_t, and at the power cap the multicast form settles ~4 %
// lower in clock for ~1 % fewer L2 bytes per product: it is not faster, so it is not the
// default.  Both forms give bit-identical results.
bool loss_multicast(const alr_params* p) {
  if (p->dtype != ALR_BF16 || ALR_LOSS_BN != 256) return false;
  const char* v = getenv("ALR_LOSS_FORM");
  return v != nullptr && strcmp(v, "mcast") == 0 && alr::cluster_forms() != nullptr;
}

// two_rows: the single-operand modes (readout, top-k), whose units hold two row blocks.
alr::LossPlan loss_plan(const alr_params* p, int sms, bool bwd, bool two_rows = false) {
  alr::LossPlan P{};
  P.N = int(p->N);
  P.d = p->d;
  P.V = p->V;
  P.B = p->B;
  P.bn = ALR_LOSS_BN;
  P.mc = (!two_rows && loss_multicast(p)) ? 1 : 0;
  // row blocks; row-block pairs for the two-row modes and for the multicast form (which
  // places sms / 2 clusters).  Forward: the vocabulary splits are sized so that one round of
  // the grid covers 8 row blocks (152 CTAs / 8 = 19 splits: 32 units per CTA at 256 row
  // blocks) and a raster group spans two rounds (16 row blocks).  Recomputing backward: one
  // vocabulary tile per unit, raster groups of 16 row blocks as well.
  const int rb = int((p->N + 127) / 128);
  const bool pairs = P.mc || two_rows;
  P.n_rb = pairs ? (rb + 1) / 2 : rb;
  const int slots = P.mc ? sms / 2 : sms;
  const int group = pairs ? 4 : 8;
  P.n_vt = (p->V + P.bn - 1) / P.bn;
  P.group_rows = P.n_rb < group ? P.n_rb : group;
  if (bwd) {
    P.n_vs = P.n_vt;  // one tile per unit
    // 16 row blocks share each W tile (the recomputed logit gradient 46.2 against 46.4 ms
    // with 8, three alternating A/B rounds)
    P.group_rows = P.n_rb < 2 * group ? P.n_rb : 2 * group;
  } else {
    int vs = slots / P.group_rows;
    if (vs < 1) vs = 1;
    P.n_vs = vs < P.n_vt ? vs : P.n_vt;
    // two rounds per raster group: twice the row blocks share each W split, so W leaves
    // DRAM about half as often, with the same number of units per CTA (forward 49.8 against
    // 50.0 ms at the text8b size, three alternating A/B rounds)
    const int wide = 2 * group;
    P.group_rows = P.n_rb < wide ? P.n_rb : wide;
  }
  // partial records per row and split: one per epilogue column group
  P.n_parts = P.n_vs * (P.bn / (two_rows ? 128 : 64));
  P.n_units = P.n_rb * P.n_vs;
  P.grid = sms < P.n_units ? sms : P.n_units;
  return P;
}

// fp32 inputs run tf32 products, which take K-major operands only: the head is then read from
// a transposed copy W^T [V, d] placed in the workspace.
// Forward-type workspace: `fields` partial statistics per row and part, one fp64 pair per
// anchor, and W^T for fp32 inputs.
struct FwdLayout {
  size_t part_off, anchor_off, wt_off, total;
};

FwdLayout fwd_layout(const alr_params* p, int sms, int fields = alr::kPFields,
                     bool two_rows = false) {
  const alr::LossPlan P = loss_plan(p, sms, false, two_rows);
  FwdLayout L{};
  L.part_off = 0;
  L.anchor_off = round_up(size_t(fields) * P.n_parts * size_t(P.N) * sizeof(float), 1024);
  L.wt_off = L.anchor_off + round_up(2 * sizeof(double) * size_t(P.N / P.B), 1024);
  L.total = L.wt_off;
  if (p->dtype == ALR_F32) L.total += round_up(size_t(p->V) * p->d * sizeof(float), 1024);
  return L;
}

// Backward workspace: G [N, V]; for fp32 also W^T [V, d], G^T [V, N'] and H_d^T [d, N'] with
// N' = N rounded up to 4 (16-byte rows).
struct BwdLayout {
  size_t g_off, wt_off, gt_off, hdt_off, total;
  int64_t ld_n;
};

// with_g = false: the layout of the backward from kept logits, whose G is the caller's and
// which needs no W^T (G^T and H_d^T only, for fp32).
BwdLayout bwd_layout(const alr_params* p, bool with_g = true) {
  BwdLayout L{};
  const size_t es = p->dtype == ALR_BF16 ? 2 : 4;
  L.g_off = 0;
  L.total = with_g ? round_up(size_t(p->N) * size_t(p->V) * es, 1024) : 0;
  L.ld_n = (p->N + 3) / 4 * 4;
  if (p->dtype == ALR_F32) {
    L.wt_off = L.total;
    L.gt_off = L.wt_off + (with_g ? round_up(size_t(p->V) * p->d * 4, 1024) : 0);
    L.hdt_off = L.gt_off + round_up(size_t(p->V) * L.ld_n * 4, 1024);
    L.total = L.hdt_off + round_up(size_t(p->d) * L.ld_n * 4, 1024);
  }
  return L;
}

// Form of the bf16 products, chosen by the environment variable ALR_GEMM_FORM:
//   "mcast"   clusters of two CTAs, each on a 128 x 256 tile, sharing every B tile by TMA
//             multicast, the default;
//   "single"  one CTA per 128 x 256 tile, each loading its own B tiles (plain_gemm.cu);
//   "pair"    CTA pairs with M = 256 products.
// The cluster forms ("mcast", "mcast4", "pair") live in libalr_cluster.so (csrc_cluster/),
// which only a single-process run loads: in a process that is one rank of several, or where
// that library cannot be loaded, every form runs as "single" (alr_kernel_forms reports it).
// The step runs at the GB300's power cap, so the form that moves fewest bytes per product
// wins: multicast halves the B traffic out of L2 and runs 6 % faster than single CTAs at the
// same clock and power.  The pair form issues more products per clock but draws more power
// per product and settles at a clock ~20 % lower.  tf32 products always run on single CTAs.
//   "mcast4"  as "mcast" with clusters of four CTAs, each loading a quarter of the B tile.
enum GemmForm { kGemmSingle = 0, kGemmMcast = 1, kGemmPair = 2, kGemmMcast4 = 3 };

GemmForm gemm_form(int dtype) {
  if (dtype != ALR_BF16) return kGemmSingle;
  const char* v = getenv("ALR_GEMM_FORM");
  if ((v != nullptr && strcmp(v, "single") == 0) || alr::cluster_forms() == nullptr)
    return kGemmSingle;
  if (v != nullptr && strcmp(v, "pair") == 0) return kGemmPair;
  if (v != nullptr && strcmp(v, "mcast4") == 0) return kGemmMcast4;
  return kGemmMcast;
}

// Rows of a K-major B box (B columns loaded by one copy).
uint32_t gemm_b_rows(int dtype) {
  switch (gemm_form(dtype)) {
    case kGemmSingle: return 256;
    case kGemmMcast4: return 64;
    default: return 128;
  }
}

alr::GemmArgs gemm_plan(int M, int Nc, int K, float* C, int64_t ldc, int sms) {
  alr::GemmArgs g{};
  g.M = M;
  g.Nc = Nc;
  g.K = K;
  g.C = C;
  g.ldc = ldc;
  g.n_mb = (M + 127) / 128;
  g.n_nb = (Nc + 255) / 256;
  g.group_m = g.n_mb < 16 ? g.n_mb : 16;
  g.n_tiles = g.n_mb * g.n_nb;
  g.grid = sms < g.n_tiles ? sms : g.n_tiles;
  return g;
}

// Plan of the pair GEMM: 256 x 256 tiles over `pairs` resident CTA pairs.
alr::GemmArgs pair_gemm_plan(int M, int Nc, int K, float* C, int64_t ldc, int pairs) {
  alr::GemmArgs g{};
  g.M = M;
  g.Nc = Nc;
  g.K = K;
  g.C = C;
  g.ldc = ldc;
  g.n_mb = (M + 255) / 256;
  g.n_nb = (Nc + 255) / 256;
  g.group_m = g.n_mb < 8 ? g.n_mb : 8;
  g.n_tiles = g.n_mb * g.n_nb;
  g.grid = 2 * (pairs < g.n_tiles ? pairs : g.n_tiles);
  return g;
}

// C (+)= A B with the operand maps already encoded (B boxes of gemm_b_rows(dt) rows).
int launch_gemm(int dt, bool a_mn, bool b_mn, bool acc, const CUtensorMap& ma,
                const CUtensorMap& mb, int M, int Nc, int K, float* C, int64_t ldc, int sms,
                cudaStream_t s, const char* what) {
  cudaError_t e;
  const GemmForm form = gemm_form(dt);
  const alr::ClusterForms* cf = alr::cluster_forms();   // non-NULL for every cluster form
  if (form == kGemmPair) {
    const int pairs = cf->pair_gemm_max_pairs();
    if (pairs < 1) return fail(ALR_ERR_CUDA, "%s: no CTA pair of the GEMM fits on this device", what);
    alr::GemmArgs g = pair_gemm_plan(M, Nc, K, C, ldc, pairs);
    g.status = alr::device_status_ptr();
    if (g.status == nullptr) return fail(ALR_ERR_CUDA, "status word lookup failed");
    e = cf->launch_pair_gemm(a_mn, b_mn, acc, &ma, &mb, &g, s);
  } else if (form == kGemmMcast || form == kGemmMcast4) {
    const int cl = form == kGemmMcast4 ? 4 : 2;
    const int clusters = cf->gemm_max_clusters(cl);
    if (clusters < 1)
      return fail(ALR_ERR_CUDA, "%s: no CTA cluster of the GEMM fits on this device", what);
    // 128-row blocks in groups of `cl`: n_mb counts groups, raster groups of 16 row blocks
    alr::GemmArgs g = gemm_plan(M, Nc, K, C, ldc, sms);
    g.n_mb = ((M + 127) / 128 + cl - 1) / cl;
    const int gm = 16 / cl;
    g.group_m = g.n_mb < gm ? g.n_mb : gm;
    g.n_tiles = g.n_mb * g.n_nb;
    g.grid = cl * (clusters < g.n_tiles ? clusters : g.n_tiles);
    g.status = alr::device_status_ptr();
    if (g.status == nullptr) return fail(ALR_ERR_CUDA, "status word lookup failed");
    g.withhold_first_stage = g_withhold_next.exchange(0);
    e = cf->launch_gemm(cl, a_mn, b_mn, acc, &ma, &mb, &g, s);
  } else {
    alr::GemmArgs g = gemm_plan(M, Nc, K, C, ldc, sms);
    g.status = alr::device_status_ptr();
    if (g.status == nullptr) return fail(ALR_ERR_CUDA, "status word lookup failed");
    g.withhold_first_stage = g_withhold_next.exchange(0);
    e = alr::launch_plain_gemm(dt, a_mn, b_mn, acc, ma, mb, g, s);
  }
  if (e != cudaSuccess) return cuda_fail(e, what);
  return ALR_OK;
}

// Tensor map of the head operand of the fused loss kernels: MN-major tiles straight from
// W [d, V] for bf16; for fp32, W is first transposed into `wt` and read K-major.
int head_map(CUtensorMap* m, const alr_params* p, const void* W, void* wt, cudaStream_t s) {
  const uint32_t kke = k_per_row(p->dtype);
  if (p->dtype == ALR_BF16) return make_map(m, W, ALR_BF16, p->V, p->d, uint64_t(p->V) * 2, kke, kke);
  cudaError_t e = alr::launch_transpose32(static_cast<const float*>(W), static_cast<float*>(wt),
                                          p->d, p->V, p->d, s);
  if (e != cudaSuccess) return cuda_fail(e, "head transpose launch");
  return make_map(m, wt, ALR_F32, p->d, p->V, uint64_t(p->d) * 4, kke, ALR_LOSS_BN);
}

// The full-vocabulary forward; with Zd / Zt given, the fused kernel also writes both logit
// matrices (kModeFwdKeep).
int fwd_impl(const alr_params* p, const void* Hd, const void* Ht, const void* W,
             const float* row_mask, const int32_t* corpus_tok, void* Zd, void* Zt,
             uint16_t* Zd_ref, uint16_t* Zt_ref, const alr_fwd_outputs* out, void* workspace,
             size_t ws_bytes, void* stream) {
  int rc = check_params(p);
  if (rc != ALR_OK) return rc;
  if (Hd == nullptr || Ht == nullptr || W == nullptr || out == nullptr)
    return fail(ALR_ERR_INVALID_ARG, "Hd, Ht, W and out must be non-NULL");
  if (!aligned16(Hd) || !aligned16(Ht) || !aligned16(W))
    return fail(ALR_ERR_INVALID_ARG, "Hd, Ht and W must be 16-byte aligned");
  if (out->loss_row == nullptr || out->lse_d == nullptr || out->lse_t == nullptr ||
      out->argmax_d == nullptr || out->argmax_t == nullptr || out->weight == nullptr ||
      out->loss_total == nullptr || out->weight_sum == nullptr)
    return fail(ALR_ERR_INVALID_ARG, "a required forward output pointer is NULL");
  if (p->mode != ALR_MODE_ALR && corpus_tok == nullptr)
    return fail(ALR_ERR_INVALID_ARG, "the erase modes need corpus_tok");
  DevInfo info;
  if ((rc = require_sm103(&info)) != ALR_OK) return rc;
  const FwdLayout lay = fwd_layout(p, info.sms);
  if (workspace == nullptr || ws_bytes < lay.total)
    return fail(ALR_ERR_INVALID_ARG, "workspace of %zu bytes is smaller than the %zu needed",
                ws_bytes, lay.total);
  if (!aligned16(workspace)) return fail(ALR_ERR_INVALID_ARG, "workspace must be 16-byte aligned");

  const int dt = p->dtype;
  const size_t es = elem_size(dt);
  const uint32_t kke = k_per_row(dt);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  CUtensorMap m_hd, m_ht, m_w;
  if ((rc = make_map(&m_hd, Hd, dt, p->d, p->N, p->d * es, kke, 128)) != ALR_OK) return rc;
  if ((rc = make_map(&m_ht, Ht, dt, p->d, p->N, p->d * es, kke, 128)) != ALR_OK) return rc;
  if ((rc = head_map(&m_w, p, W, ws + lay.wt_off, s)) != ALR_OK) return rc;

  alr::LossArgs args{};
  args.plan = loss_plan(p, info.sms, false);
  args.part = reinterpret_cast<float*>(ws + lay.part_off);
  args.corpus_tok = p->mode != ALR_MODE_ALR ? corpus_tok : nullptr;
  args.lam = p->lambda;
  args.withhold_first_stage = g_withhold_next.exchange(0);
  args.status = alr::device_status_ptr();
  if (args.status == nullptr) return fail(ALR_ERR_CUDA, "status word lookup failed");
  args.zd_out = Zd;
  args.zt_out = Zt;
  args.zd_ref = Zd_ref;
  args.zt_ref = Zt_ref;
  // bf16 inputs keep fp16 logits through TMA stores of 16-column x 32-row boxes
  CUtensorMap m_zd = m_w, m_zt = m_w;
  if (Zd != nullptr && dt == ALR_BF16) {
    if ((rc = make_map(&m_zd, Zd, kMapF16, p->V, p->N, uint64_t(p->V) * 2, 16, 32,
                       CU_TENSOR_MAP_SWIZZLE_NONE)) != ALR_OK)
      return rc;
    if ((rc = make_map(&m_zt, Zt, kMapF16, p->V, p->N, uint64_t(p->V) * 2, 16, 32,
                       CU_TENSOR_MAP_SWIZZLE_NONE)) != ALR_OK)
      return rc;
  }
  e = alr::launch_loss_kernel(Zd != nullptr ? alr::kModeFwdKeep : alr::kModeFwd, dt, m_hd, m_ht,
                              m_w, m_zd, m_zt, args, s);
  if (e != cudaSuccess) return cuda_fail(e, "forward loss kernel launch");
  double* anchor = reinterpret_cast<double*>(ws + lay.anchor_off);
  e = alr::launch_combine(args.plan, args.part, p->mode, p->gamma, row_mask, args.corpus_tok,
                          out->loss_row, out->ent_row, out->lse_d, out->lse_t, out->argmax_d,
                          out->argmax_t, out->gap_d, out->gap_t, out->logp_x, out->weight, anchor,
                          s);
  if (e != cudaSuccess) return cuda_fail(e, "combine launch");
  e = alr::launch_finalize(anchor, int(p->N / p->B), p->lambda, out->loss_total, out->weight_sum,
                          out->wl_sum, s);
  if (e != cudaSuccess) return cuda_fail(e, "finalize launch");
  return ALR_OK;
}

}  // namespace

namespace alr {
int set_last_error(int code, const char* msg) { return fail(code, "%s", msg); }
}  // namespace alr

extern "C" {

const char* alr_version(void) { return "libalr 0.1 (sm_103a)"; }

int alr_kernel_forms(int32_t* gemm, int32_t* loss) {
  if (gemm == nullptr || loss == nullptr) return fail(ALR_ERR_INVALID_ARG, "gemm and loss must be non-NULL");
  alr_params p{};
  p.dtype = ALR_BF16;
  *gemm = int32_t(gemm_form(ALR_BF16));
  *loss = loss_multicast(&p) ? 1 : 0;
  return ALR_OK;
}

const char* alr_cluster_forms_error(void) {
  return alr::cluster_forms() != nullptr ? "" : alr::cluster_forms_error();
}

int alr_debug_withhold_next_stage(int enable) {
  g_withhold_next.store(enable ? 1 : 0);
  return ALR_OK;
}

const char* alr_last_error(void) { return g_err; }

int alr_device_supported(void) {
  DevInfo info;
  return require_sm103(&info);
}

int alr_device_status(void* stream, int clear) {
  cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
  int* w = alr::device_status_ptr();
  if (w == nullptr) return fail(ALR_ERR_CUDA, "status word lookup failed");
  int v = 0;
  if ((e = cudaMemcpy(&v, w, sizeof(int), cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "reading the status word");
  if (clear) {
    const int z = 0;
    if ((e = cudaMemcpy(w, &z, sizeof(int), cudaMemcpyHostToDevice)) != cudaSuccess)
      return cuda_fail(e, "clearing the status word");
  }
  if (v != 0) return fail(ALR_ERR_TIMEOUT, "a device pipeline wait timed out");
  return ALR_OK;
}

int alr_gather_ira_blocks(const void* feat, int32_t S, int32_t L, int32_t d, int32_t dtype,
                          const int32_t* seq, const int32_t* pos, const int32_t* valid_len,
                          int32_t A, int32_t B, void* out, float* row_valid, void* stream) {
  ALR_RANGE();
  if (dtype != ALR_BF16 && dtype != ALR_F32) return fail(ALR_ERR_UNSUPPORTED, "dtype %d", dtype);
  if (S < 1 || L < 1 || d < 1 || A < 0 || B < 1)
    return fail(ALR_ERR_INVALID_ARG, "bad sizes S=%d L=%d d=%d A=%d B=%d", S, L, d, A, B);
  if ((size_t(d) * elem_size(dtype)) % 16 != 0)
    return fail(ALR_ERR_INVALID_ARG, "d * element size must be a multiple of 16 bytes");
  if (A == 0) return ALR_OK;
  if (feat == nullptr || seq == nullptr || pos == nullptr || out == nullptr)
    return fail(ALR_ERR_INVALID_ARG, "feat, seq, pos and out must be non-NULL");
  if (!aligned16(feat) || !aligned16(out))
    return fail(ALR_ERR_INVALID_ARG, "feat and out must be 16-byte aligned");
  DevInfo info;
  int rc = require_sm103(&info);
  if (rc != ALR_OK) return rc;
  cudaError_t e = alr::launch_gather(feat, S, L, d, int(elem_size(dtype)), seq, pos, valid_len, A,
                                     B, out, row_valid, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "gather launch");
  return ALR_OK;
}

size_t alr_fwd_workspace_size(const alr_params* p) {
  if (check_params(p) != ALR_OK) return 0;
  DevInfo info;
  if (device_info(&info) != ALR_OK) return 0;
  return fwd_layout(p, info.sms).total;
}

int alr_slot_loss_fwd(const alr_params* p, const void* Hd, const void* Ht, const void* W,
                      const float* row_mask, const int32_t* corpus_tok, const alr_fwd_outputs* out,
                      void* workspace, size_t ws_bytes, void* stream) {
  ALR_RANGE();
  return fwd_impl(p, Hd, Ht, W, row_mask, corpus_tok, nullptr, nullptr, nullptr, nullptr, out,
                  workspace, ws_bytes, stream);
}

int alr_slot_loss_fwd_keep_logits(const alr_params* p, const void* Hd, const void* Ht,
                                  const void* W, const float* row_mask, const int32_t* corpus_tok,
                                  void* Zd, void* Zt, uint16_t* Zd_ref, uint16_t* Zt_ref,
                                  const alr_fwd_outputs* out, void* workspace, size_t ws_bytes,
                                  void* stream) {
  ALR_RANGE();
  int rc = check_params(p);
  if (rc != ALR_OK) return rc;
  if ((rc = check_kept(p, Zd, Zd_ref, "Zd")) != ALR_OK) return rc;
  if ((rc = check_kept(p, Zt, Zt_ref, "Zt")) != ALR_OK) return rc;
  return fwd_impl(p, Hd, Ht, W, row_mask, corpus_tok, Zd, Zt, Zd_ref, Zt_ref, out, workspace,
                  ws_bytes, stream);
}

int32_t alr_kept_ref_groups(int32_t V) {
  return V < 1 ? 0 : (V + alr::kKeepGroup - 1) / alr::kKeepGroup;
}

size_t alr_bwd_workspace_size(const alr_params* p) {
  if (check_params(p) != ALR_OK) return 0;
  return bwd_layout(p).total;
}

}  // extern "C"

namespace {

// Checks shared by the backward entry points; fills `info`.
int check_bwd_args(const alr_params* p, const void* Hd, const void* Ht, const void* W,
                   const float* weight, const float* weight_sum, const float* lse_d,
                   const float* lse_t, DevInfo* info) {
  int rc = check_params(p);
  if (rc != ALR_OK) return rc;
  if (Hd == nullptr || Ht == nullptr || W == nullptr || weight == nullptr ||
      weight_sum == nullptr || lse_d == nullptr || lse_t == nullptr)
    return fail(ALR_ERR_INVALID_ARG, "a required backward input pointer is NULL");
  if (!aligned16(Hd) || !aligned16(Ht) || !aligned16(W))
    return fail(ALR_ERR_INVALID_ARG, "Hd, Ht and W must be 16-byte aligned");
  return require_sm103(info);
}

// Compact-label inputs of the top-k path (all NULL for the full-vocabulary loss).
struct TopkLabels {
  const int32_t* idx = nullptr;
  const float* prob = nullptr;
  const float* tail = nullptr;
  const float* tail_q = nullptr;
};

// The fused logit-gradient kernel: G = lambda omega / sum omega (q - p) for the full
// vocabulary (Ht given), or the top-k + tail form (labels given), recomputing the tiles.
int logit_grad_impl(const alr_params* p, const void* Hd, const void* Ht, const void* W,
                    const float* weight, const float* weight_sum, const float* lse_d,
                    const float* lse_t, const TopkLabels& lab, void* G, void* wt,
                    const DevInfo& info, cudaStream_t s) {
  const int dt = p->dtype;
  const size_t es = elem_size(dt);
  const uint32_t kke = k_per_row(dt);
  const bool topk = lab.idx != nullptr;
  int rc;
  CUtensorMap m_hd, m_ht, m_w, m_gs;
  if ((rc = make_map(&m_hd, Hd, dt, p->d, p->N, p->d * es, kke, 128)) != ALR_OK) return rc;
  m_ht = m_hd;
  if (!topk && (rc = make_map(&m_ht, Ht, dt, p->d, p->N, p->d * es, kke, 128)) != ALR_OK) return rc;
  if ((rc = head_map(&m_w, p, W, wt, s)) != ALR_OK) return rc;
  m_gs = m_w;
  if (dt == ALR_BF16 &&
      (rc = make_map(&m_gs, G, dt, p->V, p->N, p->V * es, 16, 32, CU_TENSOR_MAP_SWIZZLE_NONE)) != ALR_OK)
    return rc;
  alr::LossArgs args{};
  args.plan = loss_plan(p, info.sms, true, topk);
  args.G = G;
  args.lse_d = lse_d;
  args.lse_t = lse_t;
  args.weight = weight;
  args.weight_sum = weight_sum;
  args.lam = p->lambda;
  args.top_idx = lab.idx;
  args.top_prob = lab.prob;
  args.tail = lab.tail;
  args.tail_q = lab.tail_q;
  args.status = alr::device_status_ptr();
  if (args.status == nullptr) return fail(ALR_ERR_CUDA, "status word lookup failed");
  cudaError_t e = alr::launch_loss_kernel(topk ? alr::kModeTopkBwd : alr::kModeBwd, dt, m_hd, m_ht,
                                          m_w, m_gs, m_gs, args, s);
  if (e != cudaSuccess) return cuda_fail(e, "logit-gradient kernel launch");
  return ALR_OK;
}

// dH_d = G W^T and, when dW is given, dW += H_d^T G (fp32 via transposed workspace copies).
int head_grads_impl(const alr_params* p, const void* Hd, const void* W, const void* G, float* dHd,
                    float* dW, uint8_t* ws, const BwdLayout& lay, const DevInfo& info,
                    cudaStream_t s) {
  const int dt = p->dtype;
  const size_t es = elem_size(dt);
  const uint32_t kke = k_per_row(dt);
  int rc;
  cudaError_t e;
  // dH_d = G W^T: A = G [N, V] K-major, B = W [d, V] K-major.
  CUtensorMap m_ga, m_wk;
  if ((rc = make_map(&m_ga, G, dt, p->V, p->N, p->V * es, kke, 128)) != ALR_OK) return rc;
  if ((rc = make_map(&m_wk, W, dt, p->V, p->d, p->V * es, kke, gemm_b_rows(dt))) != ALR_OK)
    return rc;
  if ((rc = launch_gemm(dt, false, false, false, m_ga, m_wk, int(p->N), p->d, p->V, dHd, p->d,
                        info.sms, s, "dH GEMM launch")) != ALR_OK)
    return rc;
  if (dW == nullptr) return ALR_OK;
  CUtensorMap m_ha, m_gb;
  if (dt == ALR_BF16) {
    // dW += H_d^T G: A = H_d read as [K = N, M = d] (MN-major), B = G [K = N, V] (MN-major).
    if ((rc = make_map(&m_ha, Hd, dt, p->d, p->N, p->d * es, kke, kke)) != ALR_OK) return rc;
    if ((rc = make_map(&m_gb, G, dt, p->V, p->N, p->V * es, kke, kke)) != ALR_OK) return rc;
    return launch_gemm(dt, true, true, true, m_ha, m_gb, p->d, p->V, int(p->N), dW, p->V,
                       info.sms, s, "dW GEMM launch");
  } else {
    // K-major operands from transposed copies H_d^T [d, N'] and G^T [V, N'].
    float* hdt = reinterpret_cast<float*>(ws + lay.hdt_off);
    float* gt = reinterpret_cast<float*>(ws + lay.gt_off);
    if ((e = alr::launch_transpose32(static_cast<const float*>(Hd), hdt, int(p->N), p->d,
                                     int(lay.ld_n), s)) != cudaSuccess)
      return cuda_fail(e, "H_d transpose launch");
    if ((e = alr::launch_transpose32(static_cast<const float*>(G), gt, int(p->N), p->V,
                                     int(lay.ld_n), s)) != cudaSuccess)
      return cuda_fail(e, "G transpose launch");
    if ((rc = make_map(&m_ha, hdt, dt, p->N, p->d, lay.ld_n * 4, kke, 128)) != ALR_OK) return rc;
    if ((rc = make_map(&m_gb, gt, dt, p->N, p->V, lay.ld_n * 4, kke, gemm_b_rows(dt))) != ALR_OK)
      return rc;
    return launch_gemm(dt, false, false, true, m_ha, m_gb, p->d, p->V, int(p->N), dW, p->V,
                       info.sms, s, "dW GEMM launch");
  }
}

int check_workspace(void* workspace, size_t ws_bytes, size_t need) {
  if (need > 0 && (workspace == nullptr || ws_bytes < need))
    return fail(ALR_ERR_INVALID_ARG, "workspace of %zu bytes is smaller than the %zu needed",
                ws_bytes, need);
  if (need > 0 && !aligned16(workspace))
    return fail(ALR_ERR_INVALID_ARG, "workspace must be 16-byte aligned");
  return ALR_OK;
}

// Arguments of the dH / dW products of the backward passes from kept logits.
int check_head_grad_args(const alr_params* p, const void* Hd, const void* W, const float* dHd,
                         const float* dW, void* workspace, size_t ws_bytes) {
  int rc = check_params(p);
  if (rc != ALR_OK) return rc;
  if (Hd == nullptr || W == nullptr || dHd == nullptr)
    return fail(ALR_ERR_INVALID_ARG, "Hd, W and dHd must be non-NULL");
  if (!aligned16(Hd) || !aligned16(W) || !aligned16(dHd) || (dW != nullptr && !aligned16(dW)))
    return fail(ALR_ERR_INVALID_ARG, "Hd, W, dHd and dW must be 16-byte aligned");
  return check_workspace(workspace, ws_bytes, bwd_layout(p, false).total);
}

int check_topk_labels(const alr_params* p, const int32_t* idx, const float* prob,
                      const float* tail) {
  if (p->V < alr::kTopK)
    return fail(ALR_ERR_INVALID_ARG, "V = %d is below the %d label tokens", p->V, alr::kTopK);
  if (idx == nullptr || prob == nullptr || tail == nullptr)
    return fail(ALR_ERR_INVALID_ARG, "top_idx, top_prob and tail must be non-NULL");
  return ALR_OK;
}

}  // namespace

extern "C" {

size_t alr_logit_grad_workspace_size(const alr_params* p) {
  if (check_params(p) != ALR_OK) return 0;
  return p->dtype == ALR_F32 ? round_up(size_t(p->V) * p->d * 4, 1024) : 0;
}

int alr_logit_grad(const alr_params* p, const void* Hd, const void* Ht, const void* W,
                   const float* weight, const float* weight_sum, const float* lse_d,
                   const float* lse_t, void* G, void* workspace, size_t ws_bytes, void* stream) {
  ALR_RANGE();
  DevInfo info;
  int rc = check_bwd_args(p, Hd, Ht, W, weight, weight_sum, lse_d, lse_t, &info);
  if (rc != ALR_OK) return rc;
  if (G == nullptr || !aligned16(G)) return fail(ALR_ERR_INVALID_ARG, "G must be non-NULL and 16-byte aligned");
  const size_t need = alr_logit_grad_workspace_size(p);
  if (need > 0 && (workspace == nullptr || ws_bytes < need || !aligned16(workspace)))
    return fail(ALR_ERR_INVALID_ARG, "workspace of %zu bytes is smaller than the %zu needed",
                ws_bytes, need);
  return logit_grad_impl(p, Hd, Ht, W, weight, weight_sum, lse_d, lse_t, TopkLabels{}, G,
                         workspace, info, static_cast<cudaStream_t>(stream));
}

int alr_slot_loss_bwd(const alr_params* p, const void* Hd, const void* Ht, const void* W,
                      const float* weight, const float* weight_sum, const float* lse_d,
                      const float* lse_t, float* dHd, float* dW, void* workspace, size_t ws_bytes,
                      void* stream) {
  ALR_RANGE();
  DevInfo info;
  int rc = check_bwd_args(p, Hd, Ht, W, weight, weight_sum, lse_d, lse_t, &info);
  if (rc != ALR_OK) return rc;
  if (dHd == nullptr) return fail(ALR_ERR_INVALID_ARG, "dHd is NULL");
  if (!aligned16(dHd) || (dW != nullptr && !aligned16(dW)))
    return fail(ALR_ERR_INVALID_ARG, "dHd and dW must be 16-byte aligned");
  const size_t need = alr_bwd_workspace_size(p);
  if (workspace == nullptr || ws_bytes < need)
    return fail(ALR_ERR_INVALID_ARG, "workspace of %zu bytes is smaller than the %zu needed",
                ws_bytes, need);
  if (!aligned16(workspace)) return fail(ALR_ERR_INVALID_ARG, "workspace must be 16-byte aligned");

  const BwdLayout lay = bwd_layout(p);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  void* G = ws + lay.g_off;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  rc = logit_grad_impl(p, Hd, Ht, W, weight, weight_sum, lse_d, lse_t, TopkLabels{}, G,
                       ws + lay.wt_off, info, s);
  if (rc != ALR_OK) return rc;
  return head_grads_impl(p, Hd, W, G, dHd, dW, ws, lay, info, s);
}

int alr_logit_grad_from_logits(const alr_params* p, const void* Zd, const void* Zt,
                               const uint16_t* Zd_ref, const uint16_t* Zt_ref,
                               const float* weight, const float* weight_sum, const float* lse_d,
                               const float* lse_t, void* G, void* stream) {
  ALR_RANGE();
  int rc = check_params(p);
  if (rc != ALR_OK) return rc;
  if ((rc = check_kept(p, Zd, Zd_ref, "Zd")) != ALR_OK) return rc;
  if ((rc = check_kept(p, Zt, Zt_ref, "Zt")) != ALR_OK) return rc;
  if (G == nullptr || weight == nullptr || weight_sum == nullptr || lse_d == nullptr ||
      lse_t == nullptr)
    return fail(ALR_ERR_INVALID_ARG, "a required pointer is NULL");
  if (!aligned16(G)) return fail(ALR_ERR_INVALID_ARG, "G must be 16-byte aligned");
  DevInfo info;
  if ((rc = require_sm103(&info)) != ALR_OK) return rc;
  cudaError_t e = alr::launch_logits_grad(p->dtype, Zd, Zt, Zd_ref, Zt_ref, lse_d, lse_t, weight,
                                          weight_sum, p->lambda, int(p->N), p->V, G,
                                          static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "logit-gradient launch");
  return ALR_OK;
}

size_t alr_bwd_from_logits_workspace_size(const alr_params* p) {
  if (check_params(p) != ALR_OK) return 0;
  return bwd_layout(p, false).total;
}

int alr_slot_loss_bwd_from_logits(const alr_params* p, const void* Hd, const void* W,
                                  const void* Zd, const void* Zt, const uint16_t* Zd_ref,
                                  const uint16_t* Zt_ref, const float* weight,
                                  const float* weight_sum, const float* lse_d, const float* lse_t,
                                  void* G, float* dHd, float* dW, void* workspace,
                                  size_t ws_bytes, void* stream) {
  ALR_RANGE();
  // everything is validated before the gradient kernel overwrites anything
  int rc = check_head_grad_args(p, Hd, W, dHd, dW, workspace, ws_bytes);
  if (rc != ALR_OK) return rc;
  if ((rc = alr_logit_grad_from_logits(p, Zd, Zt, Zd_ref, Zt_ref, weight, weight_sum, lse_d,
                                       lse_t, G, stream)) != ALR_OK)
    return rc;
  DevInfo info;
  if ((rc = require_sm103(&info)) != ALR_OK) return rc;
  return head_grads_impl(p, Hd, W, G, dHd, dW, static_cast<uint8_t*>(workspace),
                         bwd_layout(p, false), info, static_cast<cudaStream_t>(stream));
}

size_t alr_readout_workspace_size(const alr_params* p) {
  if (check_params(p) != ALR_OK) return 0;
  DevInfo info;
  if (device_info(&info) != ALR_OK) return 0;
  return fwd_layout(p, info.sms, alr::kRFields, true).total;
}

int alr_label_readout(const alr_params* p, const void* Ht, const void* W,
                      const int32_t* corpus_tok, int32_t* top_idx, float* top_prob, float* tail,
                      float* lse_t, int32_t* argmax_t, float* gap_t, float* logp_x,
                      void* workspace, size_t ws_bytes, void* stream) {
  ALR_RANGE();
  int rc = check_params(p);
  if (rc != ALR_OK) return rc;
  if (Ht == nullptr || W == nullptr || top_idx == nullptr || top_prob == nullptr || tail == nullptr)
    return fail(ALR_ERR_INVALID_ARG, "Ht, W, top_idx, top_prob and tail must be non-NULL");
  if (p->V < alr::kTopK)
    return fail(ALR_ERR_INVALID_ARG, "V = %d is below the %d label tokens", p->V, alr::kTopK);
  if (!aligned16(Ht) || !aligned16(W))
    return fail(ALR_ERR_INVALID_ARG, "Ht and W must be 16-byte aligned");
  DevInfo info;
  if ((rc = require_sm103(&info)) != ALR_OK) return rc;
  const FwdLayout lay = fwd_layout(p, info.sms, alr::kRFields, true);
  if ((rc = check_workspace(workspace, ws_bytes, lay.total)) != ALR_OK) return rc;
  const int dt = p->dtype;
  const size_t es = elem_size(dt);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  CUtensorMap m_h, m_w;
  if ((rc = make_map(&m_h, Ht, dt, p->d, p->N, p->d * es, k_per_row(dt), 128)) != ALR_OK) return rc;
  if ((rc = head_map(&m_w, p, W, ws + lay.wt_off, s)) != ALR_OK) return rc;
  alr::LossArgs args{};
  args.plan = loss_plan(p, info.sms, false, true);
  args.part = reinterpret_cast<float*>(ws + lay.part_off);
  args.corpus_tok = corpus_tok;
  args.status = alr::device_status_ptr();
  if (args.status == nullptr) return fail(ALR_ERR_CUDA, "status word lookup failed");
  cudaError_t e = alr::launch_loss_kernel(alr::kModeReadout, dt, m_h, m_h, m_w, m_w, m_w, args, s);
  if (e != cudaSuccess) return cuda_fail(e, "label readout kernel launch");
  e = alr::launch_readout_combine(args.plan, args.part, corpus_tok != nullptr, top_idx, top_prob,
                                  tail, lse_t, argmax_t, gap_t, logp_x, s);
  if (e != cudaSuccess) return cuda_fail(e, "readout combine launch");
  return ALR_OK;
}

size_t alr_topk_fwd_workspace_size(const alr_params* p) {
  if (check_params(p) != ALR_OK) return 0;
  DevInfo info;
  if (device_info(&info) != ALR_OK) return 0;
  return fwd_layout(p, info.sms, alr::kKFields, true).total;
}

}  // extern "C"

namespace {

// The top-k + tail forward; with Zd given the fused kernel also writes z_d (kModeTopkFwdKeep).
int topk_fwd_impl(const alr_params* p, const void* Hd, const void* W, const int32_t* top_idx,
                  const float* top_prob, const float* tail, const float* row_mask,
                  const float* weight_in, void* Zd, uint16_t* Zd_ref,
                  const alr_topk_fwd_outputs* out, void* workspace, size_t ws_bytes,
                  void* stream) {
  int rc = check_params(p);
  if (rc != ALR_OK) return rc;
  if ((rc = check_topk_labels(p, top_idx, top_prob, tail)) != ALR_OK) return rc;
  if (Hd == nullptr || W == nullptr || out == nullptr || out->loss_row == nullptr ||
      out->lse_d == nullptr || out->tail_q == nullptr || out->argmax_d == nullptr ||
      out->weight == nullptr || out->loss_total == nullptr || out->weight_sum == nullptr)
    return fail(ALR_ERR_INVALID_ARG, "a required top-k forward pointer is NULL");
  if (!aligned16(Hd) || !aligned16(W))
    return fail(ALR_ERR_INVALID_ARG, "Hd and W must be 16-byte aligned");
  DevInfo info;
  if ((rc = require_sm103(&info)) != ALR_OK) return rc;
  const FwdLayout lay = fwd_layout(p, info.sms, alr::kKFields, true);
  if ((rc = check_workspace(workspace, ws_bytes, lay.total)) != ALR_OK) return rc;
  const int dt = p->dtype;
  const size_t es = elem_size(dt);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  CUtensorMap m_h, m_w;
  if ((rc = make_map(&m_h, Hd, dt, p->d, p->N, p->d * es, k_per_row(dt), 128)) != ALR_OK) return rc;
  if ((rc = head_map(&m_w, p, W, ws + lay.wt_off, s)) != ALR_OK) return rc;
  alr::LossArgs args{};
  args.plan = loss_plan(p, info.sms, false, true);
  args.part = reinterpret_cast<float*>(ws + lay.part_off);
  args.top_idx = top_idx;
  args.zd_out = Zd;
  args.zd_ref = Zd_ref;
  args.status = alr::device_status_ptr();
  if (args.status == nullptr) return fail(ALR_ERR_CUDA, "status word lookup failed");
  CUtensorMap m_zd = m_w;
  if (Zd != nullptr && dt == ALR_BF16 &&
      (rc = make_map(&m_zd, Zd, kMapF16, p->V, p->N, uint64_t(p->V) * 2, 16, 32,
                     CU_TENSOR_MAP_SWIZZLE_NONE)) != ALR_OK)
    return rc;
  cudaError_t e = alr::launch_loss_kernel(Zd != nullptr ? alr::kModeTopkFwdKeep : alr::kModeTopkFwd,
                                          dt, m_h, m_h, m_w, m_zd, m_zd, args, s);
  if (e != cudaSuccess) return cuda_fail(e, "top-k forward kernel launch");
  double* anchor = reinterpret_cast<double*>(ws + lay.anchor_off);
  e = alr::launch_topk_combine(args.plan, args.part, top_prob, tail, row_mask, weight_in, p->gamma,
                               out->loss_row, out->lse_d, out->tail_q, out->argmax_d, out->gap_d,
                               out->weight, anchor, s);
  if (e != cudaSuccess) return cuda_fail(e, "top-k combine launch");
  e = alr::launch_finalize(anchor, int(p->N / p->B), p->lambda, out->loss_total, out->weight_sum,
                          out->wl_sum, s);
  if (e != cudaSuccess) return cuda_fail(e, "finalize launch");
  return ALR_OK;
}

}  // namespace

extern "C" {

int alr_topk_loss_fwd(const alr_params* p, const void* Hd, const void* W, const int32_t* top_idx,
                      const float* top_prob, const float* tail, const float* row_mask,
                      const float* weight_in, const alr_topk_fwd_outputs* out, void* workspace,
                      size_t ws_bytes, void* stream) {
  ALR_RANGE();
  return topk_fwd_impl(p, Hd, W, top_idx, top_prob, tail, row_mask, weight_in, nullptr, nullptr,
                       out, workspace, ws_bytes, stream);
}

int alr_topk_loss_fwd_keep_logits(const alr_params* p, const void* Hd, const void* W,
                                  const int32_t* top_idx, const float* top_prob, const float* tail,
                                  const float* row_mask, const float* weight_in, void* Zd,
                                  uint16_t* Zd_ref, const alr_topk_fwd_outputs* out,
                                  void* workspace, size_t ws_bytes, void* stream) {
  ALR_RANGE();
  int rc = check_params(p);
  if (rc != ALR_OK) return rc;
  if ((rc = check_kept(p, Zd, Zd_ref, "Zd")) != ALR_OK) return rc;
  return topk_fwd_impl(p, Hd, W, top_idx, top_prob, tail, row_mask, weight_in, Zd, Zd_ref, out,
                       workspace, ws_bytes, stream);
}

int alr_topk_logit_grad_from_logits(const alr_params* p, const void* Zd, const uint16_t* Zd_ref,
                                    const int32_t* top_idx, const float* top_prob,
                                    const float* tail, const float* weight,
                                    const float* weight_sum, const float* lse_d,
                                    const float* tail_q, void* G, void* stream) {
  ALR_RANGE();
  int rc = check_params(p);
  if (rc != ALR_OK) return rc;
  if ((rc = check_topk_labels(p, top_idx, top_prob, tail)) != ALR_OK) return rc;
  if ((rc = check_kept(p, Zd, Zd_ref, "Zd")) != ALR_OK) return rc;
  if (G == nullptr || weight == nullptr || weight_sum == nullptr || lse_d == nullptr ||
      tail_q == nullptr)
    return fail(ALR_ERR_INVALID_ARG, "a required pointer is NULL");
  if (!aligned16(G)) return fail(ALR_ERR_INVALID_ARG, "G must be 16-byte aligned");
  DevInfo info;
  if ((rc = require_sm103(&info)) != ALR_OK) return rc;
  cudaError_t e = alr::launch_topk_logits_grad(p->dtype, Zd, Zd_ref, top_idx, top_prob, tail,
                                               tail_q, lse_d, weight, weight_sum, p->lambda,
                                               int(p->N), p->V, G,
                                               static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "top-k logit-gradient launch");
  return ALR_OK;
}

int alr_topk_loss_bwd_from_logits(const alr_params* p, const void* Hd, const void* W,
                                  const void* Zd, const uint16_t* Zd_ref,
                                  const int32_t* top_idx, const float* top_prob,
                                  const float* tail, const float* weight, const float* weight_sum,
                                  const float* lse_d, const float* tail_q, void* G, float* dHd,
                                  float* dW, void* workspace, size_t ws_bytes, void* stream) {
  ALR_RANGE();
  // everything is validated before the gradient kernel overwrites anything
  int rc = check_head_grad_args(p, Hd, W, dHd, dW, workspace, ws_bytes);
  if (rc != ALR_OK) return rc;
  if ((rc = alr_topk_logit_grad_from_logits(p, Zd, Zd_ref, top_idx, top_prob, tail, weight,
                                            weight_sum, lse_d, tail_q, G, stream)) != ALR_OK)
    return rc;
  DevInfo info;
  if ((rc = require_sm103(&info)) != ALR_OK) return rc;
  return head_grads_impl(p, Hd, W, G, dHd, dW, static_cast<uint8_t*>(workspace),
                         bwd_layout(p, false), info, static_cast<cudaStream_t>(stream));
}

int alr_topk_logit_grad(const alr_params* p, const void* Hd, const void* W,
                        const int32_t* top_idx, const float* top_prob, const float* tail,
                        const float* weight, const float* weight_sum, const float* lse_d,
                        const float* tail_q, void* G, void* workspace, size_t ws_bytes,
                        void* stream) {
  ALR_RANGE();
  DevInfo info;
  int rc = check_bwd_args(p, Hd, Hd, W, weight, weight_sum, lse_d, lse_d, &info);
  if (rc != ALR_OK) return rc;
  if ((rc = check_topk_labels(p, top_idx, top_prob, tail)) != ALR_OK) return rc;
  if (tail_q == nullptr) return fail(ALR_ERR_INVALID_ARG, "tail_q is NULL");
  if (G == nullptr || !aligned16(G)) return fail(ALR_ERR_INVALID_ARG, "G must be non-NULL and 16-byte aligned");
  if ((rc = check_workspace(workspace, ws_bytes, alr_logit_grad_workspace_size(p))) != ALR_OK) return rc;
  TopkLabels lab;
  lab.idx = top_idx;
  lab.prob = top_prob;
  lab.tail = tail;
  lab.tail_q = tail_q;
  return logit_grad_impl(p, Hd, nullptr, W, weight, weight_sum, lse_d, nullptr, lab, G, workspace,
                         info, static_cast<cudaStream_t>(stream));
}

int alr_topk_loss_bwd(const alr_params* p, const void* Hd, const void* W, const int32_t* top_idx,
                      const float* top_prob, const float* tail, const float* weight,
                      const float* weight_sum, const float* lse_d, const float* tail_q,
                      float* dHd, float* dW, void* workspace, size_t ws_bytes, void* stream) {
  ALR_RANGE();
  DevInfo info;
  int rc = check_bwd_args(p, Hd, Hd, W, weight, weight_sum, lse_d, lse_d, &info);
  if (rc != ALR_OK) return rc;
  if ((rc = check_topk_labels(p, top_idx, top_prob, tail)) != ALR_OK) return rc;
  if (tail_q == nullptr || dHd == nullptr) return fail(ALR_ERR_INVALID_ARG, "tail_q and dHd must be non-NULL");
  if (!aligned16(dHd) || (dW != nullptr && !aligned16(dW)))
    return fail(ALR_ERR_INVALID_ARG, "dHd and dW must be 16-byte aligned");
  if ((rc = check_workspace(workspace, ws_bytes, alr_bwd_workspace_size(p))) != ALR_OK) return rc;
  const BwdLayout lay = bwd_layout(p);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  void* G = ws + lay.g_off;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  TopkLabels lab;
  lab.idx = top_idx;
  lab.prob = top_prob;
  lab.tail = tail;
  lab.tail_q = tail_q;
  rc = logit_grad_impl(p, Hd, nullptr, W, weight, weight_sum, lse_d, nullptr, lab, G,
                       ws + lay.wt_off, info, s);
  if (rc != ALR_OK) return rc;
  return head_grads_impl(p, Hd, W, G, dHd, dW, ws, lay, info, s);
}

int alr_loss_from_sums(const float* wl_sum, const float* weight_sum, float lambda,
                       float* loss_total, void* stream) {
  ALR_RANGE();
  if (wl_sum == nullptr || weight_sum == nullptr || loss_total == nullptr)
    return fail(ALR_ERR_INVALID_ARG, "wl_sum, weight_sum and loss_total must be non-NULL");
  if (!(lambda == lambda)) return fail(ALR_ERR_INVALID_ARG, "lambda is NaN");
  DevInfo info;
  int rc = require_sm103(&info);
  if (rc != ALR_OK) return rc;
  cudaError_t e = alr::launch_loss_from_sums(wl_sum, weight_sum, lambda, loss_total,
                                             static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "loss-from-sums launch");
  return ALR_OK;
}

int alr_ira_blocks(int32_t S, int32_t K, int32_t max_blocks, const int32_t* valid_anchors,
                   const int32_t* rollout_len, const int32_t* offsets, const int32_t* rollout_tok,
                   const int32_t* corpus_anchor_tok, int32_t* seq, int32_t* pos,
                   int32_t* valid_len, int32_t* ctx_len, int32_t* anchor_tok, void* stream) {
  ALR_RANGE();
  if (S < 0 || K < 2 || max_blocks < 1)
    return fail(ALR_ERR_INVALID_ARG, "bad sizes S=%d K=%d max_blocks=%d", S, K, max_blocks);
  if (S == 0) return ALR_OK;
  if (valid_anchors == nullptr || rollout_len == nullptr || seq == nullptr || pos == nullptr ||
      valid_len == nullptr || (max_blocks > 1 && offsets == nullptr))
    return fail(ALR_ERR_INVALID_ARG,
                "valid_anchors, rollout_len, offsets, seq, pos and valid_len must be non-NULL");
  DevInfo info;
  int rc = require_sm103(&info);
  if (rc != ALR_OK) return rc;
  cudaError_t e = alr::launch_ira_blocks(S, K, max_blocks, valid_anchors, rollout_len, offsets,
                                         rollout_tok, corpus_anchor_tok, seq, pos, valid_len,
                                         ctx_len, anchor_tok, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "IRA block plan launch");
  return ALR_OK;
}

int alr_ira_draw(int32_t S, int32_t L, int32_t K, int32_t max_blocks, const uint8_t* anchor_ok,
                 const uint32_t* keys, const uint32_t* offset_u, int32_t* n_valid,
                 int32_t* anchor_pos, int32_t* offsets, void* stream) {
  ALR_RANGE();
  if (S < 0 || L < 1 || L > ALR_IRA_MAX_LEN || K < 3 || max_blocks < 1)
    return fail(ALR_ERR_INVALID_ARG, "bad sizes S=%d L=%d (at most %d) K=%d max_blocks=%d", S, L,
                ALR_IRA_MAX_LEN, K, max_blocks);
  if (S == 0) return ALR_OK;
  if (anchor_ok == nullptr || keys == nullptr || n_valid == nullptr || anchor_pos == nullptr ||
      (max_blocks > 1 && (offset_u == nullptr || offsets == nullptr)))
    return fail(ALR_ERR_INVALID_ARG,
                "anchor_ok, keys, offset_u, n_valid, anchor_pos and offsets must be non-NULL");
  DevInfo info;
  int rc = require_sm103(&info);
  if (rc != ALR_OK) return rc;
  cudaError_t e = alr::launch_ira_draw(S, L, K, max_blocks, anchor_ok, keys, offset_u, n_valid,
                                       anchor_pos, offsets, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "IRA draw launch");
  return ALR_OK;
}

int alr_ira_context(const void* store, int32_t C, int32_t F, int32_t dtype, int32_t S, int32_t K,
                    int32_t max_blocks, const int32_t* n_valid, const int32_t* rollout_len,
                    const int32_t* offsets, const int32_t* anchor_pos, void* ctx,
                    int32_t* ctx_len, int32_t* prefix_end, void* stream) {
  ALR_RANGE();
  if (dtype != ALR_BF16 && dtype != ALR_F32) return fail(ALR_ERR_UNSUPPORTED, "dtype %d", dtype);
  if (S < 0 || K < 3 || max_blocks < 2 || C < K - 2 || F < 1)
    return fail(ALR_ERR_INVALID_ARG,
                "bad sizes S=%d K=%d max_blocks=%d C=%d (at least K-2) F=%d", S, K, max_blocks, C,
                F);
  if ((size_t(F) * elem_size(dtype)) % 16 != 0)
    return fail(ALR_ERR_INVALID_ARG, "F * element size must be a multiple of 16 bytes");
  if (S == 0) return ALR_OK;
  if (store == nullptr || n_valid == nullptr || rollout_len == nullptr || offsets == nullptr ||
      anchor_pos == nullptr || ctx == nullptr)
    return fail(ALR_ERR_INVALID_ARG,
                "store, n_valid, rollout_len, offsets, anchor_pos and ctx must be non-NULL");
  if (!aligned16(store) || !aligned16(ctx))
    return fail(ALR_ERR_INVALID_ARG, "store and ctx must be 16-byte aligned");
  DevInfo info;
  int rc = require_sm103(&info);
  if (rc != ALR_OK) return rc;
  cudaError_t e = alr::launch_ira_context(store, C, F, int(elem_size(dtype)), S, K, max_blocks,
                                          n_valid, rollout_len, offsets, anchor_pos, ctx, ctx_len,
                                          prefix_end, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "IRA context launch");
  return ALR_OK;
}

int alr_accept_len(const int32_t* argmax_d, const int32_t* argmax_t, const float* active,
                   int32_t A, int32_t B, int32_t* acc_len, int64_t* hist, void* stream) {
  ALR_RANGE();
  if (A < 0 || B < 1 || B > 32) return fail(ALR_ERR_INVALID_ARG, "bad sizes A=%d B=%d", A, B);
  if (A > 0 && (argmax_d == nullptr || argmax_t == nullptr || acc_len == nullptr))
    return fail(ALR_ERR_INVALID_ARG, "argmax_d, argmax_t and acc_len must be non-NULL");
  DevInfo info;
  int rc = require_sm103(&info);
  if (rc != ALR_OK) return rc;
  if (A == 0) {   // no anchors: an all-zero histogram, no kernel to launch
    if (hist == nullptr) return ALR_OK;
    cudaError_t e = cudaMemsetAsync(hist, 0, sizeof(int64_t) * size_t(B + 1),
                                    static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "histogram clear");
    return ALR_OK;
  }
  cudaError_t e = alr::launch_accept_len(argmax_d, argmax_t, active, A, B, acc_len, hist,
                                         static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "accept_len launch");
  return ALR_OK;
}

int alr_erase_weights(const float* logp_x, const int32_t* corpus_tok, const int32_t* argmax_t,
                      const float* row_mask, int32_t A, int32_t B, float gamma, int32_t hard,
                      float* weight, void* stream) {
  ALR_RANGE();
  if (A < 0 || B < 1 || B > 32) return fail(ALR_ERR_INVALID_ARG, "bad sizes A=%d B=%d", A, B);
  if (!(gamma > 0.f)) return fail(ALR_ERR_INVALID_ARG, "gamma must be > 0");
  if (A == 0) return ALR_OK;
  if (weight == nullptr) return fail(ALR_ERR_INVALID_ARG, "weight must be non-NULL");
  if (hard ? (corpus_tok == nullptr || argmax_t == nullptr) : (logp_x == nullptr))
    return fail(ALR_ERR_INVALID_ARG, "the %s gate needs %s", hard ? "hard" : "soft",
                hard ? "corpus_tok and argmax_t" : "logp_x");
  DevInfo info;
  int rc = require_sm103(&info);
  if (rc != ALR_OK) return rc;
  cudaError_t e = alr::launch_erase_weights(logp_x, corpus_tok, argmax_t, row_mask, A, B, gamma,
                                            hard, weight, static_cast<cudaStream_t>(stream));
  if (e != cudaSuccess) return cuda_fail(e, "erase_weights launch");
  return ALR_OK;
}

int alr_gemm(int32_t dtype, int32_t a_mn, int32_t b_mn, int32_t accumulate, const void* A,
             const void* B, float* C, int32_t M, int32_t Nc, int32_t K, void* stream) {
  ALR_RANGE();
  if (dtype != ALR_BF16 && dtype != ALR_F32) return fail(ALR_ERR_UNSUPPORTED, "dtype %d", dtype);
  if (M < 1 || Nc < 1 || K < 1) return fail(ALR_ERR_INVALID_ARG, "bad sizes M=%d Nc=%d K=%d", M, Nc, K);
  if (A == nullptr || B == nullptr || C == nullptr)
    return fail(ALR_ERR_INVALID_ARG, "A, B and C must be non-NULL");
  if (!aligned16(A) || !aligned16(B) || !aligned16(C))
    return fail(ALR_ERR_INVALID_ARG, "A, B and C must be 16-byte aligned");
  if (dtype == ALR_F32 && (a_mn || b_mn))
    return fail(ALR_ERR_UNSUPPORTED, "fp32 (tf32) operands must be K-major");
  const size_t es = elem_size(dtype);
  const int64_t a_inner = a_mn ? M : K, b_inner = b_mn ? Nc : K;
  if ((a_inner * es) % 16 != 0 || (b_inner * es) % 16 != 0 || Nc % 4 != 0)
    return fail(ALR_ERR_INVALID_ARG, "row strides must be multiples of 16 bytes and Nc %% 4 == 0");
  DevInfo info;
  int rc = require_sm103(&info);
  if (rc != ALR_OK) return rc;
  const uint32_t kke = k_per_row(dtype);
  CUtensorMap ma, mb;
  if (a_mn) rc = make_map(&ma, A, dtype, M, K, M * es, kke, kke);
  else rc = make_map(&ma, A, dtype, K, M, K * es, kke, 128);
  if (rc != ALR_OK) return rc;
  if (b_mn) rc = make_map(&mb, B, dtype, Nc, K, Nc * es, kke, kke);
  else rc = make_map(&mb, B, dtype, K, Nc, K * es, kke, gemm_b_rows(dtype));
  if (rc != ALR_OK) return rc;
  return launch_gemm(dtype, a_mn != 0, b_mn != 0, accumulate != 0, ma, mb, M, Nc, K, C, Nc,
                     info.sms, static_cast<cudaStream_t>(stream), "gemm launch");
}

}  // extern "C"
