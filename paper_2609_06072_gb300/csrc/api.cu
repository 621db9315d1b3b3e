// Host side of the C ABI declared in include/ace.h: plan validation,
// workspace layout, argument checks and kernel launches.  No entry point
// allocates device memory or synchronises (except ace_get_error).
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <new>

#include "ace_internal.cuh"

using namespace ace;

namespace {
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                  const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn tensor_map_encoder() {
  static EncodeTiledFn fn = nullptr;
  static bool tried = false;
  if (!tried) {
    tried = true;
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  }
  return fn;
}
}  // namespace

bool ace::make_tmap_bf16(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  EncodeTiledFn fn = tensor_map_encoder();
  if (!fn || rows == 0 || cols == 0) return false;
  cuuint64_t gdim[2] = {cols, rows};
  cuuint64_t gstr[1] = {cols * 2};
  cuuint32_t box[2] = {64, box_rows};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), gdim, gstr, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool ace::make_tmap_f32(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows) {
  EncodeTiledFn fn = tensor_map_encoder();
  if (!fn || rows == 0 || cols == 0) return false;
  cuuint64_t gdim[2] = {cols, rows};
  cuuint64_t gstr[1] = {cols * 4};
  cuuint32_t box[2] = {32, box_rows};
  cuuint32_t es[2] = {1, 1};
  return fn(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), gdim, gstr, box, es,
            CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

namespace {

thread_local char g_msg[512] = "";

ace_status fail(ace_status st, const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_msg, sizeof(g_msg), fmt, ap);
  va_end(ap);
  return st;
}

}  // namespace

// The thread's last host-side error message, for the other translation units.
ace_status ace::report(ace_status st, const char* msg) {
  snprintf(g_msg, sizeof(g_msg), "%s", msg);
  return st;
}

namespace {

ace_status cuda_status(cudaError_t e, const char* what) {
  if (e == cudaSuccess) return ACE_OK;
  return fail(ACE_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

ace_status check_perm(const ace_plan* plan, const ace_perm* perm) {
  if (!plan || !perm || !perm->ws) return fail(ACE_ERR_ARG, "null plan or perm");
  if (perm->T < 0 || perm->T > plan->T_max) return fail(ACE_ERR_SHAPE, "perm T=%d outside [0, %d]", perm->T, plan->T_max);
  if (perm->R != perm->T * plan->pt.k) return fail(ACE_ERR_ARG, "perm R does not match T*k");
  return ACE_OK;
}

// Row tiles per backward split.  A split's dH accumulators (tiles x rank_pad
// TMEM columns) sit below its double-buffered weight-gradient accumulators
// (2 x rank_pad), so at rank_pad 128 a split takes two tiles (down's phase-2
// dh buffer reuses the dH columns).
int pt_nt_split(int rank_pad) { return bwd_nt_split(rank_pad, false); }
int pt_nt_split_sh(int rank_pad) { return bwd_nt_split(rank_pad, true); }

struct BwdWs {
  float* dHrow[2];
  float* part_dBt[2];
  float* part_dA;
  uint16_t* dHx;
  size_t total;
};

int n_rank_pad_of(const PlanTables& pt) { return (pt.rank_off[pt.G] + 63) / 64 * 64; }

// Backward scratch: dH per row (fp32, per projection), the deterministic
// split-K partials of dB^T (per projection) and dA (down), and the
// token-major dense dH of gate/up (bf16).
BwdWs bwd_layout(const ace_plan* plan, int32_t T, void* base) {
  const PlanTables& pt = plan->pt;
  const PermLayout L = perm_layout(pt, T);
  const int64_t R = (int64_t)T * pt.k;
  const size_t dhrow = align_up(4 * (size_t)R * pt.rank_pad, 256);
  const size_t n_part = (size_t)(L.max_splits > L.max_splits_sh ? L.max_splits : L.max_splits_sh);
  const size_t pa = align_up(4 * n_part * pt.rank_pad * (size_t)(pt.d > pt.f ? pt.d : pt.f), 256);
  BwdWs w{};
  char* b = static_cast<char*>(base);
  size_t off = 0;
  for (int j = 0; j < 2; ++j) {
    w.dHrow[j] = reinterpret_cast<float*>(b + off);
    off += dhrow;
    w.part_dBt[j] = reinterpret_cast<float*>(b + off);
    off += pa;
  }
  w.part_dA = reinterpret_cast<float*>(b + off);
  off += pa;
  w.dHx = reinterpret_cast<uint16_t*>(b + off);
  off += align_up(2 * (size_t)T * 2 * n_rank_pad_of(pt), 256);
  w.total = off;
  return w;
}

}  // namespace

// H_u = A_g x_t per unique pair (g, t) of gate/up into Hbuf[j] (fp32, stride
// rank_max): token-major dense tiles when the stacked ranks of a projection
// are few (the MMA then also forms the products of the groups a token skips,
// cheaper than gathering X once per active group), else gathered per unique
// pair.
namespace ace {
ace_status launch_gate_up_h(const ace_plan* plan, const ace_perm* perm, const uint16_t* X, int nproj,
                            const uint16_t* const* A, float* const* Hbuf, cudaStream_t cs) {
  const PlanTables& pt = plan->pt;
  const PermLayout L = perm_layout(pt, perm->T);
  const int n_rank = pt.rank_off[pt.G];
  const int d_in = pt.d;
  int32_t* err = at<int32_t>(perm->ws, L.err);
  ace_status st = ACE_OK;
  if (n_rank <= kDenseHMaxRank) {
    DenseHLaunch h{};
    bool okh = make_tmap_bf16(&h.tm_x, X, (uint64_t)perm->T, (uint64_t)d_in, kTileM);
    for (int j = 0; j < nproj; ++j) okh = okh && make_tmap_bf16(&h.tm_a[j], A[j], (uint64_t)n_rank, (uint64_t)d_in, 256);
    if (!okh) return fail(ACE_ERR_UNSUPPORTED, "tensor-map encoding failed for this layout");
    h.tok_uniq = perm->tok_uniq;
    h.uniq_off = perm->uniq_off;
    for (int j = 0; j < 2; ++j) h.H[j] = Hbuf[j < nproj ? j : 0];
    h.T = perm->T;
    h.d = d_in;
    h.n_rank = n_rank;
    h.nproj = nproj;
    h.rank_max = pt.rank_max;
    h.grid = plan->num_sms;
    h.err = err;
    st = cuda_status(launch_dense_h(pt, h, cs), "forward H launch");
  } else {
    FwdHLaunch h{};
    h.tiles = at<Tile>(perm->ws, L.tiles_sh);
    h.counts = perm->counts;
    h.max_tiles = L.max_tiles;
    h.uniq_tok = perm->uniq_tok;
    h.X = X;
    for (int j = 0; j < 2; ++j) {
      const int jj = j < nproj ? j : 0;
      h.A[j] = A[jj];
      h.H[j] = Hbuf[jj];
    }
    h.d_in = d_in;
    h.nproj = nproj;
    h.n_src = perm->T;
    h.err = err;
    st = cuda_status(launch_fwd_h(pt, h, cs), "forward H launch");
  }
  return st;
}
}  // namespace ace

extern "C" {

int32_t ace_version(void) { return ACE_VERSION; }

int32_t ace_build_checks(void) { return kChecks ? 1 : 0; }

const char* ace_last_error_message(void) { return g_msg; }

ace_status ace_plan_create(ace_plan** out, const ace_layer_desc* desc) {
  if (!out || !desc) return fail(ACE_ERR_ARG, "null argument");
  *out = nullptr;
  const ace_layer_desc& D = *desc;
  if (!D.e2g || !D.rank_off) return fail(ACE_ERR_ARG, "null e2g / rank_off");
  if (D.E < 1 || D.E > ACE_MAX_EXPERTS) return fail(ACE_ERR_SHAPE, "E=%d outside [1, %d]", D.E, ACE_MAX_EXPERTS);
  if (D.G < 1 || D.G > D.E) return fail(ACE_ERR_SHAPE, "G=%d outside [1, E]", D.G);
  if (D.k < 1 || D.k > D.E || D.k > kMaxK) return fail(ACE_ERR_SHAPE, "k=%d outside [1, min(E, %d)]", D.k, kMaxK);
  if (D.T_max < 0) return fail(ACE_ERR_SHAPE, "T_max < 0");
  if ((int64_t)D.T_max * D.k > (int64_t)1 << 30) return fail(ACE_ERR_SHAPE, "T_max * k too large");
  if (D.d < 8 || D.f < 8 || D.d % 8 || D.f % 8) return fail(ACE_ERR_SHAPE, "d=%d, f=%d must be positive multiples of 8", D.d, D.f);
  int used[ACE_MAX_EXPERTS] = {0};
  for (int e = 0; e < D.E; ++e) {
    if (D.e2g[e] < 0 || D.e2g[e] >= D.G) return fail(ACE_ERR_INDEX, "e2g[%d]=%d outside [0, G)", e, D.e2g[e]);
    used[D.e2g[e]] = 1;
  }
  for (int g = 0; g < D.G; ++g)
    if (!used[g]) return fail(ACE_ERR_INDEX, "group %d has no expert", g);
  if (D.rank_off[0] != 0) return fail(ACE_ERR_ARG, "rank_off[0] must be 0");
  int rank_max = 0;
  for (int g = 0; g < D.G; ++g) {
    const int rg = D.rank_off[g + 1] - D.rank_off[g];
    if (rg < 1) return fail(ACE_ERR_ARG, "r_%d=%d < 1", g, rg);
    if (rg > ACE_MAX_RANK) return fail(ACE_ERR_UNSUPPORTED, "r_%d=%d > %d", g, rg, ACE_MAX_RANK);
    rank_max = rg > rank_max ? rg : rank_max;
  }
  int dev = 0;
  cudaError_t ce = cudaGetDevice(&dev);
  if (ce != cudaSuccess) return cuda_status(ce, "cudaGetDevice");
  int major = 0, minor = 0;
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  if (!(major == 10 && minor == 3))
    return fail(ACE_ERR_UNSUPPORTED, "device %d is sm_%d%d; this library is built for sm_103a only", dev, major, minor);
  int num_sms = 0;
  ce = cudaDeviceGetAttribute(&num_sms, cudaDevAttrMultiProcessorCount, dev);
  if (ce != cudaSuccess || num_sms <= 0) return cuda_status(ce, "multiprocessor count");
  ace_plan* p = new (std::nothrow) ace_plan();
  if (!p) return fail(ACE_ERR_ARG, "out of host memory");
  std::memset(&p->pt, 0, sizeof(p->pt));
  p->pt.E = D.E;
  p->pt.G = D.G;
  p->pt.k = D.k;
  p->pt.d = D.d;
  p->pt.f = D.f;
  p->pt.rank_max = rank_max;
  p->pt.rank_pad = rank_max <= 16 ? 16 : rank_max <= 32 ? 32 : rank_max <= 64 ? 64 : 128;
  p->pt.nt_split = pt_nt_split(p->pt.rank_pad);
  p->pt.nt_split_sh = pt_nt_split_sh(p->pt.rank_pad);
  p->pt.nsm = num_sms;
  for (int e = 0; e < D.E; ++e) p->pt.e2g[e] = (int16_t)D.e2g[e];
  {
    int pos = 0;
    for (int g = 0; g < D.G; ++g) {
      p->pt.gfirst[g] = (int16_t)pos;
      for (int e = 0; e < D.E; ++e)
        if (D.e2g[e] == g) p->pt.eorder[pos++] = (int16_t)e;
    }
  }
  for (int g = 0; g <= D.G; ++g) p->pt.rank_off[g] = D.rank_off[g];
  p->T_max = D.T_max;
  p->flags = D.flags;
  p->device = dev;
  p->num_sms = num_sms;
  *out = p;
  return ACE_OK;
}

void ace_plan_destroy(ace_plan* plan) { delete plan; }

int32_t ace_plan_rank_max(const ace_plan* plan) { return plan ? plan->pt.rank_max : 0; }

int32_t ace_plan_rank_cols(const ace_plan* plan) { return plan ? n_rank_pad_of(plan->pt) : 0; }

ace_status ace_workspace_size(const ace_plan* plan, int32_t T, size_t* perm_bytes, size_t* fwd_bytes,
                              size_t* bwd_bytes) {
  if (!plan) return fail(ACE_ERR_ARG, "null plan");
  if (T < 0 || T > plan->T_max) return fail(ACE_ERR_SHAPE, "T=%d outside [0, %d]", T, plan->T_max);
  if (perm_bytes) *perm_bytes = perm_layout(plan->pt, T).total;
  if (fwd_bytes) *fwd_bytes = 2 * align_up(4 * (size_t)T * plan->pt.k * plan->pt.rank_max, 256);
  if (bwd_bytes) *bwd_bytes = bwd_layout(plan, T, nullptr).total;
  return ACE_OK;
}

ace_status ace_permute(const ace_plan* plan, const int32_t* topk_idx, int32_t T, void* perm_ws, size_t perm_ws_bytes,
                       ace_perm* out, void* stream) {
  if (!plan || !out || !perm_ws) return fail(ACE_ERR_ARG, "null argument");
  if (T < 0 || T > plan->T_max) return fail(ACE_ERR_SHAPE, "T=%d outside [0, %d]", T, plan->T_max);
  if (T > 0 && !topk_idx) return fail(ACE_ERR_ARG, "null topk_idx");
  const PermLayout L = perm_layout(plan->pt, T);
  if (perm_ws_bytes < L.total) return fail(ACE_ERR_WORKSPACE, "perm workspace %zu < %zu bytes", perm_ws_bytes, L.total);
  if (!aligned16(perm_ws) || (topk_idx && (reinterpret_cast<uintptr_t>(topk_idx) & 3u)))
    return fail(ACE_ERR_WORKSPACE, "misaligned workspace or topk_idx");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  ace_status s = cuda_status(launch_permute(plan->pt, topk_idx, T, perm_ws, L, st), "permute launch");
  if (s != ACE_OK) return s;
  out->T = T;
  out->R = T * plan->pt.k;
  out->counts = at<int32_t>(perm_ws, L.counts);
  out->group_off = at<int32_t>(perm_ws, L.group_off);
  out->expert_off = at<int32_t>(perm_ws, L.expert_off);
  out->expert_cnt = at<int32_t>(perm_ws, L.expert_cnt);
  out->row_pair = at<int32_t>(perm_ws, L.row_pair);
  out->pair_row = at<int32_t>(perm_ws, L.pair_row);
  out->uniq_off = at<int32_t>(perm_ws, L.uniq_off);
  out->uniq_tok = at<int32_t>(perm_ws, L.uniq_tok);
  out->tok_uniq = at<int32_t>(perm_ws, L.tok_uniq);
  out->row_uniq = at<int32_t>(perm_ws, L.row_uniq);
  out->ws = perm_ws;
  return ACE_OK;
}

static ace_status fwd_common(const ace_plan* plan, const ace_perm* perm, const uint16_t* X, int nproj,
                             const uint16_t* const* A, const uint16_t* const* Bt, float s, uint16_t* const* Y,
                             float* const* H, bool shared, void* ws, size_t ws_bytes, void* stream) {
  ace_status st = check_perm(plan, perm);
  if (st != ACE_OK) return st;
  if (nproj < 1 || nproj > 2) return fail(ACE_ERR_ARG, "nproj=%d must be 1 or 2", nproj);
  if (!A || !Bt || !Y) return fail(ACE_ERR_ARG, "null A / Bt / Y array");
  if (perm->R > 0 && !X) return fail(ACE_ERR_ARG, "null input");
  if (X && !aligned16(X)) return fail(ACE_ERR_ARG, "input not 16-byte aligned");
  for (int j = 0; j < nproj; ++j) {
    if (!A[j] || !Bt[j] || (perm->R > 0 && !Y[j])) return fail(ACE_ERR_ARG, "null A / Bt / Y of projection %d", j);
    if (!aligned16(A[j]) || !aligned16(Bt[j]) || (Y[j] && !aligned16(Y[j])) || (H && H[j] && !aligned16(H[j])))
      return fail(ACE_ERR_ARG, "tensor of projection %d not 16-byte aligned", j);
  }
  if (perm->R == 0) return ACE_OK;
  const PlanTables& pt = plan->pt;
  const PermLayout L = perm_layout(pt, perm->T);
  const int64_t R = perm->R;
  const int n_rank = pt.rank_off[pt.G];
  const int d_in = shared ? pt.d : pt.f, d_out = shared ? pt.f : pt.d;
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  int32_t* err = at<int32_t>(perm->ws, L.err);
  // H per unique pair (gate/up) lives in the caller's H buffers or, if absent,
  // in the forward workspace
  float* Hbuf[2] = {nullptr, nullptr};
  for (int j = 0; j < nproj; ++j) Hbuf[j] = H ? H[j] : nullptr;
  if (shared && (!Hbuf[0] || (nproj == 2 && !Hbuf[1]))) {
    const size_t need = 2 * align_up(4 * (size_t)R * pt.rank_max, 256);
    if (!ws || ws_bytes < need || !aligned16(ws))
      return fail(ACE_ERR_WORKSPACE, "forward workspace %zu < %zu bytes (needed when H is NULL)", ws_bytes, need);
    for (int j = 0; j < nproj; ++j)
      if (!Hbuf[j]) Hbuf[j] = reinterpret_cast<float*>(static_cast<char*>(ws) + j * align_up(4 * (size_t)R * pt.rank_max, 256));
  }
  if (shared) {
    st = launch_gate_up_h(plan, perm, X, nproj, A, Hbuf, cs);
    if (st != ACE_OK) return st;
  }
  FwdRowsLaunch r{};
  bool ok = true;
  if (!shared) {
    ok = ok && make_tmap_bf16(&r.tm_x, X, (uint64_t)R, (uint64_t)d_in, kTileM);
    ok = ok && make_tmap_bf16(&r.tm_x16, X, (uint64_t)R, (uint64_t)d_in, 16);
    ok = ok && make_tmap_bf16(&r.tm_a, A[0], (uint64_t)n_rank, (uint64_t)d_in, pt.rank_pad);
  }
  for (int j = 0; j < nproj; ++j) {
    ok = ok && make_tmap_bf16(&r.tm_bt[j], Bt[j], (uint64_t)n_rank, (uint64_t)d_out, pt.rank_pad);
    ok = ok && make_tmap_bf16(&r.tm_y[j], Y[j], (uint64_t)R, (uint64_t)d_out, kTileM);
    ok = ok && make_tmap_bf16(&r.tm_y16[j], Y[j], (uint64_t)R, (uint64_t)d_out, 16);
  }
  if (!ok) return fail(ACE_ERR_UNSUPPORTED, "tensor-map encoding failed for this layout");
  r.tiles = at<Tile>(perm->ws, L.tiles_row);
  r.counts = perm->counts;
  r.sched = at<int32_t>(perm->ws, L.sched);
  r.grid = R > 0 ? plan->num_sms : 0;
  r.row_uniq = at<int32_t>(perm->ws, L.row_uniq);
  for (int j = 0; j < 2; ++j) {
    const int jj = j < nproj ? j : 0;
    r.Hu[j] = Hbuf[jj];
    r.Y[j] = Y[jj];
  }
  r.Hsave = shared ? nullptr : (H ? H[0] : nullptr);
  if (!shared) {
    // the split row tiles' H is computed up front into the saved H, or into
    // the forward workspace when H is not saved (else they run whole)
    r.Hpre = r.Hsave;
    if (!r.Hpre && ws && aligned16(ws) && ws_bytes >= 4 * (size_t)R * pt.rank_max) r.Hpre = static_cast<float*>(ws);
    r.pre = r.Hpre != nullptr;
    r.test_expiry = (plan->flags & ACE_FLAG_TEST_WAIT_EXPIRY) != 0;
  }
  r.s = s;
  r.d_in = d_in;
  r.d_out = d_out;
  r.nproj = nproj;
  r.err = err;
  return cuda_status(launch_fwd_rows(pt, r, shared, cs), "forward rows launch");
}

ace_status ace_fwd_shared(const ace_plan* plan, const ace_perm* perm, const uint16_t* X, int32_t nproj,
                          const uint16_t* const* A, const uint16_t* const* Bt, float s, uint16_t* const* Y,
                          float* const* H, void* ws, size_t ws_bytes, void* stream) {
  if (!plan || !perm) return fail(ACE_ERR_ARG, "null plan or perm");
  return fwd_common(plan, perm, X, nproj, A, Bt, s, Y, H, true, ws, ws_bytes, stream);
}

ace_status ace_fwd_row(const ace_plan* plan, const ace_perm* perm, const uint16_t* Hin, const uint16_t* A,
                       const uint16_t* Bt, float s, uint16_t* Y, float* H, void* ws, size_t ws_bytes, void* stream) {
  const uint16_t* Aa[1] = {A};
  const uint16_t* Ba[1] = {Bt};
  uint16_t* Ya[1] = {Y};
  float* Ha[1] = {H};
  return fwd_common(plan, perm, Hin, 1, Aa, Ba, s, Ya, Ha, false, ws, ws_bytes, stream);
}

ace_status ace_bwd_shared(const ace_plan* plan, const ace_perm* perm, int32_t nproj, const uint16_t* const* dY,
                          const uint16_t* X, const float* const* H, const uint16_t* const* A,
                          const uint16_t* const* Bt, float s, uint16_t* dX, float* const* dA, float* const* dBt,
                          void* ws, size_t ws_bytes, void* stream) {
  ace_status st = check_perm(plan, perm);
  if (st != ACE_OK) return st;
  if (nproj < 1 || nproj > 2) return fail(ACE_ERR_ARG, "nproj=%d must be 1 or 2", nproj);
  // token and row tensors may be null (empty) when the call has no tokens
  if (!dY || !H || !A || !Bt || !dA || !dBt || (perm->T > 0 && (!dX || !X))) return fail(ACE_ERR_ARG, "null argument");
  if ((X && !aligned16(X)) || (dX && !aligned16(dX))) return fail(ACE_ERR_ARG, "X / dX not 16-byte aligned");
  for (int j = 0; j < nproj; ++j) {
    if (!A[j] || !Bt[j] || !dA[j] || !dBt[j] || (perm->R > 0 && (!dY[j] || !H[j])))
      return fail(ACE_ERR_ARG, "null tensor of projection %d", j);
    if ((dY[j] && !aligned16(dY[j])) || (H[j] && !aligned16(H[j])) || !aligned16(A[j]) || !aligned16(Bt[j]) ||
        !aligned16(dA[j]) || !aligned16(dBt[j]))
      return fail(ACE_ERR_ARG, "tensor of projection %d not 16-byte aligned", j);
  }
  const BwdWs need = bwd_layout(plan, perm->T, nullptr);
  if (!ws || ws_bytes < need.total) return fail(ACE_ERR_WORKSPACE, "backward workspace %zu < %zu bytes", ws_bytes, need.total);
  if (!aligned16(ws)) return fail(ACE_ERR_WORKSPACE, "backward workspace misaligned");
  const PermLayout L = perm_layout(plan->pt, perm->T);
  const BwdWs w = bwd_layout(plan, perm->T, ws);
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  BwdLaunch a{};
  bool ok = true;
  for (int j = 0; j < nproj; ++j) {
    ok = ok && make_tmap_bf16(&a.tm_dy[j], dY[j], (uint64_t)perm->R, (uint64_t)plan->pt.f, kTileM);
    ok = ok && make_tmap_bf16(&a.tm_bt[j], Bt[j], (uint64_t)plan->pt.rank_off[plan->pt.G], (uint64_t)plan->pt.f,
                              plan->pt.rank_pad);
  }
  if (perm->R > 0 && !ok) return fail(ACE_ERR_UNSUPPORTED, "tensor-map encoding failed for this layout");
  a.splits_row = at<Tile>(perm->ws, L.splits_row);
  a.splits_sh = at<Tile>(perm->ws, L.splits_sh);
  a.tiles_sh = at<Tile>(perm->ws, L.tiles_sh);
  a.counts = perm->counts;
  a.max_splits_row = L.max_splits;
  a.max_splits_sh = L.max_splits_sh;
  a.max_tiles_sh = L.max_tiles;
  a.uniq_tok = perm->uniq_tok;
  a.uniq_off = perm->uniq_off;
  a.group_off = perm->group_off;
  a.pair_row = perm->pair_row;
  a.pair_g = at<int32_t>(perm->ws, L.pair_g);
  a.row_uniq = at<int32_t>(perm->ws, L.row_uniq);
  a.Xin = X;
  for (int j = 0; j < 2; ++j) {
    const int jj = j < nproj ? j : 0;
    a.H[j] = H[jj];
    a.dA[j] = dA[jj];
    a.dBt[j] = dBt[jj];
    a.dHrow[j] = w.dHrow[jj];
    a.part_dBt[j] = w.part_dBt[jj];
  }
  if (nproj == 1) a.tm_dy[1] = a.tm_dy[0], a.tm_bt[1] = a.tm_bt[0];
  a.dHx = w.dHx;
  a.n_rank_pad = n_rank_pad_of(plan->pt);
  a.s = s;
  a.dXin = nullptr;
  a.d_in = plan->pt.d;
  a.d_out = plan->pt.f;
  a.nproj = nproj;
  a.T = perm->T;
  a.deterministic = (plan->flags & ACE_FLAG_DETERMINISTIC) != 0;
  a.err = at<int32_t>(perm->ws, L.err);
  st = cuda_status(launch_bwd(plan->pt, a, true, cs), "backward launch");
  if (st != ACE_OK) return st;
  if (perm->R == 0) return ACE_OK;
  // dX += dHx . [A_j], dA_j = dHx_j^T . X  (dense, token-major)
  const PlanTables& pt = plan->pt;
  DenseBwdLaunch x{};
  const int n_rank = pt.rank_off[pt.G], nrp = n_rank_pad_of(pt);
  const uint64_t T = (uint64_t)perm->T, kw = (uint64_t)nproj * nrp;
  bool okm = make_tmap_bf16(&x.tm_dhx, w.dHx, T, kw, kTileM) && make_tmap_bf16(&x.tm_dhx_t, w.dHx, T, kw, 64) &&
             make_tmap_bf16(&x.tm_x, X, T, (uint64_t)pt.d, 64) && make_tmap_bf16(&x.tm_dx, dX, T, (uint64_t)pt.d, kTileM);
  for (int j = 0; j < nproj; ++j) {
    okm = okm && make_tmap_bf16(&x.tm_acat[j], A[j], (uint64_t)n_rank, (uint64_t)pt.d, 64);
    okm = okm && make_tmap_f32(&x.tm_da[j], dA[j], (uint64_t)n_rank, (uint64_t)pt.d, 32);
  }
  if (!okm) return fail(ACE_ERR_UNSUPPORTED, "tensor-map encoding failed for this layout");
  if (nproj == 1) x.tm_acat[1] = x.tm_acat[0], x.tm_da[1] = x.tm_da[0];
  x.dX = dX;
  for (int j = 0; j < 2; ++j) x.dA[j] = dA[j < nproj ? j : 0];
  x.T = perm->T;
  x.d = pt.d;
  x.n_rank = n_rank;
  x.n_rank_pad = nrp;
  x.nproj = nproj;
  x.grid = plan->num_sms;
  x.err = a.err;
  return cuda_status(launch_dense_bwd(x, cs), "dense dX / dA launch");
}

ace_status ace_bwd_row(const ace_plan* plan, const ace_perm* perm, const uint16_t* dY, const uint16_t* Hin,
                       const float* H, const uint16_t* A, const uint16_t* Bt, float s, uint16_t* dHin, float* dA,
                       float* dBt, void* ws, size_t ws_bytes, void* stream) {
  ace_status st = check_perm(plan, perm);
  if (st != ACE_OK) return st;
  // row tensors may be null (empty) when the call has no rows
  if (!A || !Bt || !dA || !dBt || (perm->R > 0 && (!dY || !Hin || !H || !dHin)))
    return fail(ACE_ERR_ARG, "null argument");
  if ((dY && !aligned16(dY)) || (Hin && !aligned16(Hin)) || (H && !aligned16(H)) || !aligned16(A) ||
      !aligned16(Bt) || (dHin && !aligned16(dHin)) || !aligned16(dA) || !aligned16(dBt))
    return fail(ACE_ERR_ARG, "tensor not 16-byte aligned");
  const BwdWs need = bwd_layout(plan, perm->T, nullptr);
  if (!ws || ws_bytes < need.total) return fail(ACE_ERR_WORKSPACE, "backward workspace %zu < %zu bytes", ws_bytes, need.total);
  if (!aligned16(ws)) return fail(ACE_ERR_WORKSPACE, "backward workspace misaligned");
  const PermLayout L = perm_layout(plan->pt, perm->T);
  const BwdWs w = bwd_layout(plan, perm->T, ws);
  BwdLaunch a{};
  bool ok = true;
  const uint64_t R = (uint64_t)perm->R, nr = (uint64_t)plan->pt.rank_off[plan->pt.G];
  ok = ok && make_tmap_bf16(&a.tm_dy[0], dY, R, (uint64_t)plan->pt.d, kTileM);
  ok = ok && make_tmap_bf16(&a.tm_bt[0], Bt, nr, (uint64_t)plan->pt.d, plan->pt.rank_pad);
  ok = ok && make_tmap_bf16(&a.tm_a, A, nr, (uint64_t)plan->pt.f, plan->pt.rank_pad);
  ok = ok && make_tmap_bf16(&a.tm_dh, dHin, R, (uint64_t)plan->pt.f, kTileM);
  ok = ok && make_tmap_bf16(&a.tm_h, Hin, R, (uint64_t)plan->pt.f, kTileM);
  if (perm->R > 0 && !ok) return fail(ACE_ERR_UNSUPPORTED, "tensor-map encoding failed for this layout");
  a.tm_dy[1] = a.tm_dy[0];
  a.tm_bt[1] = a.tm_bt[0];
  a.splits_row = at<Tile>(perm->ws, L.splits_row);
  a.splits_sh = at<Tile>(perm->ws, L.splits_sh);
  a.tiles_sh = at<Tile>(perm->ws, L.tiles_sh);
  a.counts = perm->counts;
  a.max_splits_row = L.max_splits;
  a.max_splits_sh = L.max_splits_sh;
  a.max_tiles_sh = L.max_tiles;
  a.uniq_tok = perm->uniq_tok;
  a.uniq_off = perm->uniq_off;
  a.group_off = perm->group_off;
  a.pair_row = perm->pair_row;
  a.pair_g = at<int32_t>(perm->ws, L.pair_g);
  a.row_uniq = at<int32_t>(perm->ws, L.row_uniq);
  a.Xin = Hin;
  for (int j = 0; j < 2; ++j) {
    a.H[j] = H;
    a.dA[j] = dA;
    a.dBt[j] = dBt;
    a.dHrow[j] = w.dHrow[0];
    a.part_dBt[j] = w.part_dBt[0];
    a.part_dA[j] = w.part_dA;
  }
  a.s = s;
  a.dXin = dHin;
  a.d_in = plan->pt.f;
  a.d_out = plan->pt.d;
  a.nproj = 1;
  a.T = perm->T;
  a.deterministic = (plan->flags & ACE_FLAG_DETERMINISTIC) != 0;
  a.err = at<int32_t>(perm->ws, L.err);
  return cuda_status(launch_bwd(plan->pt, a, false, static_cast<cudaStream_t>(stream)), "backward launch");
}

// Gate-weighted combine of down, forward: H per row (the row-tile mode of
// the H kernel), the token-major combined H, then Z += Hx . [B_g^T] with the
// dense dX GEMM.
ace_status ace_fwd_combine(const ace_plan* plan, const ace_perm* perm, const uint16_t* Hin, const float* topk_w,
                           const uint16_t* A, const uint16_t* Bt, float s, uint16_t* Z, float* H, uint16_t* Hx,
                           void* stream) {
  ace_status st = check_perm(plan, perm);
  if (st != ACE_OK) return st;
  if (!A || !Bt || (perm->T > 0 && (!Z || !Hx)) || (perm->R > 0 && (!Hin || !topk_w || !H)))
    return fail(ACE_ERR_ARG, "null argument");
  if (!aligned16(A) || !aligned16(Bt) || (H && !aligned16(H)) || (Hx && !aligned16(Hx)) || (Z && !aligned16(Z)) ||
      (Hin && !aligned16(Hin)) || (reinterpret_cast<uintptr_t>(topk_w) & 3u))
    return fail(ACE_ERR_ARG, "tensor not 16-byte aligned (topk_w: 4-byte)");
  if (perm->R == 0) return ACE_OK;
  const PlanTables& pt = plan->pt;
  const PermLayout L = perm_layout(pt, perm->T);
  const int n_rank = pt.rank_off[pt.G], nrp = n_rank_pad_of(pt);
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  int32_t* err = at<int32_t>(perm->ws, L.err);
  DenseBwdLaunch x{};
  const uint64_t T = (uint64_t)perm->T;
  bool ok = make_tmap_bf16(&x.tm_dhx, Hx, T, (uint64_t)nrp, kTileM) &&
            make_tmap_bf16(&x.tm_acat[0], Bt, (uint64_t)n_rank, (uint64_t)pt.d, 64) &&
            make_tmap_bf16(&x.tm_dx, Z, T, (uint64_t)pt.d, kTileM);
  if (!ok) return fail(ACE_ERR_UNSUPPORTED, "tensor-map encoding failed for this layout");
  FwdHLaunch h{};
  h.tiles = at<Tile>(perm->ws, L.tiles_row);
  h.counts = perm->counts;
  h.max_tiles = L.max_tiles;
  h.rows = 1;
  h.X = Hin;
  h.A[0] = h.A[1] = A;
  h.H[0] = h.H[1] = H;
  h.d_in = pt.f;
  h.nproj = 1;
  h.n_src = perm->R;
  h.err = err;
  st = cuda_status(launch_fwd_h(pt, h, cs), "combine H launch");
  if (st != ACE_OK) return st;
  CombReduceLaunch c{};
  c.H = H;
  c.w = topk_w;
  c.pair_row = perm->pair_row;
  c.pair_g = at<int32_t>(perm->ws, L.pair_g);
  c.Hx = Hx;
  c.s = s;
  c.T = perm->T;
  c.n_rank_pad = nrp;
  c.err = err;
  st = cuda_status(launch_comb_reduce(pt, c, cs), "combine reduce launch");
  if (st != ACE_OK) return st;
  x.tm_acat[1] = x.tm_acat[0];
  x.dX = Z;
  x.T = perm->T;
  x.d = pt.d;
  x.n_rank = n_rank;
  x.n_rank_pad = nrp;
  x.nproj = 1;
  x.grid = plan->num_sms;
  x.err = err;
  return cuda_status(launch_dense_dx(x, cs), "combine output launch");
}

// Gate-weighted combine of down, backward: dHc_u = B_g^T dZ[t] per unique
// pair (the forward's H kernels on dZ and B^T), the row kernel in its combine
// mode (dh, dA, the gate-weight gradient), then dB^T += Hx^T . dZ with the
// dense dA GEMM.
ace_status ace_bwd_combine(const ace_plan* plan, const ace_perm* perm, const uint16_t* dZ, const uint16_t* Hin,
                           const float* topk_w, const float* H, const uint16_t* Hx, const uint16_t* A,
                           const uint16_t* Bt, float s, uint16_t* dHin, float* dtopk_w, float* dA, float* dBt,
                           void* ws, size_t ws_bytes, void* stream) {
  ace_status st = check_perm(plan, perm);
  if (st != ACE_OK) return st;
  if (!A || !Bt || !dA || !dBt ||
      (perm->R > 0 && (!dZ || !Hin || !topk_w || !H || !Hx || !dHin || !dtopk_w)))
    return fail(ACE_ERR_ARG, "null argument");
  if (!aligned16(A) || !aligned16(Bt) || !aligned16(dA) || !aligned16(dBt) || (dZ && !aligned16(dZ)) ||
      (Hin && !aligned16(Hin)) || (H && !aligned16(H)) || (Hx && !aligned16(Hx)) || (dHin && !aligned16(dHin)) ||
      (reinterpret_cast<uintptr_t>(topk_w) & 3u) || (reinterpret_cast<uintptr_t>(dtopk_w) & 3u))
    return fail(ACE_ERR_ARG, "tensor not 16-byte aligned (topk_w, dtopk_w: 4-byte)");
  const BwdWs need = bwd_layout(plan, perm->T, nullptr);
  if (!ws || ws_bytes < need.total) return fail(ACE_ERR_WORKSPACE, "backward workspace %zu < %zu bytes", ws_bytes, need.total);
  if (!aligned16(ws)) return fail(ACE_ERR_WORKSPACE, "backward workspace misaligned");
  const PlanTables& pt = plan->pt;
  const PermLayout L = perm_layout(pt, perm->T);
  const BwdWs w = bwd_layout(plan, perm->T, ws);
  const int n_rank = pt.rank_off[pt.G], nrp = n_rank_pad_of(pt);
  const uint64_t R = (uint64_t)perm->R, T = (uint64_t)perm->T;
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  int32_t* err = at<int32_t>(perm->ws, L.err);
  float* Hc = w.dHrow[0];  // dHc per unique pair, row stride rank_max
  BwdLaunch a{};
  DenseBwdLaunch x{};
  if (perm->R > 0) {
    bool ok = make_tmap_bf16(&a.tm_a, A, (uint64_t)n_rank, (uint64_t)pt.f, pt.rank_pad) &&
              make_tmap_bf16(&a.tm_dh, dHin, R, (uint64_t)pt.f, kTileM) &&
              make_tmap_bf16(&a.tm_h, Hin, R, (uint64_t)pt.f, kTileM) &&
              make_tmap_bf16(&x.tm_dhx_t, Hx, T, (uint64_t)nrp, 64) && make_tmap_bf16(&x.tm_x, dZ, T, (uint64_t)pt.d, 64) &&
              make_tmap_f32(&x.tm_da[0], dBt, (uint64_t)n_rank, (uint64_t)pt.d, 32);
    if (!ok) return fail(ACE_ERR_UNSUPPORTED, "tensor-map encoding failed for this layout");
    // B_g^T dz once per unique (g, t) pair: the same product as the gate/up H
    const uint16_t* Bts[1] = {Bt};
    float* Hcs[1] = {Hc};
    st = launch_gate_up_h(plan, perm, dZ, 1, Bts, Hcs, cs);
    if (st != ACE_OK) return st;
  }
  a.splits_row = at<Tile>(perm->ws, L.splits_row);
  a.splits_sh = at<Tile>(perm->ws, L.splits_sh);
  a.tiles_sh = at<Tile>(perm->ws, L.tiles_sh);
  a.counts = perm->counts;
  a.max_splits_row = L.max_splits;
  a.max_splits_sh = L.max_splits_sh;
  a.max_tiles_sh = L.max_tiles;
  a.uniq_tok = perm->uniq_tok;
  a.uniq_off = perm->uniq_off;
  a.group_off = perm->group_off;
  a.pair_row = perm->pair_row;
  a.pair_g = at<int32_t>(perm->ws, L.pair_g);
  a.row_uniq = at<int32_t>(perm->ws, L.row_uniq);
  a.Xin = Hin;
  a.H[0] = Hc;
  a.H[1] = H;
  for (int j = 0; j < 2; ++j) {
    a.dA[j] = dA;
    a.dBt[j] = dBt;
    a.dHrow[j] = w.dHrow[0];
    a.part_dBt[j] = w.part_dBt[0];
    a.part_dA[j] = w.part_dA;
  }
  a.s = s;
  a.dXin = dHin;
  a.d_in = pt.f;
  a.d_out = pt.d;
  a.nproj = 1;
  a.T = perm->T;
  a.deterministic = (plan->flags & ACE_FLAG_DETERMINISTIC) != 0;
  a.comb = true;
  a.w = topk_w;
  a.dw = dtopk_w;
  a.row_pair = perm->row_pair;
  a.err = err;
  st = cuda_status(launch_bwd(pt, a, false, cs), "combine backward launch");
  if (st != ACE_OK || perm->R == 0) return st;
  x.tm_da[1] = x.tm_da[0];
  x.dA[0] = x.dA[1] = dBt;
  x.T = perm->T;
  x.d = pt.d;
  x.n_rank = n_rank;
  x.n_rank_pad = nrp;
  x.nproj = 1;
  x.grid = plan->num_sms;
  x.err = err;
  return cuda_status(launch_dense_da(x, cs), "combine dB launch");
}

ace_status ace_gather_rows(const ace_perm* perm, const uint16_t* src_pairs, uint16_t* dst_rows, int32_t cols,
                           void* stream) {
  if (!perm || !src_pairs || !dst_rows) return fail(ACE_ERR_ARG, "null argument");
  if (cols < 8 || cols % 8) return fail(ACE_ERR_SHAPE, "cols=%d must be a positive multiple of 8", cols);
  if (!aligned16(src_pairs) || !aligned16(dst_rows)) return fail(ACE_ERR_ARG, "misaligned tensor");
  return cuda_status(launch_rows_copy(perm->row_pair, src_pairs, dst_rows, perm->R, cols, true,
                                      static_cast<int32_t*>(perm->ws), static_cast<cudaStream_t>(stream)),
                     "gather launch");
}

ace_status ace_scatter_rows(const ace_perm* perm, const uint16_t* src_rows, uint16_t* dst_pairs, int32_t cols,
                            void* stream) {
  if (!perm || !src_rows || !dst_pairs) return fail(ACE_ERR_ARG, "null argument");
  if (cols < 8 || cols % 8) return fail(ACE_ERR_SHAPE, "cols=%d must be a positive multiple of 8", cols);
  if (!aligned16(src_rows) || !aligned16(dst_pairs)) return fail(ACE_ERR_ARG, "misaligned tensor");
  return cuda_status(launch_rows_copy(perm->row_pair, src_rows, dst_pairs, perm->R, cols, false,
                                      static_cast<int32_t*>(perm->ws), static_cast<cudaStream_t>(stream)),
                     "scatter launch");
}

ace_status ace_get_error(const ace_perm* perm, void* stream) {
  if (!perm || !perm->ws) return fail(ACE_ERR_ARG, "null perm");
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  ace_status s = cuda_status(cudaStreamSynchronize(st), "stream synchronize");
  if (s != ACE_OK) return s;
  int32_t flag = 0;
  s = cuda_status(cudaMemcpy(&flag, perm->ws, sizeof(flag), cudaMemcpyDeviceToHost), "read error flag");
  if (s != ACE_OK) return s;
  s = cuda_status(cudaMemset(perm->ws, 0, sizeof(flag)), "clear error flag");
  if (s != ACE_OK) return s;
  if (flag & kErrTimeout) return fail(ACE_ERR_DEVICE_TIMEOUT, "a bounded device wait gave up");
  if (flag & kErrIndex) return fail(ACE_ERR_INDEX, "invalid routing: expert id out of range or repeated in a token");
  if (flag & kErrValue) return fail(ACE_ERR_ARG, "a gate weight given to the combine is not finite");
  if (flag & kErrCheck) return fail(ACE_ERR_CHECK, "ACE_CHECKS: an index or a tile outside its range (the access was skipped)");
  return ACE_OK;
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Allocation-free forward (gate/up).  Some callers cannot allocate device
// memory: an inference server or a plug-in host that reserves the device
// memory for its own pool up front and hands a plug-in no allocator and no
// workspace.  For them the shared-input forward keeps its scratch (H per
// unique pair, both projections) in this file-scope array instead of a
// caller workspace.  Every GPU that loads the library holds the array until
// the process exits.  Calls that overlap on the GPU share it and race.  No
// word of it has to start at zero: the first kernel of a call writes every H
// word the second one reads.
namespace {
constexpr size_t kNoAllocScratchBytes = size_t(32) << 20;  // 32 MiB
__device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];
constexpr int kNoAllocMaxDevices = 64;
std::mutex g_noalloc_mu;
// The array's device address, looked up once per (device, context): a
// context created after cudaDeviceReset, or another context made current on
// the same device, holds its own copy of the array at another address.
struct NoAllocAddr {
  void* ctx;
  void* ptr;
};
NoAllocAddr g_noalloc_addr[kNoAllocMaxDevices] = {};
using CtxGetCurrentFn = int (*)(void**);  // CUresult cuCtxGetCurrent(CUcontext*)
CtxGetCurrentFn ctx_get_current() {
  static CtxGetCurrentFn fn = [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      return reinterpret_cast<CtxGetCurrentFn>(p);
    return static_cast<CtxGetCurrentFn>(nullptr);
  }();
  return fn;
}
}  // namespace

extern "C" ace_status ace_fwd_shared_noalloc(const ace_plan* plan, const ace_perm* perm, const uint16_t* X,
                                             int32_t nproj, const uint16_t* const* A, const uint16_t* const* Bt,
                                             float s, uint16_t* const* Y, void* stream) {
  ace_status st = check_perm(plan, perm);
  if (st != ACE_OK) return st;
  const size_t need = 2 * align_up(4 * (size_t)perm->R * plan->pt.rank_max, 256);
  if (need > kNoAllocScratchBytes)
    return fail(ACE_ERR_WORKSPACE,
                "ace_fwd_shared_noalloc needs %zu bytes of scratch (T*k*rank_max too large); the static limit is %zu",
                need, kNoAllocScratchBytes);
  int dev = 0;
  cudaError_t ce = cudaGetDevice(&dev);
  if (ce != cudaSuccess) return cuda_status(ce, "cudaGetDevice");
  if (dev != plan->device) return fail(ACE_ERR_ARG, "current device %d is not the plan's device %d", dev, plan->device);
  if (dev < 0 || dev >= kNoAllocMaxDevices) return fail(ACE_ERR_UNSUPPORTED, "device index %d too large", dev);
  // cudaGetDevice above made the runtime's context of `dev` current
  CtxGetCurrentFn get_ctx = ctx_get_current();
  if (!get_ctx) return fail(ACE_ERR_UNSUPPORTED, "cuCtxGetCurrent is unavailable from the driver");
  void* ctx = nullptr;
  if (get_ctx(&ctx) != 0 || !ctx) return fail(ACE_ERR_CUDA, "no current CUDA context on device %d", dev);
  void* scratch = nullptr;
  {
    std::lock_guard<std::mutex> lock(g_noalloc_mu);
    NoAllocAddr& slot = g_noalloc_addr[dev];
    if (slot.ctx != ctx || !slot.ptr) {
      // first call in this context, with its device current: the array's device address
      void* p = nullptr;
      ce = cudaGetSymbolAddress(&p, g_noalloc_scratch);
      if (ce != cudaSuccess) return cuda_status(ce, "cudaGetSymbolAddress");
      slot.ctx = ctx;
      slot.ptr = p;
    }
    scratch = slot.ptr;
  }
  return ace_fwd_shared(plan, perm, X, nproj, A, Bt, s, Y, nullptr, scratch, kNoAllocScratchBytes, stream);
}
