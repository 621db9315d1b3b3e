// Internal declarations shared by the ACE CUDA translation units.
#pragma once
#include <cstddef>
#include <cstdint>
#include <cuda.h>  // CUtensorMap (types only; the encoder is fetched at run time)
#include <cuda_runtime.h>

#include "../../include/ace.h"

namespace ace {

constexpr int kTileM = 128;        // rows (or unique pairs) per MMA tile
constexpr int kPermTB = 64;        // tokens per permutation chunk / CTA
constexpr int kMaxK = 32;          // largest top-k the kernels accept

// Device error-flag bits (the flag lives at perm workspace word 0).
constexpr int kErrIndex = 1;
constexpr int kErrTimeout = 2;
constexpr int kErrValue = 4;  // a non-finite gate weight reached the combine
constexpr int kErrCheck = 8;  // ACE_CHECKS build: an index or a tile outside its range

// ACE_CHECKS (a debug build of the same sources, libace_checks.so): every
// index a kernel reads from the permutation arrays (a token, a row, a pair,
// a unique pair) and every tile or split it takes from a tile table is
// checked against its range before it is used.  A value outside raises
// kErrCheck in the device flag (ace_get_error: ACE_ERR_CHECK) and the access
// goes to a safe index instead (a bad tile is dropped), so nothing faults or
// traps.  Shared-memory and TMEM coordinates are fixed at compile time and
// checked there (static_assert).  In the normal build the checks compile away.
#ifdef ACE_CHECKS
constexpr bool kChecks = true;
#else
constexpr bool kChecks = false;
#endif
// i when lo <= i < hi; else (ACE_CHECKS) raises kErrCheck and returns `safe`
__device__ __forceinline__ int chk_idx(int i, int lo, int hi, int safe, int32_t* err) {
  if (i < lo || i >= hi) {
    atomicOr(err, kErrCheck);
    return safe;
  }
  return i;
}
// ACE_CHK(i, lo, hi, safe, err): chk_idx in the ACE_CHECKS build; the plain
// index otherwise (lo, hi and safe are then not evaluated)
#define ACE_CHK(i, lo, hi, safe, err) (::ace::kChecks ? ::ace::chk_idx((i), (lo), (hi), (safe), (err)) : (i))

// Backward row kernel of gate/up at a padded rank of at most 32: two CTAs
// per SM (half the shared-memory budget each, two-tile splits), so one CTA's
// H staging and final dH epilogue overlap the other's dY stream.
__host__ __device__ constexpr int bwd_sh_ctas_per_sm(int rank_pad) { return rank_pad <= 32 ? 2 : 1; }
// row tiles per backward split (gate/up: shared; down and the combine: not)
__host__ __device__ constexpr int bwd_nt_split(int rank_pad, bool shared) {
  return shared && bwd_sh_ctas_per_sm(rank_pad) == 2 ? 2 : rank_pad <= 64 ? 4 : 2;
}

// Plan tables passed by value (__grid_constant__) to every kernel.
struct PlanTables {
  int32_t E, G, k, d, f;
  int32_t rank_max;  // max_g r_g
  int32_t rank_pad;  // MMA N of one projection's rank block (16/32/64/128)
  int32_t nt_split;     // tiles per backward split (down and the combine)
  int32_t nt_split_sh;  // tiles per backward split of gate/up (no phase-2 buffers in TMEM)
  int32_t nsm;       // SMs of the plan's device (the last nsm forward row tiles are split in column halves)
  int16_t e2g[ACE_MAX_EXPERTS];
  int16_t eorder[ACE_MAX_EXPERTS];  // experts in (g, e) order
  int16_t gfirst[ACE_MAX_EXPERTS];  // position in eorder of group g's first expert
  int32_t rank_off[ACE_MAX_EXPERTS + 1];
};

// A unit of work: unique pairs [start, start + cnt) of group g (shared tiles)
// or rows [start, start + cnt) of group g (row tiles, backward splits).  `id`
// is the tile's or split's index, except for forward row tiles, where it
// names the output columns: 0 all, 1 the first half, 2 the second half.
struct Tile {
  int32_t g, start, cnt, id;
};
// ACE_CHECKS: true when the tile lies in group range [0, G), has at most
// max_cnt items and its items lie in [0, limit); else raises kErrCheck.  The
// normal build always returns true.
__device__ __forceinline__ bool chk_tile(const Tile& t, int G, int max_cnt, int limit, int32_t* err) {
  if (kChecks && (t.g < 0 || t.g >= G || t.cnt < 0 || t.cnt > max_cnt || t.start < 0 || t.start > limit - t.cnt)) {
    atomicOr(err, kErrCheck);
    return false;
  }
  return true;
}

// Byte layout of the permutation workspace for T tokens.
struct PermLayout {
  size_t err, counts, sched, group_off, expert_off, expert_cnt, uniq_off, tot_u, row_pair, pair_row, pair_g, row_uniq,
      uniq_tok, tok_uniq;
  size_t chunk_cntE, chunk_cntU, chunk_baseE, chunk_baseU, chunk_err;
  size_t tiles_sh, tiles_row, splits_row, splits_sh;
  size_t total;
  int32_t n_chunks, max_tiles, max_splits, max_splits_sh;
};

// counts[] slots
constexpr int kCntU = 0, kCntRows = 1, kCntTilesSh = 2, kCntTilesRow = 3, kCntSplitsRow = 4;
constexpr int kCntRowSplit = 5;  // index of the first split entry of the row tiles
constexpr int kCntSplitsSh = 6;  // backward splits of gate/up
constexpr int kSplitParts = 4;   // column parts of each split row tile (the last wave's tiles)
// sched[] slots: work counter and finished-CTA counter of the dynamically
// scheduled forward row kernel; the permutation zeroes them and the last CTA
// of every launch resets them, so each launch starts from zero
constexpr int kSchedFwdRows = 0, kSchedFwdDone = 1;

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

inline PermLayout perm_layout(const PlanTables& pt, int32_t T) {
  PermLayout L{};
  const int64_t R = (int64_t)T * pt.k;
  L.n_chunks = (T + kPermTB - 1) / kPermTB;
  L.max_tiles = (int32_t)((R + kTileM - 1) / kTileM + pt.G);
  // pieces of kTileM * nt rows, rounded up to whole waves of nsm CTAs
  auto max_pieces = [&](int nt) {
    const int64_t split_rows = (int64_t)kTileM * nt;
    const int64_t min_splits = (R + split_rows - 1) / split_rows + pt.G;
    return (int32_t)((min_splits + pt.nsm - 1) / pt.nsm * pt.nsm);
  };
  L.max_splits = max_pieces(pt.nt_split);
  L.max_splits_sh = max_pieces(pt.nt_split_sh);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    size_t o = off;
    off = align_up(off + bytes, 256);
    return o;
  };
  L.err = take(4 * 8);
  L.counts = take(4 * 8);
  L.sched = take(4 * (8 + (size_t)pt.nsm));  // 8 counters, then one H-ready flag per split row tile
  L.group_off = take(4 * (size_t)(pt.G + 1));
  L.expert_off = take(4 * (size_t)pt.E);
  L.expert_cnt = take(4 * (size_t)pt.E);
  L.uniq_off = take(4 * (size_t)(pt.G + 1));
  L.tot_u = take(4 * (size_t)pt.G);
  L.row_pair = take(4 * (size_t)R);
  L.pair_row = take(4 * (size_t)R);
  L.pair_g = take(4 * (size_t)R);
  L.row_uniq = take(4 * (size_t)R);
  L.uniq_tok = take(4 * (size_t)R);
  L.tok_uniq = take(4 * (size_t)R);
  L.chunk_cntE = take(4 * (size_t)L.n_chunks * pt.E);
  L.chunk_cntU = take(4 * (size_t)L.n_chunks * pt.G);
  L.chunk_baseE = take(4 * (size_t)L.n_chunks * pt.E);
  L.chunk_baseU = take(4 * (size_t)L.n_chunks * pt.G);
  L.chunk_err = take(4 * (size_t)(L.n_chunks + 1));
  L.tiles_sh = take(sizeof(Tile) * (size_t)L.max_tiles);
  L.tiles_row = take(sizeof(Tile) * (size_t)(L.max_tiles + (kSplitParts - 1) * pt.nsm));
  L.splits_row = take(sizeof(Tile) * (size_t)L.max_splits);
  L.splits_sh = take(sizeof(Tile) * (size_t)L.max_splits_sh);
  L.total = off;
  return L;
}

// Launches a kernel with programmatic stream serialization: its CTAs may be
// scheduled (and run their prologue) while the previous kernel on the stream
// drains; the kernel's pdl_wait() orders its memory accesses after it.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_k(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                            Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, static_cast<Args&&>(args)...);
}

template <typename T>
inline T* at(void* base, size_t off) {
  return reinterpret_cast<T*>(static_cast<char*>(base) + off);
}

// Sets the message ace_last_error_message returns and passes st through.
ace_status report(ace_status st, const char* msg);

// Launchers implemented in the .cu files (host side).  Each returns the
// cudaError_t of its launches.
cudaError_t launch_permute(const PlanTables& pt, const int32_t* topk_idx, int32_t T, void* ws, const PermLayout& L,
                           cudaStream_t st);
// Zeroes n (<= kZeroMax) device buffers in one launch (null / empty ones skipped).
constexpr int kZeroMax = 6;
cudaError_t launch_zero(void* const* ptrs, const size_t* bytes, int n, cudaStream_t st);
cudaError_t launch_rows_copy(const int32_t* row_pair, const uint16_t* src, uint16_t* dst, int64_t R, int32_t cols,
                             bool gather, int32_t* err, cudaStream_t st);

// H = A_g x per unique (g, t) pair of gate/up (deduplicated; X rows gathered),
// or with `rows` H = A_g h per row over the forward row tiles.
struct FwdHLaunch {
  const Tile* tiles;  // unique-pair tiles (rows: the forward row tiles)
  const int32_t* counts;
  int32_t max_tiles;
  int32_t rows;       // 1: row tiles, source row = output row; 0: unique pairs, source row = uniq_tok[u]
  const int32_t* uniq_tok;
  const uint16_t* X;
  const uint16_t* A[2];
  float* H[2];        // [R, rank_max] fp32, row u
  int32_t d_in, nproj;
  int32_t n_src;      // rows of X (T for unique pairs, R for row tiles)
  int32_t* err;
};
cudaError_t launch_fwd_h(const PlanTables& pt, const FwdHLaunch& a, cudaStream_t st);

// Token-major H of the gate/up forward (gemm.cu): the same H_u as
// launch_fwd_h, from 128-token blocks of X read once by TMA.
constexpr int kDenseHMaxRank = 512;  // stacked ranks of a projection up to which H is token-major
struct DenseHLaunch {
  CUtensorMap tm_x;         // X [T, d], box 64 x 128
  CUtensorMap tm_a[2];      // A_j [n_rank, d], box 64 x 256
  const int32_t* tok_uniq;  // [T, k]: the token's unique pairs, ascending g, -1 padded
  const int32_t* uniq_off;  // [G + 1]
  float* H[2];              // [U, rank_max] fp32, row u (columns past r_g written as 0)
  int32_t T, d, n_rank, nproj, rank_max, grid;
  int32_t* err;
};
cudaError_t launch_dense_h(const PlanTables& pt, const DenseHLaunch& a, cudaStream_t st);
}  // namespace ace
struct ace_plan;
namespace ace {
// H_u of gate/up per unique pair into Hbuf[j] (api.cu): the token-major dense
// H GEMM when a projection's stacked ranks are at most kDenseHMaxRank, else
// the gathering H kernel.  Host-side status; launches on `st`.
ace_status launch_gate_up_h(const ace_plan* plan, const ace_perm* perm, const uint16_t* X, int nproj,
                            const uint16_t* const* A, float* const* Hbuf, cudaStream_t st);

// Row-tile forward: Y[row] += s * B_g H_row over contiguous rows of a group.
// MODE down: H_row = A_g h_row computed here (K loop over h);  gate/up:
// H_row = H_u gathered from the unique-pair H of launch_fwd_h.
struct FwdRowsLaunch {
  CUtensorMap tm_x;       // down: Hin [R, d_in], box 64 x 128
  CUtensorMap tm_x16;     // down: Hin, box 64 x 16 (short tiles)
  CUtensorMap tm_a;       // down: A [n_rank, d_in], box 64 x rank_pad
  CUtensorMap tm_bt[2];   // Bt [n_rank, d_out], box 64 x rank_pad
  CUtensorMap tm_y[2];    // Y [R, d_out], box 64 x 128
  CUtensorMap tm_y16[2];  // Y, box 64 x 16 (short tiles)
  const Tile* tiles;         // row tiles (<= 128 rows of one group), in row order
  const int32_t* counts;     // counts[kCntTilesRow] = number of row tiles
  int32_t* sched;            // [kSchedFwdRows] work counter, [kSchedFwdDone] finished CTAs; zero at launch
  int32_t grid;              // persistent CTAs (the SM count)
  const int32_t* row_uniq;
  const float* Hu[2];    // gate/up: H per unique pair
  uint16_t* Y[2];
  float* Hsave;          // down: H per row out (may be null)
  float* Hpre;           // down: where the split row tiles' H is computed first (Hsave or scratch), or null
  int32_t pre;           // down: split row tiles take their H from Hpre (computed up front), not a K loop
  int32_t proj_split;    // gate/up: the two projections are separate work items (NPROJ = 1 kernel)
  int32_t test_expiry;   // ACE_FLAG_TEST_WAIT_EXPIRY: the up-front H's ready flags are never raised and
                         // the wait on them gives up after 2 ms
  float s;
  int32_t d_in, d_out, nproj;
  int32_t* err;
};
cudaError_t launch_fwd_rows(const PlanTables& pt, const FwdRowsLaunch& a, bool shared, cudaStream_t st);

// 2-D bf16 tensor map (row-major [rows, cols]) with a 64-column x box_rows box
// and 128-byte swizzle.  Returns false when the encoder is unavailable or
// rejects the layout.
bool make_tmap_bf16(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows);
// 2-D fp32 tensor map with a 32-column x box_rows box and 128-byte swizzle.
bool make_tmap_f32(CUtensorMap* m, const void* base, uint64_t rows, uint64_t cols, uint32_t box_rows);

struct BwdLaunch {
  CUtensorMap tm_dy[2];    // dY [R, d_out], box 64 x 128
  CUtensorMap tm_bt[2];    // Bt [n_rank, d_out], box 64 x rank_pad
  CUtensorMap tm_a;        // down: A [n_rank, d_in], box 64 x rank_pad
  CUtensorMap tm_dh;       // down: dHin [R, d_in], box 64 x 128
  CUtensorMap tm_h;        // down: Hin [R, d_in], box 64 x 128
  const Tile* splits_row;  // row splits (the dY streaming kernel: down, combine)
  const Tile* splits_sh;   // row splits of gate/up (nt_split_sh tiles each)
  const Tile* tiles_sh;    // unique-pair tiles (dH per unique pair)
  const int32_t* counts;
  int32_t max_splits_row, max_splits_sh, max_tiles_sh;
  const int32_t* uniq_tok;
  const int32_t* uniq_off;
  const int32_t* group_off;
  const int32_t* pair_row;
  const int32_t* pair_g;
  const int32_t* row_uniq;
  const uint16_t* Xin;   // gate/up: X [T, d]; down: Hin [R, f]
  const float* H[2];     // saved H (gate/up: per unique pair; down: per row), stride rank_max
  float s;
  uint16_t* dXin;        // down: dHin [R, f] in/out
  uint16_t* dHx;         // scratch: token-major dense dH [T, nproj * n_rank_pad] (gate/up)
  int32_t n_rank_pad;    // n_rank rounded up to a multiple of 64
  float* dHrow[2];       // scratch: fp32 dH per row [R, rank_pad] (gate/up)
  float* dA[2];
  float* dBt[2];
  float* part_dBt[2];    // deterministic dB^T partials [max_splits, rank_pad, d_out]
  float* part_dA[2];     // deterministic dA partials (down) [max_splits, rank_pad, d_in]
  int32_t d_in, d_out, nproj, T;
  bool deterministic;
  // gate-weighted combine of down (with shared == false): H[0] = dHc per
  // unique pair, H[1] = the forward's H per row, dB^T left to the dense GEMM
  bool comb;
  const float* w;           // combine: gate weights [T*k], pair order
  float* dw;                // combine: gate-weight gradient [T*k] out, pair order
  const int32_t* row_pair;  // combine: pair of each row
  int32_t* err;
};
cudaError_t launch_bwd(const PlanTables& pt, const BwdLaunch& a, bool shared, cudaStream_t st);

// Dense gate/up backward over the token-major dH matrix (see gemm.cu).
struct DenseBwdLaunch {
  CUtensorMap tm_dhx;      // dHx [T, nproj * n_rank_pad], box 64 x 128
  CUtensorMap tm_dhx_t;    // same tensor, box 64 x 64
  CUtensorMap tm_acat[2];  // A_j [n_rank, d], box 64 x 64
  CUtensorMap tm_x;        // X [T, d], box 64 x 64
  CUtensorMap tm_dx;       // dX [T, d], box 64 x 128
  CUtensorMap tm_da[2];    // dA_j [n_rank, d] fp32, box 32 x 32 (bulk reduce-add)
  uint16_t* dX;
  float* dA[2];
  int32_t T, d, n_rank, n_rank_pad, nproj;
  int32_t grid;  // persistent CTAs of the dX GEMM (the SM count)
  int32_t* err;
  // dX then dA in one call (launch_dense_bwd): dA reads nothing dX writes,
  // so dX signals its dependents as soon as its own inputs are ready and dA
  // waits on the grid dependency only at its end; dA's CTAs then fill the
  // SMs that dX's last round leaves idle.  (dA's inputs were complete before
  // dX's wait returned, and dX's CTAs signal only after it; the late wait
  // keeps dA from completing before dX.)
  int32_t early_signal, no_wait;
};
// dA must be zero on entry (the GEMM adds its tiles into it).
cudaError_t launch_dense_bwd(const DenseBwdLaunch& a, cudaStream_t st);
// The two halves of launch_dense_bwd on their own: dX += dHx . A (tm_dhx,
// tm_acat, tm_dx) and dA += dHx^T . X (tm_dhx_t, tm_x, tm_da).
cudaError_t launch_dense_dx(const DenseBwdLaunch& a, cudaStream_t st);
cudaError_t launch_dense_da(const DenseBwdLaunch& a, cudaStream_t st);

// Token-major combined H of the gate-weighted combine of down (combine.cu):
//   Hx[t][rank_off[g] + k] = s * sum_{j: g(e_tj) = g} w[t*k+j] * H[pair_row[t*k+j]][k]
// for k < r_g, every other column of [0, n_rank_pad) zero; bf16, row stride
// n_rank_pad.  Pairs are added in ascending j (deterministic).
struct CombReduceLaunch {
  const float* H;          // [R, rank_max] fp32 per row
  const float* w;          // [T*k] gate weights, pair order
  const int32_t* pair_row;
  const int32_t* pair_g;
  uint16_t* Hx;            // [T, n_rank_pad] bf16 out
  float s;
  int32_t T, n_rank_pad;
  int32_t* err;            // device error flag (kErrValue on a non-finite gate weight)
};
cudaError_t launch_comb_reduce(const PlanTables& pt, const CombReduceLaunch& a, cudaStream_t st);

// Expert FFN pieces (ffn.cu).
// out[row] (+)= in[row] . W_e^T over the rows of each expert e; W is [E * N, K]
// (W_e^T rows), or with w_kn [E * K, N] (W_e itself: the input gradient).
// With in2 and W2 (same shapes) the second product is added in the same
// accumulator: out[row] (+)= in[row] . W_e^T + in2[row] . W2_e^T.
cudaError_t launch_expert_gemm(const void* in, const void* W, const int32_t* expert_off, const int32_t* expert_cnt,
                               uint16_t* out, int E, int64_t R, int N, int K, int grid, int32_t* err,
                               cudaStream_t st, bool w_kn = false, bool accumulate = false,
                               const void* in2 = nullptr, const void* W2 = nullptr);
// Expert FFN forward with the adapters fused into the base GEMMs
// (ffn_fused.cu): gate/up writes u, v, h = SiLU(v) u; down writes y.
struct FfnFusedLaunch {
  CUtensorMap tm_in;     // gate/up: x [R, d], down: h [R, f], in row order; box 64 x 128
  CUtensorMap tm_w[2];   // gate/up: W_up, W_gate [E*f, d], box 64 x 128; down: W_down [E*d, f], box 64 x 256
  CUtensorMap tm_bt[2];  // gate/up: B^T of up, gate [n_rank, f]; down: [n_rank, d]; box 64 x rank_pad
  const int32_t* row_uniq;
  const int32_t* expert_off;
  const int32_t* expert_cnt;
  const int32_t* counts;  // the permutation's counts (ACE_CHECKS bounds)
  const float* Hs[2];    // gate/up: H of up, gate per unique pair; down: H per row; stride rank_max
  uint16_t* U;           // gate/up outputs [R, f] bf16 (row order): u, v, h
  uint16_t* V;
  uint16_t* Hh;
  uint16_t* Y;           // down output [R, d] bf16
  float s;
  int32_t N, K, grid;    // output columns, reduction length, persistent CTAs
  int32_t* err;
};
cudaError_t launch_ffn_fused(const PlanTables& pt, const FfnFusedLaunch& a, bool gate_up, cudaStream_t st);
cudaError_t launch_gather_tokens(const int32_t* row_pair, const int32_t* counts, int k, int T, const uint16_t* X,
                                 uint16_t* dst, int64_t R, int cols, int nsm, cudaStream_t st);
cudaError_t launch_swiglu(const uint16_t* u, const uint16_t* v, uint16_t* h, int64_t n, cudaStream_t st);

}  // namespace ace

// The plan behind the opaque ace_plan handle (host memory).
struct ace_plan {
  ace::PlanTables pt;
  int32_t T_max;
  uint32_t flags;
  int device;
  int num_sms;  // persistent kernels launch one CTA per SM
};
