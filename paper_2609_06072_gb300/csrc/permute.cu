// Route-permute: the (token, slot) pairs of the top-k routing R(x) (Sec. 3.1)
// are counted per expert, exclusive-scanned in (g(e), e) order and scattered,
// stable in t, into group-contiguous rows; the active (token, group) pairs
// A(x) of Sec. 3.5 are deduplicated into a (g, t)-sorted unique list.
//
// Three launches, no inter-CTA waiting:
//   k_perm_count   per 64-token chunk: pairs per expert, unique pairs per group
//   k_perm_colscan one CTA per expert and per group: prefix over the chunks
//                  of that column and its total; CTA 0 also gathers the
//                  routing-error flags
//   k_perm_scatter per chunk: segment offsets from the totals (a warp scan in
//                  (g, e) order), rank of each pair inside its expert
//                  (bitmask popcounts over the chunk's earlier tokens) -> row;
//                  three extra CTAs write the offsets and the tile tables
// Integer-only and order-independent, so bit-exact and deterministic.
#include <algorithm>
#include <cstdint>

#include "ace_internal.cuh"
#include "ace_ptx.cuh"

namespace ace {
namespace {

// Reads token t's k expert ids into e[0..k) (KB >= k; the loops unroll so e
// stays in registers); false when an id is out of range or repeated within
// the token.
template <int KB>
__device__ __forceinline__ bool read_token(const int32_t* __restrict__ idx, int t, int k, int E, int (&e)[KB]) {
  bool ok = true;
#pragma unroll
  for (int j = 0; j < KB; ++j) {
    e[j] = -1;
    if (j < k) {
      const int v = idx[(int64_t)t * k + j];
      e[j] = v;
      if (v < 0 || v >= E) ok = false;
    }
  }
#pragma unroll
  for (int j = 1; j < KB; ++j)
#pragma unroll
    for (int jj = 0; jj < j; ++jj)
      if (j < k && e[j] == e[jj]) ok = false;
  return ok;
}

// Bit j set when slot j is the first of the token's slots routed into its group.
template <int KB>
__device__ __forceinline__ uint32_t first_of_group(const int (&g)[KB], int k) {
  uint32_t m = 0;
#pragma unroll
  for (int j = 0; j < KB; ++j) {
    bool first = j < k;
#pragma unroll
    for (int jj = 0; jj < j; ++jj)
      if (g[jj] == g[j]) first = false;
    if (first) m |= 1u << j;
  }
  return m;
}

template <int KB>
__global__ void __launch_bounds__(kPermTB) k_perm_count(const __grid_constant__ PlanTables pt,
                                                        const int32_t* __restrict__ idx, int T,
                                                        int32_t* __restrict__ chunk_cntE,
                                                        int32_t* __restrict__ chunk_cntU,
                                                        int32_t* __restrict__ chunk_err) {
  extern __shared__ int32_t sm[];
  int32_t* cntE = sm;                // [E]
  int32_t* cntU = sm + pt.E;         // [G]
  int32_t* e2g = sm + pt.E + pt.G;   // [E] expert -> group, staged from the plan
  __shared__ int32_t err_s;
  const int tid = threadIdx.x;
  pdl_wait();
  pdl_trigger();
  for (int i = tid; i < pt.E + pt.G; i += blockDim.x) sm[i] = 0;
  for (int i = tid; i < pt.E; i += blockDim.x) e2g[i] = pt.e2g[i];
  if (tid == 0) err_s = 0;
  __syncthreads();
  const int t = blockIdx.x * kPermTB + tid;
  if (t < T) {
    int e[KB];
    if (!read_token<KB>(idx, t, pt.k, pt.E, e)) {
      atomicOr(&err_s, kErrIndex);
    } else {
      int g[KB];
#pragma unroll
      for (int j = 0; j < KB; ++j) g[j] = j < pt.k ? e2g[e[j]] : -1 - j;
      const uint32_t first = first_of_group<KB>(g, pt.k);
#pragma unroll
      for (int j = 0; j < KB; ++j) {
        if (j < pt.k) atomicAdd(&cntE[e[j]], 1);
        if ((first >> j) & 1u) atomicAdd(&cntU[g[j]], 1);
      }
    }
  }
  __syncthreads();
  const int c = blockIdx.x;
  for (int i = tid; i < pt.E; i += blockDim.x) chunk_cntE[(int64_t)c * pt.E + i] = cntE[i];
  for (int i = tid; i < pt.G; i += blockDim.x) chunk_cntU[(int64_t)c * pt.G + i] = cntU[i];
  if (tid == 0) chunk_err[c] = err_s;
}

// Group whose pieces [pre[g], pre[g + 1]) contain piece i (pre ascending, G + 1 entries).
__device__ __forceinline__ int piece_group(const int32_t* pre, int G, int i) {
  int lo = 0, hi = G;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (pre[mid] <= i)
      lo = mid;
    else
      hi = mid;
  }
  return lo;
}

// Writes the tiles of every group: group g has ceil(n_g / per) tiles of at
// most `per` items; returns the total (thread 0's view after the call).  The
// threads share the tiles (not the groups), so a large group costs no more
// than many small ones.
__device__ int build_tiles(const int32_t* n_g, const int32_t* off_g, int G, int per, Tile* __restrict__ out,
                           int32_t* scratch /* smem [G+1] */) {
  const int tid = threadIdx.x;
  for (int g = tid; g < G; g += blockDim.x) scratch[g + 1] = (n_g[g] + per - 1) / per;
  __syncthreads();
  if (tid == 0) {
    scratch[0] = 0;
    for (int g = 0; g < G; ++g) scratch[g + 1] += scratch[g];
  }
  __syncthreads();
  for (int p = tid; p < scratch[G]; p += blockDim.x) {
    const int g = piece_group(scratch, G, p), i = p - scratch[g], n = n_g[g];
    Tile tl;
    tl.g = g;
    tl.start = off_g[g] + i * per;
    tl.cnt = min(per, n - i * per);
    tl.id = p;
    out[p] = tl;
  }
  __syncthreads();
  int total = scratch[G];
  __syncthreads();
  return total;
}

// Forward row tiles in dispatch order: every group's rows in tiles of 128
// (id 0: all output columns), except that each of the last `tail` tiles of the
// list (split b) becomes kSplitParts entries covering one part of the columns
// each (ids 1 + P b + p), so the work left when SMs run dry comes in parts.
// *split_first receives the index of the first split entry.
__device__ int build_row_tiles(const int32_t* n_g, const int32_t* off_g, int G, int tail, Tile* __restrict__ out,
                               int32_t* scratch /* smem [G+1] */, int32_t* split_first) {
  const int n = build_tiles(n_g, off_g, G, kTileM, out, scratch);
  const int ns = min(n, tail), first = n - ns;
  if (threadIdx.x == 0) split_first[0] = first;
  for (int j = threadIdx.x; j < first; j += blockDim.x) out[j].id = 0;
  // read the tiles to split before any of them is overwritten
  Tile mine[8];
  int cnt = 0;
  for (int j = first + (int)threadIdx.x; j < n && cnt < 8; j += blockDim.x) mine[cnt++] = out[j];
  __syncthreads();
  cnt = 0;
  for (int j = first + (int)threadIdx.x; j < n && cnt < 8; j += blockDim.x) {
    Tile t = mine[cnt++];
    // split b = j - first: ids 1 + P b + p for its column parts p < P
    for (int p = 0; p < kSplitParts; ++p) {
      t.id = 1 + kSplitParts * (j - first) + p;
      out[first + kSplitParts * (j - first) + p] = t;
    }
  }
  __syncthreads();
  return n + (kSplitParts - 1) * ns;
}

// Sum of ceil(n_g / per) over the groups (every thread gets the total).
__device__ int count_pieces(const int32_t* n_g, int G, int per, int32_t* red /* smem [32] */) {
  int v = 0;
  for (int g = threadIdx.x; g < G; g += blockDim.x) v += (n_g[g] + per - 1) / per;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  int tot = 0;
  for (int w = 0; w < (int)(blockDim.x + 31) / 32; ++w) tot += red[w];
  return tot;
}

// Backward splits: every group's rows in near-equal pieces of at most `cap`
// rows.  When pieces of `cap` rows leave the last wave of `nsm` CTAs less than
// 90% full, the piece size shrinks so that the pieces fill whole waves:
// per = ceil(R / (waves * nsm - G)) gives at most R / per + G <= waves * nsm
// pieces.  Returns the number of splits.
__device__ int build_splits(const int32_t* n_g, const int32_t* off_g, int G, int cap, int nsm,
                            Tile* __restrict__ out, int32_t* scratch /* smem [G+1] */, int32_t* red) {
  const int min_total = count_pieces(n_g, G, cap, red);
  const int target = (min_total + nsm - 1) / nsm * nsm;
  int per = cap;
  if (min_total > 0 && 10 * (min_total - (target - nsm)) < 9 * nsm) {
    // the shortest pieces whose count still fits the whole waves of the
    // target (the count only falls as the pieces lengthen); every thread
    // takes the same branches, so the block reductions stay aligned
    int lo = 1, hi = cap;
    while (lo < hi) {
      const int mid = (lo + hi) / 2;
      if (count_pieces(n_g, G, mid, red) <= target)
        hi = mid;
      else
        lo = mid + 1;
    }
    per = hi;
  }
  const int tid = threadIdx.x;
  for (int g = tid; g < G; g += blockDim.x) scratch[g + 1] = (n_g[g] + per - 1) / per;
  __syncthreads();
  if (tid == 0) {
    scratch[0] = 0;
    for (int g = 0; g < G; ++g) scratch[g + 1] += scratch[g];
  }
  __syncthreads();
  for (int p = tid; p < scratch[G]; p += blockDim.x) {
    const int g = piece_group(scratch, G, p), i = p - scratch[g], n = n_g[g], np = scratch[g + 1] - scratch[g];
    const int b0 = (int)((int64_t)i * n / np), b1 = (int)((int64_t)(i + 1) * n / np);
    Tile tl;
    tl.g = g;
    tl.start = off_g[g] + b0;
    tl.cnt = b1 - b0;
    tl.id = p;
    out[p] = tl;
  }
  __syncthreads();
  const int total = scratch[G];
  __syncthreads();
  return total;
}

__device__ __forceinline__ int warp_incl_scan(int v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int x = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += x;
  }
  return v;
}

// Column col of the [C x ncol] chunk-count matrix (experts, then groups):
// base[c][col] = sum of cnt[c'][col] over c' < c, and the column total.
__global__ void __launch_bounds__(256) k_perm_colscan(const __grid_constant__ PlanTables pt, int n_chunks,
                                                      const int32_t* __restrict__ chunk_cntE,
                                                      const int32_t* __restrict__ chunk_cntU,
                                                      const int32_t* __restrict__ chunk_err,
                                                      int32_t* __restrict__ chunk_baseE,
                                                      int32_t* __restrict__ chunk_baseU, int32_t* __restrict__ totE,
                                                      int32_t* __restrict__ totU, int32_t* __restrict__ err,
                                                      int32_t* __restrict__ sched) {
  __shared__ int32_t wsum[8];
  __shared__ int32_t err_s;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  pdl_wait();
  pdl_trigger();
  const bool isE = (int)blockIdx.x < pt.E;
  const int ncol = isE ? pt.E : pt.G, col = isE ? blockIdx.x : blockIdx.x - pt.E;
  const int32_t* cnt = isE ? chunk_cntE : chunk_cntU;
  int32_t* base = isE ? chunk_baseE : chunk_baseU;
  if (tid == 0) err_s = 0;
  int carry = 0;
  for (int c0 = 0; c0 < n_chunks; c0 += 256) {
    const int c = c0 + tid;
    const int v = c < n_chunks ? cnt[(int64_t)c * ncol + col] : 0;
    const int x = warp_incl_scan(v);
    if (lane == 31) wsum[warp] = x;
    __syncthreads();
    if (warp == 0) {
      int w = lane < 8 ? wsum[lane] : 0;
      w = warp_incl_scan(w);
      if (lane < 8) wsum[lane] = w;
    }
    __syncthreads();
    if (c < n_chunks) base[(int64_t)c * ncol + col] = carry + (warp > 0 ? wsum[warp - 1] : 0) + x - v;
    carry += wsum[7];
    __syncthreads();
  }
  if (tid == 0) (isE ? totE : totU)[col] = carry;
  if (blockIdx.x == 0) {
    for (int i = tid; i < 8 + pt.nsm; i += blockDim.x) sched[i] = 0;  // row-kernel counters and flags start at zero
    int e = 0;
    for (int c = tid; c < n_chunks; c += 256) e |= chunk_err[c];
    if (e) atomicOr(&err_s, e);
    __syncthreads();
    if (tid == 0) *err = err_s ? kErrIndex : 0;
  }
}

__device__ __forceinline__ int prefix_bits(const uint32_t* mask, int tid) {
  int r = 0;
  const int w = tid >> 5;
  for (int i = 0; i < w; ++i) r += __popc(mask[i]);
  return r + __popc(mask[w] & ((1u << (tid & 31)) - 1u));
}

constexpr int kTableCtas = 4;  // scatter CTAs that build the offsets and tile tables

struct ScatterOut {
  int32_t* row_pair;
  int32_t* pair_row;
  int32_t* pair_g;
  int32_t* row_uniq;
  int32_t* uniq_tok;
  int32_t* tok_uniq;
  int32_t* counts;
  int32_t* group_off;
  int32_t* uniq_off;
  int32_t* expert_off;
  Tile* tiles_sh;
  Tile* tiles_row;
  Tile* splits_row;
  Tile* splits_sh;
};

template <int KB>
__global__ void __launch_bounds__(kPermTB) k_perm_scatter(const __grid_constant__ PlanTables pt,
                                                          const int32_t* __restrict__ idx, int T,
                                                          const int32_t* __restrict__ chunk_baseE,
                                                          const int32_t* __restrict__ chunk_baseU,
                                                          const int32_t* __restrict__ totE,
                                                          const int32_t* __restrict__ totU, const ScatterOut o) {
  constexpr int W = kPermTB / 32;
  extern __shared__ uint32_t msk[];
  uint32_t* mE = msk;                    // [E][W]
  uint32_t* mU = msk + (size_t)pt.E * W; // [G][W]
  __shared__ int32_t eoff[ACE_MAX_EXPERTS];      // first row of each expert segment
  __shared__ int32_t uoff[ACE_MAX_EXPERTS + 1];  // first unique pair of each group
  __shared__ int32_t goff[ACE_MAX_EXPERTS + 1];  // first row of each group
  __shared__ int32_t baseE[ACE_MAX_EXPERTS];     // this chunk's rows before it, per expert
  __shared__ int32_t baseU[ACE_MAX_EXPERTS];     // this chunk's unique pairs before it, per group
  __shared__ int32_t e2g[ACE_MAX_EXPERTS];
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int E = pt.E, G = pt.G;
  pdl_wait();
  pdl_trigger();
  const int c = blockIdx.x;
  const int t = c * kPermTB + tid;
  const int k = pt.k;
  // the token's expert ids, in flight while the offsets are computed
  int e[KB];
  bool ok = false;
  const int n_chunk_ctas = (int)gridDim.x - kTableCtas;
  if (c < n_chunk_ctas && t < T) ok = read_token<KB>(idx, t, k, E, e);
  for (int i = tid; i < (E + G) * W; i += blockDim.x) msk[i] = 0;
  if (c < n_chunk_ctas) {
    for (int i = tid; i < E; i += blockDim.x) {
      baseE[i] = chunk_baseE[(int64_t)c * E + i];
      e2g[i] = pt.e2g[i];
    }
    for (int i = tid; i < G; i += blockDim.x) baseU[i] = chunk_baseU[(int64_t)c * G + i];
  }
  // segment offsets: rows in (g, e) order (warp 0), unique pairs in g order (warp 1)
  if (warp == 0) {
    int carry = 0;
    for (int i0 = 0; i0 < E; i0 += 32) {
      const int i = i0 + lane, e = i < E ? pt.eorder[i] : 0;
      const int v = i < E ? totE[e] : 0, x = warp_incl_scan(v);
      if (i < E) eoff[e] = carry + x - v;
      carry += __shfl_sync(0xffffffffu, x, 31);
    }
    if (lane == 0) goff[G] = carry;
  } else if (warp == 1) {
    int carry = 0;
    for (int g0 = 0; g0 < G; g0 += 32) {
      const int g = g0 + lane;
      const int v = g < G ? totU[g] : 0, x = warp_incl_scan(v);
      if (g < G) uoff[g] = carry + x - v;
      carry += __shfl_sync(0xffffffffu, x, 31);
    }
    if (lane == 0) uoff[G] = carry;
  }
  __syncthreads();
  for (int g = tid; g < G; g += blockDim.x) goff[g] = eoff[pt.eorder[pt.gfirst[g]]];
  __syncthreads();
  if (c >= n_chunk_ctas) {
    // the CTAs that own no chunk write, in parallel with the chunks' scatter,
    // the offsets and the tile tables the other calls read: one table each
    __shared__ int32_t rows_g[ACE_MAX_EXPERTS];
    __shared__ int32_t scratch[ACE_MAX_EXPERTS + 1];
    const int job = c - n_chunk_ctas;
    for (int g = tid; g < G; g += blockDim.x) rows_g[g] = goff[g + 1] - goff[g];
    if (job == 0) {
      for (int g = tid; g <= G; g += blockDim.x) {
        o.group_off[g] = goff[g];
        o.uniq_off[g] = uoff[g];
      }
      for (int e = tid; e < E; e += blockDim.x) o.expert_off[e] = eoff[e];
      if (tid == 0) {
        o.counts[kCntU] = uoff[G];
        o.counts[kCntRows] = goff[G];
      }
    }
    __syncthreads();
    if (job == 0) {
      const int n = build_tiles(totU, uoff, G, kTileM, o.tiles_sh, scratch);
      if (tid == 0) o.counts[kCntTilesSh] = n;
    } else if (job == 1) {
      // the last wave's tiles are cut into column parts only when every part
      // gets at least one 64-column chunk (a quarter of d's chunks for down,
      // half of f's for gate/up)
      const bool parts = (pt.d + 63) / 64 >= kSplitParts && (pt.f + 63) / 64 >= 2;
      const int n = build_row_tiles(rows_g, goff, G, parts ? min(pt.nsm, 8 * (int)blockDim.x) : 0, o.tiles_row, scratch,
                                    o.counts + kCntRowSplit);
      if (tid == 0) o.counts[kCntTilesRow] = n;
    } else {
      // backward splits: down / combine (job 2), gate/up (job 3)
      __shared__ int32_t red[32];
      const bool sh = job == 3;
      // gate/up runs its two projections side by side (grid.y = 2), so its
      // splits fill whole waves: gate/up's two projections run side by side,
      // so a wave holds ctas_per_sm * nsm / 2 splits of each
      const int wave = sh ? max(1, bwd_sh_ctas_per_sm(pt.rank_pad) * pt.nsm / 2) : pt.nsm;
      const int n = build_splits(rows_g, goff, G, kTileM * (sh ? pt.nt_split_sh : pt.nt_split), wave,
                                 sh ? o.splits_sh : o.splits_row, scratch, red);
      if (tid == 0) o.counts[sh ? kCntSplitsSh : kCntSplitsRow] = n;
    }
    return;
  }
  if (ok) {
    const uint32_t bit = 1u << (tid & 31);
#pragma unroll
    for (int j = 0; j < KB; ++j)
      if (j < k) {
        atomicOr(&mE[e[j] * W + (tid >> 5)], bit);
        atomicOr(&mU[e2g[e[j]] * W + (tid >> 5)], bit);
      }
  }
  __syncthreads();
  if (t >= T) return;
  if (!ok) {
    for (int j = 0; j < k; ++j) {
      o.tok_uniq[(int64_t)t * k + j] = -1;
      o.pair_g[(int64_t)t * k + j] = -1;
    }
    return;
  }
  int g[KB];
#pragma unroll
  for (int j = 0; j < KB; ++j) g[j] = j < k ? e2g[e[j]] : -1 - j;
  const uint32_t first = first_of_group<KB>(g, k);
#pragma unroll
  for (int j = 0; j < KB; ++j) {
    if (j >= k) break;
    const int row = eoff[e[j]] + baseE[e[j]] + prefix_bits(&mE[e[j] * W], tid);
    const int u = uoff[g[j]] + baseU[g[j]] + prefix_bits(&mU[g[j] * W], tid);
    const int p = t * k + j;
    o.pair_row[p] = row;
    o.pair_g[p] = g[j];
    o.row_pair[row] = p;
    o.row_uniq[row] = u;
    if ((first >> j) & 1u) {
      // position among the token's distinct groups in ascending order
      int n_below = 0;
#pragma unroll
      for (int jj = 0; jj < KB; ++jj)
        if (((first >> jj) & 1u) && g[jj] < g[j]) ++n_below;
      o.uniq_tok[u] = t;
      o.tok_uniq[(int64_t)t * k + n_below] = u;
    }
  }
  for (int j = __popc(first); j < k; ++j) o.tok_uniq[(int64_t)t * k + j] = -1;
}

// Zeroes up to kZeroMax buffers (16-byte aligned, sizes multiples of 16) in
// one launch.
struct ZeroList {
  uint4* p[kZeroMax];
  int64_t n16[kZeroMax];  // 16-byte words of each
  int n;
};
__global__ void __launch_bounds__(256) k_zero(const __grid_constant__ ZeroList z) {
  pdl_wait();
  pdl_trigger();
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int b = 0; b < z.n; ++b)
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < z.n16[b]; i += stride)
      z.p[b][i] = make_uint4(0, 0, 0, 0);
}

__global__ void k_rows_copy(const int32_t* __restrict__ row_pair, const uint4* __restrict__ src,
                            uint4* __restrict__ dst, int64_t R, int vec_per_row, bool gather, int32_t* err) {
  pdl_wait();
  pdl_trigger();
  const int64_t n = R * vec_per_row;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t row = i / vec_per_row, v = i % vec_per_row;
    const int64_t p = ACE_CHK(row_pair[row], 0, (int)R, 0, err);
    if (gather)
      dst[row * vec_per_row + v] = src[p * vec_per_row + v];
    else
      dst[p * vec_per_row + v] = src[row * vec_per_row + v];
  }
}

}  // namespace

cudaError_t launch_permute(const PlanTables& pt, const int32_t* topk_idx, int32_t T, void* ws, const PermLayout& L,
                           cudaStream_t st) {
  const int C = L.n_chunks;
  if (C > 0) {
    size_t sm1 = sizeof(int32_t) * (2 * pt.E + pt.G);
    cudaError_t e = launch_k(pt.k <= 8 ? k_perm_count<8> : k_perm_count<kMaxK>, C, kPermTB, sm1, st, pt, topk_idx, T, at<int32_t>(ws, L.chunk_cntE),
                             at<int32_t>(ws, L.chunk_cntU), at<int32_t>(ws, L.chunk_err));
    if (e != cudaSuccess) return e;
  }
  cudaError_t e = launch_k(k_perm_colscan, pt.E + pt.G, 256, 0, st, pt, C, at<int32_t>(ws, L.chunk_cntE),
                           at<int32_t>(ws, L.chunk_cntU), at<int32_t>(ws, L.chunk_err), at<int32_t>(ws, L.chunk_baseE),
                           at<int32_t>(ws, L.chunk_baseU), at<int32_t>(ws, L.expert_cnt), at<int32_t>(ws, L.tot_u),
                           at<int32_t>(ws, L.err), at<int32_t>(ws, L.sched));
  if (e != cudaSuccess) return e;
  ScatterOut o;
  o.row_pair = at<int32_t>(ws, L.row_pair);
  o.pair_row = at<int32_t>(ws, L.pair_row);
  o.pair_g = at<int32_t>(ws, L.pair_g);
  o.row_uniq = at<int32_t>(ws, L.row_uniq);
  o.uniq_tok = at<int32_t>(ws, L.uniq_tok);
  o.tok_uniq = at<int32_t>(ws, L.tok_uniq);
  o.counts = at<int32_t>(ws, L.counts);
  o.group_off = at<int32_t>(ws, L.group_off);
  o.uniq_off = at<int32_t>(ws, L.uniq_off);
  o.expert_off = at<int32_t>(ws, L.expert_off);
  o.tiles_sh = at<Tile>(ws, L.tiles_sh);
  o.tiles_row = at<Tile>(ws, L.tiles_row);
  o.splits_row = at<Tile>(ws, L.splits_row);
  o.splits_sh = at<Tile>(ws, L.splits_sh);
  size_t sm3 = sizeof(uint32_t) * (size_t)(pt.E + pt.G) * (kPermTB / 32);
  // one CTA per chunk, plus the ones that write the offsets and tables
  return launch_k(pt.k <= 8 ? k_perm_scatter<8> : k_perm_scatter<kMaxK>, C + kTableCtas, kPermTB, sm3, st, pt, topk_idx, T, at<int32_t>(ws, L.chunk_baseE),
                  at<int32_t>(ws, L.chunk_baseU), at<int32_t>(ws, L.expert_cnt), at<int32_t>(ws, L.tot_u), o);
}

cudaError_t launch_zero(void* const* ptrs, const size_t* bytes, int n, cudaStream_t st) {
  ZeroList z{};
  int64_t total = 0;
  for (int i = 0; i < n && i < kZeroMax; ++i) {
    if (!ptrs[i] || bytes[i] == 0) continue;
    z.p[z.n] = static_cast<uint4*>(ptrs[i]);
    z.n16[z.n] = (int64_t)(bytes[i] / 16);
    total += z.n16[z.n];
    ++z.n;
  }
  if (z.n == 0) return cudaSuccess;
  const int blocks = (int)std::min<int64_t>((total + 255) / 256, 152 * 4);
  return launch_k(k_zero, blocks, 256, 0, st, z);
}

cudaError_t launch_rows_copy(const int32_t* row_pair, const uint16_t* src, uint16_t* dst, int64_t R, int32_t cols,
                             bool gather, int32_t* err, cudaStream_t st) {
  if (R == 0) return cudaSuccess;
  const int vpr = cols / 8;
  const int64_t n = R * vpr;
  int blocks = (int)std::min<int64_t>((n + 255) / 256, 152 * 16);
  return launch_k(k_rows_copy, blocks, 256, 0, st, row_pair, reinterpret_cast<const uint4*>(src),
                  reinterpret_cast<uint4*>(dst), R, vpr, gather, err);
}

}  // namespace ace
