// Route-permute: the (token, slot) pairs of the top-k routing R(x) (Sec. 3.1)
// are counted per expert, exclusive-scanned in (g(e), e) order and scattered,
// stable in t, into group-contiguous rows; the active (token, group) pairs
// A(x) of Sec. 3.5 are deduplicated into a (g, t)-sorted unique list.
//
// Three launches, no inter-CTA waiting:
//   k_perm_count   per 64-token chunk: pairs per expert, unique pairs per group
//   k_perm_scan    one CTA: totals, segment offsets, per-chunk bases, the
//                  unique-pair tile, row tile and row split tables
//   k_perm_scatter per chunk: rank of each pair inside its expert (bitmask
//                  popcounts over the chunk's earlier tokens) -> row
// Integer-only and order-independent, so bit-exact and deterministic.
#include <algorithm>
#include <cstdint>

#include "ace_internal.cuh"

namespace ace {
namespace {

// Reads token t's k expert ids; returns false (and leaves `e` partially
// filled) when an id is out of range or repeated within the token.
__device__ __forceinline__ bool read_token(const int32_t* __restrict__ idx, int t, int k, int E, int* e) {
  bool ok = true;
  for (int j = 0; j < k; ++j) {
    int v = idx[(int64_t)t * k + j];
    e[j] = v;
    if (v < 0 || v >= E) ok = false;
  }
  if (!ok) return false;
  for (int j = 1; j < k; ++j)
    for (int jj = 0; jj < j; ++jj)
      if (e[j] == e[jj]) return false;
  return true;
}

__global__ void __launch_bounds__(kPermTB) k_perm_count(const __grid_constant__ PlanTables pt,
                                                        const int32_t* __restrict__ idx, int T,
                                                        int32_t* __restrict__ chunk_cntE,
                                                        int32_t* __restrict__ chunk_cntU,
                                                        int32_t* __restrict__ chunk_err) {
  extern __shared__ int32_t sm[];
  int32_t* cntE = sm;                // [E]
  int32_t* cntU = sm + pt.E;         // [G]
  __shared__ int32_t err_s;
  const int tid = threadIdx.x;
  for (int i = tid; i < pt.E + pt.G; i += blockDim.x) sm[i] = 0;
  if (tid == 0) err_s = 0;
  __syncthreads();
  const int t = blockIdx.x * kPermTB + tid;
  if (t < T) {
    int e[kMaxK];
    if (!read_token(idx, t, pt.k, pt.E, e)) {
      atomicOr(&err_s, kErrIndex);
    } else {
      for (int j = 0; j < pt.k; ++j) {
        atomicAdd(&cntE[e[j]], 1);
        int g = pt.e2g[e[j]];
        bool first = true;
        for (int jj = 0; jj < j; ++jj)
          if (pt.e2g[e[jj]] == g) first = false;
        if (first) atomicAdd(&cntU[g], 1);
      }
    }
  }
  __syncthreads();
  const int c = blockIdx.x;
  for (int i = tid; i < pt.E; i += blockDim.x) chunk_cntE[(int64_t)c * pt.E + i] = cntE[i];
  for (int i = tid; i < pt.G; i += blockDim.x) chunk_cntU[(int64_t)c * pt.G + i] = cntU[i];
  if (tid == 0) chunk_err[c] = err_s;
}

// Writes the tiles of every group: group g has ceil(n_g / per) tiles of at
// most `per` items; returns the total (thread 0's view after the call).
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
  for (int g = tid; g < G; g += blockDim.x) {
    int n = n_g[g], base = scratch[g];
    for (int i = 0; i * per < n; ++i) {
      Tile tl;
      tl.g = g;
      tl.start = off_g[g] + i * per;
      tl.cnt = min(per, n - i * per);
      tl.id = base + i;
      out[base + i] = tl;
    }
  }
  __syncthreads();
  int total = scratch[G];
  __syncthreads();
  return total;
}

// Per-column prefix over chunks of a [C x ncol] count matrix, parallel over
// (column, part) with P parts per column.  Pass 1 writes each column's total;
// pass 2 writes base[c][col] = col_base[col] + sum_{c' < c} cnt[c'][col].
__device__ void column_totals(const int32_t* __restrict__ cnt, int C, int ncol, int32_t* part_sum /*smem 1024*/,
                              int32_t* total /*smem [ncol]*/) {
  const int tid = threadIdx.x;
  int P = 1;
  while (P * 2 * ncol <= (int)blockDim.x && P < 32) P *= 2;
  const int len = (C + P - 1) / P;
  if (tid < ncol * P) {
    const int col = tid / P, part = tid % P;
    int s = 0;
    for (int c = part * len; c < min(C, (part + 1) * len); ++c) s += cnt[(int64_t)c * ncol + col];
    part_sum[tid] = s;
  }
  __syncthreads();
  for (int col = tid; col < ncol; col += blockDim.x) {
    int run = 0;
    for (int part = 0; part < P; ++part) {
      const int v = part_sum[col * P + part];
      part_sum[col * P + part] = run;
      run += v;
    }
    total[col] = run;
  }
  __syncthreads();
}
__device__ void column_bases(const int32_t* __restrict__ cnt, int C, int ncol, const int32_t* part_sum,
                             const int32_t* col_base, int32_t* __restrict__ base) {
  const int tid = threadIdx.x;
  int P = 1;
  while (P * 2 * ncol <= (int)blockDim.x && P < 32) P *= 2;
  const int len = (C + P - 1) / P;
  if (tid < ncol * P) {
    const int col = tid / P, part = tid % P;
    int run = col_base[col] + part_sum[tid];
    for (int c = part * len; c < min(C, (part + 1) * len); ++c) {
      base[(int64_t)c * ncol + col] = run;
      run += cnt[(int64_t)c * ncol + col];
    }
  }
  __syncthreads();
}

__global__ void __launch_bounds__(1024) k_perm_scan(const __grid_constant__ PlanTables pt, int n_chunks,
                                                    const int32_t* __restrict__ chunk_cntE,
                                                    const int32_t* __restrict__ chunk_cntU,
                                                    const int32_t* __restrict__ chunk_err,
                                                    int32_t* __restrict__ chunk_baseE,
                                                    int32_t* __restrict__ chunk_baseU, int32_t* __restrict__ err,
                                                    int32_t* __restrict__ counts, int32_t* __restrict__ group_off,
                                                    int32_t* __restrict__ expert_off,
                                                    int32_t* __restrict__ expert_cnt,
                                                    int32_t* __restrict__ uniq_off, Tile* __restrict__ tiles_sh,
                                                    Tile* __restrict__ tiles_row, Tile* __restrict__ splits_row) {
  __shared__ int32_t totE[ACE_MAX_EXPERTS];
  __shared__ int32_t rowsG[ACE_MAX_EXPERTS];
  __shared__ int32_t totU[ACE_MAX_EXPERTS];
  __shared__ int32_t gofs[ACE_MAX_EXPERTS + 1];
  __shared__ int32_t uofs[ACE_MAX_EXPERTS + 1];
  __shared__ int32_t scratch[ACE_MAX_EXPERTS + 1];
  __shared__ int32_t eoff[ACE_MAX_EXPERTS];
  __shared__ int32_t partE[1024];
  __shared__ int32_t partU[1024];
  __shared__ int32_t err_s;
  const int tid = threadIdx.x;
  const int E = pt.E, G = pt.G;
  if (tid == 0) err_s = 0;
  for (int g = tid; g < G; g += blockDim.x) rowsG[g] = 0;
  __syncthreads();
  for (int c = tid; c < n_chunks; c += blockDim.x)
    if (chunk_err[c]) atomicOr(&err_s, chunk_err[c]);
  column_totals(chunk_cntE, n_chunks, E, partE, totE);
  column_totals(chunk_cntU, n_chunks, G, partU, totU);
  for (int e = tid; e < E; e += blockDim.x) atomicAdd(&rowsG[pt.e2g[e]], totE[e]);
  __syncthreads();
  if (tid == 0) {
    gofs[0] = 0;
    uofs[0] = 0;
    for (int g = 0; g < G; ++g) {
      gofs[g + 1] = gofs[g] + rowsG[g];
      uofs[g + 1] = uofs[g] + totU[g];
    }
    *err = err_s ? kErrIndex : 0;
    counts[kCntU] = uofs[G];
    counts[kCntRows] = gofs[G];
  }
  __syncthreads();
  for (int g = tid; g <= G; g += blockDim.x) {
    group_off[g] = gofs[g];
    uniq_off[g] = uofs[g];
  }
  for (int e = tid; e < E; e += blockDim.x) {
    const int g = pt.e2g[e];
    int start = gofs[g];
    for (int e2 = 0; e2 < e; ++e2)
      if (pt.e2g[e2] == g) start += totE[e2];
    eoff[e] = start;
    expert_off[e] = start;
    expert_cnt[e] = totE[e];
  }
  __syncthreads();
  column_bases(chunk_cntE, n_chunks, E, partE, eoff, chunk_baseE);
  column_bases(chunk_cntU, n_chunks, G, partU, uofs, chunk_baseU);
  int n = build_tiles(totU, uofs, G, kTileM, tiles_sh, scratch);
  if (tid == 0) counts[kCntTilesSh] = n;
  n = build_tiles(rowsG, gofs, G, kTileM, tiles_row, scratch);
  if (tid == 0) counts[kCntTilesRow] = n;
  n = build_tiles(rowsG, gofs, G, kTileM * pt.nt_split, splits_row, scratch);
  if (tid == 0) counts[kCntSplitsRow] = n;
}

__device__ __forceinline__ int prefix_bits(const uint32_t* mask, int tid) {
  int r = 0;
  const int w = tid >> 5;
  for (int i = 0; i < w; ++i) r += __popc(mask[i]);
  return r + __popc(mask[w] & ((1u << (tid & 31)) - 1u));
}

__global__ void __launch_bounds__(kPermTB) k_perm_scatter(const __grid_constant__ PlanTables pt,
                                                          const int32_t* __restrict__ idx, int T,
                                                          const int32_t* __restrict__ chunk_baseE,
                                                          const int32_t* __restrict__ chunk_baseU,
                                                          int32_t* __restrict__ row_pair,
                                                          int32_t* __restrict__ pair_row,
                                                          int32_t* __restrict__ pair_g,
                                                          int32_t* __restrict__ row_uniq,
                                                          int32_t* __restrict__ uniq_tok,
                                                          int32_t* __restrict__ tok_uniq) {
  constexpr int W = kPermTB / 32;
  extern __shared__ uint32_t msk[];
  uint32_t* mE = msk;                    // [E][W]
  uint32_t* mU = msk + (size_t)pt.E * W; // [G][W]
  const int tid = threadIdx.x;
  for (int i = tid; i < (pt.E + pt.G) * W; i += blockDim.x) msk[i] = 0;
  __syncthreads();
  const int c = blockIdx.x;
  const int t = c * kPermTB + tid;
  const int k = pt.k;
  int e[kMaxK];
  bool ok = false;
  if (t < T) {
    ok = read_token(idx, t, k, pt.E, e);
    if (ok) {
      const uint32_t bit = 1u << (tid & 31);
      for (int j = 0; j < k; ++j) {
        atomicOr(&mE[e[j] * W + (tid >> 5)], bit);
        atomicOr(&mU[pt.e2g[e[j]] * W + (tid >> 5)], bit);
      }
    }
  }
  __syncthreads();
  if (t >= T) return;
  if (!ok) {
    for (int j = 0; j < k; ++j) {
      tok_uniq[(int64_t)t * k + j] = -1;
      pair_g[(int64_t)t * k + j] = -1;
    }
    return;
  }
  int rows_j[kMaxK];
  for (int j = 0; j < k; ++j) {
    const int row = chunk_baseE[(int64_t)c * pt.E + e[j]] + prefix_bits(&mE[e[j] * W], tid);
    const int p = t * k + j;
    rows_j[j] = row;
    pair_row[p] = row;
    pair_g[p] = pt.e2g[e[j]];
    row_pair[row] = p;
  }
  // distinct groups of the token, ascending
  int n_u = 0;
  int last = -1;
  while (true) {
    int nxt = 0x7fffffff;
    for (int j = 0; j < k; ++j) {
      int g = pt.e2g[e[j]];
      if (g > last && g < nxt) nxt = g;
    }
    if (nxt == 0x7fffffff) break;
    const int u = chunk_baseU[(int64_t)c * pt.G + nxt] + prefix_bits(&mU[nxt * W], tid);
    uniq_tok[u] = t;
    tok_uniq[(int64_t)t * k + n_u] = u;
    for (int j = 0; j < k; ++j)
      if (pt.e2g[e[j]] == nxt) row_uniq[rows_j[j]] = u;
    ++n_u;
    last = nxt;
  }
  for (int j = n_u; j < k; ++j) tok_uniq[(int64_t)t * k + j] = -1;
}

__global__ void k_rows_copy(const int32_t* __restrict__ row_pair, const uint4* __restrict__ src,
                            uint4* __restrict__ dst, int64_t R, int vec_per_row, bool gather) {
  const int64_t n = R * vec_per_row;
  for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t row = i / vec_per_row, v = i % vec_per_row;
    const int64_t p = row_pair[row];
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
    size_t sm1 = sizeof(int32_t) * (pt.E + pt.G);
    k_perm_count<<<C, kPermTB, sm1, st>>>(pt, topk_idx, T, at<int32_t>(ws, L.chunk_cntE),
                                          at<int32_t>(ws, L.chunk_cntU), at<int32_t>(ws, L.chunk_err));
  }
  k_perm_scan<<<1, 1024, 0, st>>>(pt, C, at<int32_t>(ws, L.chunk_cntE), at<int32_t>(ws, L.chunk_cntU),
                                  at<int32_t>(ws, L.chunk_err), at<int32_t>(ws, L.chunk_baseE),
                                  at<int32_t>(ws, L.chunk_baseU), at<int32_t>(ws, L.err),
                                  at<int32_t>(ws, L.counts), at<int32_t>(ws, L.group_off),
                                  at<int32_t>(ws, L.expert_off), at<int32_t>(ws, L.expert_cnt),
                                  at<int32_t>(ws, L.uniq_off), at<Tile>(ws, L.tiles_sh), at<Tile>(ws, L.tiles_row),
                                  at<Tile>(ws, L.splits_row));
  if (C > 0) {
    size_t sm3 = sizeof(uint32_t) * (size_t)(pt.E + pt.G) * (kPermTB / 32);
    k_perm_scatter<<<C, kPermTB, sm3, st>>>(pt, topk_idx, T, at<int32_t>(ws, L.chunk_baseE),
                                            at<int32_t>(ws, L.chunk_baseU), at<int32_t>(ws, L.row_pair),
                                            at<int32_t>(ws, L.pair_row), at<int32_t>(ws, L.pair_g),
                                            at<int32_t>(ws, L.row_uniq), at<int32_t>(ws, L.uniq_tok),
                                            at<int32_t>(ws, L.tok_uniq));
  }
  return cudaGetLastError();
}

cudaError_t launch_rows_copy(const int32_t* row_pair, const uint16_t* src, uint16_t* dst, int64_t R, int32_t cols,
                             bool gather, cudaStream_t st) {
  if (R == 0) return cudaSuccess;
  const int vpr = cols / 8;
  const int64_t n = R * vpr;
  int blocks = (int)std::min<int64_t>((n + 255) / 256, 152 * 16);
  k_rows_copy<<<blocks, 256, 0, st>>>(row_pair, reinterpret_cast<const uint4*>(src), reinterpret_cast<uint4*>(dst),
                                      R, vpr, gather);
  return cudaGetLastError();
}

}  // namespace ace
