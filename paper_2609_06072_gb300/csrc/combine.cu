// Gate-weighted combine of the down projection (Sec. 3.1: the router weight
// p_e(x) scales each routed expert's output before the sum over R(x); Sec.
// 3.4: expert e uses the group adapter of g(e)).  Within one group the
// weighted sum moves inside the adapter,
//   sum_{e in g, R(t)} p_e B_g (A_g h_e) = B_g (sum_{e in g, R(t)} p_e A_g h_e),
// so the token's output needs one N-side product per active group (the
// reuse of Sec. 3.5, applied to the combined output).  The forward is
//   1. H_row = A_g h_row          (k_fwd_h over the row tiles, fwd.cu)
//   2. Hx[t] = s sum_j p_tj H_row (this file: token-major, one column block
//                                  per group, bf16)
//   3. z[t] += Hx[t] . [B_g^T]    (k_gemm_dx of gemm.cu, K = stacked ranks)
// and Hx is kept for the backward's dB^T = Hx^T . dz (k_gemm_da).
#include <cstdint>

#include "ace_internal.cuh"
#include "ace_ptx.cuh"

namespace ace {
namespace {

constexpr int kReduceThreads = 256;  // one warp per token

// Hx[t] for one token per warp: lane l owns the 8-column blocks
// c = 8 (l + 32 i) of the row; for each of the token's pairs (ascending j)
// the block's columns inside the pair's group add w * H_row.  Lane j < k
// first reads pair j's group, row and weight, and the warp shares them by
// shuffles; a block inside one group whose H row piece is 16-byte aligned is
// read in two 16-byte loads.
__global__ void __launch_bounds__(kReduceThreads) k_comb_reduce(const __grid_constant__ PlanTables pt,
                                                                const __grid_constant__ CombReduceLaunch a) {
  pdl_wait();
  pdl_trigger();
  const int t = blockIdx.x * (kReduceThreads / 32) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (t >= a.T) return;  // warp-uniform
  const int k = pt.k;
  int g_l = -1, row_l = 0;
  float w_l = 0.f;
  if (lane < k) {
    const int64_t p = (int64_t)t * k + lane;
    g_l = ACE_CHK(a.pair_g[p], -1, pt.G, -1, a.err);
    if (g_l >= 0) {  // an invalid token has no rows (the error flag is set)
      row_l = ACE_CHK(a.pair_row[p], 0, a.T * k, 0, a.err);
      w_l = a.w[p];
      if (!isfinite(w_l)) atomicOr(a.err, kErrValue);
    }
  }
  const bool vec = (pt.rank_max & 3) == 0;
  for (int c0 = 0; c0 < a.n_rank_pad; c0 += 8 * 32) {  // warp-uniform trips
    const int c = c0 + 8 * lane;
    float acc[8];
#pragma unroll
    for (int q = 0; q < 8; ++q) acc[q] = 0.f;
    for (int j = 0; j < k; ++j) {
      const int g = __shfl_sync(0xffffffffu, g_l, j);
      const int row = __shfl_sync(0xffffffffu, row_l, j);
      const float wv = __shfl_sync(0xffffffffu, w_l, j);
      if (g < 0 || c >= a.n_rank_pad) continue;
      const int r0 = pt.rank_off[g], r1 = pt.rank_off[g + 1];
      if (c + 8 <= r0 || c >= r1) continue;
      const float* h = a.H + (int64_t)row * pt.rank_max - r0;
      if (vec && c >= r0 && c + 8 <= r1 && (r0 & 3) == 0) {
        const float4 x0 = *reinterpret_cast<const float4*>(h + c);
        const float4 x1 = *reinterpret_cast<const float4*>(h + c + 4);
        acc[0] += wv * x0.x;
        acc[1] += wv * x0.y;
        acc[2] += wv * x0.z;
        acc[3] += wv * x0.w;
        acc[4] += wv * x1.x;
        acc[5] += wv * x1.y;
        acc[6] += wv * x1.z;
        acc[7] += wv * x1.w;
      } else {
#pragma unroll
        for (int q = 0; q < 8; ++q)
          if (c + q >= r0 && c + q < r1) acc[q] += wv * h[c + q];
      }
    }
    if (c >= a.n_rank_pad) continue;
    uint4 o;
    o.x = pack_bf16x2(a.s * acc[0], a.s * acc[1]);
    o.y = pack_bf16x2(a.s * acc[2], a.s * acc[3]);
    o.z = pack_bf16x2(a.s * acc[4], a.s * acc[5]);
    o.w = pack_bf16x2(a.s * acc[6], a.s * acc[7]);
    *reinterpret_cast<uint4*>(a.Hx + (int64_t)t * a.n_rank_pad + c) = o;
  }
}

}  // namespace

cudaError_t launch_comb_reduce(const PlanTables& pt, const CombReduceLaunch& a, cudaStream_t st) {
  if (a.T <= 0) return cudaSuccess;
  const int per = kReduceThreads / 32;
  return launch_k(k_comb_reduce, (a.T + per - 1) / per, kReduceThreads, 0, st, pt, a);
}

}  // namespace ace
