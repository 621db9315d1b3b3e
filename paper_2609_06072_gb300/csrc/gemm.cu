// Dense tcgen05 GEMMs of the gate/up backward over the token-major dH matrix
//   dHx [T, nproj * n_rank_pad] bf16,  dHx[t][j * n_rank_pad + rank_off[g] + k]
//     = (dH_{u(t,g)})_k for projection j when token t routes into group g,
//       zero otherwise
// (Sec. 3.4: the group adapter collects the gradient of every token routed to
// any expert of the group).  With it both remaining gradients are plain
// products over contiguous rows:
//   k_gemm_dx:  dX[t] += sum_j dHx_j[t] . A_j            (M = T, N = d, K = rank)
//   k_gemm_da:  dA_j   = dHx_j^T . X                      (M = rank, N = d, K = T)
// Each output tile is computed with its whole K loop by one CTA, so both are
// deterministic.  Warp-specialised: TMA producer warp, MMA warp, 8 epilogue
// warps.  Operands arrive by TMA in 128-byte-swizzled boxes.
#include <algorithm>
#include <cstdint>

#include "ace_internal.cuh"
#include "ace_ptx.cuh"

namespace ace {
namespace {

constexpr int kThreads = 320;
constexpr int kEpiThreads = 256;
constexpr int kEpiBar = 1;
constexpr int kBlk = 128 * 128;       // [128 rows x 64 bf16]
constexpr int kHalfBlk = 64 * 128;    // [64 rows x 64 bf16]

// ------------------------------------------------------------------ dX
// Persistent: one CTA per SM walks the [128-token x 256-column] output tiles
// (column-fastest, so concurrent CTAs share dHx rows in L2); the tiles left
// over after the last whole round go out as column halves, so that round
// takes half as long and reaches twice as many SMs.  Two TMEM
// accumulators let the epilogue of one tile overlap the K loop of the next.
// Each epilogue warp owns 32 rows x 128 columns, done in two passes of 64
// columns through its own swizzled shared-memory block: the old dX is read
// with coalesced loads (pass 0 into the block, pass 1 into registers, both
// while the K loop still runs), the accumulator rows are added there (thread =
// row) and the block is written back with coalesced stores.  (The small block
// leaves room for four pipeline stages.)
constexpr int kDxN = 256;                               // d columns per tile
constexpr int kDxStage = kBlk + (kDxN / 64) * kHalfBlk; // dHx [128 t x 64 k] + A [64 k x 256 d]
constexpr int kDxS = 4;
constexpr int kDxWarpBlk = 32 * 128;                    // [32 rows x 64 bf16] per epilogue warp
constexpr int kDxSmem = kDxS * kDxStage + 8 * kDxWarpBlk + 1024;
// byte offset of 16-byte chunk c (0..7) of row r (0..31) in a warp block
__device__ __forceinline__ uint32_t dx_off(int r, int c) { return (uint32_t)(r * 128 + ((c ^ (r & 7)) << 4)); }

// Work item `it` of this CTA: a whole tile (half = -1) for the first
// ntile / grid rounds, then one column half of a left-over tile.  False past
// the end.
__device__ __forceinline__ bool dx_item(int it, int ntile, int& tile, int& half) {
  const int grid = gridDim.x, full = ntile / grid, rem = ntile % grid;
  if (it < full) {
    tile = it * grid + blockIdx.x;
    half = -1;
    return true;
  }
  const int h = (it - full) * grid + blockIdx.x;
  if (h >= 2 * rem) return false;
  tile = full * grid + h / 2;
  half = h & 1;
  return true;
}

__global__ void __launch_bounds__(kThreads, 1) k_gemm_dx(const __grid_constant__ DenseBwdLaunch a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t full[kDxS], empty[kDxS], acc_full[2], acc_empty[2];
  __shared__ uint32_t tslot;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int ncol = (a.d + kDxN - 1) / kDxN, ntile = ((a.T + 127) / 128) * ncol;
  const int ksteps = a.n_rank_pad / 64;
  const int NK = a.nproj * ksteps;
  const uint32_t s0 = smem_u32(smem);
  if (tid == 0) {
    for (int i = 0; i < kDxS; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 8);  // every epilogue warp
    }
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, 2 * kDxN);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait();
  const uint32_t tmem = tslot;
  bool bad = false;
  if (warp == 0) {
    if (lane == 0) {
      int i = 0, tile, half;
      for (int it = 0; dx_item(it, ntile, tile, half) && !bad; ++it) {
        const int t0 = (tile / ncol) * 128, c0 = (tile % ncol) * kDxN + (half > 0 ? kDxN / 2 : 0);
        const int nq = half < 0 ? kDxN / 64 : kDxN / 128;  // 64-column boxes of A
        for (int kb = 0; kb < NK; ++kb, ++i) {
          const int s = i % kDxS, u = i / kDxS;
          if (u >= 1 && !mbar_wait(&empty[s], (u - 1) & 1)) {
            bad = true;
            break;
          }
          const int j = kb / ksteps, ks = kb % ksteps;
          const uint32_t base = s0 + s * kDxStage;
          mbar_arrive_expect_tx(&full[s], kBlk + nq * kHalfBlk);
          tma_load_2d(base, &a.tm_dhx, j * a.n_rank_pad + ks * 64, t0, &full[s]);
          for (int q = 0; q < nq; ++q)
            tma_load_2d(base + kBlk + q * kHalfBlk, &a.tm_acat[j], c0 + q * 64, ks * 64, &full[s]);
        }
      }
      // every copy issued has landed before the CTA can exit
      for (int k = max(0, i - kDxS); k < i; ++k)
        if (!mbar_wait(&full[k % kDxS], (k / kDxS) & 1)) bad = true;
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(128, kDxN, 0, 1);
      constexpr uint32_t idesc_half = idesc_bf16_f32(128, kDxN / 2, 0, 1);
      int i = 0, tile, half;
      for (int it = 0; dx_item(it, ntile, tile, half) && !bad; ++it) {
        const int b = it & 1;
        const uint32_t id = half < 0 ? idesc : idesc_half;
        if (it >= 2 && !mbar_wait(&acc_empty[b], ((it - 2) >> 1) & 1)) {
          bad = true;
          break;
        }
        tc_fence_after();
        for (int kb = 0; kb < NK; ++kb, ++i) {
          const int s = i % kDxS;
          if (!mbar_wait(&full[s], (i / kDxS) & 1)) {
            bad = true;
            break;
          }
          tc_fence_after();
          const uint32_t base = s0 + s * kDxStage;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_bf16(tmem + b * kDxN, sdesc_sw128(base + kk * 32, 16, 1024),
                        sdesc_sw128(base + kBlk + kk * 2048, kHalfBlk, 1024), id, (kb > 0 || kk > 0) ? 1u : 0u);
          tc_commit(&empty[s]);
        }
        if (!bad) tc_commit(&acc_full[b]);
      }
    }
  } else {
    const int quarter = warp & 3, ehalf = (warp - 2) >> 2;  // this warp: 32 rows x 128 columns
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    const uint32_t wb = s0 + kDxS * kDxStage + (warp - 2) * kDxWarpBlk;
    int tile, half;
    for (int it = 0; dx_item(it, ntile, tile, half); ++it) {
      const int b = it & 1;
      const int tq = (tile / ncol) * 128 + quarter * 32;  // first token of this warp's rows
      // first column of this warp's block; of a half tile only the ehalf 0
      // warps have one (the accumulator's first 128 columns)
      const int cb = (tile % ncol) * kDxN + (half < 0 ? ehalf : half) * 128;
      const bool idle = half >= 0 && ehalf == 1;
      if (idle) {
        if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[b], (it >> 1) & 1))) {
          bad = true;
          break;
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&acc_empty[b]);
        continue;
      }
      // old dX of the block, four 128-byte rows per instruction: columns
      // [0, 64) into the block, [64, 128) into registers
      uint4 later[8];
#pragma unroll
      for (int k2 = 0; k2 < 8; ++k2) {
        const int r = k2 * 4 + (lane >> 3), c = lane & 7, t = tq + r, col = cb + c * 8;
        const uint4 v = (t < a.T && col < a.d) ? *reinterpret_cast<const uint4*>(a.dX + (int64_t)t * a.d + col)
                                               : make_uint4(0, 0, 0, 0);
        later[k2] = (t < a.T && col + 64 < a.d) ? *reinterpret_cast<const uint4*>(a.dX + (int64_t)t * a.d + col + 64)
                                                : make_uint4(0, 0, 0, 0);
        sts128(wb + dx_off(r, c), v);
      }
      if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[b], (it >> 1) & 1))) {
        bad = true;
        break;
      }
      tc_fence_after();
#pragma unroll
      for (int pass = 0; pass < 2; ++pass) {
        if (pass == 1) {
#pragma unroll
          for (int k2 = 0; k2 < 8; ++k2) sts128(wb + dx_off(k2 * 4 + (lane >> 3), lane & 7), later[k2]);
          __syncwarp();
        }
#pragma unroll
        for (int h = 0; h < 2; ++h) {  // 32-column groups of the pass's 64
          uint32_t r[32];
          const uint32_t ta = tmem + lane_base + b * kDxN + ehalf * 128 + pass * 64 + h * 32;
          tmem_ld16(ta, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
          tmem_ld16(ta + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const uint32_t addr = wb + dx_off(lane, h * 4 + q);
            const uint4 y = lds128(addr);
            const uint32_t* dq = &r[q * 8];
            const float2 f0 = unpack_bf16x2(y.x), f1 = unpack_bf16x2(y.y), f2 = unpack_bf16x2(y.z),
                         f3 = unpack_bf16x2(y.w);
            uint4 o;
            o.x = pack_bf16x2(f0.x + __uint_as_float(dq[0]), f0.y + __uint_as_float(dq[1]));
            o.y = pack_bf16x2(f1.x + __uint_as_float(dq[2]), f1.y + __uint_as_float(dq[3]));
            o.z = pack_bf16x2(f2.x + __uint_as_float(dq[4]), f2.y + __uint_as_float(dq[5]));
            o.w = pack_bf16x2(f3.x + __uint_as_float(dq[6]), f3.y + __uint_as_float(dq[7]));
            sts128(addr, o);
          }
        }
        if (pass == 1) {  // the accumulator is read out
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&acc_empty[b]);
        }
        __syncwarp();
#pragma unroll
        for (int k2 = 0; k2 < 8; ++k2) {
          const int r = k2 * 4 + (lane >> 3), c = lane & 7, t = tq + r, col = cb + pass * 64 + c * 8;
          if (t < a.T && col < a.d)
            *reinterpret_cast<uint4*>(a.dX + (int64_t)t * a.d + col) = lds128(wb + dx_off(r, c));
        }
        __syncwarp();
      }
      __syncwarp();
    }
  }
  __syncwarp();
  tc_fence_before();
  if (__syncthreads_or(bad) && tid == 0) atomicOr(a.err, kErrTimeout);
  // signal dependents only as this CTA finishes: an earlier launch of the
  // next kernel (a whole SM per CTA) measured slower
  pdl_trigger();
  if (warp == 0) tmem_dealloc(tmem, 2 * kDxN);
}

// ------------------------------------------------------------------ dX on CTA pairs
// The same product on clusters of two CTAs whose tensor cores share one
// M = 256 MMA (cta_group::2): a pair computes a [256-token x 256-column] tile,
// each CTA holding the dHx rows of its 128 tokens and 128 of the 256 weight
// columns, so a CTA receives 32 KB per K step for the work that takes 48 KB
// on a single CTA, and six stages fit in flight.  Both CTAs' loads count on
// the leader's stage barrier; the leader issues the MMAs and its commits
// arrive in both CTAs; each CTA's epilogue reads its own 128 accumulator rows
// and tells the leader when they are read.  Two accumulators of 256 columns,
// so a tile's epilogue overlaps the next tile's K loop; the tiles left after
// the last whole round go out as column halves (N = 128).
constexpr int kD2S = 6;
constexpr int kD2Stage = kBlk + 2 * kHalfBlk;  // dHx [128 t x 64 k] + A [64 k x 128 d]
constexpr int kD2Smem = kD2S * kD2Stage + 8 * kDxWarpBlk + 1024;
constexpr uint32_t kD2Tmem = 512;

// Work item `it` of pair `pair` (of npair): as dx_item, over pair tiles.
__device__ __forceinline__ bool d2_item(int it, int ntile, int pair, int npair, int& tile, int& half) {
  const int full = ntile / npair, rem = ntile % npair;
  if (it < full) {
    tile = it * npair + pair;
    half = -1;
    return true;
  }
  const int h = (it - full) * npair + pair;
  if (h >= 2 * rem) return false;
  tile = full * npair + h / 2;
  half = h & 1;
  return true;
}

__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    k_gemm2_dx(const __grid_constant__ DenseBwdLaunch a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t full[kD2S], empty[kD2S], acc_full[2], acc_empty[2];
  __shared__ uint32_t tslot;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const uint32_t rank = cluster_ctarank();
  const int npair = gridDim.x / 2, pair = blockIdx.x / 2;
  const int ncol = (a.d + kDxN - 1) / kDxN, ntile = ((a.T + 255) / 256) * ncol;
  const int ksteps = a.n_rank_pad / 64;
  const int NK = a.nproj * ksteps;
  const uint32_t s0 = smem_u32(smem);
  if (tid == 0) {
    for (int i = 0; i < kD2S; ++i) {
      mbar_init(&full[i], 1);   // the leader's arm; both CTAs' bytes
      mbar_init(&empty[i], 1);  // the leader's commit
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 16);  // every epilogue warp of both CTAs
    }
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc_pair(&tslot, kD2Tmem);
  tc_fence_before();
  __syncthreads();
  cluster_sync();  // the peer's barriers exist before anything arrives on them
  tc_fence_after();
  pdl_wait();
  if (a.early_signal) pdl_trigger();  // the dA GEMM that follows does not read dX
  const uint32_t tmem = tslot;
  bool bad = false;
  if (warp == 0) {
    // ------------------------------------------------------------ producer (both CTAs)
    if (lane == 0) {
      int i = 0, tile, half;
      for (int it = 0; d2_item(it, ntile, pair, npair, tile, half) && !bad; ++it) {
        const int t0 = (tile / ncol) * 256 + (int)rank * 128;
        // this CTA's half of the item's columns (a whole tile: 128 of 256; a column half: 64 of 128)
        const int cw = half < 0 ? 128 : 64;
        const int c0 = (tile % ncol) * kDxN + (half > 0 ? kDxN / 2 : 0) + (int)rank * cw;
        for (int kb = 0; kb < NK; ++kb, ++i) {
          const int s = i % kD2S, u = i / kD2S;
          if (u >= 1 && !mbar_wait(&empty[s], (u - 1) & 1)) {
            bad = true;
            break;
          }
          const int j = kb / ksteps, ks = kb % ksteps;
          const uint32_t base = s0 + s * kD2Stage;
          const uint32_t bar = mapa_shared(smem_u32(&full[s]), 0);
          if (rank == 0) mbar_arrive_expect_tx(&full[s], 2 * (kBlk + (cw / 64) * kHalfBlk));
          tma_load_2d_pair(base, &a.tm_dhx, j * a.n_rank_pad + ks * 64, t0, bar);
          tma_load_2d_pair(base + kBlk, &a.tm_acat[j], c0, ks * 64, bar);
          if (cw == 128) tma_load_2d_pair(base + kBlk + kHalfBlk, &a.tm_acat[j], c0 + 64, ks * 64, bar);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer (leader)
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(256, kDxN, 0, 1);
      constexpr uint32_t idesc_half = idesc_bf16_f32(256, kDxN / 2, 0, 1);
      int i = 0, tile, half;
      for (int it = 0; d2_item(it, ntile, pair, npair, tile, half) && !bad; ++it) {
        const int b = it & 1;
        const uint32_t id = half < 0 ? idesc : idesc_half;
        if (it >= 2 && !mbar_wait(&acc_empty[b], ((it - 2) >> 1) & 1)) {
          bad = true;
          break;
        }
        tc_fence_after();
        for (int kb = 0; kb < NK; ++kb, ++i) {
          const int s = i % kD2S;
          if (!mbar_wait(&full[s], (i / kD2S) & 1)) {
            bad = true;
            break;
          }
          tc_fence_after();
          const uint32_t base = s0 + s * kD2Stage;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_bf16_pair(tmem + b * kDxN, sdesc_sw128(base + kk * 32, 16, 1024),
                             sdesc_sw128(base + kBlk + kk * 2048, kHalfBlk, 1024), id, (kb > 0 || kk > 0) ? 1u : 0u);
          tc_commit_pair(&empty[s]);
        }
        if (!bad) tc_commit_pair(&acc_full[b]);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue (both CTAs): this CTA's 128 tokens
    const int quarter = warp & 3, ehalf = (warp - 2) >> 2;  // this warp: 32 rows x 128 columns
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    const uint32_t wb = s0 + kD2S * kD2Stage + (warp - 2) * kDxWarpBlk;
    const uint32_t acc_empty_leader[2] = {mapa_shared(smem_u32(&acc_empty[0]), 0),
                                          mapa_shared(smem_u32(&acc_empty[1]), 0)};
    int tile, half;
    for (int it = 0; d2_item(it, ntile, pair, npair, tile, half); ++it) {
      const int b = it & 1;
      const int tq = (tile / ncol) * 256 + (int)rank * 128 + quarter * 32;  // first token of this warp's rows
      // first column of this warp's block; of a column half only the ehalf 0
      // warps have one (the accumulator's first 128 columns)
      const int cb = (tile % ncol) * kDxN + (half < 0 ? ehalf : half) * 128;
      if (half >= 0 && ehalf == 1) {
        if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[b], (it >> 1) & 1))) {
          bad = true;
          break;
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster(acc_empty_leader[b]);
        continue;
      }
      uint4 later[8];
#pragma unroll
      for (int k2 = 0; k2 < 8; ++k2) {
        const int r = k2 * 4 + (lane >> 3), c = lane & 7, t = tq + r, col = cb + c * 8;
        const uint4 v = (t < a.T && col < a.d) ? *reinterpret_cast<const uint4*>(a.dX + (int64_t)t * a.d + col)
                                               : make_uint4(0, 0, 0, 0);
        later[k2] = (t < a.T && col + 64 < a.d) ? *reinterpret_cast<const uint4*>(a.dX + (int64_t)t * a.d + col + 64)
                                                : make_uint4(0, 0, 0, 0);
        sts128(wb + dx_off(r, c), v);
      }
      if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[b], (it >> 1) & 1))) {
        bad = true;
        break;
      }
      tc_fence_after();
#pragma unroll
      for (int pass = 0; pass < 2; ++pass) {
        if (pass == 1) {
#pragma unroll
          for (int k2 = 0; k2 < 8; ++k2) sts128(wb + dx_off(k2 * 4 + (lane >> 3), lane & 7), later[k2]);
          __syncwarp();
        }
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          uint32_t r[32];
          const uint32_t ta = tmem + lane_base + b * kDxN + ehalf * 128 + pass * 64 + h * 32;
          tmem_ld16(ta, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
          tmem_ld16(ta + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const uint32_t addr = wb + dx_off(lane, h * 4 + q);
            const uint4 y = lds128(addr);
            const uint32_t* dq = &r[q * 8];
            const float2 f0 = unpack_bf16x2(y.x), f1 = unpack_bf16x2(y.y), f2 = unpack_bf16x2(y.z),
                         f3 = unpack_bf16x2(y.w);
            uint4 o;
            o.x = pack_bf16x2(f0.x + __uint_as_float(dq[0]), f0.y + __uint_as_float(dq[1]));
            o.y = pack_bf16x2(f1.x + __uint_as_float(dq[2]), f1.y + __uint_as_float(dq[3]));
            o.z = pack_bf16x2(f2.x + __uint_as_float(dq[4]), f2.y + __uint_as_float(dq[5]));
            o.w = pack_bf16x2(f3.x + __uint_as_float(dq[6]), f3.y + __uint_as_float(dq[7]));
            sts128(addr, o);
          }
        }
        if (pass == 1) {  // this warp's accumulator rows are read out: tell the leader
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive_cluster(acc_empty_leader[b]);
        }
        __syncwarp();
#pragma unroll
        for (int k2 = 0; k2 < 8; ++k2) {
          const int r = k2 * 4 + (lane >> 3), c = lane & 7, t = tq + r, col = cb + pass * 64 + c * 8;
          if (t < a.T && col < a.d)
            *reinterpret_cast<uint4*>(a.dX + (int64_t)t * a.d + col) = lds128(wb + dx_off(r, c));
        }
        __syncwarp();
      }
      __syncwarp();
    }
  }
  __syncwarp();
  tc_fence_before();
  if (__syncthreads_or(bad) && tid == 0) atomicOr(a.err, kErrTimeout);
  cluster_sync();  // no arrival or copy of the pair is still headed for this CTA
  pdl_trigger();
  if (warp == 0) tmem_dealloc_pair(tmem, kD2Tmem);
}

// ------------------------------------------------------------------ dA
// Output tiles of [128 stacked rank rows x 256 columns]; when the tiles alone
// leave SMs idle the token (K) loop is split in two halves, and each CTA adds
// its fp32 tile into the zeroed dA with bulk tensor reduce-adds.  Each element
// then receives at most two addends on top of 0, and a + b == b + a in
// floating point, so the result does not depend on their order.
constexpr int kDaN = 256;                                        // d columns per tile
constexpr int kDaStage = 2 * kHalfBlk + (kDaN / 64) * kHalfBlk;  // dHx^T [64 t x 128 k] + X [64 t x 256 d]
constexpr int kDaS = 4;
constexpr int kDaWarpStg = 32 * 128;                             // [32 rows x 32 fp32] per epilogue warp
constexpr int kDaSmem = kDaS * kDaStage + 8 * kDaWarpStg + 1024;

__host__ __device__ inline int da_ksplit(int tiles, int grid) { return tiles * 2 <= grid ? 2 : 1; }

__global__ void __launch_bounds__(kThreads, 1) k_gemm_da(const __grid_constant__ DenseBwdLaunch a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t full[kDaS], empty[kDaS], acc_full;
  __shared__ uint32_t tslot;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int mt = (a.nproj * a.n_rank_pad + 127) / 128, nt = (a.d + kDaN - 1) / kDaN;
  const int ks = da_ksplit(mt * nt, a.grid);
  const int tile = blockIdx.x / ks, half = blockIdx.x % ks;
  const int m0 = (tile / nt) * 128;  // row of the stacked [nproj * n_rank_pad] rank dimension
  const int c0 = (tile % nt) * kDaN;
  const int nkb = (a.T + 63) / 64;
  const int kb0 = half * nkb / ks, kb1 = (half + 1) * nkb / ks, NK = kb1 - kb0;
  const uint32_t s0 = smem_u32(smem);
  if (tid == 0) {
    for (int i = 0; i < kDaS; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    mbar_init(&acc_full, 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, kDaN);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  // no_wait (launch_dense_bwd): the inputs were complete before the dX GEMM's
  // own wait returned, so the wait moves to the end (below), where it keeps
  // this grid from completing before the dX GEMM
  if (!a.no_wait) pdl_wait();
  const uint32_t tmem = tslot;
  bool bad = false;
  if (warp == 0) {
    if (lane == 0) {
      int i = 0;
      for (; i < NK; ++i) {
        const int s = i % kDaS, u = i / kDaS;
        if (u >= 1 && !mbar_wait(&empty[s], (u - 1) & 1)) {
          bad = true;
          break;
        }
        const int t0 = (kb0 + i) * 64;
        const uint32_t base = s0 + s * kDaStage;
        mbar_arrive_expect_tx(&full[s], kDaStage);
        tma_load_2d(base, &a.tm_dhx_t, m0, t0, &full[s]);
        tma_load_2d(base + kHalfBlk, &a.tm_dhx_t, m0 + 64, t0, &full[s]);
        for (int q = 0; q < kDaN / 64; ++q)
          tma_load_2d(base + 2 * kHalfBlk + q * kHalfBlk, &a.tm_x, c0 + q * 64, t0, &full[s]);
      }
      for (int k = max(0, i - kDaS); k < i; ++k)
        if (!mbar_wait(&full[k % kDaS], (k / kDaS) & 1)) bad = true;
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(128, kDaN, 1, 1);
      for (int i = 0; i < NK; ++i) {
        const int s = i % kDaS;
        if (!mbar_wait(&full[s], (i / kDaS) & 1)) {
          bad = true;
          break;
        }
        tc_fence_after();
        const uint32_t base = s0 + s * kDaStage;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          tc_mma_bf16(tmem, sdesc_sw128(base + kk * 2048, kHalfBlk, 1024),
                      sdesc_sw128(base + 2 * kHalfBlk + kk * 2048, kHalfBlk, 1024), idesc, (i > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&empty[s]);
      }
      if (!bad) tc_commit(&acc_full);
    }
  } else {
    const int quarter = warp & 3, ehalf = (warp - 2) >> 2;  // this warp: 32 rank rows x 128 columns
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    const uint32_t stg = s0 + kDaS * kDaStage + (warp - 2) * kDaWarpStg;
    const int r0 = m0 + quarter * 32, j = r0 / a.n_rank_pad, rr0 = r0 % a.n_rank_pad;
    bool ok = NK == 0 || mbar_wait(&acc_full, 0);
    ok = __all_sync(0xffffffffu, ok);
    if (ok && NK > 0 && j < a.nproj && rr0 < a.n_rank) {
      tc_fence_after();
#pragma unroll 1
      for (int h = 0; h < 4; ++h) {  // 32-column groups of this warp's 128
        const int col = c0 + ehalf * 128 + h * 32;
        uint32_t v[32];
        tmem_ld16(tmem + lane_base + ehalf * 128 + h * 32, *reinterpret_cast<uint32_t(*)[16]>(&v[0]));
        tmem_ld16(tmem + lane_base + ehalf * 128 + h * 32 + 16, *reinterpret_cast<uint32_t(*)[16]>(&v[16]));
        tmem_ld_wait();
        if (lane == 0) bulk_wait_read0();  // the previous group's box has been read
        __syncwarp();
        // row = lane, 128-byte swizzle of the tensor map
#pragma unroll
        for (int q = 0; q < 8; ++q)
          sts128(stg + lane * 128 + ((q ^ (lane & 7)) << 4), make_uint4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]));
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0 && col < a.d) {
          tma_reduce_add_2d(&a.tm_da[j], stg, col, rr0);
          bulk_commit();
        }
      }
      if (lane == 0) bulk_wait0();
    }
    if (!ok) bad = true;
  }
  __syncwarp();
  tc_fence_before();
  if (__syncthreads_or(bad) && tid == 0) atomicOr(a.err, kErrTimeout);
  if (a.no_wait) pdl_wait();
  // signal dependents only as this CTA finishes: an earlier launch of the
  // next kernel (a whole SM per CTA) measured slower
  pdl_trigger();
  if (warp == 0) tmem_dealloc(tmem, kDaN);
}

// ------------------------------------------------------------------ H
// Token-major H of the gate/up forward: H_u = A_g x_t for every active pair
// u = (g, t) (Sec. 3.5), for a block of 128 consecutive tokens against 256
// stacked rank rows of A_j at a time.  X is read once per token block by TMA
// instead of once per active group of each token, and the MMA also forms the
// products of the groups a token does not route to, which the epilogue drops:
// each H_u is still computed once and written once, into the same
// per-unique-pair layout as the gathering kernel of fwd.cu.  Persistent over
// [128-token x 256-rank] tiles (rank blocks fastest, so concurrent CTAs share
// the X block in L2), two TMEM accumulators, four 48 KB stages.
constexpr int kHN = 256;                                // rank rows per tile
constexpr int kHStageB = kBlk + (kHN / 64) * kHalfBlk;  // X [128 t x 64 d] + A [256 r x 64 d]
constexpr int kHS = 4;
constexpr int kHSmem = kHS * kHStageB + 1024;

// Largest i with off[i] <= v over off[0..n] (off ascending, off[0] <= v).
__device__ __forceinline__ int upper_idx(const int32_t* off, int n, int v) {
  int lo = 0, hi = n;
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (off[mid] <= v)
      lo = mid;
    else
      hi = mid;
  }
  return lo;
}

template <int KB>
__global__ void __launch_bounds__(kThreads, 1) k_gemm_h(const __grid_constant__ PlanTables pt,
                                                        const __grid_constant__ DenseHLaunch a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t full[kHS], empty[kHS], acc_full[2], acc_empty[2];
  __shared__ uint32_t tslot;
  __shared__ int32_t uoff_s[ACE_MAX_EXPERTS + 1], roff_s[ACE_MAX_EXPERTS + 1];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int G = pt.G, k = pt.k;
  const int ncb = (a.n_rank + kHN - 1) / kHN, nper = a.nproj * ncb;
  const int ntile = ((a.T + 127) / 128) * nper;
  const int NK = (a.d + 63) / 64;
  const uint32_t s0 = smem_u32(smem);
  if (tid == 0) {
    for (int i = 0; i < kHS; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 8);  // every epilogue warp
    }
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, 2 * kHN);
  for (int i = tid; i <= G; i += blockDim.x) roff_s[i] = pt.rank_off[i];
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait();
  for (int i = tid; i <= G; i += blockDim.x) uoff_s[i] = a.uniq_off[i];
  __syncthreads();
  const uint32_t tmem = tslot;
  bool bad = false;
  if (warp == 0) {
    if (lane == 0) {
      int i = 0;
      for (int tile = blockIdx.x; tile < ntile && !bad; tile += gridDim.x) {
        const int t0 = (tile / nper) * 128, j = (tile % nper) / ncb, r0 = (tile % ncb) * kHN;
        for (int kb = 0; kb < NK; ++kb, ++i) {
          const int s = i % kHS, u = i / kHS;
          if (u >= 1 && !mbar_wait(&empty[s], (u - 1) & 1)) {
            bad = true;
            break;
          }
          const uint32_t base = s0 + s * kHStageB;
          mbar_arrive_expect_tx(&full[s], kHStageB);
          tma_load_2d(base, &a.tm_x, kb * 64, t0, &full[s]);
          tma_load_2d(base + kBlk, &a.tm_a[j], kb * 64, r0, &full[s]);
        }
      }
      // every copy issued has landed before the CTA can exit
      for (int k2 = max(0, i - kHS); k2 < i; ++k2)
        if (!mbar_wait(&full[k2 % kHS], (k2 / kHS) & 1)) bad = true;
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(128, kHN, 0, 0);
      int i = 0, it = 0;
      for (int tile = blockIdx.x; tile < ntile && !bad; tile += gridDim.x, ++it) {
        const int b = it & 1;
        if (it >= 2 && !mbar_wait(&acc_empty[b], ((it - 2) >> 1) & 1)) {
          bad = true;
          break;
        }
        tc_fence_after();
        for (int kb = 0; kb < NK; ++kb, ++i) {
          const int s = i % kHS;
          if (!mbar_wait(&full[s], (i / kHS) & 1)) {
            bad = true;
            break;
          }
          tc_fence_after();
          const uint32_t base = s0 + s * kHStageB;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_bf16(tmem + b * kHN, sdesc_sw128(base + kk * 32, 16, 1024),
                        sdesc_sw128(base + kBlk + kk * 32, 16, 1024), idesc, (kb > 0 || kk > 0) ? 1u : 0u);
          tc_commit(&empty[s]);
        }
        if (!bad) tc_commit(&acc_full[b]);
      }
    }
  } else {
    // this warp: TMEM lane quarter `quarter` (32 tokens) x 128 of the tile's 256 rank columns
    const int quarter = warp & 3, ehalf = (warp - 2) >> 2;
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    int it = 0;
    for (int tile = blockIdx.x; tile < ntile; tile += gridDim.x, ++it) {
      const int b = it & 1;
      const int t = (tile / nper) * 128 + quarter * 32 + lane, j = (tile % nper) / ncb;
      const int c_lo = (tile % ncb) * kHN + ehalf * 128;  // first rank column of this warp
      // this token's active pairs and their groups (ascending g)
      int uu[KB], gu[KB];
#pragma unroll
      for (int n = 0; n < KB; ++n) {
        uu[n] = (t < a.T && n < k) ? ACE_CHK(a.tok_uniq[(int64_t)t * k + n], -1, uoff_s[G], -1, a.err) : -1;
        gu[n] = uu[n] >= 0 ? upper_idx(uoff_s, G, uu[n]) : -1;
      }
      if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[b], (it >> 1) & 1))) {
        bad = true;
        break;
      }
      tc_fence_after();
      float* __restrict__ Hj = a.H[j];
      for (int c16 = 0; c16 < 8; ++c16) {
        const int c = c_lo + c16 * 16;
        if (c >= a.n_rank) break;  // warp-uniform
        uint32_t r[16];
        tmem_ld16(tmem + lane_base + b * kHN + ehalf * 128 + c16 * 16, r);
        tmem_ld_wait();
        // the groups whose rank rows meet columns [c, c + 16)
        const int g_lo = upper_idx(roff_s, G, c), g_hi = upper_idx(roff_s, G, min(c + 15, a.n_rank - 1));
        for (int gg = g_lo; gg <= g_hi; ++gg) {
          int u = -1;
#pragma unroll
          for (int n = 0; n < KB; ++n)
            if (gu[n] == gg) u = uu[n];
          if (u < 0) continue;
          const int off = roff_s[gg], end = roff_s[gg + 1];
          float* hrow = Hj + (int64_t)u * a.rank_max - off;
          if (c >= off && c + 16 <= end && ((a.rank_max | off) & 3) == 0) {  // 16-byte aligned, all in the group
#pragma unroll
            for (int q = 0; q < 4; ++q)
              *reinterpret_cast<float4*>(hrow + c + 4 * q) =
                  make_float4(__uint_as_float(r[4 * q]), __uint_as_float(r[4 * q + 1]), __uint_as_float(r[4 * q + 2]),
                              __uint_as_float(r[4 * q + 3]));
          } else {
#pragma unroll
            for (int q = 0; q < 16; ++q)
              if (c + q >= off && c + q < end) hrow[c + q] = __uint_as_float(r[q]);
          }
          if (end <= c + 16)  // the group ends here: zero its row's columns past r_g
            for (int q = end - off; q < a.rank_max; ++q) hrow[off + q] = 0.f;
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[b]);
    }
  }
  __syncwarp();
  tc_fence_before();
  if (__syncthreads_or(bad) && tid == 0) atomicOr(a.err, kErrTimeout);
  pdl_trigger();
  if (warp == 0) tmem_dealloc(tmem, 2 * kHN);
}

}  // namespace

cudaError_t launch_dense_h(const PlanTables& pt, const DenseHLaunch& a, cudaStream_t st) {
  if (a.T == 0) return cudaSuccess;
  auto kern = pt.k <= 8 ? k_gemm_h<8> : k_gemm_h<kMaxK>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kHSmem);
  if (e != cudaSuccess) return e;
  const int tiles = ((a.T + 127) / 128) * a.nproj * ((a.n_rank + kHN - 1) / kHN);
  return launch_k(kern, std::min(tiles, a.grid), kThreads, kHSmem, st, pt, a);
}

cudaError_t launch_dense_dx(const DenseBwdLaunch& a, cudaStream_t st) {
  if (a.T == 0) return cudaSuccess;
  if (a.T >= 256 && a.grid >= 2) {
    // CTA pairs: one per two SMs
    cudaError_t e = cudaFuncSetAttribute(k_gemm2_dx, cudaFuncAttributeMaxDynamicSharedMemorySize, kD2Smem);
    if (e != cudaSuccess) return e;
    const int pairs = std::min(((a.T + 255) / 256) * ((a.d + kDxN - 1) / kDxN), a.grid / 2);
    return launch_k(k_gemm2_dx, 2 * pairs, kThreads, kD2Smem, st, a);
  }
  cudaError_t e = cudaFuncSetAttribute(k_gemm_dx, cudaFuncAttributeMaxDynamicSharedMemorySize, kDxSmem);
  if (e != cudaSuccess) return e;
  const int dx_tiles = ((a.T + 127) / 128) * ((a.d + kDxN - 1) / kDxN);
  return launch_k(k_gemm_dx, std::min(dx_tiles, a.grid), kThreads, kDxSmem, st, a);
}

cudaError_t launch_dense_da(const DenseBwdLaunch& a, cudaStream_t st) {
  if (a.T == 0) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(k_gemm_da, cudaFuncAttributeMaxDynamicSharedMemorySize, kDaSmem);
  if (e != cudaSuccess) return e;
  // dA accumulates bulk reduce-adds: the caller has zeroed it (with the
  // backward's other accumulation targets, in one launch)
  const int da_tiles = ((a.nproj * a.n_rank_pad + 127) / 128) * ((a.d + kDaN - 1) / kDaN);
  return launch_k(k_gemm_da, da_tiles * da_ksplit(da_tiles, a.grid), kThreads, kDaSmem, st, a);
}

cudaError_t launch_dense_bwd(const DenseBwdLaunch& a, cudaStream_t st) {
  DenseBwdLaunch x = a, d = a;
  // the pair kernel signals early; the one-CTA dX kernel (T < 256) keeps the
  // plain chain
  x.early_signal = a.T >= 256 && a.grid >= 2;
  d.no_wait = x.early_signal;
  cudaError_t e = launch_dense_dx(x, st);
  return e != cudaSuccess ? e : launch_dense_da(d, st);
}

}  // namespace ace
