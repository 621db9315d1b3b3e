// Routed expert FFN forward with the group-shared adapters fused into the
// base expert GEMMs (App. "Implementation and Profiling of Grouped Adapter
// Execution": the gated FFN u = (W^up + dW^up) x, v = (W^gate + dW^gate) x,
// h = SiLU(v) * u, y = (W^down + dW^down) h, with dW = s B_g A_g the shared
// adapter of the expert's group, Sec. 3.3-3.5).
//
// k_ffn_fused<RP, GU>: persistent, one CTA per SM, over work items of 128
// rows of one expert (rows are contiguous per expert inside the group
// segments) times an output chunk.  One fp32 TMEM accumulator per item (two,
// so an item's epilogue overlaps the next item's K loop) receives
//   the base product over K = d (gate/up) or K = f (down), 64 columns a
//   stage, tcgen05 M = 128 N = 256, operands K-major, then
//   the adapter as two more K steps of K = r_g: (s H) . B_g^T, with H the
//   deduplicated A_g x of the row's unique pair (gate/up) or the row's A_g h
//   (down), staged as a bf16 operand.
// Gate/up (GU): an item covers 128 columns of f for both projections: TMEM
//   columns [0, 128) take u (W_up, adapter of up), [128, 256) take v (W_gate,
//   adapter of gate); the epilogue writes u, v and h = SiLU(v) u (bf16) --
//   the SiLU gating never leaves the kernel.  The token rows x come in row
//   order (gathered once before the kernel), so every operand comes by TMA.
// Down (DN): an item covers 256 columns of d; h rows come by TMA; the
//   epilogue writes y (bf16).
// Warps: 0 TMA producer, 1 MMA issuer, 2-9 epilogue (thread = row, two
// warps per TMEM lane quarter), 10-13 aux (H staging).
// Every wait is bounded; a wait that gives up raises the error flag and the
// CTA winds down.
#include <algorithm>
#include <cstdint>

#include "ace_internal.cuh"
#include "ace_ptx.cuh"

namespace ace {
namespace {

constexpr int kXThreads = 14 * 32;
constexpr int kXBlk = 128 * 128;              // [128 rows x 64 bf16] SW128 block
constexpr int kXStage = kXBlk + 2 * kXBlk;    // A [128 x 64] + B [256 x 64]
constexpr int kXEpiWarps = 8;                 // epilogue warps

template <int RP, bool GU>
struct FxCfg {
  static constexpr int kN = GU ? 128 : 256;                  // output columns of an item (per projection)
  // bf16 H operand(s) [128 x RP]: gate/up keeps both projections' in one
  // 64-column block side by side when they fit (columns [0, RP) and [RP, 2 RP))
  static constexpr bool kPacked = GU && 2 * RP <= 64;
  static constexpr int kHB = ((RP + 63) / 64) * kXBlk;       // one operand in its own blocks
  static constexpr int kHbytes = kPacked ? kXBlk : (GU ? 2 : 1) * kHB;
  static constexpr int kBudget = 227 * 1024 - 4096 - 1024;   // static shared memory and the alignment slack
  static constexpr int kS0 = (kBudget - kHbytes) / kXStage;
  static constexpr int S = kS0 > 4 ? 4 : kS0;
  static constexpr int kSmem = S * kXStage + kHbytes + 1024;
  static_assert(S >= 2, "pipeline depth");
  static_assert(2 * RP * 128 <= 2 * kXBlk, "adapter B^T chunk fits a stage's B region");
};

// Largest i with off[i] <= v over off[0..n] (off ascending, off[0] <= v).
__device__ __forceinline__ int upper_pos(const int32_t* off, int n, int v) {
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

template <int RP, bool GU>
__global__ void __launch_bounds__(kXThreads, 1) k_ffn_fused(const __grid_constant__ PlanTables pt,
                                                            const __grid_constant__ FfnFusedLaunch a) {
  using C = FxCfg<RP, GU>;
  constexpr int S = C::S, kN = C::kN;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t full[S], empty[S], acc_full[2], acc_empty[2], h_ready, h_free;
  __shared__ uint32_t tslot;
  __shared__ int32_t tpre[ACE_MAX_EXPERTS + 1];  // row tiles before expert e
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int E = pt.E, N = a.N, nchunk = (N + kN - 1) / kN, NK = (a.K + 63) / 64;
  const uint32_t s0 = smem_u32(smem);
  const uint32_t sH = s0 + S * kXStage;
  if (tid == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], kXEpiWarps);
    }
    mbar_init(&h_ready, 4);
    mbar_init(&h_free, 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, 512);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait();
  if (tid == 0) {
    tpre[0] = 0;
    for (int e = 0; e < E; ++e) tpre[e + 1] = tpre[e] + (a.expert_cnt[e] + 127) / 128;
  }
  __syncthreads();
  const int ntile = tpre[E] * nchunk;
  // item -> (expert, first row, rows, first output column)
  auto decode = [&](int tile, int& e, int& row0, int& cnt, int& n0) {
    const int rt = tile / nchunk;
    n0 = (tile % nchunk) * kN;
    e = upper_pos(tpre, E, rt);
    while (e + 1 < E && tpre[e + 1] <= rt) ++e;  // skip experts with no rows
    const int i = rt - tpre[e];
    row0 = a.expert_off[e] + i * 128;
    cnt = min(128, a.expert_cnt[e] - i * 128);
    if (kChecks && (row0 < 0 || cnt < 0 || row0 > a.counts[kCntRows] - cnt)) {
      atomicOr(a.err, kErrCheck);  // an expert segment outside the rows: the item is dropped
      row0 = 0;
      cnt = 0;
    }
  };
  const uint32_t tmem = tslot;
  bool bad = false;

  if (warp == 0) {
    // ------------------------------------------------------------ TMA producer
    if (lane == 0) {
      int i = 0;
      for (int tile = blockIdx.x; tile < ntile && !bad; tile += gridDim.x) {
        int e, row0, cnt, n0;
        decode(tile, e, row0, cnt, n0);
        const int g = pt.e2g[e], r0 = pt.rank_off[g];
        for (int q = 0; q < NK + 2 && !bad; ++q, ++i) {
          const int s = i % S, u = i / S;
          if (u >= 1 && !mbar_wait(&empty[s], (u - 1) & 1)) {
            bad = true;
            break;
          }
          const uint32_t base = s0 + s * kXStage;
          if (q < NK) {  // base K step
            const int k0 = q * 64;
            mbar_arrive_expect_tx(&full[s], 3 * kXBlk);
            tma_load_2d(base, &a.tm_in, k0, row0, &full[s]);
            if (GU) {  // B rows: 128 of W_up, then 128 of W_gate
              tma_load_2d(base + kXBlk, &a.tm_w[0], k0, e * N + n0, &full[s]);
              tma_load_2d(base + 2 * kXBlk, &a.tm_w[1], k0, e * N + n0, &full[s]);
            } else {
              tma_load_2d(base + kXBlk, &a.tm_w[0], k0, e * N + n0, &full[s]);
            }
          } else {  // adapter step: the 128-column B^T chunk of half hq
            const int hq = q - NK;
            const CUtensorMap* bt = &a.tm_bt[GU ? hq : 0];
            const int c0 = GU ? n0 : n0 + hq * 128;
            mbar_arrive_expect_tx(&full[s], 2 * RP * 128);
            tma_load_2d(base + kXBlk, bt, c0, r0, &full[s]);
            tma_load_2d(base + kXBlk + RP * 128, bt, c0 + 64, r0, &full[s]);
          }
        }
      }
      // every copy issued has landed before the CTA can exit
      for (int k = max(0, i - S); k < i; ++k)
        if (!mbar_wait(&full[k % S], (k / S) & 1)) bad = true;
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t id_base = idesc_bf16_f32(128, 256, 0, 0);
      constexpr uint32_t id_ad = idesc_bf16_f32(128, 128, 0, 1);
      int i = 0, it = 0;
      for (int tile = blockIdx.x; tile < ntile && !bad; tile += gridDim.x, ++it) {
        const int b = it & 1;
        if (it >= 2 && !mbar_wait(&acc_empty[b], ((it - 2) >> 1) & 1)) {
          bad = true;
          break;
        }
        tc_fence_after();
        const uint32_t acc = tmem + b * 256;
        for (int q = 0; q < NK + 2 && !bad; ++q, ++i) {
          const int s = i % S;
          if (q == NK && !mbar_wait(&h_ready, it & 1)) {
            bad = true;
            break;
          }
          if (!mbar_wait(&full[s], (i / S) & 1)) {
            bad = true;
            break;
          }
          tc_fence_after();
          const uint32_t base = s0 + s * kXStage;
          if (q < NK) {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc_mma_bf16(acc, sdesc_sw128(base + kk * 32, 16, 1024), sdesc_sw128(base + kXBlk + kk * 32, 16, 1024),
                          id_base, (q > 0 || kk > 0) ? 1u : 0u);
          } else {
            const int hq = q - NK;  // accumulator half: gate/up its projection, down its columns
            const uint32_t hop = C::kPacked ? sH + hq * RP * 2 : sH + (GU ? hq : 0) * C::kHB;
#pragma unroll
            for (int kk = 0; kk < RP / 16; ++kk)
              tc_mma_bf16(acc + hq * 128, sdesc_sw128(hop + (kk >> 2) * kXBlk + (kk & 3) * 32, 16, 1024),
                          sdesc_sw128(base + kXBlk + kk * 2048, RP * 128, 1024), id_ad, 1u);
          }
          tc_commit(&empty[s]);
        }
        if (bad) break;
        tc_commit(&h_free);
        tc_commit(&acc_full[b]);
      }
      // the last commits land before the CTA exits
      if (!bad && it > 0 && !mbar_wait(&h_free, (it - 1) & 1)) bad = true;
    }
  } else if (warp < 2 + kXEpiWarps) {
    // ------------------------------------------------------------ epilogue
    const int quarter = warp & 3, ehalf = (warp - 2) >> 2;
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    const int m = quarter * 32 + lane;
    int it = 0;
    for (int tile = blockIdx.x; tile < ntile; tile += gridDim.x, ++it) {
      const int b = it & 1;
      int e, row0, cnt, n0;
      decode(tile, e, row0, cnt, n0);
      if (!__all_sync(0xffffffffu, mbar_wait(&acc_full[b], (it >> 1) & 1))) {
        bad = true;
        break;
      }
      tc_fence_after();
      const bool live = m < cnt;
      const int64_t row = (int64_t)row0 + m;
      constexpr int kCols = GU ? 64 : 128;  // columns of this warp's share
      for (int c16 = 0; c16 < kCols / 16; ++c16) {
        const int col = ehalf * kCols + c16 * 16;  // within the item
        if (n0 + col >= N) break;                 // warp-uniform
        uint32_t r[16];
        tmem_ld16(tmem + lane_base + b * 256 + col, r);
        if (GU) {
          uint32_t rv[16];
          tmem_ld16(tmem + lane_base + b * 256 + 128 + col, rv);
          tmem_ld_wait();
          float u[16], v[16], h[16];
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            u[q] = __uint_as_float(r[q]);
            v[q] = __uint_as_float(rv[q]);
            h[q] = v[q] / (1.f + __expf(-v[q])) * u[q];
          }
          if (live) {
            const int64_t o = row * N + n0 + col;
#pragma unroll
            for (int h8 = 0; h8 < 2; ++h8) {
              if (n0 + col + h8 * 8 >= N) break;
              uint4 wu, wv, wh;
              wu.x = pack_bf16x2(u[h8 * 8 + 0], u[h8 * 8 + 1]);
              wu.y = pack_bf16x2(u[h8 * 8 + 2], u[h8 * 8 + 3]);
              wu.z = pack_bf16x2(u[h8 * 8 + 4], u[h8 * 8 + 5]);
              wu.w = pack_bf16x2(u[h8 * 8 + 6], u[h8 * 8 + 7]);
              wv.x = pack_bf16x2(v[h8 * 8 + 0], v[h8 * 8 + 1]);
              wv.y = pack_bf16x2(v[h8 * 8 + 2], v[h8 * 8 + 3]);
              wv.z = pack_bf16x2(v[h8 * 8 + 4], v[h8 * 8 + 5]);
              wv.w = pack_bf16x2(v[h8 * 8 + 6], v[h8 * 8 + 7]);
              wh.x = pack_bf16x2(h[h8 * 8 + 0], h[h8 * 8 + 1]);
              wh.y = pack_bf16x2(h[h8 * 8 + 2], h[h8 * 8 + 3]);
              wh.z = pack_bf16x2(h[h8 * 8 + 4], h[h8 * 8 + 5]);
              wh.w = pack_bf16x2(h[h8 * 8 + 6], h[h8 * 8 + 7]);
              *reinterpret_cast<uint4*>(a.U + o + h8 * 8) = wu;
              *reinterpret_cast<uint4*>(a.V + o + h8 * 8) = wv;
              *reinterpret_cast<uint4*>(a.Hh + o + h8 * 8) = wh;
            }
          }
        } else {
          tmem_ld_wait();
          if (live) {
            const int64_t o = row * N + n0 + col;
#pragma unroll
            for (int h8 = 0; h8 < 2; ++h8) {
              if (n0 + col + h8 * 8 >= N) break;
              uint4 w;
              w.x = pack_bf16x2(__uint_as_float(r[h8 * 8 + 0]), __uint_as_float(r[h8 * 8 + 1]));
              w.y = pack_bf16x2(__uint_as_float(r[h8 * 8 + 2]), __uint_as_float(r[h8 * 8 + 3]));
              w.z = pack_bf16x2(__uint_as_float(r[h8 * 8 + 4]), __uint_as_float(r[h8 * 8 + 5]));
              w.w = pack_bf16x2(__uint_as_float(r[h8 * 8 + 6]), __uint_as_float(r[h8 * 8 + 7]));
              *reinterpret_cast<uint4*>(a.Y + o + h8 * 8) = w;
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&acc_empty[b]);
    }
  } else {
    // ------------------------------------------------------------ aux: H staging
    const int t = tid - (2 + kXEpiWarps) * 32;  // 0..127: the item row this thread serves
    int it = 0;
    for (int tile = blockIdx.x; tile < ntile && !bad; tile += gridDim.x, ++it) {
      int e, row0, cnt, n0;
      decode(tile, e, row0, cnt, n0);
      const bool live = t < cnt;
      const int g = pt.e2g[e], r0 = pt.rank_off[g], rg = pt.rank_off[g + 1] - r0;
      // the adapter's H operand(s): s * H of the row (bf16), zero past r_g,
      // once the previous item's adapter MMAs are done with the buffer
      if (it >= 1 && !__all_sync(0xffffffffu, mbar_wait(&h_free, (it - 1) & 1))) {
        bad = true;
        break;
      }
      tc_fence_after();
      const int hrow = live ? (GU ? ACE_CHK(a.row_uniq[row0 + t], 0, a.counts[kCntU], 0, a.err) : row0 + t) : -1;
#pragma unroll
      for (int j = 0; j < (GU ? 2 : 1); ++j) {
        const float* hp = a.Hs[j] + (int64_t)(hrow < 0 ? 0 : hrow) * pt.rank_max;
        for (int c8 = 0; c8 < RP; c8 += 8) {
          float v[8];
#pragma unroll
          for (int qq = 0; qq < 8; ++qq) v[qq] = (hrow >= 0 && c8 + qq < rg) ? a.s * hp[c8 + qq] : 0.f;
          uint4 o;
          o.x = pack_bf16x2(v[0], v[1]);
          o.y = pack_bf16x2(v[2], v[3]);
          o.z = pack_bf16x2(v[4], v[5]);
          o.w = pack_bf16x2(v[6], v[7]);
          if (C::kPacked)
            sts128(sH + sw128_off(t, (j * RP + c8) >> 3), o);
          else
            sts128(sH + j * C::kHB + (c8 >> 6) * kXBlk + sw128_off(t, (c8 & 63) >> 3), o);
        }
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&h_ready);
    }
  }
  __syncwarp();
  tc_fence_before();
  if (__syncthreads_or(bad) && tid == 0) atomicOr(a.err, kErrTimeout);
  pdl_trigger();
  if (warp == 0) tmem_dealloc(tmem, 512);
}

template <int RP, bool GU>
cudaError_t launch_t(const PlanTables& pt, const FfnFusedLaunch& a, cudaStream_t st) {
  using C = FxCfg<RP, GU>;
  auto kern = k_ffn_fused<RP, GU>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
  if (e != cudaSuccess || a.grid <= 0) return e;
  return launch_k(kern, a.grid, kXThreads, C::kSmem, st, pt, a);
}

}  // namespace

cudaError_t launch_ffn_fused(const PlanTables& pt, const FfnFusedLaunch& a, bool gate_up, cudaStream_t st) {
  switch (pt.rank_pad) {
    case 16: return gate_up ? launch_t<16, true>(pt, a, st) : launch_t<16, false>(pt, a, st);
    case 32: return gate_up ? launch_t<32, true>(pt, a, st) : launch_t<32, false>(pt, a, st);
    case 64: return gate_up ? launch_t<64, true>(pt, a, st) : launch_t<64, false>(pt, a, st);
    case 128: return gate_up ? launch_t<128, true>(pt, a, st) : launch_t<128, false>(pt, a, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace ace
