// Fused LoRA forward of one group tile (Sec. 3.3-3.5, App. implementation):
//
//   H = X_tile . A_g^T        tcgen05, K = d_in, N = nproj * rank_pad  (TMEM)
//   H_save <- H (fp32)        for the backward
//   D = bf16(H) . B_g^T       tcgen05, K = rank_pad, N = 128-column chunks of d_out
//   Y[row] += s * D[u]        bf16 read-modify-write of every routed row
//
// SHARED (gate / up): a tile is up to 128 unique (g, t) pairs of one group;
// X rows are gathered by token and c_g(x) is computed once per pair, then
// added to every row (g, e, t) of that token in the group -- the reuse of
// Sec. 3.5.  Gate and up share the X gather and one MMA with N = 2 * rank_pad.
// ROW (down): a tile is up to 128 consecutive rows of one group.
//
// Operands are staged by cp.async (gathered rows cannot use a tiled tensor
// map) into 128-byte-swizzled shared memory; one thread issues the MMAs and
// commits them to an mbarrier; every wait is bounded.
#include <cstdint>

#include "ace_internal.cuh"
#include "ace_ptx.cuh"

namespace ace {
namespace {

constexpr int kStages = 3;
constexpr int kThreads = 256;  // warps w and w+4 share TMEM lanes 32*(w%4)..
constexpr int kBlk = kTileM * 128;

template <int RP, int NPROJ>
struct FwdCfg {
  // D chunk: 256 TMEM columns = NPROJ x kNc output columns; each warp half
  // (w / 4) owns 128 of them (one projection, or half of the chunk).
  static constexpr int kNc = NPROJ == 2 ? 128 : 256;
  static constexpr int kStageX = kTileM * 128;             // 128 rows x 64 bf16
  static constexpr int kStageA = NPROJ * RP * 128;         // NPROJ*RP rows x 64 bf16
  static constexpr int kStage = kStageX + kStageA;
  static constexpr int kHs = ((NPROJ * RP + 63) / 64) * kBlk;
  static constexpr int kBs = NPROJ * RP * kNc * 2;          // MN-major blocks of 64 columns
  static constexpr int kPhase1 = kStages * kStage;
  static constexpr int kPhase2 = kHs + 2 * kBs;
  static constexpr int kSmem = (kPhase1 > kPhase2 ? kPhase1 : kPhase2) + 1024;
  static constexpr int kTmemCols = 256;
};

template <int RP, int NPROJ, bool SHARED>
__global__ void __launch_bounds__(kThreads, 2) k_fwd(const __grid_constant__ PlanTables pt,
                                                  const __grid_constant__ FwdLaunch a) {
  using C = FwdCfg<RP, NPROJ>;
  constexpr int kNc = C::kNc;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bar_k[kStages];
  __shared__ __align__(8) uint64_t bar_d;
  __shared__ uint32_t tslot;
  __shared__ int32_t src_row[kTileM];

  const int n_tiles = a.counts[a.count_slot];
  if ((int)blockIdx.x >= n_tiles) return;
  const Tile tl = a.tiles[blockIdx.x];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int quarter = warp & 3, half = warp >> 2;
  const int m = quarter * 32 + lane;  // TMEM lane = tile row (unique pair or row)
  const int g = tl.g, r0 = pt.rank_off[g], rg = pt.rank_off[g + 1] - r0;
  const int d_in = a.d_in, d_out = a.d_out;

  if (tid < kTileM) src_row[tid] = tid < tl.cnt ? (SHARED ? a.uniq_tok[tl.start + tid] : tl.start + tid) : -1;
  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) mbar_init(&bar_k[i], 1);
    mbar_init(&bar_d, 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tslot;
  const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;

  // ---------------------------------------------------------- phase 1: H
  const int NK = (d_in + 63) / 64;
  auto load_stage = [&](int kt, int slot) {
    const uint32_t sX = smem_u32(smem + slot * C::kStage);
    const uint32_t sA = sX + C::kStageX;
    const int k0 = kt * 64;
#pragma unroll
    for (int i = 0; i < 1024 / kThreads; ++i) {
      const int idx = i * kThreads + tid, r = idx >> 3, c = idx & 7;
      const int sr = src_row[r], kc = k0 + c * 8;
      const bool v = sr >= 0 && kc < d_in;
      cp_async16(sX + sw128_off(r, c), v ? a.X + (int64_t)sr * d_in + kc : a.X, v);
    }
#pragma unroll
    for (int idx = tid; idx < NPROJ * RP * 8; idx += kThreads) {
      const int rr = idx >> 3, c = idx & 7, j = rr / RP, kr = rr % RP, kc = k0 + c * 8;
      const bool v = kr < rg && kc < d_in;
      cp_async16(sA + sw128_off(rr, c), v ? a.A[j] + (int64_t)(r0 + kr) * d_in + kc : a.A[0], v);
    }
  };

  constexpr uint32_t idesc_h = idesc_bf16_f32(128, NPROJ * RP, 0, 0);
#pragma unroll
  for (int s = 0; s < kStages - 1; ++s) {
    if (s < NK) load_stage(s, s);
    cp_async_commit();
  }
  bool bad = false, aborted = false;  // bad: this thread's wait gave up; aborted: CTA-uniform
  for (int kt = 0; kt < NK; ++kt) {
    const int slot = kt % kStages;
    cp_async_wait<kStages - 2>();
    fence_proxy_async_smem();
    if (__syncthreads_or(bad)) {
      aborted = true;
      break;
    }
    if (tid == 0) {
      tc_fence_after();
      const uint32_t sX = smem_u32(smem + slot * C::kStage), sA = sX + C::kStageX;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        tc_mma_bf16(tmem, sdesc_sw128(sX + kk * 32, 16, 1024), sdesc_sw128(sA + kk * 32, 16, 1024), idesc_h,
                    (kt > 0 || kk > 0) ? 1u : 0u);
      tc_commit(&bar_k[slot]);
    }
    const int nxt = kt + kStages - 1;
    if (nxt < NK) {
      if (kt >= 1 && !mbar_wait(&bar_k[nxt % kStages], ((kt - 1) / kStages) & 1)) bad = true;
      if (!bad) load_stage(nxt, nxt % kStages);
    }
    cp_async_commit();
  }
  cp_async_wait<0>();
  if (NK > 0 && !aborted && !bad && !mbar_wait(&bar_k[(NK - 1) % kStages], ((NK - 1) / kStages) & 1)) bad = true;
  tc_fence_before();
  aborted = __syncthreads_or(bad || aborted);
  tc_fence_after();
  if (aborted) {
    if (tid == 0) atomicOr(a.err, kErrTimeout);
    if (warp == 0) tmem_dealloc(tmem, C::kTmemCols);
    return;
  }

  // ---------------------------------------------------------- H -> H_save, Hs
  uint8_t* Hs = smem;
  uint8_t* Bs = smem + C::kHs;
  const bool row_valid = m < tl.cnt;
  // warp half h extracts columns [h * NPROJ*RP/2, (h+1) * NPROJ*RP/2) (16-column units)
  constexpr int kHcols = NPROJ * RP;
  for (int c0 = half * 16; c0 < kHcols; c0 += 32) {
    uint32_t r[16];
    tmem_ld16(tmem + lane_base + c0, r);
    tmem_ld_wait();
    const int j = c0 / RP, kb = c0 % RP;
    if (row_valid && a.H[j] != nullptr) {
      float* hrow = a.H[j] + (int64_t)(tl.start + m) * pt.rank_max;
#pragma unroll
      for (int q = 0; q < 16; ++q)
        if (kb + q < pt.rank_max) hrow[kb + q] = __uint_as_float(r[q]);
    }
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      const int col = c0 + h * 8, blk = col >> 6, ch = (col & 63) >> 3;
      uint4 v;
      v.x = pack_bf16x2(__uint_as_float(r[h * 8 + 0]), __uint_as_float(r[h * 8 + 1]));
      v.y = pack_bf16x2(__uint_as_float(r[h * 8 + 2]), __uint_as_float(r[h * 8 + 3]));
      v.z = pack_bf16x2(__uint_as_float(r[h * 8 + 4]), __uint_as_float(r[h * 8 + 5]));
      v.w = pack_bf16x2(__uint_as_float(r[h * 8 + 6]), __uint_as_float(r[h * 8 + 7]));
      *reinterpret_cast<uint4*>(Hs + blk * kBlk + sw128_off(m, ch)) = v;
    }
  }
  tc_fence_before();

  // target rows of this thread's unique pair (or its own row)
  int rows[kMaxK];
  int nrows = 0;
  if (row_valid) {
    if (SHARED) {
      const int t = src_row[m], k = pt.k;
      for (int j = 0; j < k; ++j)
        if (a.pair_g[(int64_t)t * k + j] == g) rows[nrows++] = a.pair_row[(int64_t)t * k + j];
    } else {
      rows[nrows++] = tl.start + m;
    }
  }

  // ---------------------------------------------------------- phase 2: D, RMW
  constexpr uint32_t idesc_d = idesc_bf16_f32(128, kNc, 0, 1);
  const float s = a.s;
  const int jproj = NPROJ == 2 ? half : 0;      // projection of this warp half
  const int coff = NPROJ == 2 ? 0 : half * 128;  // column offset inside the chunk
  uint16_t* __restrict__ Yj = a.Y[jproj];
  auto load_b = [&](int n0, int buf) {
    const uint32_t sB = smem_u32(Bs + buf * C::kBs);
    for (int idx = tid; idx < NPROJ * RP * (kNc / 8); idx += kThreads) {
      const int j = idx / (RP * (kNc / 8)), rem = idx % (RP * (kNc / 8)), kr = rem / (kNc / 8), cc = rem % (kNc / 8);
      const int col = n0 + cc * 8;
      const bool v = kr < rg && col < d_out;
      cp_async16(sB + j * RP * kNc * 2 + (cc >> 3) * RP * 128 + sw128_off(kr, cc & 7),
                 v ? a.Bt[j] + (int64_t)(r0 + kr) * d_out + col : a.Bt[0], v);
    }
  };
  const int nch = (d_out + kNc - 1) / kNc;
  load_b(0, 0);
  cp_async_commit();
  // rows per thread differ; TMEM loads are warp-collective, so every lane of
  // a warp runs the warp's largest row count
  const int nr_warp = __reduce_max_sync(0xffffffffu, nrows);
  for (int c = 0; c < nch; ++c) {
    const int n0 = c * kNc;
    cp_async_wait<0>();
    fence_proxy_async_smem();
    if (__syncthreads_or(bad)) {
      aborted = true;
      break;
    }
    if (tid == 0) {
      tc_fence_after();
      const uint32_t sH = smem_u32(Hs), sB = smem_u32(Bs + (c & 1) * C::kBs);
#pragma unroll
      for (int j = 0; j < NPROJ; ++j)
#pragma unroll
        for (int i = 0; i < RP / 16; ++i) {
          const int kk = (j * RP) / 16 + i;
          tc_mma_bf16(tmem + j * kNc, sdesc_sw128(sH + (kk >> 2) * kBlk + (kk & 3) * 32, 16, 1024),
                      sdesc_sw128(sB + j * RP * kNc * 2 + i * 2048, RP * 128, 1024), idesc_d, i > 0 ? 1u : 0u);
        }
      tc_commit(&bar_d);
    }
    if (c + 1 < nch) load_b(n0 + kNc, (c + 1) & 1);
    cp_async_commit();
    const int col0 = n0 + coff;
    bool waited = false;
    for (int ri = 0; ri < (nr_warp > 0 ? nr_warp : 1); ++ri) {
      // this row's 128 columns (issued before the MMA wait on the first row)
      const bool live = ri < nrows;
      uint16_t* yp = Yj + (int64_t)(live ? rows[ri] : 0) * d_out + col0;
      uint4 y[16];
#pragma unroll
      for (int q = 0; q < 16; ++q)
        y[q] = (live && col0 + q * 8 < d_out) ? *reinterpret_cast<const uint4*>(yp + q * 8) : make_uint4(0, 0, 0, 0);
      if (!waited) {
        if (!mbar_wait(&bar_d, c & 1)) bad = true;
        tc_fence_after();
        waited = true;
      }
#pragma unroll
      for (int sc = 0; sc < 128; sc += 32) {
        uint32_t r[32];
        tmem_ld16(tmem + lane_base + half * 128 + sc, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
        tmem_ld16(tmem + lane_base + half * 128 + sc + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
        tmem_ld_wait();
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int qq = sc / 8 + q;
          if (live && col0 + qq * 8 < d_out) {
            const uint32_t* dq = &r[q * 8];
            const float2 f0 = unpack_bf16x2(y[qq].x), f1 = unpack_bf16x2(y[qq].y), f2 = unpack_bf16x2(y[qq].z),
                         f3 = unpack_bf16x2(y[qq].w);
            uint4 o;
            o.x = pack_bf16x2(f0.x + s * __uint_as_float(dq[0]), f0.y + s * __uint_as_float(dq[1]));
            o.y = pack_bf16x2(f1.x + s * __uint_as_float(dq[2]), f1.y + s * __uint_as_float(dq[3]));
            o.z = pack_bf16x2(f2.x + s * __uint_as_float(dq[4]), f2.y + s * __uint_as_float(dq[5]));
            o.w = pack_bf16x2(f3.x + s * __uint_as_float(dq[6]), f3.y + s * __uint_as_float(dq[7]));
            *reinterpret_cast<uint4*>(yp + qq * 8) = o;
          }
        }
      }
    }
    tc_fence_before();
  }
  cp_async_wait<0>();
  tc_fence_before();
  aborted = __syncthreads_or(bad || aborted);
  if (aborted && tid == 0) atomicOr(a.err, kErrTimeout);
  if (warp == 0) tmem_dealloc(tmem, C::kTmemCols);
}

template <int RP, int NPROJ, bool SHARED>
cudaError_t launch_fwd_t(const PlanTables& pt, const FwdLaunch& a, cudaStream_t st) {
  using C = FwdCfg<RP, NPROJ>;
  auto kern = k_fwd<RP, NPROJ, SHARED>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
  if (e != cudaSuccess) return e;
  if (a.max_tiles <= 0) return cudaSuccess;
  kern<<<a.max_tiles, kThreads, C::kSmem, st>>>(pt, a);
  return cudaGetLastError();
}

template <bool SHARED>
cudaError_t dispatch_fwd(const PlanTables& pt, const FwdLaunch& a, cudaStream_t st) {
  const int rp = pt.rank_pad;
  if (a.nproj == 2) {
    switch (rp) {
      case 16: return launch_fwd_t<16, 2, SHARED>(pt, a, st);
      case 32: return launch_fwd_t<32, 2, SHARED>(pt, a, st);
      case 64: return launch_fwd_t<64, 2, SHARED>(pt, a, st);
      case 128: return launch_fwd_t<128, 2, SHARED>(pt, a, st);
    }
  } else {
    switch (rp) {
      case 16: return launch_fwd_t<16, 1, SHARED>(pt, a, st);
      case 32: return launch_fwd_t<32, 1, SHARED>(pt, a, st);
      case 64: return launch_fwd_t<64, 1, SHARED>(pt, a, st);
      case 128: return launch_fwd_t<128, 1, SHARED>(pt, a, st);
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace

cudaError_t launch_fwd(const PlanTables& pt, const FwdLaunch& a, bool shared, cudaStream_t st) {
  return shared ? dispatch_fwd<true>(pt, a, st) : dispatch_fwd<false>(pt, a, st);
}

}  // namespace ace
