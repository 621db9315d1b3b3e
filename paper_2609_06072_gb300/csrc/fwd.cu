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
constexpr int kNc = 128;  // output columns per D chunk

template <int RP, int NPROJ>
struct FwdCfg {
  static constexpr int kStageX = kTileM * 128;             // 128 rows x 64 bf16
  static constexpr int kStageA = NPROJ * RP * 128;         // NPROJ*RP rows x 64 bf16
  static constexpr int kStage = kStageX + kStageA;
  static constexpr int kHs = ((NPROJ * RP + 63) / 64) * kTileM * 128;
  static constexpr int kBs = NPROJ * RP * 256;             // NPROJ x [RP x 128 cols], MN-major
  static constexpr int kPhase1 = kStages * kStage;
  static constexpr int kPhase2 = kHs + kBs;
  static constexpr int kSmem = (kPhase1 > kPhase2 ? kPhase1 : kPhase2) + 1024;
  static constexpr int kTmemCols = NPROJ * kNc;            // >= NPROJ * RP
};

template <int RP, int NPROJ, bool SHARED>
__global__ void __launch_bounds__(128) k_fwd(const __grid_constant__ PlanTables pt, const __grid_constant__ FwdLaunch a) {
  using C = FwdCfg<RP, NPROJ>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bar_k[kStages];
  __shared__ __align__(8) uint64_t bar_d;
  __shared__ uint32_t tslot;
  __shared__ int32_t src_row[kTileM];
  __shared__ int32_t s_abort;

  const int n_tiles = a.counts[a.count_slot];
  if ((int)blockIdx.x >= n_tiles) return;
  const Tile tl = a.tiles[blockIdx.x];
  const int tid = threadIdx.x, warp = tid >> 5;
  const int g = tl.g, r0 = pt.rank_off[g], rg = pt.rank_off[g + 1] - r0;
  const int d_in = a.d_in, d_out = a.d_out;

  src_row[tid] = tid < tl.cnt ? (SHARED ? a.uniq_tok[tl.start + tid] : tl.start + tid) : -1;
  if (tid == 0) {
    for (int i = 0; i < kStages; ++i) mbar_init(&bar_k[i], 1);
    mbar_init(&bar_d, 1);
    s_abort = 0;
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tslot;
  const uint32_t lane_base = (uint32_t)(warp * 32) << 16;

  // ---------------------------------------------------------- phase 1: H
  const int NK = (d_in + 63) / 64;
  auto load_stage = [&](int kt, int slot) {
    const uint32_t sX = smem_u32(smem + slot * C::kStage);
    const uint32_t sA = sX + C::kStageX;
    const int k0 = kt * 64;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int idx = i * 128 + tid, m = idx >> 3, c = idx & 7;
      const int sr = src_row[m], kc = k0 + c * 8;
      const bool v = sr >= 0 && kc < d_in;
      const uint16_t* src = v ? a.X + (int64_t)sr * d_in + kc : a.X;
      cp_async16(sX + sw128_off(m, c), src, v);
    }
#pragma unroll
    for (int idx = tid; idx < NPROJ * RP * 8; idx += 128) {
      const int rr = idx >> 3, c = idx & 7, j = rr / RP, kr = rr % RP, kc = k0 + c * 8;
      const bool v = kr < rg && kc < d_in;
      const uint16_t* src = v ? a.A[j] + (int64_t)(r0 + kr) * d_in + kc : a.A[0];
      cp_async16(sA + sw128_off(rr, c), src, v);
    }
  };

  constexpr uint32_t idesc_h = idesc_bf16_f32(128, NPROJ * RP, 0, 0);
#pragma unroll
  for (int s = 0; s < kStages - 1; ++s) {
    if (s < NK) load_stage(s, s);
    cp_async_commit();
  }
  bool ok = true;
  for (int kt = 0; kt < NK; ++kt) {
    const int slot = kt % kStages;
    cp_async_wait<kStages - 2>();
    fence_proxy_async_smem();
    __syncthreads();
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
      const int nslot = nxt % kStages;
      if (kt >= 1) {  // slot last used by k-step kt-1
        if (!mbar_wait(&bar_k[nslot], ((kt - 1) / kStages) & 1)) { ok = false; atomicOr(&s_abort, 1); }
      }
      if (ok) load_stage(nxt, nslot);
    }
    cp_async_commit();
  }
  cp_async_wait<0>();
  if (NK > 0 && ok) {
    if (!mbar_wait(&bar_k[(NK - 1) % kStages], ((NK - 1) / kStages) & 1)) atomicOr(&s_abort, 1);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (s_abort) {
    if (tid == 0) atomicOr(a.err, kErrTimeout);
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, C::kTmemCols);
    return;
  }

  // ---------------------------------------------------------- H -> H_save, Hs
  uint8_t* Hs = smem;
  uint8_t* Bs = smem + C::kHs;
  const int m = tid;  // TMEM lane of this thread = tile row
  const bool row_valid = m < tl.cnt;
#pragma unroll
  for (int c0 = 0; c0 < NPROJ * RP; c0 += 16) {
    uint32_t r[16];
    tmem_ld16(tmem + lane_base + c0, r);
    tmem_ld_wait();
    const int j = c0 / RP, kb = c0 % RP;
    if (row_valid && NK > 0 && a.H[j] != nullptr) {
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
      if (NK == 0) v = make_uint4(0, 0, 0, 0);
      *reinterpret_cast<uint4*>(Hs + blk * (kTileM * 128) + sw128_off(m, ch)) = v;
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
  int chunk = 0;
  for (int n0 = 0; n0 < d_out; n0 += kNc, ++chunk) {
    const uint32_t sB = smem_u32(Bs);
    for (int idx = tid; idx < NPROJ * RP * 16; idx += 128) {
      const int j = idx / (RP * 16), rem = idx % (RP * 16), kr = rem >> 4, cc = rem & 15;
      const int col = n0 + cc * 8;
      const bool v = kr < rg && col < d_out;
      const uint16_t* src = v ? a.Bt[j] + (int64_t)(r0 + kr) * d_out + col : a.Bt[0];
      cp_async16(sB + j * RP * 256 + (cc >> 3) * RP * 128 + sw128_off(kr, cc & 7), src, v);
    }
    cp_async_commit();
    cp_async_wait<0>();
    fence_proxy_async_smem();
    __syncthreads();
    if (tid == 0) {
      tc_fence_after();
      const uint32_t sH = smem_u32(Hs);
#pragma unroll
      for (int j = 0; j < NPROJ; ++j)
#pragma unroll
        for (int i = 0; i < RP / 16; ++i) {
          const int kk = (j * RP) / 16 + i;
          tc_mma_bf16(tmem + j * kNc, sdesc_sw128(sH + (kk >> 2) * (kTileM * 128) + (kk & 3) * 32, 16, 1024),
                      sdesc_sw128(sB + j * RP * 256 + i * 2048, RP * 128, 1024), idesc_d, i > 0 ? 1u : 0u);
        }
      tc_commit(&bar_d);
    }
    if (!mbar_wait(&bar_d, chunk & 1)) atomicOr(&s_abort, 1);
    tc_fence_after();
    __syncthreads();
    if (s_abort) break;
#pragma unroll
    for (int j = 0; j < NPROJ; ++j) {
#pragma unroll
      for (int sc = 0; sc < kNc; sc += 32) {
        uint32_t r[32];
        tmem_ld16(tmem + lane_base + j * kNc + sc, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
        tmem_ld16(tmem + lane_base + j * kNc + sc + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
        tmem_ld_wait();
        const int col0 = n0 + sc;
        if (col0 < d_out) {
          for (int ri = 0; ri < nrows; ++ri) {
            uint16_t* yp = a.Y[j] + (int64_t)rows[ri] * d_out + col0;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              if (col0 + q * 8 < d_out) {
                uint4 y = *reinterpret_cast<const uint4*>(yp + q * 8);
                float2 f0 = unpack_bf16x2(y.x), f1 = unpack_bf16x2(y.y), f2 = unpack_bf16x2(y.z),
                       f3 = unpack_bf16x2(y.w);
                const uint32_t* dq = &r[q * 8];
                y.x = pack_bf16x2(f0.x + s * __uint_as_float(dq[0]), f0.y + s * __uint_as_float(dq[1]));
                y.y = pack_bf16x2(f1.x + s * __uint_as_float(dq[2]), f1.y + s * __uint_as_float(dq[3]));
                y.z = pack_bf16x2(f2.x + s * __uint_as_float(dq[4]), f2.y + s * __uint_as_float(dq[5]));
                y.w = pack_bf16x2(f3.x + s * __uint_as_float(dq[6]), f3.y + s * __uint_as_float(dq[7]));
                *reinterpret_cast<uint4*>(yp + q * 8) = y;
              }
            }
          }
        }
      }
    }
    tc_fence_before();
    __syncthreads();
  }
  if (s_abort && tid == 0) atomicOr(a.err, kErrTimeout);
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, C::kTmemCols);
}

template <int RP, int NPROJ, bool SHARED>
cudaError_t launch_fwd_t(const PlanTables& pt, const FwdLaunch& a, cudaStream_t st) {
  using C = FwdCfg<RP, NPROJ>;
  auto kern = k_fwd<RP, NPROJ, SHARED>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
  if (e != cudaSuccess) return e;
  if (a.max_tiles <= 0) return cudaSuccess;
  kern<<<a.max_tiles, 128, C::kSmem, st>>>(pt, a);
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
