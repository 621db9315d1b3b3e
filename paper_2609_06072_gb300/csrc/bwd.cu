// Fused LoRA backward (adjoint of the forward; Sec. 3.1.2 gradient form,
// Sec. 3.4 shared adapter updates).
//
// k_bwd: one CTA per split (up to NT tiles of 128 unique pairs / rows of one
// group).  Phase 1 streams the upstream gradient in 128-column chunks:
//     dC_i  = sum of the dY rows of each unique pair (SHARED) | dY rows (ROW)
//     dH_i += dC_i . B_g                (tcgen05, accumulated in TMEM over chunks)
//     dBt_c = sum_i H_i^T . dC_i        (tcgen05, one chunk of B_g^T's gradient)
//   and flushes dBt_c per chunk (fp32 atomics, or a per-split partial for the
//   deterministic two-stage reduction).  Phase 2 re-reads the input in chunks:
//     dA_c  = sum_i X_i^T . dH_i        (SHARED: X gathered by token)
//     dh_i += dH_i . A_g  (ROW only)    (bf16 read-modify-write of each row)
// k_dx (SHARED only, token-major, deterministic):
//     dX[t] += sum_proj sum_{u of t} dH[u] . A_{g(u)}   (fixed ascending g order)
// k_splitk_reduce: deterministic stage 2, sums the partials of each group's
// splits in split order; groups without rows get exact zeros.
#include <cstdint>

#include "ace_internal.cuh"
#include "ace_ptx.cuh"

namespace ace {
namespace {

constexpr int kNcB = 128;  // columns per chunk

template <int RP>
struct BwdCfg {
  static constexpr int NT = RP <= 32 ? 4 : (RP == 64 ? 2 : 1);
  static constexpr int kOpTile = ((RP + 63) / 64) * kTileM * 128;  // [128 x RP] bf16, SW128 blocks of 64 cols
  static constexpr int kHsm = NT * kOpTile;
  static constexpr int kActTile = kTileM * 256;                     // [128 x 128] bf16
  static constexpr int kWTile = RP * 256;                           // [RP x 128] bf16
  static constexpr int kBuf = kActTile + kWTile;
  static constexpr int kSmem = kHsm + 2 * kBuf + 1024;
  static constexpr int kTmem = 256;
};

// [rows x 128 cols] bf16 tile, two 64-column SW128 blocks of `rows` x 128 B.
__device__ __forceinline__ uint32_t tile_off(int rows, int r, int c_chunk /*0..15*/) {
  return (uint32_t)((c_chunk >> 3) * rows * 128) + sw128_off(r, c_chunk & 7);
}

// Loads rows [r0, r0 + RP) x cols [n0, n0 + 128) of a row-major bf16 matrix
// (row stride `ld`) into a weight tile; rows >= rv or cols >= ncol are zero.
template <int RP>
__device__ __forceinline__ void load_w_tile(uint32_t dst, const uint16_t* __restrict__ base, int r0, int rv, int ld,
                                            int n0, int ncol, int tid) {
  for (int idx = tid; idx < RP * 16; idx += 128) {
    const int k = idx >> 4, cc = idx & 15, col = n0 + cc * 8;
    const bool v = k < rv && col < ncol;
    const uint16_t* src = v ? base + (int64_t)(r0 + k) * ld + col : base;
    cp_async16(dst + tile_off(RP, k, cc), src, v);
  }
}

template <int RP, bool SHARED>
__global__ void __launch_bounds__(128) k_bwd(const __grid_constant__ PlanTables pt, const __grid_constant__ BwdLaunch a) {
  using C = BwdCfg<RP>;
  constexpr int NT = C::NT;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bar1[2];
  __shared__ __align__(8) uint64_t bar2[2];
  __shared__ uint32_t tslot;
  __shared__ int32_t s_abort;
  __shared__ int32_t s_tok[NT * kTileM];

  const int n_splits = a.counts[a.count_slot];
  if ((int)blockIdx.x >= n_splits) return;
  const int proj = blockIdx.y;
  const Tile sp = a.splits[blockIdx.x];
  const int tid = threadIdx.x, warp = tid >> 5;
  const int g = sp.g, r0 = pt.rank_off[g], rg = pt.rank_off[g + 1] - r0;
  const int ntiles = (sp.cnt + kTileM - 1) / kTileM;
  const int d_in = a.d_in, d_out = a.d_out, k = pt.k;
  const float s = a.s;
  const uint16_t* __restrict__ dY = a.dY[proj];
  const float* __restrict__ Hsave = a.H[proj];
  const uint16_t* __restrict__ Aw = a.A[proj];
  const uint16_t* __restrict__ Btw = a.Bt[proj];

  uint8_t* Hsm = smem;                 // NT operand tiles: H in phase 1, dH in phase 2
  uint8_t* buf0 = smem + C::kHsm;      // two pipeline buffers (activation tile + weight tile)
  auto act = [&](int b) { return smem_u32(buf0 + b * C::kBuf); };
  auto wt = [&](int b) { return smem_u32(buf0 + b * C::kBuf + C::kActTile); };
  auto opt = [&](int i) { return smem_u32(Hsm + i * C::kOpTile); };

  for (int i = tid; i < NT * kTileM; i += 128) {
    const int ti = i / kTileM, m = i % kTileM;
    const int cnt_i = min(kTileM, sp.cnt - ti * kTileM);
    s_tok[i] = (ti < ntiles && m < cnt_i) ? (SHARED ? a.uniq_tok[sp.start + ti * kTileM + m] : sp.start + ti * kTileM + m)
                                          : -1;
  }
  if (tid == 0) {
    mbar_init(&bar1[0], 1);
    mbar_init(&bar1[1], 1);
    mbar_init(&bar2[0], 1);
    mbar_init(&bar2[1], 1);
    s_abort = 0;
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, C::kTmem);
  // H operand tiles: bf16(H_save) of every tile, zero beyond r_g
  for (int i = 0; i < ntiles; ++i) {
    const int cnt_i = min(kTileM, sp.cnt - i * kTileM);
    const int m = tid;
    for (int c8 = 0; c8 < RP; c8 += 8) {
      float v[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        const int kk = c8 + q;
        v[q] = (m < cnt_i && kk < rg) ? Hsave[(int64_t)(sp.start + i * kTileM + m) * pt.rank_max + kk] : 0.f;
      }
      uint4 w;
      w.x = pack_bf16x2(v[0], v[1]);
      w.y = pack_bf16x2(v[2], v[3]);
      w.z = pack_bf16x2(v[4], v[5]);
      w.w = pack_bf16x2(v[6], v[7]);
      *reinterpret_cast<uint4*>(Hsm + i * C::kOpTile + (c8 >> 6) * (kTileM * 128) + sw128_off(m, (c8 & 63) >> 3)) = w;
    }
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tslot;
  const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
  const uint32_t t_dbt = tmem + NT * RP;

  // ------------------------------------------------------------- phase 1
  constexpr uint32_t id_dh = idesc_bf16_f32(128, RP, 0, 0);
  constexpr uint32_t id_w = idesc_bf16_f32(128, RP, 1, 1);
  int it = 0;
  const int nchunk1 = (d_out + kNcB - 1) / kNcB;
  for (int c = 0; c < nchunk1; ++c) {
    const int n0 = c * kNcB;
    for (int i = 0; i < ntiles; ++i, ++it) {
      const int b = it & 1;
      if (it >= 2 && !mbar_wait(&bar1[b], ((it - 2) >> 1) & 1)) atomicOr(&s_abort, 1);
      load_w_tile<RP>(wt(b), Btw, r0, rg, d_out, n0, d_out, tid);
      const uint32_t dst = act(b);
      if (SHARED) {
        // dC row of this thread's unique pair: sum of its dY rows (slot order)
        const int t = s_tok[i * kTileM + tid];
        uint8_t* base = buf0 + b * C::kBuf;
#pragma unroll
        for (int half = 0; half < 2; ++half) {
          float acc[64];
#pragma unroll
          for (int q = 0; q < 64; ++q) acc[q] = 0.f;
          const int colh = n0 + half * 64;
          if (t >= 0) {
            for (int j = 0; j < k; ++j) {
              if (a.pair_g[(int64_t)t * k + j] != g) continue;
              const uint16_t* src = dY + (int64_t)a.pair_row[(int64_t)t * k + j] * d_out + colh;
              uint4 y[8];
#pragma unroll
              for (int q = 0; q < 8; ++q)
                y[q] = (colh + q * 8 < d_out) ? __ldg(reinterpret_cast<const uint4*>(src + q * 8)) : make_uint4(0, 0, 0, 0);
#pragma unroll
              for (int q = 0; q < 8; ++q) {
                const float2 f0 = unpack_bf16x2(y[q].x), f1 = unpack_bf16x2(y[q].y), f2 = unpack_bf16x2(y[q].z),
                             f3 = unpack_bf16x2(y[q].w);
                acc[q * 8 + 0] += f0.x; acc[q * 8 + 1] += f0.y; acc[q * 8 + 2] += f1.x; acc[q * 8 + 3] += f1.y;
                acc[q * 8 + 4] += f2.x; acc[q * 8 + 5] += f2.y; acc[q * 8 + 6] += f3.x; acc[q * 8 + 7] += f3.y;
              }
            }
          }
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            uint4 w;
            w.x = pack_bf16x2(acc[q * 8 + 0], acc[q * 8 + 1]);
            w.y = pack_bf16x2(acc[q * 8 + 2], acc[q * 8 + 3]);
            w.z = pack_bf16x2(acc[q * 8 + 4], acc[q * 8 + 5]);
            w.w = pack_bf16x2(acc[q * 8 + 6], acc[q * 8 + 7]);
            *reinterpret_cast<uint4*>(base + tile_off(kTileM, tid, half * 8 + q)) = w;
          }
        }
      } else {
#pragma unroll 4
        for (int q = 0; q < 16; ++q) {
          const int idx = q * 128 + tid, m = idx >> 4, cc = idx & 15, col = n0 + cc * 8;
          const int row = s_tok[i * kTileM + m];
          const bool v = row >= 0 && col < d_out;
          const uint16_t* src = v ? dY + (int64_t)row * d_out + col : dY;
          cp_async16(dst + tile_off(kTileM, m, cc), src, v);
        }
      }
      cp_async_commit();
      cp_async_wait<0>();
      fence_proxy_async_smem();
      __syncthreads();
      if (tid == 0) {
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < kNcB / 16; ++kk) {
          // dH_i += dC . B_g (A: dC K-major, B: Bt chunk K-major)
          tc_mma_bf16(tmem + i * RP, sdesc_sw128(dst + (kk >> 2) * (kTileM * 128) + (kk & 3) * 32, 16, 1024),
                      sdesc_sw128(wt(b) + (kk >> 2) * (RP * 128) + (kk & 3) * 32, 16, 1024), id_dh,
                      (c > 0 || kk > 0) ? 1u : 0u);
        }
#pragma unroll
        for (int kk = 0; kk < kTileM / 16; ++kk) {
          // dBt_c^T += dC^T . H_i (A: dC as MN-major, B: H as MN-major)
          tc_mma_bf16(t_dbt, sdesc_sw128(dst + kk * 2048, kTileM * 128, 1024),
                      sdesc_sw128(opt(i) + kk * 2048, kTileM * 128, 1024), id_w, (i > 0 || kk > 0) ? 1u : 0u);
        }
        tc_commit(&bar1[b]);
      }
    }
    // all MMAs of this chunk done -> flush dBt chunk (lane = output column)
    if (!mbar_wait(&bar1[(it - 1) & 1], ((it - 1) >> 1) & 1)) atomicOr(&s_abort, 1);
    tc_fence_after();
    __syncthreads();
    if (s_abort) break;
    const int col = n0 + tid;
#pragma unroll
    for (int c0 = 0; c0 < RP; c0 += 16) {
      uint32_t r[16];
      tmem_ld16(t_dbt + lane_base + c0, r);
      tmem_ld_wait();
      if (col < d_out) {
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          const int kk = c0 + q;
          if (kk < rg) {
            const float v = s * __uint_as_float(r[q]);
            if (a.deterministic)
              a.part_dBt[proj][((int64_t)sp.id * RP + kk) * d_out + col] = v;
            else
              atomicAdd(&a.dBt[proj][(int64_t)(r0 + kk) * d_out + col], v);
          }
        }
      }
    }
    tc_fence_before();
    __syncthreads();
  }
  if (s_abort) {
    if (tid == 0) atomicOr(a.err, kErrTimeout);
    tc_fence_before();
    __syncthreads();
    if (warp == 0) tmem_dealloc(tmem, C::kTmem);
    return;
  }

  // dH (final, scaled by s) -> bf16 operand tiles (+ global scratch for dX)
  for (int i = 0; i < ntiles; ++i) {
    const int cnt_i = min(kTileM, sp.cnt - i * kTileM);
#pragma unroll
    for (int c0 = 0; c0 < RP; c0 += 16) {
      uint32_t r[16];
      tmem_ld16(tmem + lane_base + i * RP + c0, r);
      tmem_ld_wait();
      uint4 w[2];
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        w[h].x = pack_bf16x2(s * __uint_as_float(r[h * 8 + 0]), s * __uint_as_float(r[h * 8 + 1]));
        w[h].y = pack_bf16x2(s * __uint_as_float(r[h * 8 + 2]), s * __uint_as_float(r[h * 8 + 3]));
        w[h].z = pack_bf16x2(s * __uint_as_float(r[h * 8 + 4]), s * __uint_as_float(r[h * 8 + 5]));
        w[h].w = pack_bf16x2(s * __uint_as_float(r[h * 8 + 6]), s * __uint_as_float(r[h * 8 + 7]));
        const int col = c0 + h * 8;
        *reinterpret_cast<uint4*>(Hsm + i * C::kOpTile + (col >> 6) * (kTileM * 128) + sw128_off(tid, (col & 63) >> 3)) =
            w[h];
      }
      if (SHARED && tid < cnt_i) {
        uint4* dst = reinterpret_cast<uint4*>(a.dH[proj] + (int64_t)(sp.start + i * kTileM + tid) * RP + c0);
        dst[0] = w[0];
        dst[1] = w[1];
      }
    }
  }
  tc_fence_before();

  // ------------------------------------------------------------- phase 2
  constexpr uint32_t id_dh2 = idesc_bf16_f32(128, kNcB, 0, 1);
  const uint32_t t_da = SHARED ? tmem : tmem + kNcB;
  const uint16_t* __restrict__ Xin = a.Xin;
  int it2 = 0;
  const int nchunk2 = (d_in + kNcB - 1) / kNcB;
  for (int c = 0; c < nchunk2; ++c) {
    const int n0 = c * kNcB;
    for (int i = 0; i < ntiles; ++i, ++it2) {
      const int b = it2 & 1;
      if (it2 >= 2 && !mbar_wait(&bar2[b], ((it2 - 2) >> 1) & 1)) atomicOr(&s_abort, 1);
      const uint32_t dst = act(b);
#pragma unroll 4
      for (int q = 0; q < 16; ++q) {
        const int idx = q * 128 + tid, m = idx >> 4, cc = idx & 15, col = n0 + cc * 8;
        const int src_row = s_tok[i * kTileM + m];
        const bool v = src_row >= 0 && col < d_in;
        const uint16_t* src = v ? Xin + (int64_t)src_row * d_in + col : Xin;
        cp_async16(dst + tile_off(kTileM, m, cc), src, v);
      }
      if (!SHARED) load_w_tile<RP>(wt(b), Aw, r0, rg, d_in, n0, d_in, tid);
      cp_async_commit();
      cp_async_wait<0>();
      fence_proxy_async_smem();
      __syncthreads();
      if (tid == 0) {
        tc_fence_after();
        if (!SHARED) {
#pragma unroll
          for (int kk = 0; kk < RP / 16; ++kk)  // dh_i chunk = dH_i . A_g chunk
            tc_mma_bf16(tmem, sdesc_sw128(opt(i) + (kk >> 2) * (kTileM * 128) + (kk & 3) * 32, 16, 1024),
                        sdesc_sw128(wt(b) + kk * 2048, RP * 128, 1024), id_dh2, kk > 0 ? 1u : 0u);
        }
#pragma unroll
        for (int kk = 0; kk < kTileM / 16; ++kk)  // dA_c^T += X_i^T . dH_i
          tc_mma_bf16(t_da, sdesc_sw128(dst + kk * 2048, kTileM * 128, 1024),
                      sdesc_sw128(opt(i) + kk * 2048, kTileM * 128, 1024), id_w, (i > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&bar2[b]);
      }
      if (!SHARED) {
        if (!mbar_wait(&bar2[b], (it2 >> 1) & 1)) atomicOr(&s_abort, 1);
        tc_fence_after();
        __syncthreads();
        if (s_abort) break;
        const int row = s_tok[i * kTileM + tid];
#pragma unroll
        for (int sc = 0; sc < kNcB; sc += 32) {
          uint32_t r[32];
          tmem_ld16(tmem + lane_base + sc, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
          tmem_ld16(tmem + lane_base + sc + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
          tmem_ld_wait();
          const int col0 = n0 + sc;
          if (row >= 0 && col0 < d_in) {
            uint16_t* yp = a.dXin + (int64_t)row * d_in + col0;
#pragma unroll
            for (int q = 0; q < 4; ++q) {
              if (col0 + q * 8 < d_in) {
                uint4 y = *reinterpret_cast<const uint4*>(yp + q * 8);
                float2 f0 = unpack_bf16x2(y.x), f1 = unpack_bf16x2(y.y), f2 = unpack_bf16x2(y.z),
                       f3 = unpack_bf16x2(y.w);
                const uint32_t* dq = &r[q * 8];
                y.x = pack_bf16x2(f0.x + __uint_as_float(dq[0]), f0.y + __uint_as_float(dq[1]));
                y.y = pack_bf16x2(f1.x + __uint_as_float(dq[2]), f1.y + __uint_as_float(dq[3]));
                y.z = pack_bf16x2(f2.x + __uint_as_float(dq[4]), f2.y + __uint_as_float(dq[5]));
                y.w = pack_bf16x2(f3.x + __uint_as_float(dq[6]), f3.y + __uint_as_float(dq[7]));
                *reinterpret_cast<uint4*>(yp + q * 8) = y;
              }
            }
          }
        }
        tc_fence_before();
        __syncthreads();
      }
    }
    if (s_abort) break;
    if (SHARED) {
      if (!mbar_wait(&bar2[(it2 - 1) & 1], ((it2 - 1) >> 1) & 1)) atomicOr(&s_abort, 1);
      tc_fence_after();
      __syncthreads();
      if (s_abort) break;
    }
    const int col = n0 + tid;
#pragma unroll
    for (int c0 = 0; c0 < RP; c0 += 16) {
      uint32_t r[16];
      tmem_ld16(t_da + lane_base + c0, r);
      tmem_ld_wait();
      if (col < d_in) {
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          const int kk = c0 + q;
          if (kk < rg) {
            const float v = __uint_as_float(r[q]);
            if (a.deterministic)
              a.part_dA[proj][((int64_t)sp.id * RP + kk) * d_in + col] = v;
            else
              atomicAdd(&a.dA[proj][(int64_t)(r0 + kk) * d_in + col], v);
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
  if (warp == 0) tmem_dealloc(tmem, C::kTmem);
}

// ---------------------------------------------------------------- dX
template <int RP>
struct DxCfg {
  static constexpr int kNd = 256;
  static constexpr int kOpTile = ((RP + 63) / 64) * kTileM * 128;
  static constexpr int kWTile = RP * kNd * 2;  // 4 blocks of [RP x 128 B]
  static constexpr int kBuf = kOpTile + kWTile;
  static constexpr int kSmem = 2 * kBuf + 1024;
};

template <int RP>
__global__ void __launch_bounds__(128) k_dx(const __grid_constant__ PlanTables pt, const __grid_constant__ DxLaunch a,
                                          const int32_t* __restrict__ uniq_off) {
  using C = DxCfg<RP>;
  constexpr int kNd = C::kNd;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bar[2];
  __shared__ uint32_t tslot;
  __shared__ int32_t s_abort;
  __shared__ int32_t s_uoff[ACE_MAX_EXPERTS + 1];
  const int tid = threadIdx.x, warp = tid >> 5;
  const int t0 = blockIdx.x * kTileM, c0 = blockIdx.y * kNd;
  const int d = a.d, k = pt.k, G = pt.G;
  const int t = t0 + tid;
  for (int i = tid; i <= G; i += 128) s_uoff[i] = uniq_off[i];
  if (tid == 0) {
    mbar_init(&bar[0], 1);
    mbar_init(&bar[1], 1);
    s_abort = 0;
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, 256);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tslot;
  const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
  constexpr uint32_t idesc = idesc_bf16_f32(128, kNd, 0, 1);

  int it = 0;
  for (int j = 0; j < a.nproj; ++j) {
    int pos = 0;  // position in this token's ascending-g list of unique pairs
    for (int g = 0; g < G; ++g) {
      int u = -1;
      if (t < a.T) {
        while (pos < k) {
          const int uu = a.tok_uniq[(int64_t)t * k + pos];
          if (uu < 0 || uu >= s_uoff[g + 1]) break;
          ++pos;
          if (uu >= s_uoff[g]) { u = uu; break; }
        }
      }
      if (!__syncthreads_or(u >= 0)) continue;
      const int b = it & 1;
      if (it >= 2 && !mbar_wait(&bar[b], ((it - 2) >> 1) & 1)) atomicOr(&s_abort, 1);
      const uint32_t sop = smem_u32(smem + b * C::kBuf);
      const uint32_t sw = sop + C::kOpTile;
      // dH rows of this token for group g (zero if absent)
      const uint16_t* dHj = a.dH[j];
#pragma unroll
      for (int c8 = 0; c8 < RP; c8 += 8) {
        const bool v = u >= 0;
        const uint16_t* src = v ? dHj + (int64_t)u * RP + c8 : dHj;
        cp_async16(sop + (c8 >> 6) * (kTileM * 128) + sw128_off(tid, (c8 & 63) >> 3), src, v);
      }
      // A_g rows x [c0, c0 + 256): MN-major blocks of 64 columns
      const int r0 = pt.rank_off[g], rg = pt.rank_off[g + 1] - r0;
      for (int idx = tid; idx < RP * (kNd / 8); idx += 128) {
        const int kr = idx / (kNd / 8), cc = idx % (kNd / 8), col = c0 + cc * 8;
        const bool v = kr < rg && col < d;
        const uint16_t* src = v ? a.A[j] + (int64_t)(r0 + kr) * d + col : a.A[0];
        cp_async16(sw + (cc >> 3) * (RP * 128) + sw128_off(kr, cc & 7), src, v);
      }
      cp_async_commit();
      cp_async_wait<0>();
      fence_proxy_async_smem();
      __syncthreads();
      if (tid == 0) {
        tc_fence_after();
#pragma unroll
        for (int kk = 0; kk < RP / 16; ++kk)
          tc_mma_bf16(tmem, sdesc_sw128(sop + (kk >> 2) * (kTileM * 128) + (kk & 3) * 32, 16, 1024),
                      sdesc_sw128(sw + kk * 2048, RP * 128, 1024), idesc, (it > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&bar[b]);
      }
      ++it;
    }
  }
  if (it > 0) {
    if (!mbar_wait(&bar[(it - 1) & 1], ((it - 1) >> 1) & 1)) atomicOr(&s_abort, 1);
    tc_fence_after();
    __syncthreads();
    if (!s_abort) {
#pragma unroll 1
      for (int sc = 0; sc < kNd; sc += 32) {
        uint32_t r[32];
        tmem_ld16(tmem + lane_base + sc, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
        tmem_ld16(tmem + lane_base + sc + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
        tmem_ld_wait();
        const int col0 = c0 + sc;
        if (t < a.T && col0 < d) {
          uint16_t* yp = a.dX + (int64_t)t * d + col0;
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            if (col0 + q * 8 < d) {
              uint4 y = *reinterpret_cast<const uint4*>(yp + q * 8);
              float2 f0 = unpack_bf16x2(y.x), f1 = unpack_bf16x2(y.y), f2 = unpack_bf16x2(y.z), f3 = unpack_bf16x2(y.w);
              const uint32_t* dq = &r[q * 8];
              y.x = pack_bf16x2(f0.x + __uint_as_float(dq[0]), f0.y + __uint_as_float(dq[1]));
              y.y = pack_bf16x2(f1.x + __uint_as_float(dq[2]), f1.y + __uint_as_float(dq[3]));
              y.z = pack_bf16x2(f2.x + __uint_as_float(dq[4]), f2.y + __uint_as_float(dq[5]));
              y.w = pack_bf16x2(f3.x + __uint_as_float(dq[6]), f3.y + __uint_as_float(dq[7]));
              *reinterpret_cast<uint4*>(yp + q * 8) = y;
            }
          }
        }
      }
    }
  } else {
    __syncthreads();
  }
  if (s_abort && tid == 0) atomicOr(a.err, kErrTimeout);
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, 256);
}

// ---------------------------------------------------------------- stage 2
__global__ void __launch_bounds__(256) k_splitk_reduce(const __grid_constant__ PlanTables pt,
                                                       const Tile* __restrict__ splits,
                                                       const int32_t* __restrict__ counts, int slot,
                                                       const float* __restrict__ part, int RP, int width,
                                                       float* __restrict__ out) {
  const int i = blockIdx.x;  // global rank row
  int g = 0;
  while (pt.rank_off[g + 1] <= i) ++g;
  const int kk = i - pt.rank_off[g];
  const int c = (blockIdx.y * 256 + threadIdx.x) * 4;
  if (c >= width) return;
  const int n = counts[slot];
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int sidx = 0; sidx < n; ++sidx) {
    const Tile sp = splits[sidx];
    if (sp.g != g) continue;
    const float4 v = *reinterpret_cast<const float4*>(part + ((int64_t)sp.id * RP + kk) * width + c);
    acc.x += v.x;
    acc.y += v.y;
    acc.z += v.z;
    acc.w += v.w;
  }
  *reinterpret_cast<float4*>(out + (int64_t)i * width + c) = acc;
}

template <int RP, bool SHARED>
cudaError_t launch_bwd_t(const PlanTables& pt, const BwdLaunch& a, cudaStream_t st) {
  using C = BwdCfg<RP>;
  auto kern = k_bwd<RP, SHARED>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
  if (e != cudaSuccess) return e;
  const int n_rank = pt.rank_off[pt.G];
  const int nproj = SHARED ? a.nproj : 1;
  if (!a.deterministic) {
    for (int j = 0; j < nproj; ++j) {
      e = cudaMemsetAsync(a.dA[j], 0, sizeof(float) * (size_t)n_rank * a.d_in, st);
      if (e != cudaSuccess) return e;
      e = cudaMemsetAsync(a.dBt[j], 0, sizeof(float) * (size_t)n_rank * a.d_out, st);
      if (e != cudaSuccess) return e;
    }
  }
  if (a.max_splits > 0 && a.T > 0) {
    dim3 grid(a.max_splits, nproj);
    kern<<<grid, 128, C::kSmem, st>>>(pt, a);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
  }
  if (a.deterministic) {
    for (int j = 0; j < nproj; ++j) {
      dim3 g1(n_rank, (a.d_in / 4 + 255) / 256), g2(n_rank, (a.d_out / 4 + 255) / 256);
      k_splitk_reduce<<<g1, 256, 0, st>>>(pt, a.splits, a.counts, a.count_slot, a.part_dA[j], RP, a.d_in, a.dA[j]);
      k_splitk_reduce<<<g2, 256, 0, st>>>(pt, a.splits, a.counts, a.count_slot, a.part_dBt[j], RP, a.d_out, a.dBt[j]);
    }
    e = cudaGetLastError();
  }
  return e;
}

template <int RP>
cudaError_t launch_dx_t(const PlanTables& pt, const DxLaunch& a, const int32_t* uniq_off, cudaStream_t st) {
  using C = DxCfg<RP>;
  auto kern = k_dx<RP>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::kSmem);
  if (e != cudaSuccess) return e;
  dim3 grid((a.T + kTileM - 1) / kTileM, (a.d + C::kNd - 1) / C::kNd);
  kern<<<grid, 128, C::kSmem, st>>>(pt, a, uniq_off);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_bwd(const PlanTables& pt, const BwdLaunch& a, bool shared, cudaStream_t st) {
  switch (pt.rank_pad) {
    case 16: return shared ? launch_bwd_t<16, true>(pt, a, st) : launch_bwd_t<16, false>(pt, a, st);
    case 32: return shared ? launch_bwd_t<32, true>(pt, a, st) : launch_bwd_t<32, false>(pt, a, st);
    case 64: return shared ? launch_bwd_t<64, true>(pt, a, st) : launch_bwd_t<64, false>(pt, a, st);
    case 128: return shared ? launch_bwd_t<128, true>(pt, a, st) : launch_bwd_t<128, false>(pt, a, st);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_dx(const PlanTables& pt, const DxLaunch& a, cudaStream_t st) {
  if (a.T == 0) return cudaSuccess;
  switch (pt.rank_pad) {
    case 16: return launch_dx_t<16>(pt, a, a.uniq_off, st);
    case 32: return launch_dx_t<32>(pt, a, a.uniq_off, st);
    case 64: return launch_dx_t<64>(pt, a, a.uniq_off, st);
    case 128: return launch_dx_t<128>(pt, a, a.uniq_off, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace ace
