// Fused LoRA backward (adjoint of the forward; gradient form of Sec. 3.1.2,
// shared adapter updates of Sec. 3.4).
//
// k_bwd_rows<RP, MODE>: one CTA per split of up to NT row tiles (128
// consecutive rows of one group).  Phase 1 streams the upstream gradient in
// 128-column chunks through a 3-stage cp.async ring:
//     dH_i  += dY_i . B_g                 (tcgen05, TMEM, accumulated over chunks)
//     dBt_c  = sum_i H_{u(row)}^T . dY_i  (tcgen05, one 128-column chunk of dB_g^T)
//   dBt_c is flushed while the next chunk's MMAs run (double-buffered TMEM):
//   fp32 atomics, or a per-split partial for the deterministic two-stage sum.
//   MODE_DOWN then runs phase 2 over chunks of the input h:
//     dA_c  += h_i^T . dH_i   and   dh_i += dH_i . A_g   (bf16 RMW of the rows)
//   MODE_SHARED writes dH per row (fp32 scratch); for gate/up the rows of one
//   unique pair (g, t) share H_u, and dC_u . B_g = sum_rows dY_row . B_g, so
//   streaming contiguous rows moves exactly the bytes of the deduplicated form.
// k_dh_reduce: dH_u = sum of the dH rows of unique pair u (fixed slot order).
// k_bwd_dA: gate and up fused; per split of unique pairs, X rows gathered by
//   token: dA_c += X_i^T . dH_u,i for both projections.
// k_dx: token-major, deterministic: dX[t] += sum_proj sum_{u of t} dH_u . A_g(u),
//   groups in ascending order.
// k_splitk_reduce: deterministic stage 2 (split order); empty groups -> zeros.
#include <cstdint>

#include "ace_internal.cuh"
#include "ace_ptx.cuh"

namespace ace {
namespace {

constexpr int kNcB = 128;   // columns per chunk
constexpr int kS = 3;       // pipeline stages
constexpr int kBlk = kTileM * 128;  // one [128 x 64] bf16 SW128 block (16 KB)
constexpr int MODE_DOWN = 0, MODE_SHARED = 1;

// Operand slots of [128 x RP] bf16 (H or dH tiles).  For RP <= 64 several
// slots share one 128-byte-swizzled block side by side (column offset
// (q % TPB) * RP); for RP = 128 a slot spans two blocks.
template <int RP>
struct Slots {
  static constexpr int TPB = RP >= 64 ? 1 : 64 / RP;
  static constexpr int kSlotBlocks = RP > 64 ? 2 : 1;
  static __host__ __device__ constexpr int bytes(int nslots) {
    return ((nslots + TPB - 1) / TPB) * kSlotBlocks * kBlk;
  }
  // byte offset of the 16-byte chunk holding elements (m, k..k+7), k % 8 == 0
  static __device__ __forceinline__ uint32_t elem(int q, int m, int k) {
    const int blk = (q / TPB) * kSlotBlocks + (k >> 6);
    const int col = (q % TPB) * (RP >= 64 ? 0 : RP) + (k & 63);
    return (uint32_t)(blk * kBlk) + sw128_off(m, col >> 3);
  }
  // MN-major view [N' = k x K' = m], K' step kk of 16 rows
  static __device__ __forceinline__ uint64_t desc_mn(uint32_t base, int q, int kk) {
    const uint32_t a = base + (uint32_t)((q / TPB) * kSlotBlocks * kBlk + (q % TPB) * (RP >= 64 ? 0 : RP) * 2);
    return sdesc_sw128(a + kk * 2048, kBlk, 1024);
  }
  // K-major view [M = m x K = k], K step kk of 16 columns
  static __device__ __forceinline__ uint64_t desc_k(uint32_t base, int q, int kk) {
    const uint32_t a = base + (uint32_t)((q / TPB) * kSlotBlocks * kBlk + (kk >> 2) * kBlk +
                                         (q % TPB) * (RP >= 64 ? 0 : RP) * 2 + (kk & 3) * 32);
    return sdesc_sw128(a, 16, 1024);
  }
};

// [rows x 128 cols] bf16 tile = two 64-column SW128 blocks of `rows` x 128 B.
__device__ __forceinline__ uint32_t tile_off(int rows, int r, int c_chunk /*0..15*/) {
  return (uint32_t)((c_chunk >> 3) * rows * 128) + sw128_off(r, c_chunk & 7);
}

// rows [r0, r0 + RP) x cols [n0, n0 + 128) of a row-major bf16 matrix into a
// weight tile; rows >= rv or cols >= ncol are zero.
template <int RP>
__device__ __forceinline__ void load_w_tile(uint32_t dst, const uint16_t* __restrict__ base, int r0, int rv, int ld,
                                            int n0, int ncol, int tid) {
#pragma unroll
  for (int idx = tid; idx < RP * 16; idx += 128) {
    const int k = idx >> 4, cc = idx & 15, col = n0 + cc * 8;
    const bool v = k < rv && col < ncol;
    cp_async16(dst + tile_off(RP, k, cc), v ? base + (int64_t)(r0 + k) * ld + col : base, v);
  }
}

// 128 rows x 128 columns of a row-major bf16 matrix, row ids from `rows`
// (-1 = zero row), into an activation tile.
__device__ __forceinline__ void load_act_tile(uint32_t dst, const uint16_t* __restrict__ base, const int32_t* rows,
                                              int ld, int n0, int ncol, int tid) {
#pragma unroll
  for (int q = 0; q < 16; ++q) {
    const int idx = q * 128 + tid, m = idx >> 4, cc = idx & 15, col = n0 + cc * 8;
    const int r = rows[m];
    const bool v = r >= 0 && col < ncol;
    cp_async16(dst + tile_off(kTileM, m, cc), v ? base + (int64_t)r * ld + col : base, v);
  }
}

__device__ __forceinline__ uint4 add_bf16x8(uint4 y, const uint32_t* d, float scale) {
  const float2 f0 = unpack_bf16x2(y.x), f1 = unpack_bf16x2(y.y), f2 = unpack_bf16x2(y.z), f3 = unpack_bf16x2(y.w);
  uint4 o;
  o.x = pack_bf16x2(f0.x + scale * __uint_as_float(d[0]), f0.y + scale * __uint_as_float(d[1]));
  o.y = pack_bf16x2(f1.x + scale * __uint_as_float(d[2]), f1.y + scale * __uint_as_float(d[3]));
  o.z = pack_bf16x2(f2.x + scale * __uint_as_float(d[4]), f2.y + scale * __uint_as_float(d[5]));
  o.w = pack_bf16x2(f3.x + scale * __uint_as_float(d[6]), f3.y + scale * __uint_as_float(d[7]));
  return o;
}

// Flush one [128 cols x RP] fp32 accumulator (TMEM lane = column) of a weight
// gradient: atomics into out[(r0 + k) * ld + col] or a per-split partial.
template <int RP>
__device__ __forceinline__ void flush_wgrad(uint32_t taddr, int n0, int ld, int rg, int r0, float scale, bool det,
                                            float* __restrict__ part, int split_id, float* __restrict__ out,
                                            int tid) {
  const int col = n0 + tid;
#pragma unroll
  for (int c0 = 0; c0 < RP; c0 += 16) {
    uint32_t r[16];
    tmem_ld16(taddr + c0, r);
    tmem_ld_wait();
    if (col < ld) {
#pragma unroll
      for (int q = 0; q < 16; ++q) {
        const int kk = c0 + q;
        if (kk < rg) {
          const float v = scale * __uint_as_float(r[q]);
          if (det)
            part[((int64_t)split_id * RP + kk) * ld + col] = v;
          else
            atomicAdd(&out[(int64_t)(r0 + kk) * ld + col], v);
        }
      }
    }
  }
}

template <int RP, int MODE>
struct RowsCfg {
  static constexpr int NT = RP <= 32 ? 4 : (RP == 64 ? 2 : 1);
  static constexpr int kOps = Slots<RP>::bytes(NT);
  static constexpr int kAct = kTileM * 256;
  static constexpr int kW = RP * 256;
  static constexpr int kStage = kAct + kW;
  static constexpr int kSmem = kOps + kS * kStage + 1024;
  static constexpr int kTmem = RP <= 64 ? 256 : 512;
};

template <int RP, int MODE>
__global__ void __launch_bounds__(128, 1) k_bwd_rows(const __grid_constant__ PlanTables pt,
                                                     const __grid_constant__ BwdLaunch a) {
  using C = RowsCfg<RP, MODE>;
  using SL = Slots<RP>;
  constexpr int NT = C::NT;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bar[kS];
  __shared__ uint32_t tslot;
  __shared__ int32_t s_row[NT * kTileM];

  const int n_splits = a.counts[a.count_slot];
  if ((int)blockIdx.x >= n_splits) return;
  const int proj = blockIdx.y;
  const Tile sp = a.splits[blockIdx.x];
  const int tid = threadIdx.x, warp = tid >> 5;
  const int g = sp.g, r0 = pt.rank_off[g], rg = pt.rank_off[g + 1] - r0;
  const int ntiles = (sp.cnt + kTileM - 1) / kTileM;
  const int d_in = a.d_in, d_out = a.d_out;
  const float s = a.s;
  const uint16_t* __restrict__ dY = a.dY[proj];

  const uint32_t ops = smem_u32(smem);
  const uint32_t stage0 = ops + C::kOps;
  auto act = [&](int slot) { return stage0 + slot * C::kStage; };
  auto wt = [&](int slot) { return stage0 + slot * C::kStage + C::kAct; };

  for (int i = tid; i < NT * kTileM; i += 128) {
    const int ti = i / kTileM, m = i % kTileM;
    s_row[i] = (ti < ntiles && m < sp.cnt - ti * kTileM) ? sp.start + ti * kTileM + m : -1;
  }
  if (tid == 0) {
    for (int i = 0; i < kS; ++i) mbar_init(&bar[i], 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, C::kTmem);
  __syncthreads();
  // H operand slots: bf16 of the saved H of each row (per unique pair for gate/up)
  for (int i = 0; i < ntiles; ++i) {
    const int row = s_row[i * kTileM + tid];
    const int hrow = row < 0 ? -1 : (MODE == MODE_SHARED ? a.row_uniq[row] : row);
    const float* hp = a.H[proj] + (int64_t)(hrow < 0 ? 0 : hrow) * pt.rank_max;
#pragma unroll
    for (int c8 = 0; c8 < RP; c8 += 8) {
      float v[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) v[q] = (hrow >= 0 && c8 + q < rg) ? hp[c8 + q] : 0.f;
      uint4 w;
      w.x = pack_bf16x2(v[0], v[1]);
      w.y = pack_bf16x2(v[2], v[3]);
      w.z = pack_bf16x2(v[4], v[5]);
      w.w = pack_bf16x2(v[6], v[7]);
      *reinterpret_cast<uint4*>(smem + SL::elem(i, tid, c8)) = w;
    }
  }
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tslot;
  bool bad = false, aborted = false;  // bad: this thread's wait gave up; aborted: CTA-uniform
  const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
  const uint32_t t_dbt = tmem + NT * RP;  // two buffers of RP columns

  // ------------------------------------------------------------- phase 1
  constexpr uint32_t id_dh = idesc_bf16_f32(128, RP, 0, 0);
  constexpr uint32_t id_w = idesc_bf16_f32(128, RP, 1, 1);
  const int nch1 = (d_out + kNcB - 1) / kNcB;
  const int NI1 = nch1 * ntiles;
  auto load1 = [&](int it, int slot) {
    const int c = it / ntiles, i = it % ntiles;
    load_w_tile<RP>(wt(slot), a.Bt[proj], r0, rg, d_out, c * kNcB, d_out, tid);
    load_act_tile(act(slot), dY, &s_row[i * kTileM], d_out, c * kNcB, d_out, tid);
  };
#pragma unroll
  for (int j = 0; j < kS - 1; ++j) {
    if (j < NI1) load1(j, j);
    cp_async_commit();
  }
  for (int it = 0; it < NI1; ++it) {
    const int c = it / ntiles, i = it % ntiles, slot = it % kS;
    cp_async_wait<kS - 2>();
    fence_proxy_async_smem();
    if (__syncthreads_or(bad)) {
      aborted = true;
      break;
    }
    if (tid == 0) {
      tc_fence_after();
      const uint32_t A0 = act(slot), W0 = wt(slot);
#pragma unroll
      for (int kk = 0; kk < kNcB / 16; ++kk)  // dH_i += dY_i . B_g
        tc_mma_bf16(tmem + i * RP, sdesc_sw128(A0 + (kk >> 2) * kBlk + (kk & 3) * 32, 16, 1024),
                    sdesc_sw128(W0 + (kk >> 2) * (RP * 128) + (kk & 3) * 32, 16, 1024), id_dh,
                    (c > 0 || kk > 0) ? 1u : 0u);
#pragma unroll
      for (int kk = 0; kk < kTileM / 16; ++kk)  // dBt_c^T += dY_i^T . H_i
        tc_mma_bf16(t_dbt + (c & 1) * RP, sdesc_sw128(A0 + kk * 2048, kBlk, 1024), SL::desc_mn(ops, i, kk), id_w,
                    (i > 0 || kk > 0) ? 1u : 0u);
      tc_commit(&bar[slot]);
    }
    if (i == 0 && c > 0) {  // flush chunk c-1 while chunk c runs
      if (!mbar_wait(&bar[(it - 1) % kS], ((it - 1) / kS) & 1)) bad = true;
      tc_fence_after();
      flush_wgrad<RP>(t_dbt + ((c - 1) & 1) * RP + lane_base, (c - 1) * kNcB, d_out, rg, r0, s, a.deterministic,
                      a.part_dBt[proj], sp.id, a.dBt[proj], tid);
      tc_fence_before();
    }
    const int nxt = it + kS - 1;
    if (nxt < NI1) {
      if (it >= 1 && !mbar_wait(&bar[(it - 1) % kS], ((it - 1) / kS) & 1)) bad = true;
      load1(nxt, nxt % kS);
    }
    cp_async_commit();
  }
  cp_async_wait<0>();
  if (NI1 > 0 && !aborted && !bad && !mbar_wait(&bar[(NI1 - 1) % kS], ((NI1 - 1) / kS) & 1)) bad = true;
  aborted = __syncthreads_or(bad || aborted);
  if (NI1 > 0 && !aborted) {
    tc_fence_after();
    flush_wgrad<RP>(t_dbt + ((nch1 - 1) & 1) * RP + lane_base, (nch1 - 1) * kNcB, d_out, rg, r0, s, a.deterministic,
                    a.part_dBt[proj], sp.id, a.dBt[proj], tid);
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (aborted) {
    if (tid == 0) atomicOr(a.err, kErrTimeout);
    if (warp == 0) tmem_dealloc(tmem, C::kTmem);
    return;
  }

  // dH (scaled by s): MODE_SHARED -> fp32 scratch per row; MODE_DOWN -> bf16 operand slots
  for (int i = 0; i < ntiles; ++i) {
    const int row = s_row[i * kTileM + tid];
#pragma unroll
    for (int c0 = 0; c0 < RP; c0 += 16) {
      uint32_t r[16];
      tmem_ld16(tmem + lane_base + i * RP + c0, r);
      tmem_ld_wait();
      if (MODE == MODE_SHARED) {
        if (row >= 0) {
          float4* dst = reinterpret_cast<float4*>(a.dHrow[proj] + (int64_t)row * RP + c0);
#pragma unroll
          for (int q = 0; q < 4; ++q)
            dst[q] = make_float4(s * __uint_as_float(r[4 * q]), s * __uint_as_float(r[4 * q + 1]),
                                 s * __uint_as_float(r[4 * q + 2]), s * __uint_as_float(r[4 * q + 3]));
        }
      } else {
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          uint4 w = make_uint4(0, 0, 0, 0);
          if (row >= 0) {
            w.x = pack_bf16x2(s * __uint_as_float(r[h * 8 + 0]), s * __uint_as_float(r[h * 8 + 1]));
            w.y = pack_bf16x2(s * __uint_as_float(r[h * 8 + 2]), s * __uint_as_float(r[h * 8 + 3]));
            w.z = pack_bf16x2(s * __uint_as_float(r[h * 8 + 4]), s * __uint_as_float(r[h * 8 + 5]));
            w.w = pack_bf16x2(s * __uint_as_float(r[h * 8 + 6]), s * __uint_as_float(r[h * 8 + 7]));
          }
          *reinterpret_cast<uint4*>(smem + SL::elem(i, tid, c0 + h * 8)) = w;
        }
      }
    }
  }
  if (MODE == MODE_DOWN) {
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    // ----------------------------------------------------------- phase 2
    constexpr uint32_t id_dh2 = idesc_bf16_f32(128, kNcB, 0, 1);
    const uint32_t t_d = tmem;                 // dh chunk, 128 columns
    const uint32_t t_da = tmem + kNcB;         // two buffers of RP columns
    const int nch2 = (d_in + kNcB - 1) / kNcB;
    const int NI2 = nch2 * ntiles;
    auto load2 = [&](int it, int slot) {
      const int c = it / ntiles, i = it % ntiles;
      load_w_tile<RP>(wt(slot), a.A[proj], r0, rg, d_in, c * kNcB, d_in, tid);
      load_act_tile(act(slot), a.Xin, &s_row[i * kTileM], d_in, c * kNcB, d_in, tid);
    };
    // barrier phases continue from phase 1: iteration j of phase 2 is global NI1 + j
#pragma unroll
    for (int j = 0; j < kS - 1; ++j) {
      if (j < NI2) {
        const int gj = NI1 + j;
        if (gj >= kS && !mbar_wait(&bar[gj % kS], ((gj - kS) / kS) & 1)) bad = true;
        load2(j, gj % kS);
      }
      cp_async_commit();
    }
    for (int it = 0; it < NI2; ++it) {
      const int c = it / ntiles, i = it % ntiles, git = NI1 + it, slot = git % kS;
      cp_async_wait<kS - 2>();
      fence_proxy_async_smem();
      if (__syncthreads_or(bad)) {
        aborted = true;
        break;
      }
      if (tid == 0) {
        tc_fence_after();
        const uint32_t A0 = act(slot), W0 = wt(slot);
#pragma unroll
        for (int kk = 0; kk < RP / 16; ++kk)  // dh chunk = dH_i . A_g
          tc_mma_bf16(t_d, SL::desc_k(ops, i, kk), sdesc_sw128(W0 + kk * 2048, RP * 128, 1024), id_dh2,
                      kk > 0 ? 1u : 0u);
#pragma unroll
        for (int kk = 0; kk < kTileM / 16; ++kk)  // dA_c^T += h_i^T . dH_i
          tc_mma_bf16(t_da + (c & 1) * RP, sdesc_sw128(A0 + kk * 2048, kBlk, 1024), SL::desc_mn(ops, i, kk), id_w,
                      (i > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&bar[slot]);
      }
      // this thread's dh row chunk (issued before waiting on the MMA)
      const int row = s_row[i * kTileM + tid];
      const int n0 = c * kNcB;
      uint4 y[16];
      uint16_t* yp = a.dXin + (int64_t)(row < 0 ? 0 : row) * d_in + n0;
#pragma unroll
      for (int q = 0; q < 16; ++q)
        y[q] = (row >= 0 && n0 + q * 8 < d_in) ? *reinterpret_cast<const uint4*>(yp + q * 8) : make_uint4(0, 0, 0, 0);
      if (!mbar_wait(&bar[slot], (git / kS) & 1)) bad = true;
      tc_fence_after();
      if (i == 0 && c > 0)
        flush_wgrad<RP>(t_da + ((c - 1) & 1) * RP + lane_base, (c - 1) * kNcB, d_in, rg, r0, 1.f, a.deterministic,
                        a.part_dA[proj], sp.id, a.dA[proj], tid);
#pragma unroll
      for (int sc = 0; sc < kNcB; sc += 32) {
        uint32_t r[32];
        tmem_ld16(t_d + lane_base + sc, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
        tmem_ld16(t_d + lane_base + sc + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
        tmem_ld_wait();
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int qq = sc / 8 + q;
          if (row >= 0 && n0 + qq * 8 < d_in)
            *reinterpret_cast<uint4*>(yp + qq * 8) = add_bf16x8(y[qq], &r[q * 8], 1.f);
        }
      }
      tc_fence_before();
      const int nxt = it + kS - 1;
      if (nxt < NI2) load2(nxt, (NI1 + nxt) % kS);  // its slot's previous MMA (git - 1) is complete
      cp_async_commit();
    }
    cp_async_wait<0>();
    aborted = __syncthreads_or(bad || aborted);
    if (NI2 > 0 && !aborted) {
      tc_fence_after();
      flush_wgrad<RP>(t_da + ((nch2 - 1) & 1) * RP + lane_base, (nch2 - 1) * kNcB, d_in, rg, r0, 1.f,
                      a.deterministic, a.part_dA[proj], sp.id, a.dA[proj], tid);
    }
  }
  tc_fence_before();
  aborted = __syncthreads_or(bad || aborted);
  if (aborted && tid == 0) atomicOr(a.err, kErrTimeout);
  if (warp == 0) tmem_dealloc(tmem, C::kTmem);
}

// ---------------------------------------------------------------- dH_u
template <int RP>
__global__ void __launch_bounds__(128) k_dh_reduce(const __grid_constant__ PlanTables pt,
                                                   const __grid_constant__ BwdLaunch a) {
  const int n_tiles = a.counts[kCntTilesSh];
  if ((int)blockIdx.x >= n_tiles) return;
  const int proj = blockIdx.y;
  const Tile tl = a.tiles_sh[blockIdx.x];
  const int m = threadIdx.x;
  if (m >= tl.cnt) return;
  const int u = tl.start + m, t = a.uniq_tok[u], k = pt.k;
  float acc[RP];
#pragma unroll
  for (int q = 0; q < RP; ++q) acc[q] = 0.f;
  for (int j = 0; j < k; ++j) {
    if (a.pair_g[(int64_t)t * k + j] != tl.g) continue;
    const float4* src = reinterpret_cast<const float4*>(a.dHrow[proj] + (int64_t)a.pair_row[(int64_t)t * k + j] * RP);
#pragma unroll
    for (int q = 0; q < RP / 4; ++q) {
      const float4 v = src[q];
      acc[4 * q] += v.x;
      acc[4 * q + 1] += v.y;
      acc[4 * q + 2] += v.z;
      acc[4 * q + 3] += v.w;
    }
  }
  uint4* dst = reinterpret_cast<uint4*>(a.dH[proj] + (int64_t)u * RP);
#pragma unroll
  for (int q = 0; q < RP / 8; ++q) {
    uint4 w;
    w.x = pack_bf16x2(acc[8 * q], acc[8 * q + 1]);
    w.y = pack_bf16x2(acc[8 * q + 2], acc[8 * q + 3]);
    w.z = pack_bf16x2(acc[8 * q + 4], acc[8 * q + 5]);
    w.w = pack_bf16x2(acc[8 * q + 6], acc[8 * q + 7]);
    dst[q] = w;
  }
}

// ---------------------------------------------------------------- dA (gate/up)
template <int RP, int NPROJ>
struct DaCfg {
  static constexpr int NT = RP <= 32 ? 4 : (RP == 64 ? 2 : 1);
  static constexpr int kOps = Slots<RP>::bytes(NT * NPROJ);
  static constexpr int kStage = kTileM * 256;
  static constexpr int kSmem = kOps + kS * kStage + 1024;
  static constexpr int kTmem = NPROJ * 2 * RP <= 256 ? 256 : 512;
};

template <int RP, int NPROJ>
__global__ void __launch_bounds__(128, 1) k_bwd_dA(const __grid_constant__ PlanTables pt,
                                                   const __grid_constant__ BwdLaunch a) {
  using C = DaCfg<RP, NPROJ>;
  using SL = Slots<RP>;
  constexpr int NT = C::NT;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bar[kS];
  __shared__ uint32_t tslot;
  __shared__ int32_t s_tok[NT * kTileM];

  const int n_splits = a.counts[a.count_slot];
  if ((int)blockIdx.x >= n_splits) return;
  const Tile sp = a.splits[blockIdx.x];
  const int tid = threadIdx.x, warp = tid >> 5;
  const int g = sp.g, r0 = pt.rank_off[g], rg = pt.rank_off[g + 1] - r0;
  const int ntiles = (sp.cnt + kTileM - 1) / kTileM;
  const int d = a.d_in;
  const uint32_t ops = smem_u32(smem);
  const uint32_t stage0 = ops + C::kOps;

  for (int i = tid; i < NT * kTileM; i += 128) {
    const int ti = i / kTileM, m = i % kTileM;
    s_tok[i] = (ti < ntiles && m < sp.cnt - ti * kTileM) ? a.uniq_tok[sp.start + ti * kTileM + m] : -1;
  }
  if (tid == 0) {
    for (int i = 0; i < kS; ++i) mbar_init(&bar[i], 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, C::kTmem);
  // dH_u slots (bf16 scratch rows), slot q = i * NPROJ + j
  for (int i = 0; i < ntiles; ++i) {
    const int cnt_i = sp.cnt - i * kTileM;
    const int u = sp.start + i * kTileM + tid;
    for (int j = 0; j < NPROJ; ++j) {
#pragma unroll
      for (int c8 = 0; c8 < RP; c8 += 8) {
        const bool v = tid < cnt_i;
        cp_async16(ops + SL::elem(i * NPROJ + j, tid, c8), v ? a.dH[j] + (int64_t)u * RP + c8 : a.dH[0], v);
      }
    }
  }
  cp_async_commit();
  __syncthreads();
  const uint32_t tmem = tslot;
  bool bad = false, aborted = false;  // bad: this thread's wait gave up; aborted: CTA-uniform
  const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
  constexpr uint32_t id_w = idesc_bf16_f32(128, RP, 1, 1);
  const int nch = (d + kNcB - 1) / kNcB;
  const int NI = nch * ntiles;
  auto load = [&](int it, int slot) {
    load_act_tile(stage0 + slot * C::kStage, a.Xin, &s_tok[(it % ntiles) * kTileM], d, (it / ntiles) * kNcB, d, tid);
  };
#pragma unroll
  for (int j = 0; j < kS - 1; ++j) {
    if (j < NI) load(j, j);
    cp_async_commit();
  }
  for (int it = 0; it < NI; ++it) {
    const int c = it / ntiles, i = it % ntiles, slot = it % kS;
    cp_async_wait<kS - 2>();
    fence_proxy_async_smem();
    if (__syncthreads_or(bad)) {
      aborted = true;
      break;
    }
    if (tid == 0) {
      tc_fence_after();
      const uint32_t A0 = stage0 + slot * C::kStage;
#pragma unroll
      for (int j = 0; j < NPROJ; ++j)
#pragma unroll
        for (int kk = 0; kk < kTileM / 16; ++kk)
          tc_mma_bf16(tmem + (j * 2 + (c & 1)) * RP, sdesc_sw128(A0 + kk * 2048, kBlk, 1024),
                      SL::desc_mn(ops, i * NPROJ + j, kk), id_w, (i > 0 || kk > 0) ? 1u : 0u);
      tc_commit(&bar[slot]);
    }
    if (i == 0 && c > 0) {
      if (!mbar_wait(&bar[(it - 1) % kS], ((it - 1) / kS) & 1)) bad = true;
      tc_fence_after();
      for (int j = 0; j < NPROJ; ++j)
        flush_wgrad<RP>(tmem + (j * 2 + ((c - 1) & 1)) * RP + lane_base, (c - 1) * kNcB, d, rg, r0, 1.f,
                        a.deterministic, a.part_dA[j], sp.id, a.dA[j], tid);
      tc_fence_before();
    }
    const int nxt = it + kS - 1;
    if (nxt < NI) {
      if (it >= 1 && !mbar_wait(&bar[(it - 1) % kS], ((it - 1) / kS) & 1)) bad = true;
      load(nxt, nxt % kS);
    }
    cp_async_commit();
  }
  cp_async_wait<0>();
  if (NI > 0 && !aborted && !bad && !mbar_wait(&bar[(NI - 1) % kS], ((NI - 1) / kS) & 1)) bad = true;
  aborted = __syncthreads_or(bad || aborted);
  if (NI > 0 && !aborted) {
    tc_fence_after();
    for (int j = 0; j < NPROJ; ++j)
      flush_wgrad<RP>(tmem + (j * 2 + ((nch - 1) & 1)) * RP + lane_base, (nch - 1) * kNcB, d, rg, r0, 1.f,
                      a.deterministic, a.part_dA[j], sp.id, a.dA[j], tid);
  }
  if (aborted && tid == 0) atomicOr(a.err, kErrTimeout);
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, C::kTmem);
}

// ---------------------------------------------------------------- dX
template <int RP>
struct DxCfg {
  static constexpr int kNd = 256;
  static constexpr int kOp = (RP > 64 ? 2 : 1) * kBlk;
  static constexpr int kW = RP * kNd * 2;  // 4 blocks of [RP x 128 B]
  static constexpr int kStage = kOp + kW;
  static constexpr int kSmem = kS * kStage + 1024;
};

template <int RP>
__global__ void __launch_bounds__(128) k_dx(const __grid_constant__ PlanTables pt, const __grid_constant__ DxLaunch a) {
  using C = DxCfg<RP>;
  constexpr int kNd = C::kNd;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bar[kS];
  __shared__ uint32_t tslot;
  __shared__ int32_t s_uoff[ACE_MAX_EXPERTS + 1];
  __shared__ int32_t s_kb[ACE_MAX_EXPERTS];  // groups active in this token tile
  __shared__ int32_t s_nkb;
  const int tid = threadIdx.x, warp = tid >> 5;
  const int t0 = blockIdx.x * kTileM, c0 = blockIdx.y * kNd;
  const int d = a.d, k = pt.k, G = pt.G;
  const int t = t0 + tid;
  for (int i = tid; i <= G; i += 128) s_uoff[i] = a.uniq_off[i];
  if (tid == 0) {
    for (int i = 0; i < kS; ++i) mbar_init(&bar[i], 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, 256);
  __syncthreads();
  // token's unique pairs (ascending g) and the active groups of the tile
  int my_u[kMaxK];
  int nu = 0;
  if (t < a.T) {
    for (int j = 0; j < k; ++j) {
      const int u = a.tok_uniq[(int64_t)t * k + j];
      if (u < 0) break;
      my_u[nu++] = u;
    }
  }
  if (tid == 0) s_nkb = 0;
  __syncthreads();
  // groups with at least one token of this tile, ascending
  for (int g = 0; g < G; ++g) {
    bool has = false;
    for (int q = 0; q < nu; ++q) has |= (my_u[q] >= s_uoff[g] && my_u[q] < s_uoff[g + 1]);
    if (__syncthreads_or(has) && tid == 0) s_kb[s_nkb++] = g;
  }
  __syncthreads();
  const int ng = s_nkb;
  const int NI = ng * a.nproj;
  const uint32_t stage0 = smem_u32(smem);
  const uint32_t tmem = tslot;
  bool bad = false, aborted = false;  // bad: this thread's wait gave up; aborted: CTA-uniform
  const uint32_t lane_base = (uint32_t)(warp * 32) << 16;
  constexpr uint32_t idesc = idesc_bf16_f32(128, kNd, 0, 1);
  auto load = [&](int it, int slot) {
    const int j = it / ng, g = s_kb[it % ng];
    const uint32_t sop = stage0 + slot * C::kStage, sw = sop + C::kOp;
    int u = -1;
    for (int q = 0; q < nu; ++q)
      if (my_u[q] >= s_uoff[g] && my_u[q] < s_uoff[g + 1]) u = my_u[q];
    const uint16_t* dHj = a.dH[j];
#pragma unroll
    for (int c8 = 0; c8 < RP; c8 += 8) {
      const bool v = u >= 0;
      cp_async16(sop + (c8 >> 6) * kBlk + sw128_off(tid, (c8 & 63) >> 3), v ? dHj + (int64_t)u * RP + c8 : dHj, v);
    }
    const int r0 = pt.rank_off[g], rg = pt.rank_off[g + 1] - r0;
#pragma unroll 4
    for (int idx = tid; idx < RP * (kNd / 8); idx += 128) {
      const int kr = idx / (kNd / 8), cc = idx % (kNd / 8), col = c0 + cc * 8;
      const bool v = kr < rg && col < d;
      cp_async16(sw + (cc >> 3) * (RP * 128) + sw128_off(kr, cc & 7), v ? a.A[j] + (int64_t)(r0 + kr) * d + col : a.A[0],
                 v);
    }
  };
#pragma unroll
  for (int j = 0; j < kS - 1; ++j) {
    if (j < NI) load(j, j);
    cp_async_commit();
  }
  for (int it = 0; it < NI; ++it) {
    const int slot = it % kS;
    cp_async_wait<kS - 2>();
    fence_proxy_async_smem();
    if (__syncthreads_or(bad)) {
      aborted = true;
      break;
    }
    if (tid == 0) {
      tc_fence_after();
      const uint32_t sop = stage0 + slot * C::kStage, sw = sop + C::kOp;
#pragma unroll
      for (int kk = 0; kk < RP / 16; ++kk)
        tc_mma_bf16(tmem, sdesc_sw128(sop + (kk >> 2) * kBlk + (kk & 3) * 32, 16, 1024),
                    sdesc_sw128(sw + kk * 2048, RP * 128, 1024), idesc, (it > 0 || kk > 0) ? 1u : 0u);
      tc_commit(&bar[slot]);
    }
    const int nxt = it + kS - 1;
    if (nxt < NI) {
      if (it >= 1 && !mbar_wait(&bar[(it - 1) % kS], ((it - 1) / kS) & 1)) bad = true;
      load(nxt, nxt % kS);
    }
    cp_async_commit();
  }
  cp_async_wait<0>();
  if (NI > 0) {
    if (!aborted && !bad && !mbar_wait(&bar[(NI - 1) % kS], ((NI - 1) / kS) & 1)) bad = true;
    tc_fence_after();
    aborted = __syncthreads_or(bad || aborted);
    if (!aborted) {
#pragma unroll 1
      for (int sc = 0; sc < kNd; sc += 64) {
        const int col0 = c0 + sc;
        uint4 y[8];
        uint16_t* yp = a.dX + (int64_t)(t < a.T ? t : 0) * d + col0;
#pragma unroll
        for (int q = 0; q < 8; ++q)
          y[q] = (t < a.T && col0 + q * 8 < d) ? *reinterpret_cast<const uint4*>(yp + q * 8) : make_uint4(0, 0, 0, 0);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          uint32_t r[32];
          tmem_ld16(tmem + lane_base + sc + h * 32, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
          tmem_ld16(tmem + lane_base + sc + h * 32 + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const int qq = h * 4 + q;
            if (t < a.T && col0 + qq * 8 < d)
              *reinterpret_cast<uint4*>(yp + qq * 8) = add_bf16x8(y[qq], &r[q * 8], 1.f);
          }
        }
      }
    }
  }
  if (aborted && tid == 0) atomicOr(a.err, kErrTimeout);
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

template <typename K>
cudaError_t set_smem(K kern, int bytes) {
  return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

cudaError_t reduce_launch(const PlanTables& pt, const Tile* splits, const int32_t* counts, int slot, const float* part,
                          int RP, int width, float* out, cudaStream_t st) {
  const int n_rank = pt.rank_off[pt.G];
  dim3 grid(n_rank, (width / 4 + 255) / 256);
  k_splitk_reduce<<<grid, 256, 0, st>>>(pt, splits, counts, slot, part, RP, width, out);
  return cudaGetLastError();
}

template <int RP>
cudaError_t launch_bwd_t(const PlanTables& pt, const BwdLaunch& a, bool shared, cudaStream_t st) {
  cudaError_t e;
  const int n_rank = pt.rank_off[pt.G];
  const int nproj = shared ? a.nproj : 1;
  if (!a.deterministic) {
    for (int j = 0; j < nproj; ++j) {
      if ((e = cudaMemsetAsync(a.dA[j], 0, sizeof(float) * (size_t)n_rank * a.d_in, st)) != cudaSuccess) return e;
      if ((e = cudaMemsetAsync(a.dBt[j], 0, sizeof(float) * (size_t)n_rank * a.d_out, st)) != cudaSuccess) return e;
    }
  }
  if (a.T > 0) {
    if (!shared) {
      using C = RowsCfg<RP, MODE_DOWN>;
      auto kern = k_bwd_rows<RP, MODE_DOWN>;
      if ((e = set_smem(kern, C::kSmem)) != cudaSuccess) return e;
      kern<<<dim3(a.max_splits_row, 1), 128, C::kSmem, st>>>(pt, a);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
    } else {
      using C = RowsCfg<RP, MODE_SHARED>;
      auto kern = k_bwd_rows<RP, MODE_SHARED>;
      if ((e = set_smem(kern, C::kSmem)) != cudaSuccess) return e;
      BwdLaunch b = a;
      b.splits = a.splits_row;
      b.count_slot = kCntSplitsRow;
      b.part_dBt[0] = a.part_dBt[0];
      b.part_dBt[1] = a.part_dBt[1];
      kern<<<dim3(a.max_splits_row, nproj), 128, C::kSmem, st>>>(pt, b);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
      k_dh_reduce<RP><<<dim3(a.max_tiles_sh, nproj), 128, 0, st>>>(pt, a);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
      if (nproj == 2) {
        using D = DaCfg<RP, 2>;
        auto kd = k_bwd_dA<RP, 2>;
        if ((e = set_smem(kd, D::kSmem)) != cudaSuccess) return e;
        kd<<<a.max_splits, 128, D::kSmem, st>>>(pt, a);
      } else {
        using D = DaCfg<RP, 1>;
        auto kd = k_bwd_dA<RP, 1>;
        if ((e = set_smem(kd, D::kSmem)) != cudaSuccess) return e;
        kd<<<a.max_splits, 128, D::kSmem, st>>>(pt, a);
      }
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
  }
  if (a.deterministic) {
    for (int j = 0; j < nproj; ++j) {
      // dB^T partials are indexed by row splits, dA partials by the path's splits
      if ((e = reduce_launch(pt, a.splits_row, a.counts, kCntSplitsRow, a.part_dBt[j], RP, a.d_out, a.dBt[j], st)) !=
          cudaSuccess)
        return e;
      if ((e = reduce_launch(pt, shared ? a.splits : a.splits_row, a.counts, shared ? kCntSplitsSh : kCntSplitsRow,
                             a.part_dA[j], RP, a.d_in, a.dA[j], st)) != cudaSuccess)
        return e;
    }
  }
  return cudaSuccess;
}

template <int RP>
cudaError_t launch_dx_t(const PlanTables& pt, const DxLaunch& a, cudaStream_t st) {
  using C = DxCfg<RP>;
  auto kern = k_dx<RP>;
  cudaError_t e = set_smem(kern, C::kSmem);
  if (e != cudaSuccess) return e;
  dim3 grid((a.T + kTileM - 1) / kTileM, (a.d + C::kNd - 1) / C::kNd);
  kern<<<grid, 128, C::kSmem, st>>>(pt, a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_bwd(const PlanTables& pt, const BwdLaunch& a, bool shared, cudaStream_t st) {
  switch (pt.rank_pad) {
    case 16: return launch_bwd_t<16>(pt, a, shared, st);
    case 32: return launch_bwd_t<32>(pt, a, shared, st);
    case 64: return launch_bwd_t<64>(pt, a, shared, st);
    case 128: return launch_bwd_t<128>(pt, a, shared, st);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_dx(const PlanTables& pt, const DxLaunch& a, cudaStream_t st) {
  if (a.T == 0) return cudaSuccess;
  switch (pt.rank_pad) {
    case 16: return launch_dx_t<16>(pt, a, st);
    case 32: return launch_dx_t<32>(pt, a, st);
    case 64: return launch_dx_t<64>(pt, a, st);
    case 128: return launch_dx_t<128>(pt, a, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace ace
