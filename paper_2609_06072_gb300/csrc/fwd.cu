// Fused LoRA forward (Sec. 3.3-3.5; App. "Implementation and Profiling of
// Grouped Adapter Execution").
//
// k_fwd_h (gate/up): per tile of up to 128 unique (g, t) pairs of one group,
//   H_u = A_g x_t is computed ONCE per active group of a token (Sec. 3.5):
//   X rows gathered by token with cp.async into 128-byte-swizzled smem,
//   tcgen05 MMA with N = nproj * rank_pad (gate and up share the gather),
//   fp32 H written per unique pair.
// k_fwd_rows: persistent, one CTA per SM; each CTA takes an equal share of
//   the rows (16-row quanta) and walks it in tiles of <= 128 consecutive rows
//   of one group (expert segments are contiguous inside group segments).
//   Warp-specialised:
//     warp 0     TMA producer: row tiles of Y (and of h for down) and chunks of
//                B_g^T / A_g into a ring of shared-memory slots
//     warp 1     MMA issuer: (down) H = h . A_g^T over the K loop, then per
//                64-column chunk D = H . B_g^T into double-buffered TMEM
//     warps 2-9  epilogue, two groups of four (one warp per TMEM lane
//                quarter): H -> bf16 operand (down: from TMEM; gate/up:
//                gathered from the unique pair of each row), then group p
//                takes the chunks of parity p: Y += s * D on its own 32 rows
//                in swizzled smem (TMEM lane = row) and stores those rows.
//   For gate/up the K = r_g product B_g H_u is evaluated per routed row; the
//   K = d product A_g x -- the one that dominates -- stays deduplicated.
#include <cstdint>

#include "ace_internal.cuh"
#include "ace_ptx.cuh"

namespace ace {
namespace {

constexpr int kBlk = kTileM * 128;  // [128 rows x 64 bf16] SW128 block, 16 KB

// ------------------------------------------------------------------ k_fwd_h
constexpr int kHStages = 3;
constexpr int kHThreads = 256;

template <int RP, int NPROJ>
struct FwdHCfg {
  static constexpr int kStageA = NPROJ * RP * 128;
  static constexpr int kStage = kBlk + kStageA;
  static constexpr int kSmem = kHStages * kStage + 1024;
  static constexpr int kTmem = NPROJ * RP <= 32 ? 32 : NPROJ * RP <= 64 ? 64 : NPROJ * RP <= 128 ? 128 : 256;
};

template <int RP, int NPROJ>
__global__ void __launch_bounds__(kHThreads) k_fwd_h(const __grid_constant__ PlanTables pt,
                                                     const __grid_constant__ FwdHLaunch a) {
  using C = FwdHCfg<RP, NPROJ>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t bar_k[kHStages];
  __shared__ uint32_t tslot;
  __shared__ int32_t src_row[kTileM];

  const int n_tiles = a.counts[kCntTilesSh];
  if ((int)blockIdx.x >= n_tiles) return;
  const Tile tl = a.tiles[blockIdx.x];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int quarter = warp & 3, half = warp >> 2;
  const int m = quarter * 32 + lane;
  const int g = tl.g, r0 = pt.rank_off[g], rg = pt.rank_off[g + 1] - r0;
  const int d_in = a.d_in;

  if (tid < kTileM) src_row[tid] = tid < tl.cnt ? a.uniq_tok[tl.start + tid] : -1;
  if (tid == 0) {
    for (int i = 0; i < kHStages; ++i) mbar_init(&bar_k[i], 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, C::kTmem);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tslot;
  const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;

  const int NK = (d_in + 63) / 64;
  auto load_stage = [&](int kt, int slot) {
    const uint32_t sX = smem_u32(smem + slot * C::kStage);
    const uint32_t sA = sX + kBlk;
    const int k0 = kt * 64;
#pragma unroll
    for (int i = 0; i < 1024 / kHThreads; ++i) {
      const int idx = i * kHThreads + tid, r = idx >> 3, c = idx & 7;
      const int sr = src_row[r], kc = k0 + c * 8;
      const bool v = sr >= 0 && kc < d_in;
      cp_async16(sX + sw128_off(r, c), v ? a.X + (int64_t)sr * d_in + kc : a.X, v);
    }
#pragma unroll
    for (int idx = tid; idx < NPROJ * RP * 8; idx += kHThreads) {
      const int rr = idx >> 3, c = idx & 7, j = rr / RP, kr = rr % RP, kc = k0 + c * 8;
      const bool v = kr < rg && kc < d_in;
      cp_async16(sA + sw128_off(rr, c), v ? a.A[j] + (int64_t)(r0 + kr) * d_in + kc : a.A[0], v);
    }
  };
  constexpr uint32_t idesc_h = idesc_bf16_f32(128, NPROJ * RP, 0, 0);
#pragma unroll
  for (int s = 0; s < kHStages - 1; ++s) {
    if (s < NK) load_stage(s, s);
    cp_async_commit();
  }
  bool bad = false, aborted = false;
  for (int kt = 0; kt < NK; ++kt) {
    const int slot = kt % kHStages;
    cp_async_wait<kHStages - 2>();
    fence_proxy_async_smem();
    if (__syncthreads_or(bad)) {
      aborted = true;
      break;
    }
    if (tid == 0) {
      tc_fence_after();
      const uint32_t sX = smem_u32(smem + slot * C::kStage), sA = sX + kBlk;
#pragma unroll
      for (int kk = 0; kk < 4; ++kk)
        tc_mma_bf16(tmem, sdesc_sw128(sX + kk * 32, 16, 1024), sdesc_sw128(sA + kk * 32, 16, 1024), idesc_h,
                    (kt > 0 || kk > 0) ? 1u : 0u);
      tc_commit(&bar_k[slot]);
    }
    const int nxt = kt + kHStages - 1;
    if (nxt < NK) {
      if (kt >= 1 && !mbar_wait(&bar_k[nxt % kHStages], ((kt - 1) / kHStages) & 1)) bad = true;
      if (!bad) load_stage(nxt, nxt % kHStages);
    }
    cp_async_commit();
  }
  cp_async_wait<0>();
  if (NK > 0 && !aborted && !bad && !mbar_wait(&bar_k[(NK - 1) % kHStages], ((NK - 1) / kHStages) & 1)) bad = true;
  tc_fence_before();
  aborted = __syncthreads_or(bad || aborted);
  tc_fence_after();
  if (!aborted) {
    constexpr int kHcols = NPROJ * RP;
    for (int c0 = half * 16; c0 < kHcols; c0 += 32) {
      uint32_t r[16];
      tmem_ld16(tmem + lane_base + c0, r);
      tmem_ld_wait();
      const int j = c0 / RP, kb = c0 % RP;
      if (m < tl.cnt) {
        float* hrow = a.H[j] + (int64_t)(tl.start + m) * pt.rank_max;
#pragma unroll
        for (int q = 0; q < 16; ++q)
          if (kb + q < pt.rank_max) hrow[kb + q] = __uint_as_float(r[q]);
      }
    }
  }
  if (aborted && tid == 0) atomicOr(a.err, kErrTimeout);
  tc_fence_before();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, C::kTmem);
}

// --------------------------------------------------------------- k_fwd_rows
constexpr int kRowsThreads = 320;  // 10 warps: producer, MMA, 2 x 4 epilogue warps
constexpr int kChunk = 64;         // output columns per D chunk
constexpr int kQuant = 16;         // rows per work quantum and per small TMA box

template <int RP, int NPROJ>
struct RowsFwdCfg {
  static constexpr int kWBlk = RP * 128;                    // [RP x 64] weight block
  static constexpr int kSlot = NPROJ * (kBlk + kWBlk);      // Y tiles + B^T blocks (down K-step: h + A)
  static constexpr int kHs = ((NPROJ * RP + 63) / 64) * kBlk;
  static constexpr int kBudget = 200 * 1024;
  static constexpr int kS0 = (kBudget - kHs) / kSlot;
  static constexpr int S = kS0 > 8 ? 8 : (kS0 < 2 ? 2 : kS0);
  static constexpr int kSmem = kHs + S * kSlot + 1024;
};

// Rows of one CTA of a persistent row kernel: equal shares of 16-row quanta
// over the CTAs that have work (at least 128 rows each).
struct RowRange {
  int begin, end;
};
__device__ __forceinline__ RowRange cta_rows(int R) {
  const int ncta = min((int)gridDim.x, max(1, (R + kTileM - 1) / kTileM));
  if ((int)blockIdx.x >= ncta) return {0, 0};
  const int nq = (R + kQuant - 1) / kQuant;
  const int q0 = (int)((int64_t)blockIdx.x * nq / ncta), q1 = (int)((int64_t)(blockIdx.x + 1) * nq / ncta);
  return {min(R, q0 * kQuant), min(R, q1 * kQuant)};
}

// Walks a row range in tiles of at most 128 rows that never cross a group
// boundary (every row of a tile uses the same A_g, B_g).  goff: group_off in
// shared memory.  Every role of a CTA walks the same sequence.
struct TileWalk {
  int cur, end, g;
  __device__ __forceinline__ bool next(const int32_t* goff, Tile& t) {
    if (cur >= end) return false;
    while (goff[g + 1] <= cur) ++g;
    t.g = g;
    t.start = cur;
    t.cnt = min(kTileM, min(end, goff[g + 1]) - cur);
    t.id = 0;
    cur += t.cnt;
    return true;
  }
};

// Rows [y, y + cnt) of a 64-column box at column x: one 128-row box for a
// whole tile, else ceil(cnt / 16) boxes of 16 rows (so a short tile reads at
// most 15 rows it does not use).  Returns the bytes the copies deliver.
__device__ __forceinline__ uint32_t load_rows(uint32_t dst, const CUtensorMap* m128, const CUtensorMap* m16, int x,
                                              int y, int cnt, uint64_t* bar) {
  if (cnt == kTileM) {
    tma_load_2d(dst, m128, x, y, bar);
    return kBlk;
  }
  const int nb = (cnt + kQuant - 1) / kQuant;
  for (int b = 0; b < nb; ++b) tma_load_2d(dst + b * kQuant * 128, m16, x, y + b * kQuant, bar);
  return nb * kQuant * 128;
}
__device__ __forceinline__ uint32_t rows_bytes(int cnt) {
  return cnt == kTileM ? (uint32_t)kBlk : (uint32_t)((cnt + kQuant - 1) / kQuant) * kQuant * 128;
}

// Persistent: one CTA per SM walks its share of the rows tile by tile; the
// producer, the MMA issuer and the epilogue run ahead of one another across
// tile boundaries.  The eight epilogue warps form two groups of four (one warp
// per TMEM lane quarter); group p owns the D chunks of parity p, and each warp
// updates and stores only its own 32 rows, so a chunk needs no barrier wider
// than its group.
template <int RP, int NPROJ, bool SHARED>
__global__ void __launch_bounds__(kRowsThreads, 1) k_fwd_rows(const __grid_constant__ PlanTables pt,
                                                              const __grid_constant__ FwdRowsLaunch a) {
  using C = RowsFwdCfg<RP, NPROJ>;
  constexpr int S = C::S;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t full[S], empty[S], dfull[2], dempty[2], hacc, hs_ready;
  __shared__ uint32_t tslot;
  __shared__ int32_t goff[ACE_MAX_EXPERTS + 1];

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  for (int i = tid; i <= pt.G; i += kRowsThreads) goff[i] = a.group_off[i];
  if (tid == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&dfull[i], 1);
      mbar_init(&dempty[i], 4);  // the four warps of the group that owns the buffer
    }
    mbar_init(&hacc, 1);
    mbar_init(&hs_ready, 8);  // every epilogue warp
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, 256);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tslot;
  const RowRange rr = cta_rows(goff[pt.G]);
  const int d_in = a.d_in, d_out = a.d_out;
  const int NK = SHARED ? 0 : (d_in + 63) / 64;  // K steps of the down H GEMM
  const int nch = (d_out + kChunk - 1) / kChunk;
  const uint32_t sHs = smem_u32(smem);
  const uint32_t slot0 = sHs + C::kHs;
  const uint32_t dbase = SHARED ? 0u : 128u;  // down: H accumulator in columns [0, RP)
  bool bad = false;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      TileWalk w{rr.begin, rr.end, 0};
      Tile tl;
      int i = 0;
      while (!bad && w.next(goff, tl)) {
        const int r0 = pt.rank_off[tl.g];
        const uint32_t rb = rows_bytes(tl.cnt);
        for (int it = 0; it < NK + nch; ++it, ++i) {
          const int s = i % S, u = i / S;
          if (u >= 1 && !mbar_wait(&empty[s], (u - 1) & 1)) {
            bad = true;
            break;
          }
          const uint32_t base = slot0 + s * C::kSlot;
          if (it < NK) {
            mbar_arrive_expect_tx(&full[s], rb + C::kWBlk);
            load_rows(base, &a.tm_x, &a.tm_x16, it * 64, tl.start, tl.cnt, &full[s]);
            tma_load_2d(base + NPROJ * kBlk, &a.tm_a, it * 64, r0, &full[s]);
          } else {
            const int n0 = (it - NK) * kChunk;
            mbar_arrive_expect_tx(&full[s], NPROJ * (rb + C::kWBlk));
#pragma unroll
            for (int j = 0; j < NPROJ; ++j) {
              load_rows(base + j * kBlk, &a.tm_y[j], &a.tm_y16[j], n0, tl.start, tl.cnt, &full[s]);
              tma_load_2d(base + NPROJ * kBlk + j * C::kWBlk, &a.tm_bt[j], n0, r0, &full[s]);
            }
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
      constexpr uint32_t idesc_h = idesc_bf16_f32(128, RP, 0, 0);
      constexpr uint32_t idesc_d = idesc_bf16_f32(128, kChunk, 0, 1);
      TileWalk w{rr.begin, rr.end, 0};
      Tile tl;
      int i = 0, cc = 0, ti = 0;
      while (!bad && w.next(goff, tl)) {
        for (int it = 0; it < NK + nch; ++it, ++i) {
          const int s = i % S, u = i / S;
          if (!mbar_wait(&full[s], u & 1)) {
            bad = true;
            break;
          }
          tc_fence_after();
          const uint32_t base = slot0 + s * C::kSlot;
          if (it < NK) {
#pragma unroll
            for (int kk = 0; kk < 4; ++kk)
              tc_mma_bf16(tmem, sdesc_sw128(base + kk * 32, 16, 1024),
                          sdesc_sw128(base + NPROJ * kBlk + kk * 32, 16, 1024), idesc_h,
                          (it > 0 || kk > 0) ? 1u : 0u);
            tc_commit(&empty[s]);
            if (it == NK - 1) tc_commit(&hacc);
          } else {
            const int b = cc & 1;
            if (it == NK && !mbar_wait(&hs_ready, ti & 1)) {
              bad = true;
              break;
            }
            if (cc >= 2 && !mbar_wait(&dempty[b], ((cc - 2) >> 1) & 1)) {
              bad = true;
              break;
            }
            tc_fence_after();
#pragma unroll
            for (int j = 0; j < NPROJ; ++j)
#pragma unroll
              for (int kk = 0; kk < RP / 16; ++kk) {
                const int kg = (j * RP) / 16 + kk;
                tc_mma_bf16(tmem + dbase + (b * NPROJ + j) * kChunk,
                            sdesc_sw128(sHs + (kg >> 2) * kBlk + (kg & 3) * 32, 16, 1024),
                            sdesc_sw128(base + NPROJ * kBlk + j * C::kWBlk + kk * 2048, C::kWBlk, 1024), idesc_d,
                            kk > 0 ? 1u : 0u);
              }
            tc_commit(&dfull[b]);
            ++cc;
          }
        }
        ++ti;
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int grp = (warp - 2) >> 2;        // chunk parity of this warp's group
    const int quarter = warp & 3;           // TMEM lane quarter of this warp
    const int m = quarter * 32 + lane;      // tile row owned by this thread
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    const float s = a.s;
    TileWalk w{rr.begin, rr.end, 0};
    Tile tl;
    int i0 = 0, cc0 = 0, ti = 0;
    bool ok = true;
    // Every decision to stop is made jointly by the four warps of a group
    // (bar.red.and), so no warp is ever left waiting at its group's barrier.
    while (ok && w.next(goff, tl)) {
      const int r0 = pt.rank_off[tl.g], rg = pt.rank_off[tl.g + 1] - r0;
      const bool live = m < tl.cnt;
      // sHs is free once the previous tile's last D chunk has completed
      bool w_ok = ti == 0 || mbar_wait(&dfull[(cc0 - 1) & 1], ((cc0 - 1) >> 1) & 1);
      // H -> bf16 operand (row m), columns split between the two groups
      if (!SHARED) {
        w_ok = w_ok && mbar_wait(&hacc, ti & 1);
        w_ok = __all_sync(0xffffffffu, w_ok);
        tc_fence_after();
        for (int c0 = grp * 16; c0 < RP && w_ok; c0 += 32) {
          uint32_t r[16];
          tmem_ld16(tmem + lane_base + c0, r);
          tmem_ld_wait();
          float v[16];
#pragma unroll
          for (int q = 0; q < 16; ++q) v[q] = (live && c0 + q < rg) ? __uint_as_float(r[q]) : 0.f;
          if (live && a.Hsave != nullptr) {
            float* hrow = a.Hsave + (int64_t)(tl.start + m) * pt.rank_max;
#pragma unroll
            for (int q = 0; q < 16; ++q)
              if (c0 + q < pt.rank_max) hrow[c0 + q] = v[q];
          }
#pragma unroll
          for (int h = 0; h < 2; ++h) {
            const int col = c0 + h * 8;
            uint4 o;
            o.x = pack_bf16x2(v[h * 8 + 0], v[h * 8 + 1]);
            o.y = pack_bf16x2(v[h * 8 + 2], v[h * 8 + 3]);
            o.z = pack_bf16x2(v[h * 8 + 4], v[h * 8 + 5]);
            o.w = pack_bf16x2(v[h * 8 + 6], v[h * 8 + 7]);
            sts128(sHs + (col >> 6) * kBlk + sw128_off(m, (col & 63) >> 3), o);
          }
        }
      } else if (w_ok) {
        const int u = live ? a.row_uniq[tl.start + m] : -1;
#pragma unroll
        for (int j = 0; j < NPROJ; ++j) {
          const float* hp = a.Hu[j] + (int64_t)(u < 0 ? 0 : u) * pt.rank_max;
          for (int c8 = grp * 8; c8 < RP; c8 += 16) {
            float v[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) v[q] = (u >= 0 && c8 + q < rg) ? hp[c8 + q] : 0.f;
            uint4 o;
            o.x = pack_bf16x2(v[0], v[1]);
            o.y = pack_bf16x2(v[2], v[3]);
            o.z = pack_bf16x2(v[4], v[5]);
            o.w = pack_bf16x2(v[6], v[7]);
            const int col = j * RP + c8;
            sts128(sHs + (col >> 6) * kBlk + sw128_off(m, (col & 63) >> 3), o);
          }
        }
      }
      fence_proxy_async_smem();
      tc_fence_before();
      ok = named_bar_and(1 + grp, 128, w_ok);
      if (!ok) break;
      if (lane == 0) mbar_arrive(&hs_ready);
      // the chunks of this group's parity: Y += s * D on this warp's 32 rows, then row stores
      for (int c = (grp ^ cc0) & 1; c < nch; c += 2) {
        const int cc = cc0 + c, i = i0 + NK + c, sl = i % S, b = cc & 1, n0 = c * kChunk;
        bool c_ok = mbar_wait(&full[sl], (i / S) & 1) && mbar_wait(&dfull[b], (cc >> 1) & 1);
        c_ok = __all_sync(0xffffffffu, c_ok);
        const uint32_t base = slot0 + sl * C::kSlot;
        if (c_ok) {
          tc_fence_after();
#pragma unroll
          for (int j = 0; j < NPROJ; ++j) {
            const uint32_t ta = tmem + lane_base + dbase + (b * NPROJ + j) * kChunk;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              uint32_t r[32];
              tmem_ld16(ta + h * 32, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
              tmem_ld16(ta + h * 32 + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
              tmem_ld_wait();
#pragma unroll
              for (int q = 0; q < 4; ++q) {
                const uint32_t addr = base + j * kBlk + sw128_off(m, h * 4 + q);
                const uint4 y = lds128(addr);
                const uint32_t* dq = &r[q * 8];
                const float2 f0 = unpack_bf16x2(y.x), f1 = unpack_bf16x2(y.y), f2 = unpack_bf16x2(y.z),
                             f3 = unpack_bf16x2(y.w);
                uint4 o;
                o.x = pack_bf16x2(f0.x + s * __uint_as_float(dq[0]), f0.y + s * __uint_as_float(dq[1]));
                o.y = pack_bf16x2(f1.x + s * __uint_as_float(dq[2]), f1.y + s * __uint_as_float(dq[3]));
                o.z = pack_bf16x2(f2.x + s * __uint_as_float(dq[4]), f2.y + s * __uint_as_float(dq[5]));
                o.w = pack_bf16x2(f3.x + s * __uint_as_float(dq[6]), f3.y + s * __uint_as_float(dq[7]));
                sts128(addr, o);
              }
            }
          }
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&dempty[b]);
          // this warp's 32 rows, 128 contiguous bytes each: 4 rows per instruction
#pragma unroll
          for (int j = 0; j < NPROJ; ++j)
#pragma unroll
            for (int it = 0; it < 8; ++it) {
              const int row = quarter * 32 + it * 4 + (lane >> 3), ch = lane & 7, col = n0 + ch * 8;
              if (row < tl.cnt && col < d_out) {
                const uint4 v = lds128(base + j * kBlk + sw128_off(row, ch));
                *reinterpret_cast<uint4*>(a.Y[j] + (int64_t)(tl.start + row) * d_out + col) = v;
              }
            }
          fence_proxy_async_smem();
        }
        ok = named_bar_and(1 + grp, 128, c_ok);
        if (!ok) break;
        if (warp == 2 + 4 * grp && lane == 0) mbar_arrive(&empty[sl]);
      }
      i0 += NK + nch;
      cc0 += nch;
      ++ti;
    }
    if (!ok) bad = true;
  }
  __syncwarp();  // reconverge the single-lane roles before the CTA barrier
  tc_fence_before();
  if (__syncthreads_or(bad) && tid == 0) atomicOr(a.err, kErrTimeout);
  if (warp == 0) tmem_dealloc(tmem, 256);
}

template <typename K>
cudaError_t set_smem(K kern, int bytes) {
  return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

template <int RP, int NPROJ>
cudaError_t launch_h_t(const PlanTables& pt, const FwdHLaunch& a, cudaStream_t st) {
  using C = FwdHCfg<RP, NPROJ>;
  auto kern = k_fwd_h<RP, NPROJ>;
  cudaError_t e = set_smem(kern, C::kSmem);
  if (e != cudaSuccess || a.max_tiles <= 0) return e;
  kern<<<a.max_tiles, kHThreads, C::kSmem, st>>>(pt, a);
  return cudaGetLastError();
}

template <int RP, int NPROJ, bool SHARED>
cudaError_t launch_rows_t(const PlanTables& pt, const FwdRowsLaunch& a, cudaStream_t st) {
  using C = RowsFwdCfg<RP, NPROJ>;
  auto kern = k_fwd_rows<RP, NPROJ, SHARED>;
  cudaError_t e = set_smem(kern, C::kSmem);
  if (e != cudaSuccess || a.grid <= 0) return e;
  kern<<<a.grid, kRowsThreads, C::kSmem, st>>>(pt, a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_fwd_h(const PlanTables& pt, const FwdHLaunch& a, cudaStream_t st) {
  const bool two = a.nproj == 2;
  switch (pt.rank_pad) {
    case 16: return two ? launch_h_t<16, 2>(pt, a, st) : launch_h_t<16, 1>(pt, a, st);
    case 32: return two ? launch_h_t<32, 2>(pt, a, st) : launch_h_t<32, 1>(pt, a, st);
    case 64: return two ? launch_h_t<64, 2>(pt, a, st) : launch_h_t<64, 1>(pt, a, st);
    case 128: return two ? launch_h_t<128, 2>(pt, a, st) : launch_h_t<128, 1>(pt, a, st);
  }
  return cudaErrorInvalidValue;
}

cudaError_t launch_fwd_rows(const PlanTables& pt, const FwdRowsLaunch& a, bool shared, cudaStream_t st) {
  if (!shared) {
    switch (pt.rank_pad) {
      case 16: return launch_rows_t<16, 1, false>(pt, a, st);
      case 32: return launch_rows_t<32, 1, false>(pt, a, st);
      case 64: return launch_rows_t<64, 1, false>(pt, a, st);
      case 128: return launch_rows_t<128, 1, false>(pt, a, st);
    }
  } else if (a.nproj == 2) {
    switch (pt.rank_pad) {
      case 16: return launch_rows_t<16, 2, true>(pt, a, st);
      case 32: return launch_rows_t<32, 2, true>(pt, a, st);
      case 64: return launch_rows_t<64, 2, true>(pt, a, st);
      case 128: return launch_rows_t<128, 2, true>(pt, a, st);
    }
  } else {
    switch (pt.rank_pad) {
      case 16: return launch_rows_t<16, 1, true>(pt, a, st);
      case 32: return launch_rows_t<32, 1, true>(pt, a, st);
      case 64: return launch_rows_t<64, 1, true>(pt, a, st);
      case 128: return launch_rows_t<128, 1, true>(pt, a, st);
    }
  }
  return cudaErrorInvalidValue;
}

}  // namespace ace
