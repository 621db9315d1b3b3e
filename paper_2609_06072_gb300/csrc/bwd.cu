// Fused LoRA backward (adjoint of the forward; gradient form of Sec. 3.1.2,
// shared adapter updates of Sec. 3.4).
//
// k_bwd_rows<RP, MODE>: one CTA per split of up to NT row tiles (128
//   consecutive rows of one group), warp-specialised (TMA producer warp, MMA
//   warp, 4 epilogue warps).  Phase 1 streams the upstream gradient dY in
//   128-column chunks:
//     dH_i  += dY_i . B_g                 (TMEM, accumulated over chunks)
//     dBt_c  = sum_i H_{u(row)}^T . dY_i  (TMEM, double-buffered per chunk)
//   and the epilogue flushes each dBt chunk (fp32 atomics, or a per-split
//   partial for the deterministic two-stage sum) while the next chunk runs.
//   The epilogue then writes dH (scaled by s).  MODE_DOWN continues over
//   128-column chunks of the input h:
//     dh_i  += dH_i . A_g                 (dh tiles staged by TMA, added in
//                                          swizzled smem, coalesced stores)
//     dA_c   = sum_i h_i^T . dH_i         (flushed like dB^T)
//   For gate/up (MODE_SHARED) the rows of one unique pair (g, t) share H_u and
//   dC_u . B_g = sum_rows dY_row . B_g, so streaming contiguous rows moves the
//   bytes of the deduplicated form.  dH_u, the sum of its rows' dH, lands in
//   the token-major dense dHx consumed by the dense dX / dA GEMMs of gemm.cu:
//   in the fast mode each row adds its dH there with bf16 vector reductions;
//   in the deterministic mode the rows go to fp32 scratch and
// k_dh_reduce sums them per unique pair in a fixed slot order.
// MODE_COMB (the down projection's delta taken through the gate-weighted
//   combine) has no phase 1: the token gradient dz reaches the rows through
//   the unique-pair product dHc_u = B_g^T dz_t (computed before, by the dense
//   H GEMM on dz), so the epilogue stages dH_row = s p_row dHc_u directly as
//   the phase-2 operand and writes the gate-weight gradient
//   dp_row = s dHc_u . H_row on the way; phase 2 (dh, dA) is MODE_DOWN's.
//   dB^T comes from the dense dA GEMM of gemm.cu on the token-major combined H.
// k_splitk_reduce: deterministic stage 2 of dB^T / dA (split order); empty groups
//   -> exact zeros.
#include <cstdint>

#include "ace_internal.cuh"
#include "ace_ptx.cuh"

namespace ace {
namespace {

constexpr int kNcB = 128;           // columns per chunk
constexpr int kBlk = kTileM * 128;  // one [128 x 64] bf16 SW128 block (16 KB)
constexpr int MODE_DOWN = 0, MODE_SHARED = 1, MODE_COMB = 2;
constexpr int kThreadsWS = 320;     // producer, MMA, 8 epilogue warps (two per TMEM lane quarter)
constexpr int kEpiThreads = 256;
constexpr int kEpiBar = 1;
constexpr int kIssueBar = 2;        // epilogue -> producer: the H prefetches are out

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

__device__ __forceinline__ uint4 pack8(const float* v) {
  uint4 w;
  w.x = pack_bf16x2(v[0], v[1]);
  w.y = pack_bf16x2(v[2], v[3]);
  w.z = pack_bf16x2(v[4], v[5]);
  w.w = pack_bf16x2(v[6], v[7]);
  return w;
}

// Adds v[0..16), the values of 16 consecutive bf16 columns starting O
// columns past an 8-column boundary (win0 = that boundary), into global
// memory with 16-byte vector reductions only: one per aligned 8-column
// window that meets the first `nvalid` columns.  Window positions outside
// them receive +0, which leaves a neighbour's bf16 value unchanged (x + 0 = x),
// so a group whose rank offset is not a multiple of 8 needs no 16-bit
// atomics (those would run as compare-and-swap loops).
template <int O>
__device__ __forceinline__ void red_windows(uint16_t* win0, const float* v, int nvalid) {
#pragma unroll
  for (int w = 0; w < (O == 0 ? 2 : 3); ++w) {
    const int qlo = 8 * w - O;  // index into v of the window's first column
    const int lo = qlo < 0 ? 0 : qlo;
    if (lo >= nvalid) continue;
    float u[8];
#pragma unroll
    for (int p = 0; p < 8; ++p) {
      const int q = qlo + p;
      u[p] = (q >= 0 && q < 16 && q < nvalid) ? v[q] : 0.f;
    }
    red_add_bf16x8(win0 + 8 * w, pack8(u));
  }
}

// Flush one [128 cols x RP] fp32 accumulator of a weight gradient (TMEM lane
// `col_lane` = column n0 + col_lane): atomics into out, a per-split partial,
// or a plain store of the final value.
enum FlushMode { kAtomic = 0, kPartial = 1, kStore = 2 };
template <int RP>
__device__ __forceinline__ void flush_wgrad(uint32_t taddr, int n0, int ld, int rg, int r0, float scale, int mode,
                                            float* __restrict__ part, int split_id, float* __restrict__ out,
                                            int col_lane, bool zero = false, int c_begin = 0, int c_step = 16) {
  const int col = n0 + col_lane;
  for (int c0 = c_begin; c0 < RP; c0 += c_step) {
    uint32_t r[16];
    tmem_ld16(taddr + c0, r);
    tmem_ld_wait();
    if (col < ld) {
#pragma unroll
      for (int q = 0; q < 16; ++q) {
        const int kk = c0 + q;
        if (kk < rg) {
          const float v = zero ? 0.f : scale * __uint_as_float(r[q]);
          if (mode == kPartial)
            part[((int64_t)split_id * RP + kk) * ld + col] = v;
          else if (mode == kAtomic)
            atomicAdd(&out[(int64_t)(r0 + kk) * ld + col], v);
          else
            out[(int64_t)(r0 + kk) * ld + col] = v;
        }
      }
    }
  }
}

// ----------------------------------------------------------------- k_bwd_rows
template <int RP, int MODE>
struct RowsCfg {
  // row tiles per split: the split's dH accumulators (NT x RP TMEM columns)
  // sit below the weight-gradient accumulators (2 x RP from kTB); at RP = 128
  // two tiles fill the 512 columns, and the phase-2 dh buffer of down and the
  // combine takes the dH columns once dH is staged as the phase-2 operand
  static constexpr int NT = bwd_nt_split(RP, MODE == MODE_SHARED);
  static constexpr int kPerSM = MODE == MODE_SHARED ? bwd_sh_ctas_per_sm(RP) : 1;  // resident CTAs per SM
  static constexpr int kOps = Slots<RP>::bytes(NT);
  static constexpr int kWBlk = RP * 128;
  static constexpr int kSlotA = 2 * kBlk + 2 * kWBlk;  // dY tile + B^T chunk (down phase 2: A chunk + h tile)
  static constexpr int kSlotB = 2 * kBlk;                      // down: dh tile for the RMW
  // down / combine: dh tiles of the RMW (one at RP = 128, where two would not
  // fit beside the ring)
  static constexpr int SB = MODE != MODE_SHARED ? (RP > 64 ? 1 : 2) : 0;
  static constexpr int kBudget = 220 * 1024 / kPerSM;
  static constexpr int kSA0 = (kBudget - kOps - SB * kSlotB) / kSlotA;
  static constexpr int SA = kSA0 > 6 ? 6 : (kSA0 < 2 ? 2 : kSA0);
  static constexpr int kSmem = kOps + SA * kSlotA + SB * kSlotB + 1024;
  // dH accumulators of the split's tiles below kTB; dB^T (phase 1) / dA
  // (phase 2) accumulators, 2 x RP columns, from kTB
  static constexpr int kTB = NT * RP > 128 ? 256 : 128;
  static constexpr int ND = (RP > 64 || kTB > 128) ? 1 : 2;  // down: dh D buffers of 128 columns
  static constexpr int kDB = RP > 64 ? 0 : (kTB > 128 ? 384 : 256);
  static constexpr int kTmem = (MODE != MODE_SHARED || RP > 64 || kTB > 128) ? 512 : 256;
  static_assert(kSmem <= 227 * 1024, "shared memory per CTA");
  static_assert(kPerSM == 1 || kPerSM * (kSmem + 3 * 1024) <= 228 * 1024, "resident CTAs per SM");
  static_assert(ND * kNcB + (kDB == 0 ? 0 : kDB) <= 512 && (kDB != 0 || ND * kNcB <= kTB), "TMEM: dh buffers");
};

template <int RP, int MODE>
__global__ void __launch_bounds__(kThreadsWS, RowsCfg<RP, MODE>::kPerSM) k_bwd_rows(const __grid_constant__ PlanTables pt,
                                                            const __grid_constant__ BwdLaunch a) {
  using C = RowsCfg<RP, MODE>;
  using SL = Slots<RP>;
  constexpr int NT = C::NT, SA = C::SA, SB = C::SB > 0 ? C::SB : 1;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t fullA[SA], emptyA[SA], fullB[SB], emptyB[SB];
  __shared__ __align__(8) uint64_t dbt_full[2], dbt_empty[2], d_full[2], d_empty[2], da_full[2], da_empty[2];
  __shared__ __align__(8) uint64_t dh_full, hs_ready, ops_ready;
  __shared__ uint32_t tslot;
  __shared__ int32_t tok_s[MODE == MODE_SHARED ? NT * kTileM : 1];  // token of each row (gate/up)
  static_assert(NT * RP <= C::kTB, "dH accumulators must fit below the dB^T columns");

  pdl_wait();
  const int n_splits = a.counts[MODE == MODE_SHARED ? kCntSplitsSh : kCntSplitsRow];
  if ((int)blockIdx.x >= n_splits) return;
  const int proj = blockIdx.y;
  const Tile sp = (MODE == MODE_SHARED ? a.splits_sh : a.splits_row)[blockIdx.x];
  if (kChecks && !chk_tile(sp, pt.G, RowsCfg<RP, MODE>::NT * kTileM, a.counts[kCntRows], a.err)) return;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int g = sp.g, r0 = pt.rank_off[g], rg = pt.rank_off[g + 1] - r0;
  const int ntiles = (sp.cnt + kTileM - 1) / kTileM;
  const int d_in = a.d_in, d_out = a.d_out;
  const int nch1 = MODE == MODE_COMB ? 0 : (d_out + kNcB - 1) / kNcB;
  const int nch2 = MODE != MODE_SHARED ? (d_in + kNcB - 1) / kNcB : 0;
  const int NI1 = nch1 * ntiles, NI2 = nch2 * ntiles;
  // Each split walks the column chunks starting at its own offset, so the
  // splits of one group that run at the same time flush their weight
  // gradients into different columns (fewer same-address atomics in L2).
  auto chunk_col = [&](int c, int nch) { return ((c + sp.id) % nch) * kNcB; };
  const uint32_t sOps = smem_u32(smem);
  const uint32_t sA0 = sOps + C::kOps;
  const uint32_t sB0 = sA0 + SA * C::kSlotA;

  if (tid == 0) {
    for (int i = 0; i < SA; ++i) {
      mbar_init(&fullA[i], 1);
      mbar_init(&emptyA[i], 1);
    }
    for (int i = 0; i < SB; ++i) {
      mbar_init(&fullB[i], 1);
      mbar_init(&emptyB[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&dbt_full[i], 1);
      mbar_init(&dbt_empty[i], 1);
      mbar_init(&d_full[i], 1);
      mbar_init(&d_empty[i], 1);
      mbar_init(&da_full[i], 1);
      mbar_init(&da_empty[i], 1);
    }
    mbar_init(&dh_full, 1);
    mbar_init(&hs_ready, 1);
    mbar_init(&ops_ready, 8);  // the epilogue warps, once the H operand is staged
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, C::kTmem);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tslot;
  bool bad = false;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    // the dY stream starts once the epilogue has sent out its H prefetches,
    // and runs two slots ahead until the H operand is staged, so the H loads
    // are not queued behind a full ring of dY
    named_bar(kIssueBar, kEpiThreads + 32);
    if (lane == 0) {
      for (int q = 0; q < NI1 + NI2 && !bad; ++q) {
        if (q == 2 && !mbar_wait(&ops_ready, 0)) {
          bad = true;
          break;
        }
        const int s = q % SA, u = q / SA;
        if (u >= 1 && !mbar_wait(&emptyA[s], (u - 1) & 1)) {
          bad = true;
          break;
        }
        const uint32_t base = sA0 + s * C::kSlotA;
        if (q < NI1) {
          const int c = q / ntiles, i = q % ntiles, n0 = chunk_col(c, nch1), row0 = sp.start + i * kTileM;
          mbar_arrive_expect_tx(&fullA[s], 2 * kBlk + 2 * C::kWBlk);
          tma_load_2d(base, &a.tm_dy[proj], n0, row0, &fullA[s]);
          tma_load_2d(base + kBlk, &a.tm_dy[proj], n0 + 64, row0, &fullA[s]);
          tma_load_2d(base + 2 * kBlk, &a.tm_bt[proj], n0, r0, &fullA[s]);
          tma_load_2d(base + 2 * kBlk + C::kWBlk, &a.tm_bt[proj], n0 + 64, r0, &fullA[s]);
        } else {
          const int j = q - NI1, c = j / ntiles, i = j % ntiles, n0 = chunk_col(c, nch2), row0 = sp.start + i * kTileM;
          mbar_arrive_expect_tx(&fullA[s], 2 * C::kWBlk + 2 * kBlk);
          tma_load_2d(base, &a.tm_a, n0, r0, &fullA[s]);
          tma_load_2d(base + C::kWBlk, &a.tm_a, n0 + 64, r0, &fullA[s]);
          tma_load_2d(base + 2 * C::kWBlk, &a.tm_h, n0, row0, &fullA[s]);
          tma_load_2d(base + 2 * C::kWBlk + kBlk, &a.tm_h, n0 + 64, row0, &fullA[s]);
          const int sb = j % SB, ub = j / SB;
          if (ub >= 1 && !mbar_wait(&emptyB[sb], (ub - 1) & 1)) {
            bad = true;
            break;
          }
          const uint32_t bb = sB0 + sb * C::kSlotB;
          mbar_arrive_expect_tx(&fullB[sb], 2 * kBlk);
          tma_load_2d(bb, &a.tm_dh, n0, row0, &fullB[sb]);
          tma_load_2d(bb + kBlk, &a.tm_dh, n0 + 64, row0, &fullB[sb]);
        }
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t id_dh = idesc_bf16_f32(128, RP, 0, 0);
      constexpr uint32_t id_w = idesc_bf16_f32(128, RP, 1, 1);
      if (!mbar_wait(&ops_ready, 0)) bad = true;
      for (int q = 0; q < NI1 && !bad; ++q) {
        const int c = q / ntiles, i = q % ntiles, s = q % SA, u = q / SA;
        if (!mbar_wait(&fullA[s], u & 1)) {
          bad = true;
          break;
        }
        if (i == 0 && c >= 2 && !mbar_wait(&dbt_empty[c & 1], ((c - 2) >> 1) & 1)) {
          bad = true;
          break;
        }
        tc_fence_after();
        const uint32_t base = sA0 + s * C::kSlotA;
#pragma unroll
        for (int kk = 0; kk < kNcB / 16; ++kk)  // dH_i += dY_i . B_g
          tc_mma_bf16(tmem + i * RP, sdesc_sw128(base + (kk >> 2) * kBlk + (kk & 3) * 32, 16, 1024),
                      sdesc_sw128(base + 2 * kBlk + (kk >> 2) * C::kWBlk + (kk & 3) * 32, 16, 1024), id_dh,
                      (c > 0 || kk > 0) ? 1u : 0u);
#pragma unroll
        for (int kk = 0; kk < kTileM / 16; ++kk)  // dBt_c^T += dY_i^T . H_i
          tc_mma_bf16(tmem + C::kTB + (c & 1) * RP, sdesc_sw128(base + kk * 2048, kBlk, 1024),
                      SL::desc_mn(sOps, i, kk), id_w, (i > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&emptyA[s]);
        if (i == ntiles - 1) tc_commit(&dbt_full[c & 1]);
      }
      if (!bad) tc_commit(&dh_full);
      if (MODE != MODE_SHARED && !bad) {
        constexpr uint32_t id_d = idesc_bf16_f32(128, kNcB, 0, 1);
        if (!mbar_wait(&hs_ready, 0)) bad = true;
        for (int j = 0; j < NI2 && !bad; ++j) {
          const int q = NI1 + j, c = j / ntiles, i = j % ntiles, s = q % SA, u = q / SA;
          const int b = j % C::ND;
          if (!mbar_wait(&fullA[s], u & 1)) {
            bad = true;
            break;
          }
          if (j >= C::ND && !mbar_wait(&d_empty[b], ((j - C::ND) / C::ND) & 1)) {
            bad = true;
            break;
          }
          if (i == 0 && c >= 2 && !mbar_wait(&da_empty[c & 1], ((c - 2) >> 1) & 1)) {
            bad = true;
            break;
          }
          tc_fence_after();
          const uint32_t base = sA0 + s * C::kSlotA;
#pragma unroll
          for (int kk = 0; kk < RP / 16; ++kk)  // dh chunk = dH_i . A_g chunk
            tc_mma_bf16(tmem + C::kDB + b * kNcB, SL::desc_k(sOps, i, kk),
                        sdesc_sw128(base + kk * 2048, C::kWBlk, 1024), id_d, kk > 0 ? 1u : 0u);
#pragma unroll
          for (int kk = 0; kk < kTileM / 16; ++kk)  // dA_c^T += h_i^T . dH_i
            tc_mma_bf16(tmem + C::kTB + (c & 1) * RP, sdesc_sw128(base + 2 * C::kWBlk + kk * 2048, kBlk, 1024),
                        SL::desc_mn(sOps, i, kk), id_w, (i > 0 || kk > 0) ? 1u : 0u);
          tc_commit(&emptyA[s]);
          tc_commit(&d_full[b]);
          if (i == ntiles - 1) tc_commit(&da_full[c & 1]);
        }
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int et = tid - 64;
    const int quarter = warp & 3;
    const int ehalf = (warp - 2) >> 2;  // which half of the columns this warp owns
    const int m = quarter * 32 + lane;
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    const int fmode = a.deterministic ? kPartial : kAtomic;
    // H operand slots: bf16 of the saved H of each row, staged while the
    // producer already streams the first dY tiles.  The rows' lines are
    // prefetched into L2 first, ahead of the stream.  MODE_COMB stages
    // dH_row = s p_row dHc_u instead (H[0] = dHc per unique pair, H[1] = the
    // forward's H per row) and writes dp_row = s dHc_u . H_row.
    {
      for (int idx = et; idx < sp.cnt; idx += kEpiThreads) {
        const int hrow =
            MODE != MODE_DOWN ? ACE_CHK(a.row_uniq[sp.start + idx], 0, a.counts[kCntU], 0, a.err) : sp.start + idx;
        const float* hp = a.H[proj] + (int64_t)hrow * pt.rank_max;
        for (int c = 0; c < RP && c < pt.rank_max; c += 32) prefetch_l2(hp + c);
        if (MODE == MODE_COMB) {
          const float* hs = a.H[1] + (int64_t)(sp.start + idx) * pt.rank_max;
          for (int c = 0; c < RP && c < pt.rank_max; c += 32) prefetch_l2(hs + c);
        }
      }
      named_bar_arrive(kIssueBar, kEpiThreads + 32);
      const bool vec = (pt.rank_max & 3) == 0, vec2 = (pt.rank_max & 1) == 0;
      // v[0..32) = src[c0 .. c0 + 32), zero past rank_max or for a dead row;
      // 16- or 8-byte loads where the row stride rank_max keeps them aligned
      auto load32 = [&](const float* src, int c0, bool live, float* v) {
        if (vec2 && !vec) {
#pragma unroll
          for (int q = 0; q < 16; ++q) {
            const int c = c0 + 2 * q;
            const float2 x = (live && c < pt.rank_max) ? *reinterpret_cast<const float2*>(src + c) : make_float2(0.f, 0.f);
            v[2 * q] = x.x;
            v[2 * q + 1] = x.y;
          }
        } else if (vec) {
#pragma unroll
          for (int q = 0; q < 8; ++q) {
            const int c = c0 + 4 * q;
            const float4 x = (live && c < pt.rank_max) ? *reinterpret_cast<const float4*>(src + c)
                                                       : make_float4(0.f, 0.f, 0.f, 0.f);
            v[4 * q] = x.x;
            v[4 * q + 1] = x.y;
            v[4 * q + 2] = x.z;
            v[4 * q + 3] = x.w;
          }
        } else {
#pragma unroll
          for (int q = 0; q < 32; ++q) v[q] = (live && c0 + q < pt.rank_max) ? src[c0 + q] : 0.f;
        }
      };
      for (int idx = et; idx < ntiles * kTileM; idx += kEpiThreads) {
        const int i = idx / kTileM, mm = idx % kTileM;
        const int row = sp.start + idx;
        const int hrow =
            idx >= sp.cnt ? -1 : (MODE != MODE_DOWN ? ACE_CHK(a.row_uniq[row], 0, a.counts[kCntU], 0, a.err) : row);
        const float* hp = a.H[proj] + (int64_t)(hrow < 0 ? 0 : hrow) * pt.rank_max;
        if (MODE == MODE_SHARED) tok_s[idx] = hrow < 0 ? -1 : ACE_CHK(a.uniq_tok[hrow], 0, a.T, 0, a.err);
        const int pair =
            (MODE == MODE_COMB && hrow >= 0) ? ACE_CHK(a.row_pair[row], 0, a.counts[kCntRows], 0, a.err) : 0;
        const float wscale = (MODE == MODE_COMB && hrow >= 0) ? a.s * a.w[pair] : 0.f;
        float dp = 0.f;
#pragma unroll
        for (int c0 = 0; c0 < RP; c0 += 32) {
          float v[32];
          load32(hp, c0, hrow >= 0, v);
#pragma unroll
          for (int q = 0; q < 32; ++q)
            if (c0 + q >= rg) v[q] = 0.f;
          if (MODE == MODE_COMB) {
            float hs[32];
            load32(a.H[1] + (int64_t)(hrow >= 0 ? row : 0) * pt.rank_max, c0, hrow >= 0, hs);
#pragma unroll
            for (int q = 0; q < 32; ++q) {
              dp += v[q] * hs[q];
              v[q] *= wscale;
            }
          }
#pragma unroll
          for (int c8 = 0; c8 < 4; ++c8)
            if (c0 + 8 * c8 < RP) sts128(sOps + SL::elem(i, mm, c0 + 8 * c8), pack8(v + 8 * c8));
        }
        if (MODE == MODE_COMB && hrow >= 0) a.dw[pair] = a.s * dp;
      }
      fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(&ops_ready);
    }
    bool ok = true;
    for (int c = 0; c < nch1 && ok; ++c) {
      ok = named_bar_and(kEpiBar, kEpiThreads, mbar_wait(&dbt_full[c & 1], (c >> 1) & 1));
      if (!ok) break;
      tc_fence_after();
      flush_wgrad<RP>(tmem + lane_base + C::kTB + (c & 1) * RP, chunk_col(c, nch1), d_out, rg, r0, a.s, fmode,
                      a.part_dBt[proj], sp.id, a.dBt[proj], m, false, ehalf * 16, 32);
      tc_fence_before();
      named_bar(kEpiBar, kEpiThreads);
      if (et == 0) mbar_arrive(&dbt_empty[c & 1]);
    }
    if (ok) ok = named_bar_and(kEpiBar, kEpiThreads, mbar_wait(&dh_full, 0));
    if (ok) {
      tc_fence_after();
      // dH (scaled by s): gate/up -> fp32 per row; down -> bf16 operand slots
      // (the combine staged its dH with the operand slots above)
      for (int i = 0; i < (MODE == MODE_COMB ? 0 : ntiles); ++i) {
        const bool live = i * kTileM + m < sp.cnt;
        const int64_t row = sp.start + i * kTileM + m;
#pragma unroll
        for (int c0 = ehalf * 16; c0 < RP; c0 += 32) {
          uint32_t r[16];
          tmem_ld16(tmem + lane_base + i * RP + c0, r);
          tmem_ld_wait();
          float v[16];
#pragma unroll
          // columns >= r_g come from the next group's rank rows of the B^T box: zero them
          for (int q = 0; q < 16; ++q) v[q] = (live && c0 + q < rg) ? a.s * __uint_as_float(r[q]) : 0.f;
          if (MODE == MODE_SHARED) {
            if (live && a.deterministic) {
              float4* dst = reinterpret_cast<float4*>(a.dHrow[proj] + row * RP + c0);
#pragma unroll
              for (int q = 0; q < 4; ++q) dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
            } else if (live) {
              // dHx[t][proj * n_rank_pad + r0 + k] += dH_row[k], k < r_g, by
              // 16-byte vector reductions over the aligned 8-column windows
              uint16_t* row_dst = a.dHx + (int64_t)tok_s[i * kTileM + m] * (a.nproj * a.n_rank_pad) +
                                  proj * a.n_rank_pad;
              const int col0 = r0 + c0, o = col0 & 7;
              uint16_t* win0 = row_dst + (col0 - o);
              switch (o) {
                case 0: red_windows<0>(win0, v, rg - c0); break;
                case 1: red_windows<1>(win0, v, rg - c0); break;
                case 2: red_windows<2>(win0, v, rg - c0); break;
                case 3: red_windows<3>(win0, v, rg - c0); break;
                case 4: red_windows<4>(win0, v, rg - c0); break;
                case 5: red_windows<5>(win0, v, rg - c0); break;
                case 6: red_windows<6>(win0, v, rg - c0); break;
                default: red_windows<7>(win0, v, rg - c0); break;
              }
            }
          } else {
            sts128(sOps + SL::elem(i, m, c0), pack8(v));
            sts128(sOps + SL::elem(i, m, c0 + 8), pack8(v + 8));
          }
        }
      }
      fence_proxy_async_smem();
      tc_fence_before();
      named_bar(kEpiBar, kEpiThreads);
      if (et == 0) mbar_arrive(&hs_ready);
    }
    if (MODE != MODE_SHARED) {
      for (int j = 0; j < NI2 && ok; ++j) {
        const int c = j / ntiles, i = j % ntiles, b = j % C::ND, sb = j % SB, n0 = chunk_col(c, nch2);
        bool w_ok = mbar_wait(&fullB[sb], (j / SB) & 1);
        w_ok = w_ok && mbar_wait(&d_full[b], (j / C::ND) & 1);
        ok = named_bar_and(kEpiBar, kEpiThreads, w_ok);
        if (!ok) break;
        tc_fence_after();
        const uint32_t bb = sB0 + sb * C::kSlotB;
#pragma unroll
        for (int hh = 0; hh < 2; ++hh) {
          const int h = ehalf * 2 + hh;
          uint32_t r[32];
          const uint32_t ta = tmem + lane_base + C::kDB + b * kNcB + h * 32;
          tmem_ld16(ta, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
          tmem_ld16(ta + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
          tmem_ld_wait();
#pragma unroll
          for (int q = 0; q < 4; ++q) {
            const uint32_t addr = bb + tile_off(kTileM, m, h * 4 + q);
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
        tc_fence_before();
        named_bar(kEpiBar, kEpiThreads);
        if (et == 0) mbar_arrive(&d_empty[b]);
        const int cnt_i = sp.cnt - i * kTileM;
#pragma unroll 4
        for (int it = et; it < kTileM * 16; it += kEpiThreads) {
          const int row = it >> 4, ch = it & 15, col = n0 + ch * 8;
          if (row < cnt_i && col < d_in) {
            const uint4 v = lds128(bb + tile_off(kTileM, row, ch));
            *reinterpret_cast<uint4*>(a.dXin + (int64_t)(sp.start + i * kTileM + row) * d_in + col) = v;
          }
        }
        fence_proxy_async_smem();
        named_bar(kEpiBar, kEpiThreads);
        if (et == 0) mbar_arrive(&emptyB[sb]);
        if (i == ntiles - 1) {  // dA chunk c of this split is complete
          ok = named_bar_and(kEpiBar, kEpiThreads, mbar_wait(&da_full[c & 1], (c >> 1) & 1));
          if (!ok) break;
          tc_fence_after();
          flush_wgrad<RP>(tmem + lane_base + C::kTB + (c & 1) * RP, n0, d_in, rg, r0, 1.f, fmode, a.part_dA[proj],
                          sp.id, a.dA[proj], m, false, ehalf * 16, 32);
          tc_fence_before();
          named_bar(kEpiBar, kEpiThreads);
          if (et == 0) mbar_arrive(&da_empty[c & 1]);
        }
      }
    }
    if (!ok) bad = true;
  }
  __syncwarp();
  tc_fence_before();
  if (__syncthreads_or(bad) && tid == 0) atomicOr(a.err, kErrTimeout);
  // signal dependents only as this CTA finishes: an earlier launch of the
  // next kernel (a whole SM per CTA) measured slower
  pdl_trigger();
  if (warp == 0) tmem_dealloc(tmem, C::kTmem);
}

// ---------------------------------------------------------------- dH_u
// dH_u = sum of the dH rows of unique pair u (fixed slot order), written into
// the token-major dense matrix dHx[t][j * n_rank_pad + rank_off[g] + k].  One
// thread per (unique pair, 8 columns): the RP / 8 threads of a pair read its
// rows' 32-byte pieces side by side, and many pairs' loads are in flight.
template <int RP>
__global__ void __launch_bounds__(128) k_dh_reduce(const __grid_constant__ PlanTables pt,
                                                   const __grid_constant__ BwdLaunch a) {
  constexpr int CH = RP / 8;  // threads per unique pair
  pdl_wait();
  pdl_trigger();
  const int n_tiles = a.counts[kCntTilesSh];
  const int tile = blockIdx.x / CH;
  if (tile >= n_tiles) return;
  const int proj = blockIdx.y;
  const Tile tl = a.tiles_sh[tile];
  if (kChecks && !chk_tile(tl, pt.G, kTileM, a.counts[kCntU], a.err)) return;
  const int m = (blockIdx.x % CH) * (128 / CH) + threadIdx.x / CH, q = threadIdx.x % CH;
  if (m >= tl.cnt) return;
  const int u = tl.start + m, t = ACE_CHK(a.uniq_tok[u], 0, a.T, 0, a.err), k = pt.k, g = tl.g;
  const int r0 = pt.rank_off[g], rg = pt.rank_off[g + 1] - r0;
  int rows[kMaxK];
  int n = 0;
  for (int j = 0; j < k; ++j)
    if (a.pair_g[(int64_t)t * k + j] == g)
      rows[n++] = ACE_CHK(a.pair_row[(int64_t)t * k + j], 0, a.counts[kCntRows], 0, a.err);
  float acc[8];
#pragma unroll
  for (int c = 0; c < 8; ++c) acc[c] = 0.f;
  for (int i = 0; i < n; ++i) {
    const float4* src = reinterpret_cast<const float4*>(a.dHrow[proj] + (int64_t)rows[i] * RP + q * 8);
    const float4 v0 = src[0], v1 = src[1];
    acc[0] += v0.x;
    acc[1] += v0.y;
    acc[2] += v0.z;
    acc[3] += v0.w;
    acc[4] += v1.x;
    acc[5] += v1.y;
    acc[6] += v1.z;
    acc[7] += v1.w;
  }
  if (q * 8 >= rg) return;
  const int kw = a.nproj * a.n_rank_pad;
  uint16_t* dst = a.dHx + (int64_t)t * kw + proj * a.n_rank_pad + r0 + q * 8;
  if ((r0 & 7) == 0 && q * 8 + 8 <= rg) {
    *reinterpret_cast<uint4*>(dst) = pack8(acc);
  } else {
#pragma unroll
    for (int c = 0; c < 8; ++c)
      if (q * 8 + c < rg) {
        const __nv_bfloat16 h = __float2bfloat16_rn(acc[c]);
        dst[c] = *reinterpret_cast<const uint16_t*>(&h);
      }
  }
}

// ---------------------------------------------------------------- stage 2
__global__ void __launch_bounds__(256) k_splitk_reduce(const __grid_constant__ PlanTables pt,
                                                       const Tile* __restrict__ splits,
                                                       const int32_t* __restrict__ counts, int slot,
                                                       const float* __restrict__ part, int RP, int width,
                                                       float* __restrict__ out) {
  pdl_wait();
  pdl_trigger();
  const int i = blockIdx.x;  // global rank row
  int g = 0;
  while (pt.rank_off[g + 1] <= i) ++g;
  const int kk = i - pt.rank_off[g];
  const int n = counts[slot];
  // the split table lists the splits group by group (ascending g): find the
  // range of group g in one pass of the block over the table
  __shared__ int s_lo, s_hi;
  if (threadIdx.x == 0) s_lo = s_hi = 0;
  __syncthreads();
  for (int t = threadIdx.x; t < n; t += blockDim.x)
    if (splits[t].g == g) {
      if (t == 0 || splits[t - 1].g != g) s_lo = t;
      if (t == n - 1 || splits[t + 1].g != g) s_hi = t + 1;
    }
  __syncthreads();
  const int lo = s_lo, hi = s_hi;
  const int c = (blockIdx.y * 256 + threadIdx.x) * 4;
  if (c >= width) return;
  const float* base = part + (int64_t)kk * width + c;
  const int64_t stride = (int64_t)RP * width;  // one split's partial
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  // in split order, four partials in flight at a time
  int sidx = lo;
  for (; sidx + 4 <= hi; sidx += 4) {
    float4 v[4];
#pragma unroll
    for (int q = 0; q < 4; ++q) v[q] = *reinterpret_cast<const float4*>(base + (int64_t)splits[sidx + q].id * stride);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      acc.x += v[q].x;
      acc.y += v[q].y;
      acc.z += v[q].z;
      acc.w += v[q].w;
    }
  }
  for (; sidx < hi; ++sidx) {
    const float4 v = *reinterpret_cast<const float4*>(base + (int64_t)splits[sidx].id * stride);
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

template <int RP, int MODE>
cudaError_t launch_rows(const PlanTables& pt, const BwdLaunch& a, int nproj, cudaStream_t st) {
  using C = RowsCfg<RP, MODE>;
  auto kern = k_bwd_rows<RP, MODE>;
  cudaError_t e = set_smem(kern, C::kSmem);
  if (e != cudaSuccess) return e;
  const int grid = MODE == MODE_SHARED ? a.max_splits_sh : a.max_splits_row;
  return launch_k(kern, dim3(grid, nproj), kThreadsWS, C::kSmem, st, pt, a);
}

// Combine backward: one launch zeroes dB^T (the dense dA GEMM of gemm.cu
// adds its tiles into it afterwards) and, in the fast mode, dA; then the row
// kernel and, in the deterministic mode, stage 2 of dA.
template <int RP>
cudaError_t launch_comb_t(const PlanTables& pt, const BwdLaunch& a, cudaStream_t st) {
  const int n_rank = pt.rank_off[pt.G];
  void* zp[kZeroMax] = {};
  size_t zb[kZeroMax] = {};
  int nz = 0;
  zp[nz] = a.dBt[0], zb[nz++] = sizeof(float) * (size_t)n_rank * a.d_out;
  if (!a.deterministic) zp[nz] = a.dA[0], zb[nz++] = sizeof(float) * (size_t)n_rank * a.d_in;
  cudaError_t e = launch_zero(zp, zb, nz, st);
  if (e != cudaSuccess) return e;
  if ((e = launch_rows<RP, MODE_COMB>(pt, a, 1, st)) != cudaSuccess) return e;
  if (!a.deterministic) return cudaSuccess;
  dim3 grid(n_rank, (a.d_in / 4 + 255) / 256);
  return launch_k(k_splitk_reduce, grid, 256, 0, st, pt, a.splits_row, a.counts, kCntSplitsRow, a.part_dA[0], (int)RP,
                  a.d_in, a.dA[0]);
}

template <int RP>
cudaError_t launch_bwd_t(const PlanTables& pt, const BwdLaunch& a, bool shared, cudaStream_t st) {
  if (a.comb) return launch_comb_t<RP>(pt, a, st);
  cudaError_t e;
  const int n_rank = pt.rank_off[pt.G];
  const int nproj = shared ? a.nproj : 1;
  // one launch zeroes every accumulation target of the call: the fast-mode
  // atomic dB^T (and down dA), and for gate/up the dense dH and the dA that
  // the dense GEMM adds its tiles into
  void* zp[kZeroMax] = {};
  size_t zb[kZeroMax] = {};
  int nz = 0;
  if (!a.deterministic)
    for (int j = 0; j < nproj; ++j) zp[nz] = a.dBt[j], zb[nz++] = sizeof(float) * (size_t)n_rank * a.d_out;
  if (!shared && !a.deterministic) zp[nz] = a.dA[0], zb[nz++] = sizeof(float) * (size_t)n_rank * a.d_in;
  if (shared) {
    zp[nz] = a.dHx, zb[nz++] = sizeof(uint16_t) * (size_t)a.T * nproj * a.n_rank_pad;
    for (int j = 0; j < nproj; ++j) zp[nz] = a.dA[j], zb[nz++] = sizeof(float) * (size_t)n_rank * a.d_in;
  }
  if ((e = launch_zero(zp, zb, nz, st)) != cudaSuccess) return e;
  if (!shared) {
    if ((e = launch_rows<RP, MODE_DOWN>(pt, a, 1, st)) != cudaSuccess) return e;
  } else {
    if ((e = launch_rows<RP, MODE_SHARED>(pt, a, nproj, st)) != cudaSuccess) return e;
    if (a.deterministic &&
        (e = launch_k(k_dh_reduce<RP>, dim3(a.max_tiles_sh * (RP / 8), nproj), 128, 0, st, pt, a)) != cudaSuccess)
      return e;
  }
  if (a.deterministic) {
    const Tile* splits = shared ? a.splits_sh : a.splits_row;
    const int slot = shared ? kCntSplitsSh : kCntSplitsRow;
    for (int j = 0; j < nproj; ++j) {
      dim3 grid(n_rank, (a.d_out / 4 + 255) / 256);
      if ((e = launch_k(k_splitk_reduce, grid, 256, 0, st, pt, splits, a.counts, slot, a.part_dBt[j], (int)RP,
                        a.d_out, a.dBt[j])) != cudaSuccess)
        return e;
    }
    if (!shared) {
      dim3 grid(n_rank, (a.d_in / 4 + 255) / 256);
      if ((e = launch_k(k_splitk_reduce, grid, 256, 0, st, pt, a.splits_row, a.counts, kCntSplitsRow, a.part_dA[0],
                        (int)RP, a.d_in, a.dA[0])) != cudaSuccess)
        return e;
    }
  }
  return cudaSuccess;
}

}  // namespace

cudaError_t launch_bwd(const PlanTables& pt, const BwdLaunch& a, bool shared, cudaStream_t st) {
  if (a.T == 0) {
    // no routed rows: every weight gradient is zero
    const int n_rank = pt.rank_off[pt.G];
    const int nproj = shared ? a.nproj : 1;
    for (int j = 0; j < nproj; ++j) {
      cudaError_t e = cudaMemsetAsync(a.dA[j], 0, sizeof(float) * (size_t)n_rank * a.d_in, st);
      if (e == cudaSuccess) e = cudaMemsetAsync(a.dBt[j], 0, sizeof(float) * (size_t)n_rank * a.d_out, st);
      if (e != cudaSuccess) return e;
    }
    return cudaSuccess;
  }
  switch (pt.rank_pad) {
    case 16: return launch_bwd_t<16>(pt, a, shared, st);
    case 32: return launch_bwd_t<32>(pt, a, shared, st);
    case 64: return launch_bwd_t<64>(pt, a, shared, st);
    case 128: return launch_bwd_t<128>(pt, a, shared, st);
  }
  return cudaErrorInvalidValue;
}

}  // namespace ace
