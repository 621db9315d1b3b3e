// Fused LoRA forward (Sec. 3.3-3.5; App. "Implementation and Profiling of
// Grouped Adapter Execution").
//
// k_fwd_h (gate/up, when the token-major k_gemm_h of gemm.cu does not
//   apply): per tile of up to 128 unique (g, t) pairs of one group,
//   H_u = A_g x_t is computed ONCE per active group of a token (Sec. 3.5):
//   X rows gathered by token with cp.async into 128-byte-swizzled smem,
//   tcgen05 MMA with N = nproj * rank_pad (gate and up share the gather),
//   fp32 H written per unique pair.  With `rows` set the same kernel takes
//   the forward row tiles instead (each split tile once) and computes
//   H_row = A_g h_row for contiguous rows of h: the first step of the
//   gate-weighted combine of down.
// k_fwd_rows: persistent, one CTA per SM; tiles of <= 128 consecutive rows
//   of one group (expert segments are contiguous inside group segments) are
//   taken dynamically from a counter; the last wave's tiles come in column
//   parts (down: their H computed up front, one tile per CTA), so the SMs
//   finish together.  Warp-specialised:
//     warp 0     TMA producer: row tiles of Y (and of h for down) and chunks of
//                B_g^T / A_g into a ring of shared-memory slots
//     warp 1     MMA issuer: (down) H = h . A_g^T over the K loop, then per
//                64-column chunk D = H . B_g^T into one of four TMEM buffers
//     warps 2-17 epilogue, four groups of four (one warp per TMEM lane
//                quarter): H -> bf16 operand (down: from TMEM; gate/up:
//                gathered from the unique pair of each row), then group p
//                takes the chunks cc with cc % 4 == p: Y += s * D on its own
//                32 rows in swizzled smem (TMEM lane = row) and stores them.
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

  pdl_wait();
  Tile tl;
  if (a.rows) {
    // row tiles: whole tiles first, then kSplitParts entries per split tile
    const int n_items = a.counts[kCntTilesRow], split0 = a.counts[kCntRowSplit];
    const int b = blockIdx.x;
    if (b >= split0 + (n_items - split0) / kSplitParts) return;
    tl = a.tiles[b < split0 ? b : split0 + (b - split0) * kSplitParts];
  } else {
    if ((int)blockIdx.x >= a.counts[kCntTilesSh]) return;
    tl = a.tiles[blockIdx.x];
  }
  if (kChecks && !chk_tile(tl, pt.G, kTileM, a.counts[a.rows ? kCntRows : kCntU], a.err)) return;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int quarter = warp & 3, half = warp >> 2;
  const int m = quarter * 32 + lane;
  const int g = tl.g, r0 = pt.rank_off[g], rg = pt.rank_off[g + 1] - r0;
  const int d_in = a.d_in;

  if (tid < kTileM)
    src_row[tid] = tid < tl.cnt ? (a.rows ? tl.start + tid : ACE_CHK(a.uniq_tok[tl.start + tid], 0, a.n_src, 0, a.err))
                                : -1;
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
    // the tile goes through the (now idle) stage buffers: its rows are rows
    // [start, start + cnt) of H_j, one contiguous range of cnt * rank_max
    // floats, which the CTA then writes with consecutive threads on
    // consecutive addresses (a thread per row would write 32 rows per store)
    constexpr int kHcols = NPROJ * RP, kLd = kHcols + 4;  // smem row stride in floats (bank-conflict free)
    static_assert(kTileM * kLd * 4 <= kHStages * C::kStage, "H tile fits the stage buffers");
    float* sH = reinterpret_cast<float*>(smem);
    for (int c0 = half * 16; c0 < kHcols; c0 += 32) {
      uint32_t r[16];
      tmem_ld16(tmem + lane_base + c0, r);
      tmem_ld_wait();
      float4* dst = reinterpret_cast<float4*>(sH + m * kLd + c0);
#pragma unroll
      for (int q = 0; q < 4; ++q)
        dst[q] = make_float4(__uint_as_float(r[4 * q]), __uint_as_float(r[4 * q + 1]), __uint_as_float(r[4 * q + 2]),
                             __uint_as_float(r[4 * q + 3]));
    }
    __syncthreads();
    const int W = pt.rank_max, n = tl.cnt * W;
#pragma unroll
    for (int j = 0; j < NPROJ; ++j) {
      float* dst = a.H[j] + (int64_t)tl.start * W;
      if ((W & 3) == 0) {
        for (int e = 4 * tid; e < n; e += 4 * kHThreads) {
          const int row = e / W, col = e - row * W;
          *reinterpret_cast<float4*>(dst + e) = *reinterpret_cast<const float4*>(sH + row * kLd + j * RP + col);
        }
      } else {
        for (int e = tid; e < n; e += kHThreads) {
          const int row = e / W, col = e - row * W;
          dst[e] = sH[row * kLd + j * RP + col];
        }
      }
    }
  }
  if (aborted && tid == 0) atomicOr(a.err, kErrTimeout);
  tc_fence_before();
  __syncthreads();
  // the row kernel that follows takes a whole SM per CTA: let it launch only
  // as this grid's CTAs finish (an early launch measured slower)
  pdl_trigger();
  if (warp == 0) tmem_dealloc(tmem, C::kTmem);
}

// Columns [c0, c0 + 16) of an fp32 H row of rank_max columns (those below
// rank_max): 16-byte stores where the row stride keeps them aligned.
__device__ __forceinline__ void store_row16(float* hrow, int c0, int rank_max, const float* v) {
  if ((rank_max & 3) == 0 && c0 + 16 <= rank_max) {
#pragma unroll
    for (int q = 0; q < 4; ++q)
      *reinterpret_cast<float4*>(hrow + c0 + 4 * q) = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
  } else {
#pragma unroll
    for (int q = 0; q < 16; ++q)
      if (c0 + q < rank_max) hrow[c0 + q] = v[q];
  }
}

// --------------------------------------------------------------- k_fwd_rows
constexpr int kNGrp = 4;                        // epilogue groups (4 warps each, one per TMEM lane quarter)
constexpr int kRowsThreads = 64 + 128 * kNGrp;  // producer warp, MMA warp, epilogue warps
constexpr int kRowsTmem = 512;
constexpr int kChunk = 64;         // output columns per D chunk
constexpr int kQuant = 16;         // rows per small TMA box (short tiles)
constexpr int kQ = 4;              // depth of the tile queue

template <int RP, int NPROJ, bool SHARED>
struct RowsFwdCfg {
  static constexpr int kWBlk = RP * 128;                    // [RP x 64] weight block
  static constexpr int kSlot = NPROJ * (kBlk + kWBlk);      // Y tiles + B^T blocks (down K-step: h + A)
  static constexpr int kHs = ((NPROJ * RP + 63) / 64) * kBlk;  // bf16 H operand of one tile
  static constexpr int kBudget = 210 * 1024;
  // H operand buffers: two wherever they fit beside three ring slots
  static constexpr int NBH = 2 * kHs + 3 * kSlot <= kBudget ? 2 : 1;
  static constexpr int kS0 = (kBudget - NBH * kHs) / kSlot;
  // ring slots: down keeps at most 6 (7 or 8 measured slower, 6 the fastest)
  static constexpr int kSmax = SHARED ? 8 : 6;
  static constexpr int S = kS0 > kSmax ? kSmax : (kS0 < 2 ? 2 : kS0);
  static constexpr int kSmem = NBH * kHs + S * kSlot + 1024;
  static constexpr int kHcol = RP <= 64 ? 64 : 128;         // down: TMEM columns of one H accumulator
  static constexpr uint32_t kDBase = SHARED ? 0u : 2u * kHcol;
  static_assert(kDBase + kNGrp * NPROJ * kChunk <= kRowsTmem, "TMEM budget");
};

// Rows [y, y + cnt) of a 64-column box at column x: one 128-row box for a
// whole tile, else ceil(cnt / 16) boxes of 16 rows (so a short tile reads at
// most 15 rows it does not use).
__device__ __forceinline__ void load_rows(uint32_t dst, const CUtensorMap* m128, const CUtensorMap* m16, int x, int y,
                                          int cnt, uint64_t* bar) {
  if (cnt == kTileM) {
    tma_load_2d(dst, m128, x, y, bar);
    return;
  }
  const int nb = (cnt + kQuant - 1) / kQuant;
  for (int b = 0; b < nb; ++b) tma_load_2d(dst + b * kQuant * 128, m16, x, y + b * kQuant, bar);
}
// Output chunks [lo, hi) of a row tile: id 0 names all columns; split b has
// ids 1 + P b + p for its column parts p < P = kSplitParts.  A kernel takes
// the parts of a split tile `merge` at a time (the entries of the other parts
// are skipped): gate/up merges 2 (a part then costs a gather of H per row; 4
// parts measured slower), down with an up-front H takes single parts, down
// without one takes the tile whole (cutting it would make every part repeat
// the tile's K loop).
__device__ __forceinline__ int split_part(const Tile& t) { return (t.id - 1) % kSplitParts; }
__device__ __forceinline__ int split_index(const Tile& t) { return (t.id - 1) / kSplitParts; }
__device__ __forceinline__ bool tile_live(const Tile& t, int merge) {
  return t.cnt > 0 && !(t.id > 0 && split_part(t) % merge != 0);
}
__device__ __forceinline__ int chunk_lo(const Tile& t, int nch, int merge) {
  return t.id > 0 && merge < kSplitParts ? split_part(t) * nch / kSplitParts : 0;
}
__device__ __forceinline__ int chunk_hi(const Tile& t, int nch, int merge) {
  return t.id > 0 && merge < kSplitParts ? (split_part(t) + merge) * nch / kSplitParts : nch;
}
// Up-front H of the split row tiles (down): ready once every epilogue warp of
// the CTA that computed it has added 1.
constexpr int kPreWriters = 4 * 4;
// the H-ready wait's bound under ACE_FLAG_TEST_WAIT_EXPIRY
constexpr uint64_t kTestWaitLimitNs = 2000000ull;
__device__ __forceinline__ uint32_t rows_bytes(int cnt) {
  return cnt == kTileM ? (uint32_t)kBlk : (uint32_t)((cnt + kQuant - 1) / kQuant) * kQuant * 128;
}

// Tile queue: the producer takes row tiles from a global counter (so faster
// SMs take more tiles), skips the ones this kernel does not run, and hands
// each live tile index to the MMA warp and the epilogue warps through a small
// ring in shared memory; -1 ends.  The consumers take an entry at the start
// of the tile before it, so a claim that finds the ring full waits only for
// them to reach the start of a tile whose loads are already issued: the wait
// always ends.
struct TileQueue {
  int32_t item[kQ];
  uint64_t full[kQ], empty[kQ];
};
// Consumer side: the next tile (false at the end or if a wait gave up; *ok
// tells which).  Every lane of a warp calls it; lane 0 releases the entry.
__device__ __forceinline__ bool queue_next(TileQueue& tq, int& q, const Tile* tiles, Tile& t, bool single_lane,
                                           bool* ok, int psplit, int& pj) {
  const int e = q % kQ;
  bool w = mbar_wait(&tq.full[e], (q / kQ) & 1);
  if (!single_lane) w = __all_sync(0xffffffffu, w);
  if (!w) {
    *ok = false;
    return false;
  }
  const int item = *reinterpret_cast<volatile int32_t*>(&tq.item[e]);
  if (!single_lane) __syncwarp();
  if (single_lane || (threadIdx.x & 31) == 0) mbar_arrive(&tq.empty[e]);
  ++q;
  if (item < 0) return false;
  t = tiles[item >> psplit];
  pj = item & psplit;
  return true;
}
// Persistent: one CTA per SM; tiles of <= 128 consecutive rows of one group
// are taken dynamically.  The producer, the MMA issuer and the epilogue run
// ahead of one another across tile boundaries: for down, the K loop of the
// next tile (H = h . A_g^T into the other of two TMEM accumulators) follows
// the D chunks of the current tile in the ring; for gate/up the next tile's
// H is gathered while the current one streams (the H operand is
// double-buffered in shared memory where it fits).  (Interleaving the next
// K loop into the chunk stream measured slower.)  Down with an up-front H
// starts with the K loop of its split tile (H to global memory, no chunks);
// the split tiles' parts later stage that H like gate/up stages H_u, so the
// H accumulators count only the tiles with a K loop (kc) and the H operand
// buffers only the tiles with chunks (ci).  The epilogue warps form kNGrp
// groups of four (one warp per TMEM lane quarter); group p owns the D chunks
// cc with cc % kNGrp == p, and each warp updates and stores only its own 32
// rows, so no barrier spans more than one warp: every hand-off is an mbarrier
// (a ring slot is released by the MMA commit after a K step, or by the four
// warps of the group after a chunk, each on its own barrier).
template <int RP, int NPROJ, bool SHARED>
__global__ void __launch_bounds__(kRowsThreads, 1) k_fwd_rows(const __grid_constant__ PlanTables pt,
                                                              const __grid_constant__ FwdRowsLaunch a) {
  using C = RowsFwdCfg<RP, NPROJ, SHARED>;
  constexpr int S = C::S, NBH = C::NBH;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t full[S], emptyK[S], emptyC[S], dfull[kNGrp], dempty[kNGrp];
  __shared__ __align__(8) uint64_t hacc[2], hs_ready[2], hs_free[2];
  __shared__ __align__(8) TileQueue tq;
  __shared__ uint32_t tslot;

  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  if (tid == 0) {
    for (int i = 0; i < S; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&emptyK[i], 1);  // MMA commit after a K step
      mbar_init(&emptyC[i], 4);  // the four warps of the group that owns the chunk
    }
    for (int i = 0; i < kNGrp; ++i) {
      mbar_init(&dfull[i], 1);
      mbar_init(&dempty[i], 4);
    }
    for (int i = 0; i < kQ; ++i) {
      mbar_init(&tq.full[i], 1);
      mbar_init(&tq.empty[i], 1 + 4 * kNGrp);  // MMA thread + every epilogue warp
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&hacc[i], 1);              // down: H of the tiles of this parity accumulated
      mbar_init(&hs_ready[i], 4 * kNGrp);  // H operand of the tiles of this parity staged (every epilogue warp)
      mbar_init(&hs_free[i], 1);           // D chunks reading H buffer i done (MMA commit)
    }
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, kRowsTmem);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tslot;
  pdl_wait();
  const int n_items = a.counts[kCntTilesRow];
  // down with an up-front H: CTA b first computes the H of split row tile b
  // (K loop only) into Hpre; the split tiles' column halves then read it
  // instead of repeating the K loop, so the last work comes in halves
  const bool pre = !SHARED && a.pre != 0;
  const int merge = SHARED ? 2 : (pre ? 1 : kSplitParts);  // parts of a split tile taken together
  // gate/up with the two projections as separate work items (one projection
  // per kernel instance, NPROJ == 1): 1, else 0
  const int psplit = (SHARED && NPROJ == 1 && a.proj_split) ? 1 : 0;
  const int split0 = a.counts[kCntRowSplit], n_split = (n_items - split0) / kSplitParts;
  bool has_pre = pre && (int)blockIdx.x < n_split;
  Tile pre_t{};
  if (has_pre) pre_t = a.tiles[split0 + kSplitParts * (int)blockIdx.x];
  if (kChecks && has_pre) has_pre = chk_tile(pre_t, pt.G, kTileM, a.counts[kCntRows], a.err);
  int32_t* const hflag = a.sched + 8;
  auto needs_k = [&](const Tile& t) { return !SHARED && !(pre && t.id > 0); };
  const int d_in = a.d_in, d_out = a.d_out;
  const int NK = SHARED ? 0 : (d_in + 63) / 64;  // K steps of the down H GEMM
  const int nch = (d_out + kChunk - 1) / kChunk;
  const uint32_t sHs0 = smem_u32(smem);
  const uint32_t slot0 = sHs0 + NBH * C::kHs;
  bool bad = false;

  if (warp == 0) {
    // ------------------------------------------------------------ producer
    if (lane == 0) {
      int last[S], nK[S], nC[S];  // per slot: kind of the last use (0 none, 1 K step, 2 chunk), use counts
#pragma unroll
      for (int k = 0; k < S; ++k) last[k] = nK[k] = nC[k] = 0;
      int i = 0, q = 0;
      // take the next tile (the counter runs over the entries this kernel
      // takes: every unsplit tile, then every merge-th part entry), or the
      // end; hand it on
      // with the projections split, counter value v names projection v & 1
      // of entry v >> 1, and the queue carries (entry << 1) | projection
      const int n_take = (split0 + (n_items - split0) / merge) << psplit;
      auto grab = [&](Tile& t, int& pj) -> bool {
        int item;
        while (true) {
          const int v = atomicAdd(a.sched + kSchedFwdRows, 1);
          if (v >= n_take) {
            item = -1;
            break;
          }
          const int vt = v >> psplit;
          item = vt < split0 ? vt : split0 + (vt - split0) * merge;
          t = a.tiles[item];
          pj = v & psplit;
          if (tile_live(t, merge) && (!kChecks || chk_tile(t, pt.G, kTileM, a.counts[kCntRows], a.err))) break;
        }
        const int e = q % kQ;
        if (q >= kQ && !mbar_wait(&tq.empty[e], ((q - kQ) / kQ) & 1)) {
          bad = true;
          return false;
        }
        tq.item[e] = item < 0 ? -1 : (item << psplit) | pj;
        mbar_arrive(&tq.full[e]);
        ++q;
        return item >= 0;
      };
      auto acquire = [&](bool kstep) -> uint32_t {  // next ring slot, once its last user released it
        const int s = i % S;
        if ((last[s] == 1 && !mbar_wait(&emptyK[s], (nK[s] - 1) & 1)) ||
            (last[s] == 2 && !mbar_wait(&emptyC[s], (nC[s] - 1) & 1)))
          bad = true;
        last[s] = kstep ? 1 : 2;
        if (kstep) ++nK[s]; else ++nC[s];
        return (uint32_t)s;
      };
      auto load_k = [&](const Tile& t, int k) {
        const uint32_t s = acquire(true);
        if (bad) return;
        const uint32_t base = slot0 + s * C::kSlot;
        mbar_arrive_expect_tx(&full[s], rows_bytes(t.cnt) + C::kWBlk);
        load_rows(base, &a.tm_x, &a.tm_x16, k * 64, t.start, t.cnt, &full[s]);
        tma_load_2d(base + NPROJ * kBlk, &a.tm_a, k * 64, pt.rank_off[t.g], &full[s]);
        ++i;
      };
      auto load_c = [&](const Tile& t, int pj, int c) {
        const uint32_t s = acquire(false);
        if (bad) return;
        const uint32_t base = slot0 + s * C::kSlot;
        const int n0 = c * kChunk;
        mbar_arrive_expect_tx(&full[s], NPROJ * (rows_bytes(t.cnt) + C::kWBlk));
#pragma unroll
        for (int j = 0; j < NPROJ; ++j) {
          const int jj = j + pj;  // the tensors' projection (pj = 0 unless the projections are split)
          load_rows(base + j * kBlk, &a.tm_y[jj], &a.tm_y16[jj], n0, t.start, t.cnt, &full[s]);
          tma_load_2d(base + NPROJ * kBlk + j * C::kWBlk, &a.tm_bt[jj], n0, pt.rank_off[t.g], &full[s]);
        }
        ++i;
      };
      Tile cur, nxt;
      int pcur = 0, pnxt = 0;
      if (has_pre)
        for (int k = 0; k < NK && !bad; ++k) load_k(pre_t, k);
      bool has_cur = grab(cur, pcur);
      if (has_cur && needs_k(cur))
        for (int k = 0; k < NK && !bad; ++k) load_k(cur, k);
      while (has_cur && !bad) {
        const bool has_nxt = grab(nxt, pnxt);
        for (int c = chunk_lo(cur, nch, merge); c < chunk_hi(cur, nch, merge) && !bad; ++c) load_c(cur, pcur, c);
        if (has_nxt && needs_k(nxt))
          for (int k = 0; k < NK && !bad; ++k) load_k(nxt, k);
        cur = nxt;
        pcur = pnxt;
        has_cur = has_nxt;
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
      // ci counts the tiles with D chunks (H operand buffers, hs_ready / hs_free),
      // kc the tiles with a K loop (H accumulators, hacc)
      int i = 0, cc = 0, ci = 0, kc = 0, q = 0;
      auto mma_k = [&](int hb, int k) {  // K step k of the tile whose H accumulator is hb
        const int s = i % S;
        if (!mbar_wait(&full[s], (i / S) & 1)) {
          bad = true;
          return;
        }
        tc_fence_after();
        const uint32_t base = slot0 + s * C::kSlot;
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
          tc_mma_bf16(tmem + hb * C::kHcol, sdesc_sw128(base + kk * 32, 16, 1024),
                      sdesc_sw128(base + NPROJ * kBlk + kk * 32, 16, 1024), idesc_h, (k > 0 || kk > 0) ? 1u : 0u);
        tc_commit(&emptyK[s]);
        if (k == NK - 1) tc_commit(&hacc[hb]);
        ++i;
      };
      auto mma_c = [&](bool first, bool last) {  // a D chunk of chunk-tile ci
        const int s = i % S, b = cc % kNGrp;
        if ((first && !mbar_wait(&hs_ready[ci & 1], (ci >> 1) & 1)) ||
            (cc >= kNGrp && !mbar_wait(&dempty[b], ((cc - kNGrp) / kNGrp) & 1)) ||
            !mbar_wait(&full[s], (i / S) & 1)) {
          bad = true;
          return;
        }
        tc_fence_after();
        const uint32_t base = slot0 + s * C::kSlot;
        const uint32_t sHs = sHs0 + (ci % NBH) * C::kHs;
#pragma unroll
        for (int j = 0; j < NPROJ; ++j)
#pragma unroll
          for (int kk = 0; kk < RP / 16; ++kk) {
            const int kg = (j * RP) / 16 + kk;
            tc_mma_bf16(tmem + C::kDBase + (b * NPROJ + j) * kChunk,
                        sdesc_sw128(sHs + (kg >> 2) * kBlk + (kg & 3) * 32, 16, 1024),
                        sdesc_sw128(base + NPROJ * kBlk + j * C::kWBlk + kk * 2048, C::kWBlk, 1024), idesc_d,
                        kk > 0 ? 1u : 0u);
          }
        tc_commit(&dfull[b]);
        if (last) tc_commit(&hs_free[ci % NBH]);
        ++cc;
        ++i;
      };
      Tile cur, nxt;
      int pdummy = 0;
      bool qok = true;
      if (has_pre) {
        for (int k = 0; k < NK && !bad; ++k) mma_k(kc & 1, k);
        ++kc;
      }
      bool has_cur = queue_next(tq, q, a.tiles, cur, true, &qok, psplit, pdummy);
      if (has_cur && needs_k(cur)) {
        for (int k = 0; k < NK && !bad; ++k) mma_k(kc & 1, k);
        ++kc;
      }
      while (has_cur && !bad) {
        const bool has_nxt = queue_next(tq, q, a.tiles, nxt, true, &qok, psplit, pdummy);
        const int lo = chunk_lo(cur, nch, merge), hi = chunk_hi(cur, nch, merge);
        for (int c = lo; c < hi && !bad; ++c) mma_c(c == lo, c == hi - 1);
        ++ci;
        if (has_nxt && needs_k(nxt)) {
          for (int k = 0; k < NK && !bad; ++k) mma_k(kc & 1, k);
          ++kc;
        }
        cur = nxt;
        has_cur = has_nxt;
      }
      if (!qok) bad = true;
      // the last commits must land before the CTA exits
      if (!bad && ci > 0 && !mbar_wait(&hs_free[(ci - 1) % NBH], ((ci - 1) / NBH) & 1)) bad = true;
      if (!bad && kc > 0 && ci == 0 && !mbar_wait(&hacc[(kc - 1) & 1], ((kc - 1) >> 1) & 1)) bad = true;
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int grp = (warp - 2) >> 2;        // this warp's group: chunks cc with cc % kNGrp == grp
    const int quarter = warp & 3;           // TMEM lane quarter of this warp
    const int m = quarter * 32 + lane;      // tile row owned by this thread
    const uint32_t lane_base = (uint32_t)(quarter * 32) << 16;
    const float s = a.s;
    // H operand of chunk-tile ci (tile t, K-tile kt or -1) into buffer
    // ci % NBH: this warp's rows, its group's share of the columns
    auto stage_h = [&](const Tile& t, int pj, int ci, int kt) {
      const uint32_t sHs = sHs0 + (ci % NBH) * C::kHs;
      if (quarter * 32 >= t.cnt) return;  // no live row: these H rows feed only D rows nobody reads
      const bool live = m < t.cnt;
      const int rg = pt.rank_off[t.g + 1] - pt.rank_off[t.g];
      if (!SHARED && kt >= 0) {
        tc_fence_after();
        for (int c0 = grp * 16; c0 < RP; c0 += 16 * kNGrp) {
          uint32_t r[16];
          tmem_ld16(tmem + lane_base + (kt & 1) * C::kHcol + c0, r);
          tmem_ld_wait();
          float v[16];
#pragma unroll
          for (int qq = 0; qq < 16; ++qq) v[qq] = (live && c0 + qq < rg) ? __uint_as_float(r[qq]) : 0.f;
          if (live && a.Hsave != nullptr) store_row16(a.Hsave + (int64_t)(t.start + m) * pt.rank_max, c0, pt.rank_max, v);
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
      } else {
        // gate/up: H of the row's unique pair; down split tile: its up-front H row
        const int u = live ? (SHARED ? ACE_CHK(a.row_uniq[t.start + m], 0, a.counts[kCntU], 0, a.err) : t.start + m) : -1;
        if ((pt.rank_max & 3) != 0) {
          // rows not 16-byte aligned: 8 columns at a time (measured faster
          // here than all loads up front)
#pragma unroll
          for (int j = 0; j < NPROJ; ++j) {
            const float* hp = (SHARED ? a.Hu[j + pj] : a.Hpre) + (int64_t)(u < 0 ? 0 : u) * pt.rank_max;
            for (int c8 = grp * 8; c8 < RP; c8 += 8 * kNGrp) {
              float w[8];
#pragma unroll
              for (int qq = 0; qq < 8; ++qq) w[qq] = (u >= 0 && c8 + qq < rg) ? hp[c8 + qq] : 0.f;
              uint4 o;
              o.x = pack_bf16x2(w[0], w[1]);
              o.y = pack_bf16x2(w[2], w[3]);
              o.z = pack_bf16x2(w[4], w[5]);
              o.w = pack_bf16x2(w[6], w[7]);
              const int col = j * RP + c8;
              sts128(sHs + (col >> 6) * kBlk + sw128_off(m, (col & 63) >> 3), o);
            }
          }
          return;
        }
        // rows 16-byte aligned (rank_max % 4 == 0): every load of the thread
        // is issued before the first is used, 16 bytes each (one round trip
        // per tile instead of one per 8 columns)
        constexpr int kIt = (RP + 8 * kNGrp - 1) / (8 * kNGrp);
        float v[NPROJ][kIt][8];
#pragma unroll
        for (int j = 0; j < NPROJ; ++j) {
          const float* hp = (SHARED ? a.Hu[j + pj] : a.Hpre) + (int64_t)(u < 0 ? 0 : u) * pt.rank_max;
#pragma unroll
          for (int it = 0; it < kIt; ++it) {
            const int c8 = grp * 8 + it * 8 * kNGrp;
            float* w = v[j][it];
            if (u >= 0 && c8 < rg && c8 + 8 <= pt.rank_max) {
              const float4 x0 = *reinterpret_cast<const float4*>(hp + c8);
              const float4 x1 = *reinterpret_cast<const float4*>(hp + c8 + 4);
              w[0] = x0.x, w[1] = x0.y, w[2] = x0.z, w[3] = x0.w;
              w[4] = x1.x, w[5] = x1.y, w[6] = x1.z, w[7] = x1.w;
            } else {
#pragma unroll
              for (int qq = 0; qq < 8; ++qq) w[qq] = (u >= 0 && c8 + qq < rg) ? hp[c8 + qq] : 0.f;
            }
          }
        }
#pragma unroll
        for (int j = 0; j < NPROJ; ++j)
#pragma unroll
          for (int it = 0; it < kIt; ++it) {
            const int c8 = grp * 8 + it * 8 * kNGrp;
            if (c8 >= RP) continue;
            float* w = v[j][it];
#pragma unroll
            for (int qq = 0; qq < 8; ++qq) w[qq] = c8 + qq < rg ? w[qq] : 0.f;
            uint4 o;
            o.x = pack_bf16x2(w[0], w[1]);
            o.y = pack_bf16x2(w[2], w[3]);
            o.z = pack_bf16x2(w[4], w[5]);
            o.w = pack_bf16x2(w[6], w[7]);
            const int col = j * RP + c8;
            sts128(sHs + (col >> 6) * kBlk + sw128_off(m, (col & 63) >> 3), o);
          }
      }
    };
    // H of chunk-tile ci (tile t; kt: its K-tile number, -1 without a K
    // loop): wait until the buffer's previous tile is done with it and the H
    // exists (down: the K loop, or the up-front H of a split tile), stage,
    // publish
    auto prepare_h = [&](const Tile& t, int pj, int ci, int kt) -> bool {
      bool w = true;
      if (ci >= NBH) w = mbar_wait(&hs_free[ci % NBH], ((ci - NBH) / NBH) & 1);
      if (kt >= 0) w = w && mbar_wait(&hacc[kt & 1], (kt >> 1) & 1);
      if (!SHARED && kt < 0) {  // split tile: wait for its up-front H
        bool w2 = true;
        if (lane == 0) {
          const uint64_t t0 = globaltimer_ns(), limit = a.test_expiry ? kTestWaitLimitNs : kWaitLimitNs;
          while (ld_acquire(hflag + split_index(t)) < kPreWriters)
            if (globaltimer_ns() - t0 > limit) {
              w2 = false;
              break;
            }
        }
        w = w && __shfl_sync(0xffffffffu, w2, 0);
        if (w) (void)ld_acquire(hflag + split_index(t));  // every lane's H loads follow an acquire
      }
      if (!__all_sync(0xffffffffu, w)) return false;
      stage_h(t, pj, ci, kt);
      fence_proxy_async_smem();
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&hs_ready[ci & 1]);
      return true;
    };
    // the up-front H of split tile blockIdx.x: this warp's rows and columns
    // into Hpre, then count this warp in the tile's flag
    auto drain_pre = [&](const Tile& t, int kt) -> bool {
      if (!__all_sync(0xffffffffu, mbar_wait(&hacc[kt & 1], (kt >> 1) & 1))) return false;
      tc_fence_after();
      const bool live = m < t.cnt;
      const int rg = pt.rank_off[t.g + 1] - pt.rank_off[t.g];
      for (int c0 = grp * 16; c0 < RP; c0 += 16 * kNGrp) {
        uint32_t r[16];
        tmem_ld16(tmem + lane_base + (kt & 1) * C::kHcol + c0, r);
        tmem_ld_wait();
        if (live) {
          float v[16];
#pragma unroll
          for (int qq = 0; qq < 16; ++qq) v[qq] = c0 + qq < rg ? __uint_as_float(r[qq]) : 0.f;
          store_row16(a.Hpre + (int64_t)(t.start + m) * pt.rank_max, c0, pt.rank_max, v);
        }
      }
      tc_fence_before();
      __threadfence();
      __syncwarp();
      if (lane == 0 && !a.test_expiry) atomicAdd(hflag + blockIdx.x, 1);
      return true;
    };
    int q = 0, ib = 0, cc0 = 0, ci = 0, kc = 0;
    bool ok = true;
    Tile cur, nxt;
    int pcur = 0, pnxt = 0;
    if (has_pre) {
      ok = drain_pre(pre_t, kc);
      ++kc;
      ib += NK;
    }
    bool has_cur = ok && queue_next(tq, q, a.tiles, cur, false, &ok, psplit, pcur);
    if (has_cur) {
      int kt = -1;
      if (needs_k(cur)) {
        kt = kc++;
        ib += NK;
      }
      ok = prepare_h(cur, pcur, ci, kt);
    }
    while (has_cur && ok) {
      const bool has_nxt = queue_next(tq, q, a.tiles, nxt, false, &ok, psplit, pnxt);
      if (!ok) break;
      const bool inter = has_nxt && needs_k(nxt);
      // gate/up with two H buffers: gather the next tile's H now, while this tile streams
      const bool early = SHARED && NBH == 2 && has_nxt;
      if (early && !(ok = prepare_h(nxt, pnxt, ci + 1, -1))) break;
      const bool qlive = quarter * 32 < cur.cnt;  // this warp has live rows (warp-uniform)
      const int lo = chunk_lo(cur, nch, merge), hi = chunk_hi(cur, nch, merge);
      for (int c = lo + ((grp - cc0) % kNGrp + kNGrp) % kNGrp; c < hi; c += kNGrp) {
        const int cc = cc0 + (c - lo), i = ib + (c - lo);
        const int sl = i % S, b = cc % kNGrp, n0 = c * kChunk;
        ok = __all_sync(0xffffffffu, mbar_wait(&full[sl], (i / S) & 1) && mbar_wait(&dfull[b], (cc / kNGrp) & 1));
        if (!ok) break;
        tc_fence_after();
        const uint32_t base = slot0 + sl * C::kSlot;
        if (qlive) {
#pragma unroll
          for (int j = 0; j < NPROJ; ++j) {
            const uint32_t ta = tmem + lane_base + C::kDBase + (b * NPROJ + j) * kChunk;
#pragma unroll
            for (int h = 0; h < 2; ++h) {
              uint32_t r[32];
              tmem_ld16(ta + h * 32, *reinterpret_cast<uint32_t(*)[16]>(&r[0]));
              tmem_ld16(ta + h * 32 + 16, *reinterpret_cast<uint32_t(*)[16]>(&r[16]));
              tmem_ld_wait();
#pragma unroll
              for (int qq = 0; qq < 4; ++qq) {
                const uint32_t addr = base + j * kBlk + sw128_off(m, h * 4 + qq);
                const uint4 y = lds128(addr);
                const uint32_t* dq = &r[qq * 8];
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
        }
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(&dempty[b]);
        if (qlive) {
          // this warp's 32 rows, 128 contiguous bytes each: 4 rows per instruction
#pragma unroll
          for (int j = 0; j < NPROJ; ++j)
#pragma unroll
            for (int it = 0; it < 8; ++it) {
              const int row = quarter * 32 + it * 4 + (lane >> 3), ch = lane & 7, col = n0 + ch * 8;
              if (row < cur.cnt && col < d_out) {
                const uint4 v = lds128(base + j * kBlk + sw128_off(row, ch));
                *reinterpret_cast<uint4*>(a.Y[j + pcur] + (int64_t)(cur.start + row) * d_out + col) = v;
              }
            }
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(&emptyC[sl]);
      }
      if (!ok) break;
      if (has_nxt && !early && !(ok = prepare_h(nxt, pnxt, ci + 1, inter ? kc++ : -1))) break;
      ib += (hi - lo) + (inter ? NK : 0);
      cc0 += hi - lo;
      ++ci;
      cur = nxt;
      pcur = pnxt;
      has_cur = has_nxt;
    }
    if (!ok) bad = true;
  }
  __syncwarp();  // reconverge the single-lane roles before the CTA barrier
  tc_fence_before();
  if (__syncthreads_or(bad) && tid == 0) atomicOr(a.err, kErrTimeout);
  __shared__ int last_cta;
  if (tid == 0) {
    // the last CTA to finish (every producer has taken its final index) resets
    // the counters (and the H-ready flags) for the next launch
    __threadfence();
    last_cta = atomicAdd(a.sched + kSchedFwdDone, 1) == (int)gridDim.x - 1;
    if (last_cta) {
      atomicExch(a.sched + kSchedFwdRows, 0);
      atomicExch(a.sched + kSchedFwdDone, 0);
    }
  }
  if (pre) {
    __syncthreads();
    if (last_cta)
      for (int b = tid; b < n_split; b += blockDim.x) hflag[b] = 0;
  }
  // signal dependents only as this CTA finishes: an earlier launch of the
  // next kernel (a whole SM per CTA) measured slower
  pdl_trigger();
  if (warp == 0) tmem_dealloc(tmem, kRowsTmem);
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
  return launch_k(kern, a.max_tiles, kHThreads, C::kSmem, st, pt, a);
}

template <int RP, int NPROJ, bool SHARED>
cudaError_t launch_rows_t(const PlanTables& pt, const FwdRowsLaunch& a, cudaStream_t st) {
  using C = RowsFwdCfg<RP, NPROJ, SHARED>;
  auto kern = k_fwd_rows<RP, NPROJ, SHARED>;
  cudaError_t e = set_smem(kern, C::kSmem);
  if (e != cudaSuccess || a.grid <= 0) return e;
  return launch_k(kern, a.grid, kRowsThreads, C::kSmem, st, pt, a);
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
    // at rank_pad 128 a tile's two projections go out as separate work
    // items: their shared-memory budget then leaves room for two H operand
    // buffers and four ring slots (both projections in one item: one H
    // buffer and two slots).  At rank_pad 64 one item holding both
    // projections measured faster.
    FwdRowsLaunch b = a;
    b.proj_split = 1;
    switch (pt.rank_pad) {
      case 16: return launch_rows_t<16, 2, true>(pt, a, st);
      case 32: return launch_rows_t<32, 2, true>(pt, a, st);
      case 64: return launch_rows_t<64, 2, true>(pt, a, st);
      case 128: return launch_rows_t<128, 1, true>(pt, b, st);
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
