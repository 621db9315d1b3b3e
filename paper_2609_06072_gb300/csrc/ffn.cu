// Routed expert FFN with the group-shared adapters (App. "Implementation and
// Profiling of Grouped Adapter Execution": u = (W^up + dW^up) x,
// v = (W^gate + dW^gate) x, h = SiLU(v) * u, y = (W^down + dW^down) h), forward,
// composed from the base expert GEMMs and the adapter calls of this library:
//   X rows gathered into row order, u / v = base GEMMs per expert segment,
//   the gate/up adapter deltas added by the shared-input forward,
//   h = SiLU(v) * u, y = base GEMM of h, the down delta added by the per-row
//   forward.
// k_expert_gemm: out[row] = in[row] . W_e^T for the rows of each expert e
//   (rows contiguous per expert in row order).  Persistent over [128 rows of
//   one expert x 256 output columns] tiles; both operands K-major by TMA
//   (128-byte swizzle), four 48 KB stages, tcgen05 M = 128, N = 256 into one
//   of two TMEM accumulators, eight epilogue warps (thread = row, 128 columns
//   each) storing bf16.  A second product over the same rows (the backward's
//   dv . W_gate beside du . W_up) can follow in the same accumulator.
#include <algorithm>
#include <cstdint>

#include "ace_internal.cuh"
#include "ace_ptx.cuh"

namespace ace {
namespace {

constexpr int kFThreads = 320;           // producer, MMA, 8 epilogue warps
constexpr int kFBlk = 128 * 128;         // [128 rows x 64 bf16]
constexpr int kFN = 256;                 // output columns per tile
constexpr int kFStage = kFBlk + 2 * kFBlk;  // in [128 x 64] + W [256 x 64]
constexpr int kFS = 4;
constexpr int kFSmem = kFS * kFStage + 1024;

struct ExpertGemmLaunch {
  CUtensorMap tm_in;   // in [R, K] bf16, box 64 x 128
  CUtensorMap tm_w;    // W_e^T rows: [E * N, K] bf16, box 64 x 256; or (B_MN) W_e: [E * K, N], box 64 x 64
  // optional second product over the same rows, summed into the same
  // accumulator (its K steps follow the first's): out = in . W + in2 . W2
  CUtensorMap tm_in2, tm_w2;
  int32_t two;
  const int32_t* expert_off;
  const int32_t* expert_cnt;
  uint16_t* out;       // [R, N] bf16
  int32_t E, N, K, grid;
  int32_t accumulate;  // out[row] += instead of =
  int32_t* err;
};

// Largest i with off[i] <= v over off[0..n] (off ascending, off[0] <= v).
__device__ __forceinline__ int upper_i(const int32_t* off, int n, int v) {
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

// B_MN: the weights are given as W_e [K, N] (N contiguous; the input
// gradient through a frozen weight) instead of [N, K]; the B tile is then four
// [64 k x 64 n] boxes read MN-major.
template <bool B_MN>
__global__ void __launch_bounds__(kFThreads, 1) k_expert_gemm(const __grid_constant__ ExpertGemmLaunch a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  __shared__ __align__(8) uint64_t full[kFS], empty[kFS], acc_full[2], acc_empty[2];
  __shared__ uint32_t tslot;
  __shared__ int32_t tpre[ACE_MAX_EXPERTS + 1];  // row tiles before expert e
  __shared__ int32_t eoff[ACE_MAX_EXPERTS], ecnt[ACE_MAX_EXPERTS];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int E = a.E, nchunk = (a.N + kFN - 1) / kFN, NK1 = (a.K + 63) / 64, NK = a.two ? 2 * NK1 : NK1;
  const uint32_t s0 = smem_u32(smem);
  if (tid == 0) {
    for (int i = 0; i < kFS; ++i) {
      mbar_init(&full[i], 1);
      mbar_init(&empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&acc_full[i], 1);
      mbar_init(&acc_empty[i], 8);
    }
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(&tslot, 2 * kFN);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  pdl_wait();
  for (int e = tid; e < E; e += blockDim.x) {
    eoff[e] = a.expert_off[e];
    ecnt[e] = a.expert_cnt[e];
  }
  __syncthreads();
  if (tid == 0) {
    tpre[0] = 0;
    for (int e = 0; e < E; ++e) tpre[e + 1] = tpre[e] + (ecnt[e] + 127) / 128;
  }
  __syncthreads();
  const int ntile = tpre[E] * nchunk;
  // tile -> (expert, first row, rows, first column)
  auto decode = [&](int tile, int& e, int& row0, int& cnt, int& n0) {
    const int rt = tile / nchunk;
    n0 = (tile % nchunk) * kFN;
    e = upper_i(tpre, E, rt);
    while (e + 1 < E && tpre[e + 1] <= rt) ++e;  // skip experts with no rows
    const int i = rt - tpre[e];
    row0 = eoff[e] + i * 128;
    cnt = min(128, ecnt[e] - i * 128);
  };
  const uint32_t tmem = tslot;
  bool bad = false;
  if (warp == 0) {
    if (lane == 0) {
      int i = 0;
      for (int tile = blockIdx.x; tile < ntile && !bad; tile += gridDim.x) {
        int e, row0, cnt, n0;
        decode(tile, e, row0, cnt, n0);
        for (int kb = 0; kb < NK; ++kb, ++i) {
          const int s = i % kFS, u = i / kFS;
          if (u >= 1 && !mbar_wait(&empty[s], (u - 1) & 1)) {
            bad = true;
            break;
          }
          const uint32_t base = s0 + s * kFStage;
          const bool second = kb >= NK1;
          const int kq = second ? kb - NK1 : kb;
          const CUtensorMap* tin = second ? &a.tm_in2 : &a.tm_in;
          const CUtensorMap* tw = second ? &a.tm_w2 : &a.tm_w;
          mbar_arrive_expect_tx(&full[s], kFStage);
          tma_load_2d(base, tin, kq * 64, row0, &full[s]);
          if (B_MN) {
            for (int q = 0; q < kFN / 64; ++q)
              tma_load_2d(base + kFBlk + q * (kFBlk / 2), tw, n0 + q * 64, e * a.K + kq * 64, &full[s]);
          } else {
            tma_load_2d(base + kFBlk, tw, kq * 64, e * a.N + n0, &full[s]);
          }
        }
      }
      for (int k2 = max(0, i - kFS); k2 < i; ++k2)
        if (!mbar_wait(&full[k2 % kFS], (k2 / kFS) & 1)) bad = true;
    }
  } else if (warp == 1) {
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(128, kFN, 0, B_MN ? 1 : 0);
      int i = 0, it = 0;
      for (int tile = blockIdx.x; tile < ntile && !bad; tile += gridDim.x, ++it) {
        const int b = it & 1;
        if (it >= 2 && !mbar_wait(&acc_empty[b], ((it - 2) >> 1) & 1)) {
          bad = true;
          break;
        }
        tc_fence_after();
        for (int kb = 0; kb < NK; ++kb, ++i) {
          const int s = i % kFS;
          if (!mbar_wait(&full[s], (i / kFS) & 1)) {
            bad = true;
            break;
          }
          tc_fence_after();
          const uint32_t base = s0 + s * kFStage;
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_bf16(tmem + b * kFN, sdesc_sw128(base + kk * 32, 16, 1024),
                        B_MN ? sdesc_sw128(base + kFBlk + kk * 2048, kFBlk / 2, 1024)
                             : sdesc_sw128(base + kFBlk + kk * 32, 16, 1024),
                        idesc, (kb > 0 || kk > 0) ? 1u : 0u);
          tc_commit(&empty[s]);
        }
        if (!bad) tc_commit(&acc_full[b]);
      }
    }
  } else {
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
      uint16_t* orow = a.out + (int64_t)(row0 + m) * a.N;
      for (int c16 = 0; c16 < 8; ++c16) {
        const int col = n0 + ehalf * 128 + c16 * 16;
        if (col >= a.N) break;  // warp-uniform
        // out[row] += the product (fp32 sum, one rounding): the old values of
        // a whole 16-column piece come in two 16-byte loads, issued before the
        // accumulator is read
        const bool whole = col + 16 <= a.N;
        uint4 o0 = make_uint4(0u, 0u, 0u, 0u), o1 = o0;
        if (a.accumulate && whole && m < cnt) {
          o0 = *reinterpret_cast<const uint4*>(orow + col);
          o1 = *reinterpret_cast<const uint4*>(orow + col + 8);
        }
        uint32_t r[16];
        tmem_ld16(tmem + lane_base + b * kFN + ehalf * 128 + c16 * 16, r);
        tmem_ld_wait();
        if (m < cnt) {
          if (a.accumulate && whole) {
            const uint32_t ow[8] = {o0.x, o0.y, o0.z, o0.w, o1.x, o1.y, o1.z, o1.w};
#pragma unroll
            for (int q = 0; q < 8; ++q) {
              const float2 f = unpack_bf16x2(ow[q]);
              r[2 * q] = __float_as_uint(f.x + __uint_as_float(r[2 * q]));
              r[2 * q + 1] = __float_as_uint(f.y + __uint_as_float(r[2 * q + 1]));
            }
          } else if (a.accumulate) {
            for (int q = 0; q < 16 && col + q < a.N; ++q) {
              const float old = __uint_as_float((uint32_t)orow[col + q] << 16);
              r[q] = __float_as_uint(old + __uint_as_float(r[q]));
            }
          }
          if (whole) {
            uint4 v0, v1;
            v0.x = pack_bf16x2(__uint_as_float(r[0]), __uint_as_float(r[1]));
            v0.y = pack_bf16x2(__uint_as_float(r[2]), __uint_as_float(r[3]));
            v0.z = pack_bf16x2(__uint_as_float(r[4]), __uint_as_float(r[5]));
            v0.w = pack_bf16x2(__uint_as_float(r[6]), __uint_as_float(r[7]));
            v1.x = pack_bf16x2(__uint_as_float(r[8]), __uint_as_float(r[9]));
            v1.y = pack_bf16x2(__uint_as_float(r[10]), __uint_as_float(r[11]));
            v1.z = pack_bf16x2(__uint_as_float(r[12]), __uint_as_float(r[13]));
            v1.w = pack_bf16x2(__uint_as_float(r[14]), __uint_as_float(r[15]));
            *reinterpret_cast<uint4*>(orow + col) = v0;
            *reinterpret_cast<uint4*>(orow + col + 8) = v1;
          } else {
            for (int q = 0; q < 16 && col + q < a.N; ++q) {
              const __nv_bfloat16 h = __float2bfloat16_rn(__uint_as_float(r[q]));
              orow[col + q] = *reinterpret_cast<const uint16_t*>(&h);
            }
          }
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
  if (warp == 0) tmem_dealloc(tmem, 2 * kFN);
}

// dst[row] = X[row_pair[row] / k]: token rows into row order over the rows
// the permutation wrote (counts[kCntRows]; the rows of invalid tokens are
// never written and are skipped).  A warp copies a row, each lane eight
// 16-byte pieces at a time, all eight loads issued before the first store.
__global__ void __launch_bounds__(256) k_gather_tokens(const int32_t* __restrict__ row_pair,
                                                       const int32_t* __restrict__ counts, int k, int T,
                                                       const uint16_t* __restrict__ X, uint16_t* __restrict__ dst,
                                                       int64_t R, int cols) {
  pdl_wait();
  pdl_trigger();
  const int per = cols / 8;  // 16-byte pieces per row
  const int64_t nrow = min(R, (int64_t)counts[kCntRows]);
  const int lane = threadIdx.x & 31;
  const int64_t nwarps = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t row = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; row < nrow; row += nwarps) {
    const int64_t t = row_pair[row] / k;
    if (t < 0 || t >= T) continue;
    const uint4* __restrict__ src = reinterpret_cast<const uint4*>(X + t * cols);
    uint4* __restrict__ out = reinterpret_cast<uint4*>(dst + row * cols);
    for (int c0 = 0; c0 < per; c0 += 8 * 32) {
      uint4 v[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int c = c0 + i * 32 + lane;
        if (c < per) v[i] = src[c];
      }
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const int c = c0 + i * 32 + lane;
        if (c < per) out[c] = v[i];
      }
    }
  }
}

// h = SiLU(v) * u elementwise (bf16 in, fp32 arithmetic, bf16 out), 8 a thread
__global__ void __launch_bounds__(256) k_swiglu(const uint16_t* __restrict__ u, const uint16_t* __restrict__ v,
                                                uint16_t* __restrict__ h, int64_t n8) {
  pdl_wait();
  pdl_trigger();
  const int64_t i = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (i >= n8) return;
  const uint4 a = reinterpret_cast<const uint4*>(u)[i], b = reinterpret_cast<const uint4*>(v)[i];
  const uint32_t ua[4] = {a.x, a.y, a.z, a.w}, vb[4] = {b.x, b.y, b.z, b.w};
  uint32_t o[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float2 uu = unpack_bf16x2(ua[q]), vv = unpack_bf16x2(vb[q]);
    const float h0 = vv.x / (1.f + __expf(-vv.x)) * uu.x, h1 = vv.y / (1.f + __expf(-vv.y)) * uu.y;
    o[q] = pack_bf16x2(h0, h1);
  }
  reinterpret_cast<uint4*>(h)[i] = make_uint4(o[0], o[1], o[2], o[3]);
}

// du = dh * SiLU(v), dv = dh * u * SiLU'(v) with SiLU'(v) = sigma(v) (1 + v (1 - sigma(v)))
__global__ void __launch_bounds__(256) k_swiglu_bwd(const uint16_t* __restrict__ dh, const uint16_t* __restrict__ u,
                                                    const uint16_t* __restrict__ v, uint16_t* __restrict__ du,
                                                    uint16_t* __restrict__ dv, int64_t n8) {
  pdl_wait();
  pdl_trigger();
  const int64_t i = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (i >= n8) return;
  const uint4 g = reinterpret_cast<const uint4*>(dh)[i], a = reinterpret_cast<const uint4*>(u)[i],
              b = reinterpret_cast<const uint4*>(v)[i];
  const uint32_t gg[4] = {g.x, g.y, g.z, g.w}, ua[4] = {a.x, a.y, a.z, a.w}, vb[4] = {b.x, b.y, b.z, b.w};
  uint32_t ou[4], ov[4];
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float2 dg = unpack_bf16x2(gg[q]), uu = unpack_bf16x2(ua[q]), vv = unpack_bf16x2(vb[q]);
    const float s0 = 1.f / (1.f + __expf(-vv.x)), s1 = 1.f / (1.f + __expf(-vv.y));
    ou[q] = pack_bf16x2(dg.x * vv.x * s0, dg.y * vv.y * s1);
    ov[q] = pack_bf16x2(dg.x * uu.x * s0 * (1.f + vv.x * (1.f - s0)), dg.y * uu.y * s1 * (1.f + vv.y * (1.f - s1)));
  }
  reinterpret_cast<uint4*>(du)[i] = make_uint4(ou[0], ou[1], ou[2], ou[3]);
  reinterpret_cast<uint4*>(dv)[i] = make_uint4(ov[0], ov[1], ov[2], ov[3]);
}

// dX[t] = sum_j rows[pair_row[t k + j]] over the token's valid pairs, in
// ascending j (fp32 sum, one rounding); 8 columns a thread
__global__ void __launch_bounds__(256) k_token_sum(const uint16_t* __restrict__ rows, const int32_t* __restrict__ pair_row,
                                                   const int32_t* __restrict__ pair_g, int k, int T, int cols,
                                                   uint16_t* __restrict__ dX, int32_t* err) {
  pdl_wait();
  pdl_trigger();
  const int per = cols / 8;
  const int64_t idx = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (idx >= (int64_t)T * per) return;
  const int64_t t = idx / per;
  const int c = (int)(idx % per) * 8;
  float acc[8] = {};
  for (int j = 0; j < k; ++j) {
    const int64_t p = t * k + j;
    if (pair_g[p] < 0) continue;  // invalid token: no rows
    const uint4 w =
        *reinterpret_cast<const uint4*>(rows + (int64_t)ACE_CHK(pair_row[p], 0, T * k, 0, err) * cols + c);
    const uint32_t ww[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const float2 f = unpack_bf16x2(ww[q]);
      acc[2 * q] += f.x;
      acc[2 * q + 1] += f.y;
    }
  }
  *reinterpret_cast<uint4*>(dX + t * cols + c) = make_uint4(pack_bf16x2(acc[0], acc[1]), pack_bf16x2(acc[2], acc[3]),
                                                            pack_bf16x2(acc[4], acc[5]), pack_bf16x2(acc[6], acc[7]));
}

}  // namespace

cudaError_t launch_expert_gemm(const void* in, const void* W, const int32_t* expert_off, const int32_t* expert_cnt,
                               uint16_t* out, int E, int64_t R, int N, int K, int grid, int32_t* err,
                               cudaStream_t st, bool w_kn, bool accumulate, const void* in2, const void* W2) {
  ExpertGemmLaunch a{};
  auto maps = [&](CUtensorMap* ti, CUtensorMap* tw, const void* x, const void* w) {
    return make_tmap_bf16(ti, x, (uint64_t)R, (uint64_t)K, 128) &&
           (w_kn ? make_tmap_bf16(tw, w, (uint64_t)E * K, (uint64_t)N, 64)
                 : make_tmap_bf16(tw, w, (uint64_t)E * N, (uint64_t)K, 256));
  };
  bool ok = maps(&a.tm_in, &a.tm_w, in, W);
  a.two = in2 != nullptr && W2 != nullptr;
  if (a.two) ok = ok && maps(&a.tm_in2, &a.tm_w2, in2, W2);
  if (!ok) return cudaErrorInvalidValue;
  a.accumulate = accumulate ? 1 : 0;
  a.expert_off = expert_off;
  a.expert_cnt = expert_cnt;
  a.out = out;
  a.E = E;
  a.N = N;
  a.K = K;
  a.grid = grid;
  a.err = err;
  auto kern = w_kn ? k_expert_gemm<true> : k_expert_gemm<false>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, kFSmem);
  if (e != cudaSuccess) return e;
  return launch_k(kern, grid, kFThreads, kFSmem, st, a);
}

cudaError_t launch_gather_tokens(const int32_t* row_pair, const int32_t* counts, int k, int T, const uint16_t* X,
                                 uint16_t* dst, int64_t R, int cols, int nsm, cudaStream_t st) {
  if (R == 0) return cudaSuccess;
  // a warp per row, eight warps a block, up to 16 blocks per SM
  const int64_t blocks = std::min<int64_t>((R + 7) / 8, (int64_t)nsm * 16);
  return launch_k(k_gather_tokens, (unsigned)blocks, 256, 0, st, row_pair, counts, k, T, X, dst, R, cols);
}

cudaError_t launch_swiglu(const uint16_t* u, const uint16_t* v, uint16_t* h, int64_t n, cudaStream_t st) {
  const int64_t n8 = n / 8;
  if (n8 == 0) return cudaSuccess;
  return launch_k(k_swiglu, (unsigned)((n8 + 255) / 256), 256, 0, st, u, v, h, n8);
}

}  // namespace ace

using namespace ace;

extern "C" {

// Forward: the token rows in row order [R, d].  Backward: dh, du, dv [R, f]
// and the per-row input gradient [R, d].
static size_t ffn_ws_bytes(const PlanTables& pt, int64_t R) {
  const size_t fwd = align_up(2 * (size_t)R * pt.d, 256);
  const size_t bwd = 3 * align_up(2 * (size_t)R * pt.f, 256) + align_up(2 * (size_t)R * pt.d, 256);
  return fwd > bwd ? fwd : bwd;
}

ace_status ace_ffn_workspace_size(const ace_plan* plan, int32_t T, size_t* bytes) {
  if (!plan || !bytes) return report(ACE_ERR_ARG, "ace_ffn_workspace_size: null argument");
  if (T < 0 || T > plan->T_max) return report(ACE_ERR_SHAPE, "ace_ffn_workspace_size: T outside [0, T_max]");
  *bytes = ffn_ws_bytes(plan->pt, (int64_t)T * plan->pt.k);
  return ACE_OK;
}

ace_status ace_ffn_fwd(const ace_plan* plan, const ace_perm* perm, const uint16_t* X, const uint16_t* W_gate,
                       const uint16_t* W_up, const uint16_t* W_down, const uint16_t* const* A,
                       const uint16_t* const* Bt, float s, uint16_t* U, uint16_t* V, uint16_t* Hh, uint16_t* Y,
                       float* const* Hgu, float* Hd, void* ws, size_t ws_bytes, void* stream) {
  if (!plan || !perm || !perm->ws) return report(ACE_ERR_ARG, "ace_ffn_fwd: null plan or perm");
  if (perm->T < 0 || perm->T > plan->T_max || perm->R != perm->T * plan->pt.k)
    return report(ACE_ERR_SHAPE, "ace_ffn_fwd: perm does not match the plan");
  if (!A || !Bt || !Hgu || !W_gate || !W_up || !W_down) return report(ACE_ERR_ARG, "ace_ffn_fwd: null argument");
  for (int j = 0; j < 3; ++j)
    if (!A[j] || !Bt[j]) return report(ACE_ERR_ARG, "ace_ffn_fwd: null adapter");
  if (perm->R == 0) return ACE_OK;
  if (!X || !U || !V || !Hh || !Y || !Hgu[0] || !Hgu[1] || !Hd) return report(ACE_ERR_ARG, "ace_ffn_fwd: null tensor");
  const PlanTables& pt = plan->pt;
  const int64_t R = perm->R;
  const size_t need = ffn_ws_bytes(pt, R);
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  if (!ws || ws_bytes < need || !al16(ws)) return report(ACE_ERR_WORKSPACE, "ace_ffn_fwd: workspace too small or misaligned");
  if (!al16(X) || !al16(W_gate) || !al16(W_up) || !al16(W_down) || !al16(U) || !al16(V) || !al16(Hh) || !al16(Y))
    return report(ACE_ERR_ARG, "ace_ffn_fwd: tensor not 16-byte aligned");
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  const PermLayout L = perm_layout(pt, perm->T);
  int32_t* err = at<int32_t>(perm->ws, L.err);
  auto cuda = [](cudaError_t e, const char* what) {
    return e == cudaSuccess ? ACE_OK : report(ACE_ERR_CUDA, what);
  };
  const int n_rank = pt.rank_off[pt.G];
  // 1. H of gate and up per unique pair, A_g x once per active group of a token
  const uint16_t* Agu[2] = {A[0], A[1]};
  float* Hgu_buf[2] = {Hgu[0], Hgu[1]};
  ace_status st = launch_gate_up_h(plan, perm, X, 2, Agu, Hgu_buf, cs);
  if (st != ACE_OK) return st;
  // 2. the token rows in row order, then u, v (base + adapter) and
  // h = SiLU(v) u in one kernel
  uint16_t* Xr = static_cast<uint16_t*>(ws);
  st = cuda(launch_gather_tokens(perm->row_pair, perm->counts, pt.k, perm->T, X, Xr, R, pt.d, plan->num_sms, cs),
            "ace_ffn_fwd: gather launch");
  if (st != ACE_OK) return st;
  FfnFusedLaunch g{};
  bool ok = make_tmap_bf16(&g.tm_in, Xr, (uint64_t)R, (uint64_t)pt.d, 128) &&
            make_tmap_bf16(&g.tm_w[0], W_up, (uint64_t)pt.E * pt.f, (uint64_t)pt.d, 128) &&
            make_tmap_bf16(&g.tm_w[1], W_gate, (uint64_t)pt.E * pt.f, (uint64_t)pt.d, 128) &&
            make_tmap_bf16(&g.tm_bt[0], Bt[1], (uint64_t)n_rank, (uint64_t)pt.f, pt.rank_pad) &&
            make_tmap_bf16(&g.tm_bt[1], Bt[0], (uint64_t)n_rank, (uint64_t)pt.f, pt.rank_pad);
  if (!ok) return report(ACE_ERR_UNSUPPORTED, "ace_ffn_fwd: tensor-map encoding failed");
  g.row_uniq = at<int32_t>(perm->ws, L.row_uniq);
  g.expert_off = perm->expert_off;
  g.expert_cnt = perm->expert_cnt;
  g.counts = perm->counts;
  g.Hs[0] = Hgu[1];  // TMEM half 0: up
  g.Hs[1] = Hgu[0];  // TMEM half 1: gate
  g.U = U;
  g.V = V;
  g.Hh = Hh;
  g.s = s;
  g.N = pt.f;
  g.K = pt.d;
  g.grid = plan->num_sms;
  g.err = err;
  st = cuda(launch_ffn_fused(pt, g, true, cs), "ace_ffn_fwd: gate/up launch");
  if (st != ACE_OK) return st;
  // 3. H of down per row, A_g h
  FwdHLaunch hd{};
  hd.tiles = at<Tile>(perm->ws, L.tiles_row);
  hd.counts = perm->counts;
  hd.max_tiles = L.max_tiles;
  hd.rows = 1;
  hd.X = Hh;
  hd.A[0] = hd.A[1] = A[2];
  hd.H[0] = hd.H[1] = Hd;
  hd.d_in = pt.f;
  hd.nproj = 1;
  hd.n_src = R;
  hd.err = err;
  st = cuda(launch_fwd_h(pt, hd, cs), "ace_ffn_fwd: down H launch");
  if (st != ACE_OK) return st;
  // 4. y (base + adapter)
  FfnFusedLaunch dn{};
  ok = make_tmap_bf16(&dn.tm_in, Hh, (uint64_t)R, (uint64_t)pt.f, 128) &&
       make_tmap_bf16(&dn.tm_w[0], W_down, (uint64_t)pt.E * pt.d, (uint64_t)pt.f, 256) &&
       make_tmap_bf16(&dn.tm_bt[0], Bt[2], (uint64_t)n_rank, (uint64_t)pt.d, pt.rank_pad);
  if (!ok) return report(ACE_ERR_UNSUPPORTED, "ace_ffn_fwd: tensor-map encoding failed");
  dn.tm_w[1] = dn.tm_w[0];
  dn.tm_bt[1] = dn.tm_bt[0];
  dn.expert_off = perm->expert_off;
  dn.expert_cnt = perm->expert_cnt;
  dn.counts = perm->counts;
  dn.Hs[0] = dn.Hs[1] = Hd;
  dn.Y = Y;
  dn.s = s;
  dn.N = pt.d;
  dn.K = pt.f;
  dn.grid = plan->num_sms;
  dn.err = err;
  return cuda(launch_ffn_fused(pt, dn, false, cs), "ace_ffn_fwd: down launch");
}

ace_status ace_ffn_bwd(const ace_plan* plan, const ace_perm* perm, const uint16_t* dY, const uint16_t* X,
                       const uint16_t* W_gate, const uint16_t* W_up, const uint16_t* W_down, const uint16_t* const* A,
                       const uint16_t* const* Bt, float s, const uint16_t* U, const uint16_t* V, const uint16_t* Hh,
                       const float* const* Hgu, const float* Hd, uint16_t* dX, float* const* dA, float* const* dBt,
                       void* ws, size_t ws_bytes, void* bws, size_t bws_bytes, void* stream) {
  if (!plan || !perm || !perm->ws) return report(ACE_ERR_ARG, "ace_ffn_bwd: null plan or perm");
  if (perm->T < 0 || perm->T > plan->T_max || perm->R != perm->T * plan->pt.k)
    return report(ACE_ERR_SHAPE, "ace_ffn_bwd: perm does not match the plan");
  if (!A || !Bt || !dA || !dBt || !Hgu || !W_gate || !W_up || !W_down) return report(ACE_ERR_ARG, "ace_ffn_bwd: null argument");
  for (int j = 0; j < 3; ++j)
    if (!A[j] || !Bt[j] || !dA[j] || !dBt[j]) return report(ACE_ERR_ARG, "ace_ffn_bwd: null adapter or gradient");
  const PlanTables& pt = plan->pt;
  const int64_t R = perm->R;
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  auto cuda = [](cudaError_t e, const char* what) {
    return e == cudaSuccess ? ACE_OK : report(ACE_ERR_CUDA, what);
  };
  if (R == 0) {  // no rows: every adapter gradient is zero, and there is no token to write
    const int n_rank = pt.rank_off[pt.G];
    const int d_in[3] = {pt.d, pt.d, pt.f}, d_out[3] = {pt.f, pt.f, pt.d};
    for (int j = 0; j < 3; ++j) {
      ace_status st = cuda(cudaMemsetAsync(dA[j], 0, 4 * (size_t)n_rank * d_in[j], cs), "ace_ffn_bwd: memset");
      if (st == ACE_OK) st = cuda(cudaMemsetAsync(dBt[j], 0, 4 * (size_t)n_rank * d_out[j], cs), "ace_ffn_bwd: memset");
      if (st != ACE_OK) return st;
    }
    return ACE_OK;
  }
  if (!dY || !X || !U || !V || !Hh || !Hgu[0] || !Hgu[1] || !Hd || !dX) return report(ACE_ERR_ARG, "ace_ffn_bwd: null tensor");
  const size_t need = ffn_ws_bytes(pt, R);
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  if (!ws || ws_bytes < need || !al16(ws)) return report(ACE_ERR_WORKSPACE, "ace_ffn_bwd: workspace too small or misaligned");
  if (!al16(dY) || !al16(X) || !al16(U) || !al16(V) || !al16(Hh) || !al16(dX) || !al16(W_gate) || !al16(W_up) ||
      !al16(W_down))
    return report(ACE_ERR_ARG, "ace_ffn_bwd: tensor not 16-byte aligned");
  const PermLayout L = perm_layout(pt, perm->T);
  int32_t* err = at<int32_t>(perm->ws, L.err);
  char* w = static_cast<char*>(ws);
  const size_t rf = align_up(2 * (size_t)R * pt.f, 256);
  uint16_t* dh = reinterpret_cast<uint16_t*>(w);
  uint16_t* du = reinterpret_cast<uint16_t*>(w + rf);
  uint16_t* dv = reinterpret_cast<uint16_t*>(w + 2 * rf);
  uint16_t* dxr = reinterpret_cast<uint16_t*>(w + 3 * rf);
  // dh = dy . W_down (base), then the down adapter: dh += s A_d^T (B_d^T dy), dA_d, dB_d
  ace_status st = cuda(launch_expert_gemm(dY, W_down, perm->expert_off, perm->expert_cnt, dh, pt.E, R, pt.f, pt.d,
                                          plan->num_sms, err, cs, true, false),
                       "ace_ffn_bwd: down input-gradient GEMM launch");
  if (st != ACE_OK) return st;
  st = ace_bwd_row(plan, perm, dY, Hh, Hd, A[2], Bt[2], s, dh, dA[2], dBt[2], bws, bws_bytes, stream);
  if (st != ACE_OK) return st;
  // through the gating
  const int64_t n8 = R * pt.f / 8;
  st = cuda(launch_k(k_swiglu_bwd, (unsigned)((n8 + 255) / 256), 256, 0, cs, (const uint16_t*)dh, U, V, du, dv, n8),
            "ace_ffn_bwd: SiLU gating backward launch");
  if (st != ACE_OK) return st;
  // base input gradient per row: du . W_up + dv . W_gate in one GEMM (the
  // gate product's K steps follow the up product's in the same accumulator),
  // then summed per token
  st = cuda(launch_expert_gemm(du, W_up, perm->expert_off, perm->expert_cnt, dxr, pt.E, R, pt.d, pt.f, plan->num_sms,
                               err, cs, true, false, dv, W_gate),
            "ace_ffn_bwd: up and gate input-gradient GEMM launch");
  if (st != ACE_OK) return st;
  const int64_t nt = (int64_t)perm->T * (pt.d / 8);
  st = cuda(launch_k(k_token_sum, (unsigned)((nt + 255) / 256), 256, 0, cs, (const uint16_t*)dxr,
                     (const int32_t*)perm->pair_row, (const int32_t*)at<int32_t>(perm->ws, L.pair_g), pt.k, perm->T,
                     pt.d, dX, err),
            "ace_ffn_bwd: token sum launch");
  if (st != ACE_OK) return st;
  // the gate and up adapters: dX += their input gradient, dA, dB
  const uint16_t* Agu[2] = {A[0], A[1]};
  const uint16_t* Bgu[2] = {Bt[0], Bt[1]};
  const uint16_t* dYgu[2] = {dv, du};
  float* dAgu[2] = {dA[0], dA[1]};
  float* dBgu[2] = {dBt[0], dBt[1]};
  return ace_bwd_shared(plan, perm, 2, dYgu, X, Hgu, Agu, Bgu, s, dX, dAgu, dBgu, bws, bws_bytes, stream);
}

}  // extern "C"
