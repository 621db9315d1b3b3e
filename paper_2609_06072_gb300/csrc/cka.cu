// Linear CKA similarity of a layer's expert adapters on a probe set (Sec. 3.2,
// rank consolidation), without materialising the E representation matrices.
//
// With Z_e = X A_e^T B_e^T [N x d_out] and Xc = H X (H = I - 11^T / N),
//   Zc_i^T Zc_j = B_i M_ij B_j^T,   M_ij = A_i (Xc^T Xc) A_j^T   (r x r)
// so every Frobenius norm in CKA reduces to r x r products:
//   ||Zc_i^T Zc_j||_F^2 = tr(M_ij^T Gb_i M_ij Gb_j),  Gb_e = B_e^T B_e (r x r).
// The work is one K = N product Xc^T Xc (tensor cores: the dense dA GEMM of
// gemm.cu with the centred probe as both operands; the column means are
// taken out of X before the product, so a large mean cancels nothing),
// P = A (Xc^T Xc) and M = P A^T over the stacked expert ranks (fp32), the
// E Gram blocks Gb_e, and one small trace per expert pair.
#include <cmath>
#include <cstdint>

#include "ace_internal.cuh"
#include "ace_ptx.cuh"

namespace ace {
namespace {

constexpr int kColChunks = 64;  // row chunks of the probe column sums

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(uint16_t v) { return __uint_as_float((uint32_t)v << 16); }

// part[c][col] = sum of X[rows of chunk c][col]
__global__ void __launch_bounds__(256) k_colsum(const uint16_t* __restrict__ X, int N, int d, float* __restrict__ part) {
  const int col = blockIdx.x * 256 + threadIdx.x, c = blockIdx.y;
  if (col >= d) return;
  const int r0 = (int)((int64_t)c * N / kColChunks), r1 = (int)((int64_t)(c + 1) * N / kColChunks);
  float s = 0.f;
  for (int r = r0; r < r1; ++r) s += to_f(X[(int64_t)r * d + col]);
  part[(int64_t)c * d + col] = s;
}

// colsum[col] = sum over the chunks, in chunk order
__global__ void __launch_bounds__(256) k_colsum_total(const float* __restrict__ part, int d, float* __restrict__ colsum) {
  const int col = blockIdx.x * 256 + threadIdx.x;
  if (col >= d) return;
  float s = 0.f;
  for (int c = 0; c < kColChunks; ++c) s += part[(int64_t)c * d + col];
  colsum[col] = s;
}

// Xc = X - 1 mu^T with mu = colsum / N (fp32 arithmetic, bf16 out), 8 columns a thread
__global__ void __launch_bounds__(256) k_center_x(const uint16_t* __restrict__ X, const float* __restrict__ colsum,
                                                  int N, int d, uint16_t* __restrict__ Xc) {
  const int64_t idx = (int64_t)blockIdx.x * 256 + threadIdx.x;
  if (idx >= (int64_t)N * (d / 8)) return;
  const int64_t row = idx / (d / 8);
  const int c0 = (int)(idx % (d / 8)) * 8;
  const uint4 v = *reinterpret_cast<const uint4*>(X + row * d + c0);
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
  uint32_t o[4];
  const float inv_n = 1.f / (float)N;
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const float2 f = unpack_bf16x2(w[q]);
    o[q] = pack_bf16x2(f.x - colsum[c0 + 2 * q] * inv_n, f.y - colsum[c0 + 2 * q + 1] * inv_n);
  }
  *reinterpret_cast<uint4*>(Xc + row * d + c0) = make_uint4(o[0], o[1], o[2], o[3]);
}

// C[M x N] = A[M x K] . B with A row-major (lda) and B row-major [K x N]
// (B_NK false) or given as its transpose [N x K] (B_NK true); fp32 or bf16
// operands, fp32 accumulation.  64 x 64 tiles, 16 x 16 threads of 4 x 4.
template <typename TA, typename TB, bool B_NK>
__global__ void __launch_bounds__(256) k_sgemm(int M, int Nn, int K, const TA* __restrict__ A, int lda,
                                               const TB* __restrict__ B, int ldb, float* __restrict__ C, int ldc) {
  __shared__ float As[16][64 + 4];
  __shared__ float Bs[16][64 + 4];
  const int tid = threadIdx.x, tx = tid % 16, ty = tid / 16;
  const int m0 = blockIdx.y * 64, n0 = blockIdx.x * 64;
  float acc[4][4] = {};
  for (int k0 = 0; k0 < K; k0 += 16) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int idx = tid + q * 256, mm = idx / 16, kk = idx % 16, gm = m0 + mm, gk = k0 + kk;
      As[kk][mm] = (gm < M && gk < K) ? to_f(A[(int64_t)gm * lda + gk]) : 0.f;
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int idx = tid + q * 256;
      if (!B_NK) {
        const int kk = idx / 64, nn = idx % 64, gk = k0 + kk, gn = n0 + nn;
        Bs[kk][nn] = (gk < K && gn < Nn) ? to_f(B[(int64_t)gk * ldb + gn]) : 0.f;
      } else {
        const int nn = idx / 16, kk = idx % 16, gk = k0 + kk, gn = n0 + nn;
        Bs[kk][nn] = (gk < K && gn < Nn) ? to_f(B[(int64_t)gn * ldb + gk]) : 0.f;
      }
    }
    __syncthreads();
#pragma unroll
    for (int kk = 0; kk < 16; ++kk) {
      float av[4], bv[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) av[i] = As[kk][ty * 4 + i];
#pragma unroll
      for (int j = 0; j < 4; ++j) bv[j] = Bs[kk][tx * 4 + j];
#pragma unroll
      for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(av[i], bv[j], acc[i][j]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < 4; ++i)
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int gm = m0 + ty * 4 + i, gn = n0 + tx * 4 + j;
      if (gm < M && gn < Nn) C[(int64_t)gm * ldc + gn] = acc[i][j];
    }
}

// Gb_e[a][b] = sum_c Bt[e r + a][c] Bt[e r + b][c], one CTA per expert
__global__ void __launch_bounds__(256) k_gram_b(const uint16_t* __restrict__ Bt, int r, int d_out, float* __restrict__ Gb) {
  const int e = blockIdx.x;
  for (int p = threadIdx.x; p < r * r; p += 256) {
    const int a = p / r, b = p % r;
    const uint16_t* ra = Bt + (int64_t)(e * r + a) * d_out;
    const uint16_t* rb = Bt + (int64_t)(e * r + b) * d_out;
    float s = 0.f;
    for (int c = 0; c < d_out; ++c) s = fmaf(to_f(ra[c]), to_f(rb[c]), s);
    Gb[(int64_t)e * r * r + p] = s;
  }
}

// t_ij = tr(M_ij^T Gb_i M_ij Gb_j) = sum_ab (Gb_i M_ij)[a][b] (M_ij Gb_j)[a][b]
// for the expert pair (i, j) = (blockIdx.y, blockIdx.x); diag[i] = t_ii.
constexpr int kMaxCkaRank = 32;
__global__ void __launch_bounds__(128) k_cka_cross(const float* __restrict__ Mx, const float* __restrict__ Gb, int E,
                                                   int r, float* __restrict__ T, float* __restrict__ diag) {
  __shared__ float m[kMaxCkaRank][kMaxCkaRank + 1], gi[kMaxCkaRank][kMaxCkaRank + 1],
      gj[kMaxCkaRank][kMaxCkaRank + 1];
  __shared__ float red[4];
  const int i = blockIdx.y, j = blockIdx.x, ld = E * r;
  for (int p = threadIdx.x; p < r * r; p += 128) {
    const int a = p / r, b = p % r;
    m[a][b] = Mx[(int64_t)(i * r + a) * ld + j * r + b];
    gi[a][b] = Gb[(int64_t)i * r * r + p];
    gj[a][b] = Gb[(int64_t)j * r * r + p];
  }
  __syncthreads();
  float s = 0.f;
  for (int p = threadIdx.x; p < r * r; p += 128) {
    const int a = p / r, b = p % r;
    float x = 0.f, y = 0.f;
    for (int c = 0; c < r; ++c) {
      x = fmaf(gi[a][c], m[c][b], x);
      y = fmaf(m[a][c], gj[c][b], y);
    }
    s = fmaf(x, y, s);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    const float t = red[0] + red[1] + red[2] + red[3];
    T[(int64_t)i * E + j] = t;
    if (i == j) diag[i] = t;
  }
}

// S_ij = t_ij / sqrt(t_ii t_jj); NaN everywhere if the covariance GEMM's
// bounded wait gave up (err != 0)
__global__ void __launch_bounds__(256) k_cka_norm(float* __restrict__ S, const float* __restrict__ diag, int E,
                                                  const int32_t* __restrict__ err) {
  const int idx = blockIdx.x * 256 + threadIdx.x;
  if (idx >= E * E) return;
  const int i = idx / E, j = idx % E;
  const float den = sqrtf(diag[i]) * sqrtf(diag[j]);
  S[idx] = *err ? __int_as_float(0x7fc00000) : (den > 0.f ? S[idx] / den : 0.f);
}

// The groups' shared adapters at the consolidation step (Sec. 3.2, group-
// anchor appendix): rank row i of group g (k = i - rank_off[g]) copies row
// anchor_g * r + k of the expert-wise adapters when k < r, else A takes the
// caller's initialisation row i and B^T is zero.  One CTA per rank row.
struct ConsolidateParams {
  int32_t G, r, d_in, d_out;
  int32_t rank_off[ACE_MAX_EXPERTS + 1];
  int32_t anchor[ACE_MAX_EXPERTS];
};

__global__ void __launch_bounds__(256) k_consolidate(const __grid_constant__ ConsolidateParams p,
                                                     const uint16_t* __restrict__ A_e, const uint16_t* __restrict__ Bt_e,
                                                     const uint16_t* __restrict__ A_init, uint16_t* __restrict__ A_g,
                                                     uint16_t* __restrict__ Bt_g) {
  const int i = blockIdx.x;
  int lo = 0, hi = p.G;  // the group holding row i: largest g with rank_off[g] <= i
  while (hi - lo > 1) {
    const int mid = (lo + hi) >> 1;
    if (p.rank_off[mid] <= i)
      lo = mid;
    else
      hi = mid;
  }
  const int k = i - p.rank_off[lo];
  const bool anchor_row = k < p.r;
  const int64_t src = (int64_t)p.anchor[lo] * p.r + k;
  for (int c = threadIdx.x; c < p.d_in; c += 256)
    A_g[(int64_t)i * p.d_in + c] = anchor_row ? A_e[src * p.d_in + c] : A_init[(int64_t)i * p.d_in + c];
  for (int c = threadIdx.x; c < p.d_out; c += 256)
    Bt_g[(int64_t)i * p.d_out + c] = anchor_row ? Bt_e[src * p.d_out + c] : (uint16_t)0;
}

struct CkaWs {
  float *C, *part, *colsum, *P, *Mx, *Gb, *diag;
  uint16_t* Xc;  // the centred probe [N, d_in] bf16
  int32_t* err;
  size_t total;
};

CkaWs cka_layout(int N, int d_in, int E, int r, void* base) {
  CkaWs w{};
  char* b = static_cast<char*>(base);
  size_t off = 0;
  auto take = [&](size_t bytes) {
    char* p = b + off;
    off = align_up(off + bytes, 256);
    return p;
  };
  const size_t er = (size_t)E * r;
  w.C = reinterpret_cast<float*>(take(4 * (size_t)d_in * d_in));
  w.part = reinterpret_cast<float*>(take(4 * (size_t)kColChunks * d_in));
  w.colsum = reinterpret_cast<float*>(take(4 * (size_t)d_in));
  w.P = reinterpret_cast<float*>(take(4 * er * d_in));
  w.Mx = reinterpret_cast<float*>(take(4 * er * er));
  w.Gb = reinterpret_cast<float*>(take(4 * (size_t)E * r * r));
  w.diag = reinterpret_cast<float*>(take(4 * (size_t)E));
  w.err = reinterpret_cast<int32_t*>(take(16));
  w.Xc = reinterpret_cast<uint16_t*>(take(2 * (size_t)N * d_in));
  w.total = off;
  return w;
}

}  // namespace
}  // namespace ace

using namespace ace;

namespace {

ace_status cka_check(int32_t N, int32_t d_in, int32_t d_out, int32_t E, int32_t r) {
  if (N < 1 || d_in < 64 || d_in % 64 || d_out < 1 || E < 1 || E > ACE_MAX_EXPERTS || r < 1 || r > kMaxCkaRank)
    return report(ACE_ERR_SHAPE, "ace_cka: need N >= 1, d_in a positive multiple of 64, d_out >= 1, "
                                 "1 <= E <= ACE_MAX_EXPERTS, 1 <= r <= 32");
  return ACE_OK;
}

}  // namespace

extern "C" {

ace_status ace_cka_workspace_size(int32_t N, int32_t d_in, int32_t d_out, int32_t E, int32_t r, size_t* bytes) {
  ace_status st = cka_check(N, d_in, d_out, E, r);
  if (st != ACE_OK) return st;
  if (!bytes) return report(ACE_ERR_ARG, "ace_cka_workspace_size: null output");
  *bytes = cka_layout(N, d_in, E, r, nullptr).total;
  return ACE_OK;
}

ace_status ace_cka(int32_t N, int32_t d_in, int32_t d_out, int32_t E, int32_t r, const uint16_t* X, const uint16_t* A,
                   const uint16_t* Bt, int32_t center, float* S, void* ws, size_t ws_bytes, void* stream) {
  ace_status st = cka_check(N, d_in, d_out, E, r);
  if (st != ACE_OK) return st;
  if (!X || !A || !Bt || !S || !ws) return report(ACE_ERR_ARG, "ace_cka: null argument");
  auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
  if (!al16(X) || !al16(A) || !al16(Bt) || !al16(ws) || (reinterpret_cast<uintptr_t>(S) & 3u))
    return report(ACE_ERR_ARG, "ace_cka: misaligned tensor");
  const CkaWs w = cka_layout(N, d_in, E, r, ws);
  if (ws_bytes < w.total) return report(ACE_ERR_WORKSPACE, "ace_cka: workspace too small");
  int dev = 0, major = 0, minor = 0, nsm = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return report(ACE_ERR_CUDA, "ace_cka: cudaGetDevice failed");
  cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev);
  cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev);
  cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  if (!(major == 10 && minor == 3)) return report(ACE_ERR_UNSUPPORTED, "ace_cka: this library is built for sm_103a only");
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  // Xc^T Xc: the dense dA GEMM with the probe, centred first (center != 0),
  // as both operands
  cudaError_t e = cudaMemsetAsync(w.C, 0, 4 * (size_t)d_in * d_in, cs);
  if (e == cudaSuccess) e = cudaMemsetAsync(w.err, 0, 16, cs);
  const uint16_t* Xg = X;
  if (e == cudaSuccess && center) {
    k_colsum<<<dim3((d_in + 255) / 256, kColChunks), 256, 0, cs>>>(X, N, d_in, w.part);
    k_colsum_total<<<(d_in + 255) / 256, 256, 0, cs>>>(w.part, d_in, w.colsum);
    const int64_t nv = (int64_t)N * (d_in / 8);
    k_center_x<<<(unsigned)((nv + 255) / 256), 256, 0, cs>>>(X, w.colsum, N, d_in, w.Xc);
    e = cudaGetLastError();
    Xg = w.Xc;
  }
  DenseBwdLaunch g{};
  const uint64_t n = (uint64_t)N, di = (uint64_t)d_in;
  if (!make_tmap_bf16(&g.tm_dhx_t, Xg, n, di, 64) || !make_tmap_bf16(&g.tm_x, Xg, n, di, 64) ||
      !make_tmap_f32(&g.tm_da[0], w.C, di, di, 32))
    return report(ACE_ERR_UNSUPPORTED, "ace_cka: tensor-map encoding failed");
  g.tm_da[1] = g.tm_da[0];
  g.dA[0] = g.dA[1] = w.C;
  g.T = N;
  g.d = d_in;
  g.n_rank = d_in;
  g.n_rank_pad = d_in;
  g.nproj = 1;
  g.grid = nsm;
  g.err = w.err;
  if (e == cudaSuccess) e = launch_dense_da(g, cs);
  const int er = E * r;
  if (e == cudaSuccess) {
    // P = A . Cc  [er x d_in],  M = P . A^T  [er x er]
    k_sgemm<uint16_t, float, false><<<dim3((d_in + 63) / 64, (er + 63) / 64), 256, 0, cs>>>(er, d_in, d_in, A, d_in,
                                                                                             w.C, d_in, w.P, d_in);
    k_sgemm<float, uint16_t, true><<<dim3((er + 63) / 64, (er + 63) / 64), 256, 0, cs>>>(er, er, d_in, w.P, d_in, A,
                                                                                          d_in, w.Mx, er);
    k_gram_b<<<E, 256, 0, cs>>>(Bt, r, d_out, w.Gb);
    k_cka_cross<<<dim3(E, E), 128, 0, cs>>>(w.Mx, w.Gb, E, r, S, w.diag);
    k_cka_norm<<<(E * E + 255) / 256, 256, 0, cs>>>(S, w.diag, E, w.err);
    e = cudaGetLastError();
  }
  if (e != cudaSuccess) return report(ACE_ERR_CUDA, cudaGetErrorString(e));
  return ACE_OK;
}

ace_status ace_consolidate_adapters(int32_t E, int32_t r, int32_t d_in, int32_t d_out, const int32_t* e2g,
                                    const int32_t* anchors, int32_t G, const uint16_t* A_e, const uint16_t* Bt_e,
                                    const uint16_t* A_init, uint16_t* A_g, uint16_t* Bt_g, int32_t* rank_off,
                                    void* stream) {
  if (!e2g || !anchors || !rank_off || !A_e || !Bt_e || !A_init || !A_g || !Bt_g)
    return report(ACE_ERR_ARG, "ace_consolidate_adapters: null argument");
  if (E < 1 || E > ACE_MAX_EXPERTS || G < 1 || G > E || r < 1 || d_in < 1 || d_out < 1)
    return report(ACE_ERR_SHAPE, "ace_consolidate_adapters: need 1 <= G <= E <= ACE_MAX_EXPERTS, r, d_in, d_out >= 1");
  ConsolidateParams p{};
  p.G = G;
  p.r = r;
  p.d_in = d_in;
  p.d_out = d_out;
  int members[ACE_MAX_EXPERTS] = {0};
  for (int e = 0; e < E; ++e) {
    if (e2g[e] < 0 || e2g[e] >= G) return report(ACE_ERR_INDEX, "ace_consolidate_adapters: group out of range");
    ++members[e2g[e]];
  }
  p.rank_off[0] = 0;
  for (int g = 0; g < G; ++g) {
    if (members[g] == 0) return report(ACE_ERR_INDEX, "ace_consolidate_adapters: empty group");
    if (anchors[g] < 0 || anchors[g] >= E || e2g[anchors[g]] != g)
      return report(ACE_ERR_INDEX, "ace_consolidate_adapters: anchor is not a member of its group");
    p.anchor[g] = anchors[g];
    p.rank_off[g + 1] = p.rank_off[g] + r * members[g];
  }
  for (int g = 0; g <= G; ++g) rank_off[g] = p.rank_off[g];
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  k_consolidate<<<E * r, 256, 0, cs>>>(p, A_e, Bt_e, A_init, A_g, Bt_g);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? ACE_OK : report(ACE_ERR_CUDA, cudaGetErrorString(e));
}

}  // extern "C"
