/*
 * ace.h -- C ABI of the GB300 (sm_103a) grouped adapter execution library.
 *
 * The library implements the data-parallel hot path of ACE (arxiv 2609.06072):
 * the forward and backward passes of group-shared LoRA deltas on the MoE
 * expert gate / up / down projections.
 *
 *   Sec. 3.1  expert-wise MoE LoRA: y(x) = sum_{e in R(x)} p_e(x)(W_e x + B_e A_e x)
 *   Sec. 3.3  rank consolidation: one adapter Delta W_g = B_g A_g per group,
 *             A_g in R^{r_g x d_in}, B_g in R^{d_out x r_g}, r_g = sum_{e in G_g} r_e
 *   Sec. 3.4  every routed expert e uses Delta W_{g(e)}; the group adapter
 *             receives gradient from every pair routed into the group
 *   Sec. 3.5  grouped execution: c_g(x) = B_g (A_g x) is evaluated once per
 *             active group of a token and reused by all its routed experts
 *             of that group (gate / up, whose input x is shared)
 *   App. "Implementation and Profiling of Grouped Adapter Execution":
 *             gate/up take x, down takes the expert-specific h_e
 *
 * Beyond that path: the down delta taken through the router's gate-weighted
 * combine (ace_fwd_combine / ace_bwd_combine); rank consolidation, the step
 * that produces the expert -> group map (ace_cka, ace_group_experts,
 * ace_consolidate_adapters); and the routed expert FFN with frozen base
 * weights and the adapters together (ace_ffn_fwd / ace_ffn_bwd).
 *
 * Terms used below.  T tokens, top-k routing, pair p = t*k + j (token t,
 * slot j), R = T*k pairs.  E experts, G groups, e2g the expert->group map,
 * rank_off[G+1] the packed rank offsets (r_g = rank_off[g+1] - rank_off[g]).
 * d = hidden size (gate/up d_in, down d_out), f = expert intermediate size
 * (gate/up d_out, down d_in).  s = LoRA scale.
 *
 * Row order.  Every per-pair tensor the kernels touch is in ROW order: the
 * pairs sorted by (g(e), e, t), so expert segments are contiguous inside
 * group segments.  ace_permute produces the map (row_pair / pair_row).
 * Unique (token, group) pairs -- the set A(x) of Sec. 3.5 -- are sorted by
 * (g, t).
 *
 * Memory.  Every tensor pointer is a DEVICE pointer owned by the caller.
 * The library allocates no device memory: scratch space is a caller-owned
 * workspace sized by ace_workspace_size.  Tensors must be 16-byte aligned.
 * bf16 tensors are passed as `uint16_t*` holding the bf16 bit patterns; fp32
 * tensors as `float*`.  All matrices are row-major and dense.
 *
 * Streams / errors.  Every call is asynchronous on the caller's stream and
 * returns an ace_status.  Host-side checks (null pointers, shapes, limits,
 * workspace size, alignment) return an error WITHOUT launching.  Invalid
 * routing found on the device (expert id out of range, an expert repeated in
 * a token) sets a device flag; ace_get_error synchronises the stream, reads
 * and clears it.  No call synchronises otherwise, and none aborts, traps or
 * throws.  ace_last_error_message() gives a thread-local description of the
 * last host-side failure.
 *
 * Device.  Requires an sm_103 GPU (GB300).  Plans created on another device
 * fail with ACE_ERR_UNSUPPORTED; there is no fallback.
 */
#ifndef ACE_H_
#define ACE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define ACE_VERSION 1

typedef int32_t ace_status;
#define ACE_OK 0
#define ACE_ERR_ARG 1            /* null pointer or invalid scalar argument */
#define ACE_ERR_SHAPE 2          /* shape outside the plan or the supported limits */
#define ACE_ERR_WORKSPACE 3      /* workspace too small or misaligned */
#define ACE_ERR_INDEX 4          /* invalid routing or expert->group map */
#define ACE_ERR_UNSUPPORTED 5    /* device is not sm_103, or rank too large */
#define ACE_ERR_CUDA 6           /* a CUDA runtime call failed */
#define ACE_ERR_DEVICE_TIMEOUT 7 /* a bounded device-side wait gave up */
#define ACE_ERR_CHECK 8          /* libace_checks.so only: an index read from the
                                    permutation arrays, or a tile of a tile table,
                                    was outside its range; the access went to a safe
                                    index instead and the results are unspecified */

/* plan flags */
#define ACE_FLAG_DETERMINISTIC 1u /* dA / dB^T via fixed-order two-stage split-K (bitwise reproducible);
                                     otherwise fp32 atomics (any summation order) */
/* Test only, never for production use: exercises the bounded-wait failure
 * path.  With it, ace_fwd_row (when it computes the split row tiles' H up
 * front, i.e. with a saved H or forward scratch) never raises the ready flags
 * of that H, and the row kernel's wait on them gives up after 2 ms instead of
 * 1 s.  The call then ends early: ace_get_error returns
 * ACE_ERR_DEVICE_TIMEOUT, Y is unspecified, and the context stays usable. */
#define ACE_FLAG_TEST_WAIT_EXPIRY 2u

/* Limits. */
#define ACE_MAX_EXPERTS 512
#define ACE_MAX_RANK 128 /* max r_g of one group */

/* Layer description (host memory; copied into the plan). */
typedef struct ace_layer_desc {
  int32_t T_max;           /* largest T a call will use; T_max * k <= 2^30 */
  int32_t k;               /* top-k, 1 <= k <= E, k <= 32 */
  int32_t E;               /* experts, 1 <= E <= ACE_MAX_EXPERTS */
  int32_t G;               /* groups, 1 <= G <= E */
  const int32_t* e2g;      /* [E] expert -> group, values in [0, G); every group non-empty */
  const int32_t* rank_off; /* [G+1] rank offsets, rank_off[0] = 0, 1 <= r_g <= ACE_MAX_RANK */
  int32_t d;               /* hidden size, multiple of 8 */
  int32_t f;               /* expert intermediate size, multiple of 8 */
  uint32_t flags;          /* ACE_FLAG_* */
} ace_layer_desc;

typedef struct ace_plan ace_plan; /* opaque, host memory only */

/* Views into the permutation workspace filled by ace_permute (device pointers).
 * Row r is the r-th pair in (g(e), e, t) order.  All int32. */
typedef struct ace_perm {
  int32_t T;              /* tokens of this call */
  int32_t R;              /* T * k */
  int32_t* counts;        /* [8]: [0] U = #unique (g,t), [1] rows written */
  int32_t* group_off;     /* [G+1] first row of each group segment */
  int32_t* expert_off;    /* [E] first row of each expert segment */
  int32_t* expert_cnt;    /* [E] rows of each expert */
  int32_t* row_pair;      /* [R] pair index p = t*k + j held by row r */
  int32_t* pair_row;      /* [R] inverse of row_pair */
  int32_t* uniq_off;      /* [G+1] first unique pair of each group */
  int32_t* uniq_tok;      /* [R] token of unique pair u (first U entries valid) */
  int32_t* tok_uniq;      /* [T*k] unique pairs of token t, ascending g, then -1 */
  int32_t* row_uniq;      /* [R] unique pair (g, t) of the pair held by row r */
  void* ws;               /* the workspace these views point into */
} ace_perm;

int32_t ace_version(void);
const char* ace_last_error_message(void);

/* Create a plan on the current CUDA device.  Host-side validation of the
 * description (map in range, every group non-empty, ranks in limits). */
ace_status ace_plan_create(ace_plan** out, const ace_layer_desc* desc);
void ace_plan_destroy(ace_plan* plan);

/* Max over groups of r_g; the row stride (in elements) of every H / dH
 * buffer below. */
int32_t ace_plan_rank_max(const ace_plan* plan);

/* rank_off[G] rounded up to a multiple of 64: the row stride (in elements)
 * of the token-major combined H of ace_fwd_combine / ace_bwd_combine. */
int32_t ace_plan_rank_cols(const ace_plan* plan);

/* Workspace bytes for T tokens:
 *   perm_bytes  -- ace_permute (lives as long as the ace_perm views are used)
 *   fwd_bytes   -- forward scratch, used only when the call's H argument is NULL:
 *                  ace_fwd_shared keeps H per unique pair there, ace_fwd_row the H
 *                  of the rows of its last wave of tiles (computed first, so that
 *                  wave can run in column parts; with neither H nor scratch that
 *                  wave runs whole tiles)
 *   bwd_bytes   -- ace_bwd_shared / ace_bwd_row / ace_bwd_combine scratch
 * A NULL output pointer is skipped. */
ace_status ace_workspace_size(const ace_plan* plan, int32_t T, size_t* perm_bytes, size_t* fwd_bytes,
                              size_t* bwd_bytes);

/* Route-permute (Sec. 3.1 R(x), Sec. 3.5 A(x)).
 *   topk_idx  [T, k] int32 expert ids of each token (slot order as given)
 * Counts pairs per expert, exclusive-scans them in (g, e) order and scatters
 * the pairs, stable in t, into group-contiguous rows; builds the unique
 * (g, t) list and per-token unique lists.  Bit-exact and deterministic.
 * Invalid tokens (id out of [0,E) or a repeated id) raise the device flag
 * (ACE_ERR_INDEX from ace_get_error); their pairs are left out and the
 * outputs are then unspecified. */
ace_status ace_permute(const ace_plan* plan, const int32_t* topk_idx, int32_t T, void* perm_ws,
                       size_t perm_ws_bytes, ace_perm* out, void* stream);

/* Forward, shared input (gate / up; Sec. 3.5 and App. implementation).
 *   X       [T, d] bf16 token activations
 *   nproj   1 or 2 projections fused on the same X and the same map
 *   A[i]    [rank_off[G], d] bf16, rows rank_off[g].. hold A_g
 *   Bt[i]   [rank_off[G], f] bf16, rows rank_off[g].. hold B_g^T
 *   Y[i]    [R, f] bf16 IN/OUT in row order: Y[row] += s * B_g (A_g X[t])
 *   H[i]    [R, rank_max] fp32 OUT (NULL: kept in the forward workspace):
 *           H[u] = A_g X[t] for unique pair u (first U rows; columns >= r_g zero)
 * A_g x is computed once per unique (g, t) pair; the result B_g (A_g x) is
 * added to every row of that pair. */
ace_status ace_fwd_shared(const ace_plan* plan, const ace_perm* perm, const uint16_t* X, int32_t nproj,
                          const uint16_t* const* A, const uint16_t* const* Bt, float s, uint16_t* const* Y,
                          float* const* H, void* ws, size_t ws_bytes, void* stream);

/* Allocation-free variant of ace_fwd_shared for callers that cannot
 * allocate device memory (an inference server or plug-in host that reserves
 * the device memory for its own pool up front and gives a plug-in neither an
 * allocator nor a workspace).  The paper has no counterpart: this is a
 * deployment convenience.  Same arguments as ace_fwd_shared without H and
 * without the workspace: H is not returned, and the scratch it needs (2 x
 * T*k x rank_max fp32) lives in a 32 MiB array inside the library that every
 * GPU loading the library holds until the process exits.  Larger sizes fail
 * with ACE_ERR_WORKSPACE and launch nothing.  The first call in a CUDA
 * context (per device; again after cudaDeviceReset or when another context
 * is current) looks up the array's device address: make that call before
 * any stream capture.
 * All calls share the array: calls that overlap on the GPU race, so issue
 * them on one stream or otherwise order them.  Nothing in the array has to
 * start at zero: each call writes every scratch word it reads before reading
 * it.  Nothing is allocated. */
ace_status ace_fwd_shared_noalloc(const ace_plan* plan, const ace_perm* perm, const uint16_t* X, int32_t nproj,
                                  const uint16_t* const* A, const uint16_t* const* Bt, float s, uint16_t* const* Y,
                                  void* stream);

/* Forward, per row (down).
 *   Hin  [R, f] bf16 expert-specific inputs h_e in row order
 *   A    [rank_off[G], f] bf16 (A_g);  Bt [rank_off[G], d] bf16 (B_g^T)
 *   Y    [R, d] bf16 IN/OUT: Y[row] += s * B_g (A_g Hin[row])
 *   H    [R, rank_max] fp32 OUT or NULL: A_g Hin[row]
 *   ws   forward scratch (ace_workspace_size fwd_bytes) or NULL; read only when H is NULL */
ace_status ace_fwd_row(const ace_plan* plan, const ace_perm* perm, const uint16_t* Hin, const uint16_t* A,
                       const uint16_t* Bt, float s, uint16_t* Y, float* H, void* ws, size_t ws_bytes,
                       void* stream);

/* Backward, shared input (gate / up).  Adjoint of ace_fwd_shared:
 *   dY[i]   [R, f] bf16 row-order upstream gradients
 *   H[i]    [R, rank_max] fp32 saved by the forward (unique-pair rows)
 *   dX      [T, d] bf16 IN/OUT: dX[t] += sum_i sum_{u of t} s A_g^T (B_g^T dC_u),
 *           dC_u = sum of the dY rows of unique pair u
 *   dA[i]   [rank_off[G], d] fp32 OUT (overwritten): s sum_u (B_g^T dC_u) X[t_u]^T
 *   dBt[i]  [rank_off[G], f] fp32 OUT (overwritten): s sum_u H_u dC_u^T
 * Groups with no routed pair get exact zeros. */
ace_status ace_bwd_shared(const ace_plan* plan, const ace_perm* perm, int32_t nproj, const uint16_t* const* dY,
                          const uint16_t* X, const float* const* H, const uint16_t* const* A,
                          const uint16_t* const* Bt, float s, uint16_t* dX, float* const* dA, float* const* dBt,
                          void* ws, size_t ws_bytes, void* stream);

/* Backward, per row (down).
 *   dY    [R, d] bf16;  Hin [R, f] bf16;  H [R, rank_max] fp32 from ace_fwd_row
 *   dHin  [R, f] bf16 IN/OUT: dHin[row] += s A_g^T (B_g^T dY[row])
 *   dA    [rank_off[G], f] fp32 OUT;  dBt [rank_off[G], d] fp32 OUT */
ace_status ace_bwd_row(const ace_plan* plan, const ace_perm* perm, const uint16_t* dY, const uint16_t* Hin,
                       const float* H, const uint16_t* A, const uint16_t* Bt, float s, uint16_t* dHin, float* dA,
                       float* dBt, void* ws, size_t ws_bytes, void* stream);

/* Gate-weighted combine of the down projection, forward.  Sec. 3.1's
 * y(x) = sum_{e in R(x)} p_e(x) (W_e h_e + B_e A_e h_e) with expert e using the
 * group adapter of g(e) (Sec. 3.4): the adapter's share of the combined
 * output, in token rows.
 *   Hin     [R, f] bf16 expert inputs h_e in row order
 *   topk_w  [T, k] fp32 gate weights p, pair order (pair t*k + j); a non-finite
 *           weight sets the device flag (ACE_ERR_ARG from ace_get_error)
 *   A       [rank_off[G], f] bf16 (A_g);  Bt [rank_off[G], d] bf16 (B_g^T)
 *   Z       [T, d] bf16 IN/OUT: Z[t] += sum_j p[t,j] s B_g (A_g Hin[pair_row[t*k+j]])
 *   H       [R, rank_max] fp32 OUT: A_g Hin[row] (columns >= r_g zero)
 *   Hx      [T, ace_plan_rank_cols] bf16 OUT, the combined H:
 *           Hx[t][rank_off[g] + i] = s sum_{j: g(e_tj) = g} p[t,j] H[pair_row[t*k+j]][i]
 *           for i < r_g, every other column zero
 * By linearity the weighted sum over a token's experts of one group is taken
 * before B_g, so each token needs one product with the stacked B^T (K =
 * rank_off[G]) instead of one per routed expert.  H and Hx are the inputs
 * ace_bwd_combine needs.  Pairs of a token are summed in ascending j
 * (deterministic). */
ace_status ace_fwd_combine(const ace_plan* plan, const ace_perm* perm, const uint16_t* Hin, const float* topk_w,
                           const uint16_t* A, const uint16_t* Bt, float s, uint16_t* Z, float* H, uint16_t* Hx,
                           void* stream);

/* Backward of ace_fwd_combine for the token gradient dZ [T, d] bf16:
 *   H, Hx    from ace_fwd_combine
 *   dHin     [R, f] bf16 IN/OUT: dHin[row] += p s A_g^T (B_g^T dZ[t])
 *   dtopk_w  [T, k] fp32 OUT (overwritten): s (B_g^T dZ[t]) . (A_g Hin[row]), the
 *            adapter's share of the gate-weight gradient
 *   dA       [rank_off[G], f] fp32 OUT: s sum_rows p (B_g^T dZ[t]) Hin[row]^T
 *   dBt      [rank_off[G], d] fp32 OUT: sum_t Hx[t] dZ[t]^T over the group's columns
 *   ws       backward scratch (ace_workspace_size bwd_bytes)
 * B_g^T dZ[t] is formed once per unique (g, t) pair.  Groups with no routed
 * pair get exact zeros. */
ace_status ace_bwd_combine(const ace_plan* plan, const ace_perm* perm, const uint16_t* dZ, const uint16_t* Hin,
                           const float* topk_w, const float* H, const uint16_t* Hx, const uint16_t* A,
                           const uint16_t* Bt, float s, uint16_t* dHin, float* dtopk_w, float* dA, float* dBt,
                           void* ws, size_t ws_bytes, void* stream);

/* Linear CKA similarity of a layer's expert-wise adapters on a probe set
 * (Sec. 3.2): s_ij = ||Zc_i^T Zc_j||_F^2 / (||Zc_i^T Zc_i||_F ||Zc_j^T Zc_j||_F)
 * with Z_e = X A_e^T B_e^T and Zc_e = H Z_e, H = I - 11^T / N (center != 0) or
 * Zc_e = Z_e (center == 0; the centering appendix's other variant).
 *   X      [N, d_in] bf16 probe inputs (the same for every expert)
 *   A      [E * r, d_in] bf16, rows e*r.. hold A_e;  Bt [E * r, d_out] bf16 (B_e^T)
 *   S      [E, E] fp32 OUT
 *   ws     device workspace of ace_cka_workspace_size bytes
 * d_in a multiple of 64, r <= 32.  The representation matrices are never
 * formed: with M_ij = A_i (Xc^T Xc) A_j^T, every norm is an r x r trace; the
 * probe is centred (fp32 column means, bf16 Xc) before the product.  If
 * a bounded device wait gives up, S is filled with NaN.  Device pointers;
 * asynchronous on `stream`. */
ace_status ace_cka_workspace_size(int32_t N, int32_t d_in, int32_t d_out, int32_t E, int32_t r, size_t* bytes);
ace_status ace_cka(int32_t N, int32_t d_in, int32_t d_out, int32_t E, int32_t r, const uint16_t* X, const uint16_t* A,
                   const uint16_t* Bt, int32_t center, float* S, void* ws, size_t ws_bytes, void* stream);

/* The groups' shared adapters at the consolidation step (Sec. 3.2, group-anchor
 * appendix), from expert-wise adapters of rank r:
 *   e2g      [E] int32 HOST group of each expert (e.g. from ace_group_experts), G groups
 *   anchors  [G] int32 HOST anchor expert of each group (a member of it)
 *   A_e [E*r, d_in], Bt_e [E*r, d_out] bf16 device: the expert-wise adapters
 *   A_init   [E*r, d_in] bf16 device: LoRA initialisation rows for A (the caller's draw)
 *   A_g, Bt_g [E*r, d_in] / [E*r, d_out] bf16 device OUT: group g's rank rows
 *            rank_off[g].. start with its anchor's r rows of A_e / B_e^T; the
 *            rest take A_init's rows at the same positions and zero B^T rows
 *   rank_off [G+1] int32 HOST OUT: r_g = r |g|, the plan's rank offsets
 * At the consolidation step each group's Delta W_g therefore equals its
 * anchor's Delta W_e.  The budget is unchanged: sum_g r_g = E r. */
ace_status ace_consolidate_adapters(int32_t E, int32_t r, int32_t d_in, int32_t d_out, const int32_t* e2g,
                                    const int32_t* anchors, int32_t G, const uint16_t* A_e, const uint16_t* Bt_e,
                                    const uint16_t* A_init, uint16_t* A_g, uint16_t* Bt_g, int32_t* rank_off,
                                    void* stream);

/* Grouping of one layer's experts from their pairwise similarities, for rank
 * consolidation (Sec. 3.2; layer-wise graph construction, Louvain, fixed-
 * threshold and group-anchor appendices).  HOST memory, no GPU work:
 *   S        [E, E] fp32 host similarities (e.g. linear CKA of the adapters'
 *            outputs on a probe set), symmetrised as (S + S^T) / 2
 *   method   ACE_GROUP_LOUVAIN: Louvain on W = max(0, S' - median of the
 *            off-diagonal S'), zero diagonal, resolution `param` (the paper
 *            uses 0.8); ACE_GROUP_THRESHOLD: connected components of
 *            {(i, j): i != j, S'_ij >= param} (the paper's variant uses 0.9)
 *   e2g      [E] int32 host OUT: group of each expert, groups numbered in order
 *            of their smallest expert
 *   anchors  [E] int32 host OUT or NULL: the first G entries receive each
 *            group's CKA-centre anchor, the member with the largest sum of
 *            similarities to its group (ties to the lower index)
 *   G_out    OUT: number of groups
 * The consolidated ranks follow as r_g = sum of the members' ranks (rank_off
 * of the group plan).  Deterministic; double-precision arithmetic. */
#define ACE_GROUP_LOUVAIN 0
#define ACE_GROUP_THRESHOLD 1
ace_status ace_group_experts(const float* S, int32_t E, int32_t method, double param, int32_t* e2g,
                             int32_t* anchors, int32_t* G_out);

/* Routed expert FFN forward with the group-shared adapters (App. "Implementation
 * and Profiling of Grouped Adapter Execution"): for every row (pair t, e)
 *   u = (W_e^up + s B_g A_g) x_t,  v = (W_e^gate + s B_g A_g) x_t,
 *   h = SiLU(v) * u,  y = (W_e^down + s B_g A_g) h
 * with the plan's map for all three projections.  Composed from per-expert
 * base GEMMs and the adapter calls above (ace_fwd_shared for gate/up,
 * ace_fwd_row for down); u, v, h and y are rounded to bf16 between steps.
 *   X        [T, d] bf16 token inputs
 *   W_gate, W_up [E, f, d] bf16; W_down [E, d, f] bf16: frozen base weights
 *   A[3], Bt[3]  gate, up, down adapters (layouts as in ace_fwd_shared / ace_fwd_row)
 *   U, V, Hh [R, f] bf16 OUT (row order): u, v and h;  Y [R, d] bf16 OUT: y
 *   Hgu[2]   [R, rank_max] fp32 OUT: H of gate and up per unique pair
 *   Hd       [R, rank_max] fp32 OUT: H of down per row
 *   ws       ace_ffn_workspace_size bytes (the token rows in row order) */
ace_status ace_ffn_workspace_size(const ace_plan* plan, int32_t T, size_t* bytes);
ace_status ace_ffn_fwd(const ace_plan* plan, const ace_perm* perm, const uint16_t* X, const uint16_t* W_gate,
                       const uint16_t* W_up, const uint16_t* W_down, const uint16_t* const* A,
                       const uint16_t* const* Bt, float s, uint16_t* U, uint16_t* V, uint16_t* Hh, uint16_t* Y,
                       float* const* Hgu, float* Hd, void* ws, size_t ws_bytes, void* stream);

/* Backward of ace_ffn_fwd with frozen base weights, for the per-row output
 * gradient dY [R, d] bf16 (row order):
 *   dX       [T, d] bf16 OUT (overwritten): the token-input gradient through
 *            the three projections and the gating
 *   dA[3], dBt[3]  fp32 OUT: adapter gradients of gate, up, down
 *   U, V, Hh, Hgu, Hd  from ace_ffn_fwd;  ws: ace_ffn_workspace_size bytes;
 *   bws: the adapter backward workspace (ace_workspace_size bwd_bytes) */
ace_status ace_ffn_bwd(const ace_plan* plan, const ace_perm* perm, const uint16_t* dY, const uint16_t* X,
                       const uint16_t* W_gate, const uint16_t* W_up, const uint16_t* W_down, const uint16_t* const* A,
                       const uint16_t* const* Bt, float s, const uint16_t* U, const uint16_t* V, const uint16_t* Hh,
                       const float* const* Hgu, const float* Hd, uint16_t* dX, float* const* dA, float* const* dBt,
                       void* ws, size_t ws_bytes, void* bws, size_t bws_bytes, void* stream);

/* Row-order helpers (bf16, `cols` elements per row, cols multiple of 8):
 *   gather:  dst[row] = src[row_pair[row]]   (pair order -> row order)
 *   scatter: dst[row_pair[row]] = src[row]   (row order -> pair order) */
ace_status ace_gather_rows(const ace_perm* perm, const uint16_t* src_pairs, uint16_t* dst_rows, int32_t cols,
                           void* stream);
ace_status ace_scatter_rows(const ace_perm* perm, const uint16_t* src_rows, uint16_t* dst_pairs, int32_t cols,
                            void* stream);

/* Synchronises `stream`, then reads and clears the device error flag of the
 * permutation workspace: ACE_OK, ACE_ERR_INDEX (invalid routing),
 * ACE_ERR_DEVICE_TIMEOUT (a bounded wait gave up; results unspecified),
 * ACE_ERR_ARG (a non-finite gate weight reached ace_fwd_combine) or, in the
 * checked build, ACE_ERR_CHECK. */
ace_status ace_get_error(const ace_perm* perm, void* stream);

/* 1 in libace_checks.so, the debug build of the same sources compiled with
 * ACE_CHECKS: every kernel range-checks each index it reads from the
 * permutation arrays and each tile it takes from a tile table before using
 * it, and reports a violation as ACE_ERR_CHECK (the access goes to a safe
 * index; nothing faults or traps).  0 in libace.so, where the checks compile
 * away.  The two libraries export the same calls with the same semantics. */
int32_t ace_build_checks(void);

#ifdef __cplusplus
}
#endif
#endif /* ACE_H_ */
