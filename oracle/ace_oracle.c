/*
 * ACE grouped adapter execution -- plain fp64 CPU oracle.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call, link or
 * load this file; only the test suite, the smoke check and the CPU-baseline
 * leg of the benchmark do.  It shares no code, header, table or helper with
 * the CUDA library.
 *
 * It computes the plain definitions of the paper (arxiv 2609.06072), pair by
 * pair, with no deduplication, no permutation of the arithmetic and no
 * blocking:
 *
 *   Sec. 3.1 (expert-wise MoE LoRA):  y(x) = sum_{e in R(x)} p_e(x)(W_e x + B_e A_e x)
 *   Sec. 3.3 (rank consolidation):    Delta W_g = B_g A_g,  A_g in R^{r_g x d_in},
 *                                     B_g in R^{d_out x r_g}, r_g = sum_{e in G_g} r_e
 *   Sec. 3.4 (shared adapter output): expert e uses Delta W_{g(e)}
 *   Sec. 3.5 (grouped execution):     c_g(x) = B_g (A_g x) evaluated per active
 *                                     group and reused -- an exact rewrite, so
 *                                     the oracle simply evaluates it per pair.
 *   App. "Implementation and Profiling of Grouped Adapter Execution": gate/up
 *   take the token input x, down takes the expert-specific h_e.
 *
 * Gradients are the adjoint of that definition (Sec. 3.1.2 gives the
 * expert-wise form dL/dDeltaW_e = sum_n 1[e in R(x_n)] (.) dy x^T):
 *   dA_g  = s * sum_{pairs p in g} (B_g^T dy_p) x_p^T
 *   dB_g  = s * sum_{pairs p in g} dy_p (A_g x_p)^T          (stored transposed)
 *   dx_p  = s * A_g^T (B_g^T dy_p)   (summed over a token's pairs for gate/up)
 *
 * The gate-weighted combine of the down projection (the oracle_combine_*
 * functions) carries the router weight p_e(x) of Sec. 3.1 into the sum over
 * a token's routed experts and returns token rows; its gradients are the
 * adjoint of that sum, including the gradient of each gate weight.
 *
 * The routing permutation is a stable sort of the (token, slot) pairs by the
 * key (g(e), e, t) -- the row order the library documents -- computed with
 * the C library's qsort on unique keys.
 *
 * bf16 inputs are passed as their raw 16-bit patterns and decoded exactly;
 * all arithmetic is double precision.  Reductions run serially in a fixed
 * order per output element, so results are identical for any thread count.
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define OR_OK 0
#define OR_ERR_ARG 1
#define OR_ERR_INDEX 4

static double bf16_to_f64(uint16_t h) {
  union { uint32_t u; float f; } v;
  v.u = (uint32_t)h << 16;
  return (double)v.f;
}

int oracle_version(void) { return 1; }

/* ------------------------------------------------------------------ routing */

typedef struct { int32_t g, e, t, p; } pair_key;

static int cmp_pair_key(const void* a, const void* b) {
  const pair_key* x = (const pair_key*)a;
  const pair_key* y = (const pair_key*)b;
  if (x->g != y->g) return x->g < y->g ? -1 : 1;
  if (x->e != y->e) return x->e < y->e ? -1 : 1;
  if (x->t != y->t) return x->t < y->t ? -1 : 1;
  return 0;
}

typedef struct { int32_t g, t; } gt_key;

static int cmp_gt_key(const void* a, const void* b) {
  const gt_key* x = (const gt_key*)a;
  const gt_key* y = (const gt_key*)b;
  if (x->g != y->g) return x->g < y->g ? -1 : 1;
  if (x->t != y->t) return x->t < y->t ? -1 : 1;
  return 0;
}

/*
 * Validates the routing (Sec. 3.1: R(x) is a set of k distinct experts in
 * [0, E)) and the map g(e) in [0, G) (Sec. 3.3), then builds:
 *   group_off[G+1]   first row of each group segment (rows sorted by (g,e,t))
 *   expert_off[E]    first row of each expert segment, expert_cnt[E] its size
 *   row_pair[R]      pair index p = t*k + j held by each row; pair_row[R] its inverse
 *   uniq_off[G+1]    first unique (g,t) entry of each group   (Sec. 3.5, A(x))
 *   uniq_tok[U]      token of each unique (g,t), sorted by (g,t)
 *   uniq_rows_ptr[U+1], uniq_rows[R]  the rows of each unique pair, ascending e
 *   row_uniq[R]      unique pair of each row
 *   tok_uniq[T*k]    unique pairs of each token, ascending g, -1 padded
 *   *U_out           number of unique (g,t) pairs
 */
int oracle_permute(int32_t T, int32_t k, int32_t E, int32_t G, const int32_t* topk_idx,
                   const int32_t* e2g, int32_t* group_off, int32_t* expert_off, int32_t* expert_cnt,
                   int32_t* row_pair, int32_t* pair_row, int32_t* row_uniq, int32_t* uniq_off,
                   int32_t* uniq_tok, int32_t* uniq_rows_ptr, int32_t* uniq_rows, int32_t* tok_uniq,
                   int32_t* U_out) {
  if (T < 0 || k < 1 || E < 1 || G < 1 || k > E) return OR_ERR_ARG;
  for (int32_t e = 0; e < E; ++e)
    if (e2g[e] < 0 || e2g[e] >= G) return OR_ERR_INDEX;
  const int64_t R = (int64_t)T * k;
  for (int32_t t = 0; t < T; ++t)
    for (int32_t j = 0; j < k; ++j) {
      int32_t e = topk_idx[(int64_t)t * k + j];
      if (e < 0 || e >= E) return OR_ERR_INDEX;
      for (int32_t jj = 0; jj < j; ++jj)
        if (topk_idx[(int64_t)t * k + jj] == e) return OR_ERR_INDEX;
    }

  pair_key* keys = (pair_key*)malloc(sizeof(pair_key) * (R > 0 ? R : 1));
  gt_key* gts = (gt_key*)malloc(sizeof(gt_key) * (R > 0 ? R : 1));
  if (!keys || !gts) { free(keys); free(gts); return OR_ERR_ARG; }
  for (int64_t p = 0; p < R; ++p) {
    int32_t e = topk_idx[p];
    keys[p].g = e2g[e];
    keys[p].e = e;
    keys[p].t = (int32_t)(p / k);
    keys[p].p = (int32_t)p;
    gts[p].g = e2g[e];
    gts[p].t = (int32_t)(p / k);
  }
  qsort(keys, (size_t)R, sizeof(pair_key), cmp_pair_key);
  for (int64_t r = 0; r < R; ++r) {
    row_pair[r] = keys[r].p;
    pair_row[keys[r].p] = (int32_t)r;
  }
  /* segment offsets: counts, then exclusive scans in (g, e) order; an empty
     expert's segment is the empty range at the place it would occupy */
  for (int32_t g = 0; g <= G; ++g) group_off[g] = 0;
  for (int32_t e = 0; e < E; ++e) expert_cnt[e] = 0;
  for (int64_t r = 0; r < R; ++r) {
    group_off[keys[r].g + 1] += 1;
    expert_cnt[keys[r].e] += 1;
  }
  for (int32_t g = 0; g < G; ++g) group_off[g + 1] += group_off[g];
  for (int32_t e = 0; e < E; ++e) {
    int32_t start = group_off[e2g[e]];
    for (int32_t e2 = 0; e2 < e; ++e2)
      if (e2g[e2] == e2g[e]) start += expert_cnt[e2];
    expert_off[e] = start;
  }

  /* distinct (g,t), sorted */
  qsort(gts, (size_t)R, sizeof(gt_key), cmp_gt_key);
  int32_t U = 0;
  for (int32_t g = 0; g <= G; ++g) uniq_off[g] = 0;
  for (int64_t i = 0; i < R; ++i) {
    if (i > 0 && gts[i].g == gts[i - 1].g && gts[i].t == gts[i - 1].t) continue;
    gts[U] = gts[i];
    uniq_tok[U] = gts[i].t;
    uniq_off[gts[i].g + 1] += 1;
    ++U;
  }
  for (int32_t g = 0; g < G; ++g) uniq_off[g + 1] += uniq_off[g];
  *U_out = U;

  /* rows of each unique pair: scan rows in (g,e,t) order, so ascending e */
  int32_t* cnt = (int32_t*)calloc((size_t)U + 1, sizeof(int32_t));
  for (int64_t r = 0; r < R; ++r) {
    gt_key q = {keys[r].g, keys[r].t};
    gt_key* hit = (gt_key*)bsearch(&q, gts, (size_t)U, sizeof(gt_key), cmp_gt_key);
    int32_t u = (int32_t)(hit - gts);
    row_uniq[r] = u;
    cnt[u] += 1;
  }
  uniq_rows_ptr[0] = 0;
  for (int32_t u = 0; u < U; ++u) uniq_rows_ptr[u + 1] = uniq_rows_ptr[u] + cnt[u];
  for (int32_t u = 0; u < U; ++u) cnt[u] = 0;
  for (int64_t r = 0; r < R; ++r) {
    int32_t u = row_uniq[r];
    uniq_rows[uniq_rows_ptr[u] + cnt[u]] = (int32_t)r;
    cnt[u] += 1;
  }
  /* per-token list of its unique pairs, ascending g (u is sorted by (g,t)) */
  for (int64_t i = 0; i < R; ++i) tok_uniq[i] = -1;
  int32_t* tcnt = (int32_t*)calloc((size_t)T + 1, sizeof(int32_t));
  for (int32_t u = 0; u < U; ++u) {
    int32_t t = uniq_tok[u];
    tok_uniq[(int64_t)t * k + tcnt[t]] = u;
    tcnt[t] += 1;
  }
  free(tcnt);
  free(cnt);
  free(keys);
  free(gts);
  return OR_OK;
}

/* ------------------------------------------------------------------ forward */

/*
 * LoRA delta of one projection, per pair p = t*k + j with e = topk_idx[p],
 * g = e2g[e] (Sec. 3.3-3.5):
 *   H_p      = A_g x_p                         (r_g values)
 *   y_out[p] = y_in[p] + s * B_g H_p           (d_out values)
 * x_p = X[t] when x_per_pair == 0 (gate/up: shared input), else X[p] (down).
 * B_g is given transposed: Bt_all holds B_g^T as rows rank_off[g]..rank_off[g+1]-1.
 * y_in may be NULL (taken as zero).  When sel != NULL only the pairs
 * sel[0..n_sel) are computed and output row i holds pair sel[i] (compact).
 * h_out (may be NULL) receives H_p, padded with zeros to r_max entries.
 */
int oracle_fwd(int32_t T, int32_t k, int32_t E, int32_t G, const int32_t* topk_idx, const int32_t* e2g,
               const int32_t* rank_off, int32_t d_in, int32_t d_out, const uint16_t* X, int32_t x_per_pair,
               const uint16_t* A_all, const uint16_t* Bt_all, double s, const uint16_t* y_in, double* y_out,
               double* h_out, int32_t r_max, const int32_t* sel, int64_t n_sel) {
  if (T < 0 || k < 1 || d_in < 1 || d_out < 1) return OR_ERR_ARG;
  for (int32_t g = 0; g < G; ++g)
    if (rank_off[g + 1] - rank_off[g] < 0 || rank_off[g + 1] - rank_off[g] > 1024) return OR_ERR_ARG;
  const int64_t R = (int64_t)T * k;
  const int64_t n = sel ? n_sel : R;
  for (int64_t i = 0; i < n; ++i) {
    int64_t p = sel ? sel[i] : i;
    if (p < 0 || p >= R) return OR_ERR_INDEX;
    int32_t e = topk_idx[p];
    if (e < 0 || e >= E || e2g[e] < 0 || e2g[e] >= G) return OR_ERR_INDEX;
  }
#pragma omp parallel for schedule(dynamic, 16)
  for (int64_t i = 0; i < n; ++i) {
    int64_t p = sel ? sel[i] : i;
    int32_t g = e2g[topk_idx[p]];
    int32_t r0 = rank_off[g], rg = rank_off[g + 1] - rank_off[g];
    const uint16_t* x = X + (x_per_pair ? p : p / k) * (int64_t)d_in;
    double H[1024];
    for (int32_t i_r = 0; i_r < rg; ++i_r) {
      const uint16_t* a = A_all + (int64_t)(r0 + i_r) * d_in;
      double acc = 0.0;
      for (int32_t c = 0; c < d_in; ++c) acc += bf16_to_f64(a[c]) * bf16_to_f64(x[c]);
      H[i_r] = acc;
    }
    const int64_t o_row = sel ? i : p;
    if (h_out) {
      for (int32_t i_r = 0; i_r < r_max; ++i_r) h_out[o_row * r_max + i_r] = i_r < rg ? H[i_r] : 0.0;
    }
    for (int32_t o = 0; o < d_out; ++o) {
      double acc = 0.0;
      for (int32_t i_r = 0; i_r < rg; ++i_r) acc += bf16_to_f64(Bt_all[(int64_t)(r0 + i_r) * d_out + o]) * H[i_r];
      double base = y_in ? bf16_to_f64(y_in[p * (int64_t)d_out + o]) : 0.0;
      y_out[o_row * (int64_t)d_out + o] = base + s * acc;
    }
  }
  return OR_OK;
}

/* ----------------------------------------------------------------- backward */

/*
 * Input gradient of one projection (adjoint of oracle_fwd):
 *   x_per_pair == 0 : dx_out[t] = dx_in[t] + sum_j s * A_g^T (B_g^T dy_{t*k+j})   (token rows)
 *   x_per_pair == 1 : dx_out[p] = dx_in[p] + s * A_g^T (B_g^T dy_p)              (pair rows)
 * dy is pair-ordered [T*k, d_out].  dx_in may be NULL.  sel lists the tokens
 * (or pairs) to compute, output row i holding sel[i]; NULL = all.
 */
int oracle_bwd_dx(int32_t T, int32_t k, int32_t E, int32_t G, const int32_t* topk_idx, const int32_t* e2g,
                  const int32_t* rank_off, int32_t d_in, int32_t d_out, int32_t x_per_pair, const uint16_t* dy,
                  const uint16_t* A_all, const uint16_t* Bt_all, double s, const uint16_t* dx_in, double* dx_out,
                  const int32_t* sel, int64_t n_sel) {
  if (T < 0 || k < 1 || d_in < 1 || d_out < 1) return OR_ERR_ARG;
  const int64_t R = (int64_t)T * k;
  const int64_t n_rows = x_per_pair ? R : T;
  const int64_t n = sel ? n_sel : n_rows;
  for (int64_t i = 0; i < n; ++i) {
    int64_t q = sel ? sel[i] : i;
    if (q < 0 || q >= n_rows) return OR_ERR_INDEX;
  }
  for (int64_t p = 0; p < R; ++p) {
    int32_t e = topk_idx[p];
    if (e < 0 || e >= E || e2g[e] < 0 || e2g[e] >= G) return OR_ERR_INDEX;
  }
#pragma omp parallel for schedule(dynamic, 8)
  for (int64_t i = 0; i < n; ++i) {
    int64_t q = sel ? sel[i] : i;
    double* out = dx_out + (sel ? i : q) * (int64_t)d_in;
    for (int32_t c = 0; c < d_in; ++c) out[c] = dx_in ? bf16_to_f64(dx_in[q * (int64_t)d_in + c]) : 0.0;
    int64_t p_lo = x_per_pair ? q : q * k;
    int64_t p_hi = x_per_pair ? q + 1 : q * k + k;
    for (int64_t p = p_lo; p < p_hi; ++p) {
      int32_t g = e2g[topk_idx[p]];
      int32_t r0 = rank_off[g], rg = rank_off[g + 1] - rank_off[g];
      const uint16_t* dyp = dy + p * (int64_t)d_out;
      for (int32_t i_r = 0; i_r < rg; ++i_r) {
        const uint16_t* bt = Bt_all + (int64_t)(r0 + i_r) * d_out;
        double w = 0.0; /* (B_g^T dy_p)[i_r] */
        for (int32_t o = 0; o < d_out; ++o) w += bf16_to_f64(bt[o]) * bf16_to_f64(dyp[o]);
        const uint16_t* a = A_all + (int64_t)(r0 + i_r) * d_in;
        for (int32_t c = 0; c < d_in; ++c) out[c] += s * w * bf16_to_f64(a[c]);
      }
    }
  }
  return OR_OK;
}

/*
 * Weight gradients of one projection (shared adapter updates, Sec. 3.4: the
 * group adapter receives gradient from every pair routed to any expert of
 * its group):
 *   dA[i][c]  = s * sum_{p: g(e_p)=g(i)} (B_g^T dy_p)[i] * x_p[c]
 *   dBt[i][o] = s * sum_{p: g(e_p)=g(i)} (A_g x_p)[i]   * dy_p[o]
 * for every global rank row i (group g(i) owns rows rank_off[g]..rank_off[g+1]-1).
 * Pairs are visited in ascending p.  Groups with no pairs get exact zeros.
 * sel lists the rank rows to compute, output row ii holding rank row sel[ii];
 * NULL = all rank_off[G] rows.
 */
int oracle_bwd_w(int32_t T, int32_t k, int32_t E, int32_t G, const int32_t* topk_idx, const int32_t* e2g,
                 const int32_t* rank_off, int32_t d_in, int32_t d_out, const uint16_t* X, int32_t x_per_pair,
                 const uint16_t* dy, const uint16_t* A_all, const uint16_t* Bt_all, double s, double* dA,
                 double* dBt, const int32_t* sel, int64_t n_sel) {
  if (T < 0 || k < 1 || d_in < 1 || d_out < 1) return OR_ERR_ARG;
  const int64_t R = (int64_t)T * k;
  const int32_t n_rank = rank_off[G];
  const int64_t n = sel ? n_sel : n_rank;
  for (int64_t i = 0; i < n; ++i) {
    int64_t q = sel ? sel[i] : i;
    if (q < 0 || q >= n_rank) return OR_ERR_INDEX;
  }
  for (int64_t p = 0; p < R; ++p) {
    int32_t e = topk_idx[p];
    if (e < 0 || e >= E || e2g[e] < 0 || e2g[e] >= G) return OR_ERR_INDEX;
  }
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t ii = 0; ii < n; ++ii) {
    int32_t i = (int32_t)(sel ? sel[ii] : ii);
    int32_t g = 0;
    while (!(rank_off[g] <= i && i < rank_off[g + 1])) ++g;
    double* da = dA + (sel ? ii : (int64_t)i) * d_in;
    double* db = dBt + (sel ? ii : (int64_t)i) * d_out;
    for (int32_t c = 0; c < d_in; ++c) da[c] = 0.0;
    for (int32_t o = 0; o < d_out; ++o) db[o] = 0.0;
    const uint16_t* a = A_all + (int64_t)i * d_in;
    const uint16_t* bt = Bt_all + (int64_t)i * d_out;
    for (int64_t p = 0; p < R; ++p) {
      if (e2g[topk_idx[p]] != g) continue;
      const uint16_t* x = X + (x_per_pair ? p : p / k) * (int64_t)d_in;
      const uint16_t* dyp = dy + p * (int64_t)d_out;
      double w = 0.0, hv = 0.0;
      for (int32_t o = 0; o < d_out; ++o) w += bf16_to_f64(bt[o]) * bf16_to_f64(dyp[o]);
      for (int32_t c = 0; c < d_in; ++c) hv += bf16_to_f64(a[c]) * bf16_to_f64(x[c]);
      for (int32_t c = 0; c < d_in; ++c) da[c] += s * w * bf16_to_f64(x[c]);
      for (int32_t o = 0; o < d_out; ++o) db[o] += s * hv * bf16_to_f64(dyp[o]);
    }
  }
  return OR_OK;
}

/* --------------------------------------------- gate-weighted combine (down) */

/*
 * The down projection's adapter delta taken through the router's combine
 * (Sec. 3.1: y(x) = sum_{e in R(x)} p_e(x) (W_e h_e + B_e A_e h_e), with
 * expert e using the group adapter of g(e) as in Sec. 3.4):
 *   z_out[t] = z_in[t] + sum_j w_p * s * B_g (A_g h_p),   p = t*k + j, g = g(e_p)
 * h is pair-ordered [T*k, d_in], w the gate weights [T*k] (fp32), z token
 * rows [T, d_out].  z_in may be NULL.  sel lists the tokens to compute,
 * output row i holding token sel[i]; NULL = all.  Pairs of a token are
 * summed in ascending j.
 */
int oracle_combine_fwd(int32_t T, int32_t k, int32_t E, int32_t G, const int32_t* topk_idx, const int32_t* e2g,
                       const int32_t* rank_off, int32_t d_in, int32_t d_out, const uint16_t* h, const float* w,
                       const uint16_t* A_all, const uint16_t* Bt_all, double s, const uint16_t* z_in,
                       double* z_out, const int32_t* sel, int64_t n_sel) {
  if (T < 0 || k < 1 || d_in < 1 || d_out < 1) return OR_ERR_ARG;
  for (int32_t g = 0; g < G; ++g)
    if (rank_off[g + 1] - rank_off[g] < 0 || rank_off[g + 1] - rank_off[g] > 1024) return OR_ERR_ARG;
  const int64_t R = (int64_t)T * k;
  const int64_t n = sel ? n_sel : T;
  for (int64_t i = 0; i < n; ++i) {
    int64_t t = sel ? sel[i] : i;
    if (t < 0 || t >= T) return OR_ERR_INDEX;
  }
  for (int64_t p = 0; p < R; ++p) {
    int32_t e = topk_idx[p];
    if (e < 0 || e >= E || e2g[e] < 0 || e2g[e] >= G) return OR_ERR_INDEX;
  }
#pragma omp parallel for schedule(dynamic, 8)
  for (int64_t i = 0; i < n; ++i) {
    int64_t t = sel ? sel[i] : i;
    double* z = z_out + i * (int64_t)d_out;
    for (int32_t o = 0; o < d_out; ++o) z[o] = z_in ? bf16_to_f64(z_in[t * (int64_t)d_out + o]) : 0.0;
    for (int64_t p = t * k; p < t * k + k; ++p) {
      int32_t g = e2g[topk_idx[p]];
      int32_t r0 = rank_off[g], rg = rank_off[g + 1] - rank_off[g];
      const uint16_t* x = h + p * (int64_t)d_in;
      double H[1024];
      for (int32_t i_r = 0; i_r < rg; ++i_r) {
        const uint16_t* a = A_all + (int64_t)(r0 + i_r) * d_in;
        double acc = 0.0;
        for (int32_t c = 0; c < d_in; ++c) acc += bf16_to_f64(a[c]) * bf16_to_f64(x[c]);
        H[i_r] = acc;
      }
      const double wp = (double)w[p];
      for (int32_t o = 0; o < d_out; ++o) {
        double acc = 0.0;
        for (int32_t i_r = 0; i_r < rg; ++i_r) acc += bf16_to_f64(Bt_all[(int64_t)(r0 + i_r) * d_out + o]) * H[i_r];
        z[o] += wp * s * acc;
      }
    }
  }
  return OR_OK;
}

/*
 * Input and gate-weight gradients of oracle_combine_fwd for a token-space
 * output gradient dz [T, d_out]:
 *   dh_out[p] = dh_in[p] + w_p * s * A_g^T (B_g^T dz_t)     (pair rows [T*k, d_in])
 *   dw[p]     = s * (B_g^T dz_t) . (A_g h_p)                  (only the adapter's share)
 * dh_in may be NULL.  sel lists the pairs to compute, output row i holding
 * pair sel[i]; NULL = all.
 */
int oracle_combine_bwd_dh(int32_t T, int32_t k, int32_t E, int32_t G, const int32_t* topk_idx,
                          const int32_t* e2g, const int32_t* rank_off, int32_t d_in, int32_t d_out,
                          const uint16_t* dz, const uint16_t* h, const float* w, const uint16_t* A_all,
                          const uint16_t* Bt_all, double s, const uint16_t* dh_in, double* dh_out, double* dw,
                          const int32_t* sel, int64_t n_sel) {
  if (T < 0 || k < 1 || d_in < 1 || d_out < 1) return OR_ERR_ARG;
  for (int32_t g = 0; g < G; ++g)
    if (rank_off[g + 1] - rank_off[g] < 0 || rank_off[g + 1] - rank_off[g] > 1024) return OR_ERR_ARG;
  const int64_t R = (int64_t)T * k;
  const int64_t n = sel ? n_sel : R;
  for (int64_t i = 0; i < n; ++i) {
    int64_t p = sel ? sel[i] : i;
    if (p < 0 || p >= R) return OR_ERR_INDEX;
  }
  for (int64_t p = 0; p < R; ++p) {
    int32_t e = topk_idx[p];
    if (e < 0 || e >= E || e2g[e] < 0 || e2g[e] >= G) return OR_ERR_INDEX;
  }
#pragma omp parallel for schedule(dynamic, 16)
  for (int64_t i = 0; i < n; ++i) {
    int64_t p = sel ? sel[i] : i;
    int64_t t = p / k;
    int32_t g = e2g[topk_idx[p]];
    int32_t r0 = rank_off[g], rg = rank_off[g + 1] - rank_off[g];
    const uint16_t* dzt = dz + t * (int64_t)d_out;
    const uint16_t* x = h + p * (int64_t)d_in;
    double* out = dh_out + i * (int64_t)d_in;
    for (int32_t c = 0; c < d_in; ++c) out[c] = dh_in ? bf16_to_f64(dh_in[p * (int64_t)d_in + c]) : 0.0;
    const double wp = (double)w[p];
    double dwp = 0.0;
    for (int32_t i_r = 0; i_r < rg; ++i_r) {
      const uint16_t* bt = Bt_all + (int64_t)(r0 + i_r) * d_out;
      const uint16_t* a = A_all + (int64_t)(r0 + i_r) * d_in;
      double v = 0.0; /* (B_g^T dz_t)[i_r] */
      for (int32_t o = 0; o < d_out; ++o) v += bf16_to_f64(bt[o]) * bf16_to_f64(dzt[o]);
      double hv = 0.0; /* (A_g h_p)[i_r] */
      for (int32_t c = 0; c < d_in; ++c) hv += bf16_to_f64(a[c]) * bf16_to_f64(x[c]);
      for (int32_t c = 0; c < d_in; ++c) out[c] += wp * s * v * bf16_to_f64(a[c]);
      dwp += s * v * hv;
    }
    if (dw) dw[i] = dwp;
  }
  return OR_OK;
}

/*
 * Weight gradients of oracle_combine_fwd (shared adapter updates, Sec. 3.4):
 *   dA[i][c]  = s * sum_{p: g(e_p)=g(i)} w_p (B_g^T dz_t)[i] * h_p[c]
 *   dBt[i][o] = s * sum_{p: g(e_p)=g(i)} w_p (A_g h_p)[i]   * dz_t[o]
 * Pairs are visited in ascending p; groups with no pairs get exact zeros.
 * sel lists the rank rows to compute (output row ii = rank row sel[ii]).
 */
int oracle_combine_bwd_w(int32_t T, int32_t k, int32_t E, int32_t G, const int32_t* topk_idx,
                         const int32_t* e2g, const int32_t* rank_off, int32_t d_in, int32_t d_out,
                         const uint16_t* h, const uint16_t* dz, const float* w, const uint16_t* A_all,
                         const uint16_t* Bt_all, double s, double* dA, double* dBt, const int32_t* sel,
                         int64_t n_sel) {
  if (T < 0 || k < 1 || d_in < 1 || d_out < 1) return OR_ERR_ARG;
  const int64_t R = (int64_t)T * k;
  const int32_t n_rank = rank_off[G];
  const int64_t n = sel ? n_sel : n_rank;
  for (int64_t i = 0; i < n; ++i) {
    int64_t q = sel ? sel[i] : i;
    if (q < 0 || q >= n_rank) return OR_ERR_INDEX;
  }
  for (int64_t p = 0; p < R; ++p) {
    int32_t e = topk_idx[p];
    if (e < 0 || e >= E || e2g[e] < 0 || e2g[e] >= G) return OR_ERR_INDEX;
  }
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t ii = 0; ii < n; ++ii) {
    int32_t i = (int32_t)(sel ? sel[ii] : ii);
    int32_t g = 0;
    while (!(rank_off[g] <= i && i < rank_off[g + 1])) ++g;
    double* da = dA + ii * (int64_t)d_in;
    double* db = dBt + ii * (int64_t)d_out;
    for (int32_t c = 0; c < d_in; ++c) da[c] = 0.0;
    for (int32_t o = 0; o < d_out; ++o) db[o] = 0.0;
    const uint16_t* a = A_all + (int64_t)i * d_in;
    const uint16_t* bt = Bt_all + (int64_t)i * d_out;
    for (int64_t p = 0; p < R; ++p) {
      if (e2g[topk_idx[p]] != g) continue;
      const uint16_t* x = h + p * (int64_t)d_in;
      const uint16_t* dzt = dz + (p / k) * (int64_t)d_out;
      const double wp = (double)w[p];
      double v = 0.0, hv = 0.0;
      for (int32_t o = 0; o < d_out; ++o) v += bf16_to_f64(bt[o]) * bf16_to_f64(dzt[o]);
      for (int32_t c = 0; c < d_in; ++c) hv += bf16_to_f64(a[c]) * bf16_to_f64(x[c]);
      for (int32_t c = 0; c < d_in; ++c) da[c] += s * wp * v * bf16_to_f64(x[c]);
      for (int32_t o = 0; o < d_out; ++o) db[o] += s * wp * hv * bf16_to_f64(dzt[o]);
    }
  }
  return OR_OK;
}
