// Expert grouping for rank consolidation (Sec. 3.2; the layer-wise graph
// construction, Louvain and fixed-threshold appendices; the group-anchor
// appendix).  Host code only: the E x E similarity matrix of one layer is
// small (E <= 512), and the grouping is a one-time step before training.
//
//   graph      W_ij = max(0, S'_ij - b), S' = (S + S^T) / 2 with a zero
//              diagonal, b the median of the off-diagonal entries of S'
//   Louvain    generalized weighted modularity with resolution gamma: from
//              singletons, each node (ascending index) is taken out of its
//              group and put into the neighbouring group with the largest
//              gain k_i,in(C) - gamma k_i tot(C) / 2m, staying unless another
//              group's gain is strictly larger (ties to the lower label);
//              sweeps repeat until one moves nothing, then groups become
//              super-nodes (summed weights, internal weight as a self-loop)
//              and the level repeats until a level moves nothing
//   threshold  connected components of {(i, j): i != j, S'_ij >= t}
//   anchor     per group the member maximising sum_{j in group} S_ij (ties
//              to the lower index)
// Groups are numbered in order of their smallest expert.  All arithmetic is
// double precision.
#include <algorithm>
#include <cstdarg>
#include <cstdio>
#include <map>
#include <vector>

#include "ace_internal.cuh"

namespace {

ace_status cfail(ace_status st, const char* fmt, ...) {
  char msg[256];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(msg, sizeof(msg), fmt, ap);
  va_end(ap);
  return ace::report(st, msg);
}

using Mat = std::vector<double>;  // row-major n x n

// Symmetrised similarities with the given diagonal.
Mat symmetrise(const float* S, int E) {
  Mat s((size_t)E * E);
  for (int i = 0; i < E; ++i)
    for (int j = 0; j < E; ++j) s[(size_t)i * E + j] = 0.5 * ((double)S[(size_t)i * E + j] + (double)S[(size_t)j * E + i]);
  return s;
}

Mat similarity_graph(const Mat& s, int E) {
  std::vector<double> off;
  off.reserve((size_t)E * (E > 0 ? E - 1 : 0));
  for (int i = 0; i < E; ++i)
    for (int j = 0; j < E; ++j)
      if (i != j) off.push_back(s[(size_t)i * E + j]);
  double b = 0.0;
  if (!off.empty()) {
    std::sort(off.begin(), off.end());
    const size_t n = off.size();
    b = n % 2 ? off[n / 2] : 0.5 * (off[n / 2 - 1] + off[n / 2]);
  }
  Mat w((size_t)E * E, 0.0);
  for (int i = 0; i < E; ++i)
    for (int j = 0; j < E; ++j)
      if (i != j) w[(size_t)i * E + j] = std::max(0.0, s[(size_t)i * E + j] - b);
  return w;
}

// One Louvain level on the n-node graph w.  comm receives the group label of
// each node (labels are node indices); returns whether any node moved.
bool local_moves(const Mat& w, int n, double gamma, std::vector<int>& comm) {
  std::vector<double> k(n, 0.0);
  double two_m = 0.0;
  for (int i = 0; i < n; ++i) {
    for (int j = 0; j < n; ++j) k[i] += w[(size_t)i * n + j];
    two_m += k[i];
  }
  comm.resize(n);
  for (int i = 0; i < n; ++i) comm[i] = i;
  if (two_m <= 0.0) return false;
  std::vector<double> tot(k);
  bool moved_any = false;
  for (;;) {
    bool moved = false;
    for (int i = 0; i < n; ++i) {
      const int own = comm[i];
      tot[own] -= k[i];
      std::map<int, double> k_in;  // ordered by label: ties go to the lower one
      for (int j = 0; j < n; ++j)
        if (j != i && w[(size_t)i * n + j] > 0.0) k_in[comm[j]] += w[(size_t)i * n + j];
      k_in.emplace(own, 0.0);
      auto gain = [&](int c) { return k_in[c] - gamma * k[i] * tot[c] / two_m; };
      int best = own;
      double best_gain = gain(own);
      for (const auto& kv : k_in) {
        const double g = gain(kv.first);
        if (g > best_gain) {
          best = kv.first;
          best_gain = g;
        }
      }
      comm[i] = best;
      tot[best] += k[i];
      if (best != own) moved = moved_any = true;
    }
    if (!moved) return moved_any;
  }
}

std::vector<int> relabel(const std::vector<int>& z) {
  std::map<int, int> seen;
  std::vector<int> out(z.size());
  for (size_t i = 0; i < z.size(); ++i) {
    auto it = seen.find(z[i]);
    if (it == seen.end()) it = seen.emplace(z[i], (int)seen.size()).first;
    out[i] = it->second;
  }
  return out;
}

std::vector<int> louvain(const Mat& w0, int E, double gamma) {
  std::vector<int> member(E);
  for (int v = 0; v < E; ++v) member[v] = v;
  Mat cur = w0;
  int n = E;
  std::vector<int> comm;
  for (;;) {
    if (!local_moves(cur, n, gamma, comm)) break;
    std::map<int, int> idx;  // ascending old label -> new super-node
    for (int a = 0; a < n; ++a) idx.emplace(comm[a], 0);
    int m = 0;
    for (auto& kv : idx) kv.second = m++;
    Mat agg((size_t)m * m, 0.0);
    for (int a = 0; a < n; ++a)
      for (int b = 0; b < n; ++b) agg[(size_t)idx[comm[a]] * m + idx[comm[b]]] += cur[(size_t)a * n + b];
    for (int v = 0; v < E; ++v) member[v] = idx[comm[member[v]]];
    cur.swap(agg);
    n = m;
    if (m == 1) break;
  }
  return relabel(member);
}

std::vector<int> threshold_groups(const Mat& s, int E, double t) {
  std::vector<int> label(E, -1);
  int nxt = 0;
  for (int src = 0; src < E; ++src) {
    if (label[src] >= 0) continue;
    label[src] = nxt;
    std::vector<int> queue{src};
    for (size_t q = 0; q < queue.size(); ++q) {
      const int i = queue[q];
      for (int j = 0; j < E; ++j)
        if (j != i && label[j] < 0 && s[(size_t)i * E + j] >= t) {
          label[j] = nxt;
          queue.push_back(j);
        }
    }
    ++nxt;
  }
  return label;
}

}  // namespace

extern "C" {

ace_status ace_group_experts(const float* S, int32_t E, int32_t method, double param, int32_t* e2g,
                             int32_t* anchors, int32_t* G_out) {
  if (!S || !e2g || !G_out) return cfail(ACE_ERR_ARG, "null argument");
  if (E < 1 || E > ACE_MAX_EXPERTS) return cfail(ACE_ERR_SHAPE, "E=%d outside [1, %d]", E, ACE_MAX_EXPERTS);
  if (method != ACE_GROUP_LOUVAIN && method != ACE_GROUP_THRESHOLD)
    return cfail(ACE_ERR_ARG, "unknown grouping method %d", method);
  for (size_t i = 0; i < (size_t)E * E; ++i)
    if (!(S[i] == S[i]) || S[i] > 3.0e38f || S[i] < -3.0e38f) return cfail(ACE_ERR_ARG, "non-finite similarity");
  if (method == ACE_GROUP_LOUVAIN && !(param >= 0.0)) return cfail(ACE_ERR_ARG, "resolution must be >= 0");
  const Mat s = symmetrise(S, E);
  const std::vector<int> z =
      method == ACE_GROUP_LOUVAIN ? louvain(similarity_graph(s, E), E, param) : threshold_groups(s, E, param);
  int G = 0;
  for (int e = 0; e < E; ++e) {
    e2g[e] = z[e];
    G = std::max(G, z[e] + 1);
  }
  *G_out = G;
  if (anchors) {
    for (int g = 0; g < G; ++g) {
      int best = -1;
      double best_v = 0.0;
      for (int i = 0; i < E; ++i) {
        if (z[i] != g) continue;
        double v = 0.0;
        for (int j = 0; j < E; ++j)
          if (z[j] == g) v += (double)S[(size_t)i * E + j];
        if (best < 0 || v > best_v) {
          best = i;
          best_v = v;
        }
      }
      anchors[g] = best;
    }
  }
  return ACE_OK;
}

}  // extern "C"
