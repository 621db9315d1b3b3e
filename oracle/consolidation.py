"""fp64 CPU oracle of ACE's rank consolidation: the step that produces the
expert -> group map the grouped path takes as input (arxiv 2609.06072).

TEST INFRASTRUCTURE ONLY, like the rest of this package: the test suite may
import it; the product library never does.  Plain numpy in float64 and
pure-Python loops over experts; no blocking or reordering beyond what each
definition states.

Functions and the passages they follow:

* ``adapter_outputs``  -- Z_e = [(Delta W_e x_n)^T]_n over the probe set,
                          Delta W_e = B_e A_e (Sec. 3.2, rank consolidation).
* ``cka_matrix``       -- s_ij = ||Zc_i^T Zc_j||_F^2 / (||Zc_i^T Zc_i||_F ||Zc_j^T Zc_j||_F),
                          Zc_e = H Z_e with H = I - 11^T / N (Sec. 3.2; the
                          centering appendix also allows the uncentered form).
* ``similarity_graph`` -- symmetrise, zero the diagonal, subtract the median
                          of the off-diagonal entries, clamp at zero
                          (layer-wise graph construction appendix).
* ``modularity``, ``louvain`` -- generalized weighted modularity with
                          resolution gamma, greedy local moves then
                          aggregation into super-nodes (Louvain appendix).
* ``threshold_groups`` -- connected components of {(i, j): i != j, s_ij >= t}
                          (fixed-threshold appendix).
* ``cka_center_anchor`` -- the group member most central in within-group CKA
                          (group-anchor appendix).
* ``consolidate``      -- groups -> expert->group map, r_g = sum of member
                          ranks, and the shared adapters initialised from the
                          anchor plus LoRA initialisation for the other rank
                          rows (Sec. 3.2, group-anchor appendix).

Readings where the paper is silent: the symmetrisation is (S + S^T) / 2;
Louvain visits nodes in ascending index, sweeps until a sweep moves nothing,
compares a node's best candidate with returning to its own group and moves
only on a strictly larger gain, breaks ties toward the lowest group label,
and stops when a level moves nothing; groups are labelled in order of their
smallest expert index; the anchor maximises the sum of within-group
similarities (ties to the lowest index) and fills the first rank rows of the
shared adapter, in the member order of ascending expert index.
"""
from __future__ import annotations

from typing import List, Sequence

import numpy as np

from paper_2609_06072_gb300 import workloads as _W


def _f64(bits) -> np.ndarray:
    return _W.bf16_bits_to_f32(np.asarray(bits, dtype=np.uint16)).astype(np.float64)


# ------------------------------------------------------------------ CKA
def adapter_outputs(X_probe, A_e: Sequence, Bt_e: Sequence) -> List[np.ndarray]:
    """Z_e = X_probe A_e^T B_e^T for every expert (bf16 bit patterns in,
    float64 out): row n is (Delta W_e x_n)^T, Delta W_e = B_e A_e."""
    X = _f64(X_probe)
    return [(X @ _f64(A).T) @ _f64(Bt) for A, Bt in zip(A_e, Bt_e)]


def cka(Z_i: np.ndarray, Z_j: np.ndarray, center: bool = True) -> float:
    """Linear CKA of two representation matrices [N, d_out] by its
    definition (Frobenius norms of the cross- and self-covariances)."""
    if center:
        Z_i = Z_i - Z_i.mean(axis=0, keepdims=True)  # H Z with H = I - 11^T / N
        Z_j = Z_j - Z_j.mean(axis=0, keepdims=True)
    num = np.linalg.norm(Z_i.T @ Z_j, "fro") ** 2
    den = np.linalg.norm(Z_i.T @ Z_i, "fro") * np.linalg.norm(Z_j.T @ Z_j, "fro")
    return float(num / den) if den > 0 else 0.0


def cka_matrix(Z: Sequence[np.ndarray], center: bool = True) -> np.ndarray:
    """The E x E matrix of pairwise linear CKA similarities."""
    E = len(Z)
    S = np.empty((E, E))
    for i in range(E):
        for j in range(E):
            S[i, j] = cka(Z[i], Z[j], center)
    return S


# ------------------------------------------------------------------ graph
def similarity_graph(S: np.ndarray) -> np.ndarray:
    """W_ij = max(0, S_ij - b) on the symmetrised S with a zero diagonal,
    b the median of the off-diagonal entries."""
    S = 0.5 * (np.asarray(S, dtype=np.float64) + np.asarray(S, dtype=np.float64).T)
    E = S.shape[0]
    off = ~np.eye(E, dtype=bool)
    b = float(np.median(S[off])) if E > 1 else 0.0
    W = np.where(off, np.maximum(0.0, S - b), 0.0)
    return W


def modularity(W: np.ndarray, z: Sequence[int], gamma: float) -> float:
    """Q = 1/(2m) sum_ij (W_ij - gamma k_i k_j / (2m)) [z_i = z_j]."""
    W = np.asarray(W, dtype=np.float64)
    k = W.sum(axis=1)
    two_m = W.sum()
    if two_m <= 0:
        return 0.0
    z = np.asarray(z)
    same = z[:, None] == z[None, :]
    return float(((W - gamma * np.outer(k, k) / two_m) * same).sum() / two_m)


def _local_moves(W: np.ndarray, gamma: float):
    """One Louvain level: start from singletons, move nodes greedily.
    Returns (community of each node, whether any node moved)."""
    n = W.shape[0]
    k = W.sum(axis=1)
    two_m = W.sum()
    comm = list(range(n))
    tot = [float(k[i]) for i in range(n)]  # sum of degrees per community label
    moved_any = False
    if two_m <= 0:
        return comm, False
    while True:
        moved = False
        for i in range(n):
            own = comm[i]
            tot[own] -= k[i]  # take i out of its community
            # weight from i to each community (self-loop excluded: i is out)
            k_in = {}
            for j in range(n):
                if j != i and W[i, j] > 0:
                    k_in[comm[j]] = k_in.get(comm[j], 0.0) + W[i, j]
            k_in.setdefault(own, 0.0)

            def gain(c):
                return k_in[c] - gamma * k[i] * tot[c] / two_m

            best, best_gain = own, gain(own)
            for c in sorted(k_in):
                g = gain(c)
                if g > best_gain:
                    best, best_gain = c, g
            comm[i] = best
            tot[best] += k[i]
            if best != own:
                moved = True
                moved_any = True
        if not moved:
            return comm, moved_any


def louvain(W: np.ndarray, gamma: float = 0.8) -> np.ndarray:
    """Louvain community detection on the weighted graph W (symmetric, zero
    diagonal): local moves, then communities become super-nodes (edge weight
    = summed member weights, internal weight as a self-loop), repeated until
    a level moves nothing.  Returns group labels 0..G-1 numbered in order of
    their smallest member."""
    W = np.asarray(W, dtype=np.float64)
    n = W.shape[0]
    member = list(range(n))  # super-node of each original node
    cur = W.copy()
    while True:
        comm, moved = _local_moves(cur, gamma)
        if not moved:
            break
        labels = sorted(set(comm))
        idx = {c: a for a, c in enumerate(labels)}
        m = len(labels)
        agg = np.zeros((m, m))
        for a in range(cur.shape[0]):
            for b in range(cur.shape[0]):
                agg[idx[comm[a]], idx[comm[b]]] += cur[a, b]
        member = [idx[comm[member[v]]] for v in range(n)]
        cur = agg
        if m == 1:
            break
    return _relabel(member)


def _relabel(z: Sequence[int]) -> np.ndarray:
    out, seen = [], {}
    for c in z:
        if c not in seen:
            seen[c] = len(seen)
        out.append(seen[c])
    return np.asarray(out, dtype=np.int32)


def threshold_groups(S: np.ndarray, t: float = 0.9) -> np.ndarray:
    """Connected components of the graph with an edge (i, j), i != j, wherever
    the symmetrised similarity is >= t (breadth-first search)."""
    S = 0.5 * (np.asarray(S, dtype=np.float64) + np.asarray(S, dtype=np.float64).T)
    E = S.shape[0]
    label = [-1] * E
    nxt = 0
    for s in range(E):
        if label[s] >= 0:
            continue
        label[s] = nxt
        queue = [s]
        while queue:
            i = queue.pop(0)
            for j in range(E):
                if j != i and label[j] < 0 and S[i, j] >= t:
                    label[j] = nxt
                    queue.append(j)
        nxt += 1
    return np.asarray(label, dtype=np.int32)


# ------------------------------------------------------------------ anchor
def cka_center_anchor(S: np.ndarray, labels: Sequence[int]) -> np.ndarray:
    """For each group g (label order), the member i maximising
    sum_{j in g} S_ij; ties go to the lowest expert index."""
    S = np.asarray(S, dtype=np.float64)
    labels = np.asarray(labels)
    G = int(labels.max()) + 1 if labels.size else 0
    anchors = np.empty(G, dtype=np.int32)
    for g in range(G):
        mem = np.flatnonzero(labels == g)
        best, best_v = -1, -np.inf
        for i in mem:
            v = float(S[i, mem].sum())
            if v > best_v:
                best, best_v = int(i), v
        anchors[g] = best
    return anchors


def consolidate(labels, ranks, anchors, A_e, Bt_e, A_init_rows):
    """The shared adapters of the groups (Sec. 3.2): group g takes
    r_g = sum of its members' ranks rank rows, rows rank_off[g].. of the
    stacked A / B^T.  The first r_anchor rows are the anchor's own A_e and
    B_e^T; the remaining rows take standard LoRA initialisation: A from
    ``A_init_rows`` (the caller's random draw, one row per stacked rank row,
    used in order), B^T zero.  Returns (e2g, rank_off, A_g, Bt_g) with A_g /
    Bt_g as float64."""
    labels = np.asarray(labels, dtype=np.int32)
    ranks = np.asarray(ranks, dtype=np.int64)
    G = int(labels.max()) + 1
    r_g = np.array([int(ranks[labels == g].sum()) for g in range(G)], dtype=np.int64)
    rank_off = np.concatenate([[0], np.cumsum(r_g)]).astype(np.int32)
    d_in, d_out = np.asarray(A_e[0]).shape[1], np.asarray(Bt_e[0]).shape[1]
    A_g = np.zeros((int(rank_off[-1]), d_in))
    Bt_g = np.zeros((int(rank_off[-1]), d_out))
    init = np.asarray(A_init_rows, dtype=np.float64)
    for g in range(G):
        a = int(anchors[g])
        r0, ra = int(rank_off[g]), int(ranks[a])
        A_g[r0:r0 + ra] = _f64(A_e[a])
        Bt_g[r0:r0 + ra] = _f64(Bt_e[a])
        A_g[r0 + ra:rank_off[g + 1]] = init[r0 + ra:rank_off[g + 1]]
    return labels.copy(), rank_off, A_g, Bt_g
