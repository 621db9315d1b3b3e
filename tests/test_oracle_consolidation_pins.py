"""Pins of the consolidation oracle (CKA similarity, similarity graph,
Louvain grouping, fixed-threshold grouping, CKA-centre anchor, shared-adapter
initialisation) against what the mathematics and the paper fix: the Gram
(kernel) form of linear CKA and its low-rank Gram-product form, the
invariances CKA is chosen for, exact modularity gains by brute force,
brute-force optimal partitions on tiny graphs with planted structure, the
connected components of a library routine, and the parameter budget."""
import numpy as np
import pytest

from oracle import consolidation as C
from paper_2609_06072_gb300 import workloads as W


def bits(x):
    return W.f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


def experts(rng, E, N, d_in, d_out, r):
    X = bits(rng.standard_normal((N, d_in)))
    A = [bits(rng.standard_normal((r, d_in))) for _ in range(E)]
    Bt = [bits(rng.standard_normal((r, d_out))) for _ in range(E)]
    return X, A, Bt


# ------------------------------------------------------------------ CKA
def test_cka_equals_kernel_form():
    """Kornblith et al.: ||Zc_i^T Zc_j||_F^2 = tr(Kc_i Kc_j) with the centred
    Gram matrices Kc = H Z Z^T H, so CKA is the normalised Gram alignment."""
    rng = np.random.default_rng(0)
    X, A, Bt = experts(rng, 4, 40, 12, 9, 3)
    Z = C.adapter_outputs(X, A, Bt)
    N = Z[0].shape[0]
    H = np.eye(N) - np.ones((N, N)) / N
    K = [H @ z @ z.T @ H for z in Z]
    S = C.cka_matrix(Z)
    for i in range(4):
        for j in range(4):
            ref = np.trace(K[i] @ K[j]) / np.sqrt(np.trace(K[i] @ K[i]) * np.trace(K[j] @ K[j]))
            assert abs(S[i, j] - ref) < 1e-10


def test_cka_low_rank_gram_product_form():
    """With Z_e = X A_e^T B_e^T and Xc = H X, Zc_i^T Zc_j = B_i M_ij B_j^T with
    M_ij = A_i (Xc^T Xc) A_j^T (r x r), so every norm in CKA reduces to r x r
    products: ||Zc_i^T Zc_j||_F^2 = tr(M_ij^T (B_i^T B_i) M_ij (B_j^T B_j))."""
    rng = np.random.default_rng(1)
    X, A, Bt = experts(rng, 5, 64, 16, 11, 4)
    S = C.cka_matrix(C.adapter_outputs(X, A, Bt))
    Xf = W.bf16_bits_to_f32(X).astype(np.float64)
    Xc = Xf - Xf.mean(axis=0)
    Cx = Xc.T @ Xc
    Af = [W.bf16_bits_to_f32(a).astype(np.float64) for a in A]
    Gb = [W.bf16_bits_to_f32(b).astype(np.float64) @ W.bf16_bits_to_f32(b).astype(np.float64).T for b in Bt]

    def cross(i, j):
        M = Af[i] @ Cx @ Af[j].T
        return np.trace(M.T @ Gb[i] @ M @ Gb[j])

    for i in range(5):
        for j in range(5):
            ref = cross(i, j) / np.sqrt(cross(i, i) * cross(j, j))
            assert abs(S[i, j] - ref) < 1e-10


def test_cka_invariances_and_bounds():
    """Scale invariance (the reason the paper picks CKA) and invariance to an
    orthogonal change of output basis; S_ii = 1, symmetric, in [0, 1];
    (uncentred) outputs on disjoint probe samples have similarity exactly 0."""
    rng = np.random.default_rng(2)
    X, A, Bt = experts(rng, 3, 50, 10, 8, 2)
    Z = C.adapter_outputs(X, A, Bt)
    S = C.cka_matrix(Z)
    assert np.allclose(np.diag(S), 1.0, atol=1e-12) and np.allclose(S, S.T, atol=1e-12)
    assert np.all(S >= -1e-12) and np.all(S <= 1 + 1e-12)
    Q, _ = np.linalg.qr(rng.standard_normal((8, 8)))
    assert abs(C.cka(Z[0], 7.5 * Z[1] @ Q) - S[0, 1]) < 1e-10
    Za = np.concatenate([Z[0][:25], np.zeros((25, 8))], axis=0)
    Zb = np.concatenate([np.zeros((25, 8)), Z[1][25:]], axis=0)
    assert C.cka(Za, Zb, center=False) == 0.0 and C.cka(Za, Za, center=False) == 1.0


def test_cka_centering_matters_only_through_the_mean():
    """Uncentred CKA equals centred CKA once the representations have zero
    mean; with a large common offset it differs (the centering appendix's
    two variants)."""
    rng = np.random.default_rng(3)
    Zi, Zj = rng.standard_normal((30, 6)), rng.standard_normal((30, 6))
    Zi0, Zj0 = Zi - Zi.mean(0), Zj - Zj.mean(0)
    assert abs(C.cka(Zi0, Zj0, center=False) - C.cka(Zi, Zj, center=True)) < 1e-12
    off = 50.0 * np.ones((1, 6))
    assert abs(C.cka(Zi + off, Zj + off, center=False) - C.cka(Zi, Zj)) > 0.1


# ------------------------------------------------------------------ graph
def test_similarity_graph_hand_example():
    S = np.array([[1.0, 0.9, 0.2, 0.3],
                  [0.7, 1.0, 0.4, 0.1],
                  [0.2, 0.4, 1.0, 0.8],
                  [0.3, 0.1, 0.8, 1.0]])
    Wg = C.similarity_graph(S)
    # symmetrised off-diagonal values: 0.8, 0.2, 0.3, 0.4, 0.1, 0.8 -> median 0.35
    ref = np.array([[0, 0.45, 0, 0], [0.45, 0, 0.05, 0], [0, 0.05, 0, 0.45], [0, 0, 0.45, 0]])
    assert np.allclose(Wg, ref, atol=1e-12)


def test_modularity_closed_forms():
    rng = np.random.default_rng(4)
    Wg = C.similarity_graph(rng.uniform(0, 1, (6, 6)))
    k = Wg.sum(1)
    two_m = Wg.sum()
    assert abs(C.modularity(Wg, [0] * 6, 1.0)) < 1e-12  # one group, gamma = 1
    single = C.modularity(Wg, list(range(6)), 0.8)
    assert abs(single + 0.8 * (k ** 2).sum() / two_m ** 2) < 1e-12


def test_modularity_gain_formula():
    """Moving a node i, taken out to a singleton, into group C changes Q by
    exactly (2 / 2m) (k_i,in(C) - gamma k_i tot(C) / 2m): the gain the local
    moves rank candidates by."""
    rng = np.random.default_rng(5)
    for trial in range(20):
        n = 7
        Wg = C.similarity_graph(rng.uniform(0, 1, (n, n)))
        z = list(rng.integers(0, 3, n))
        k, two_m, gamma = Wg.sum(1), Wg.sum(), 0.8
        i = int(rng.integers(n))
        base = list(z)
        base[i] = 99  # i alone
        for c in set(z) - {99}:
            moved = list(base)
            moved[i] = c
            members = [j for j in range(n) if base[j] == c]
            k_in = Wg[i, members].sum()
            tot = k[members].sum()
            pred = 2.0 / two_m * (k_in - gamma * k[i] * tot / two_m)
            assert abs(C.modularity(Wg, moved, gamma) - C.modularity(Wg, base, gamma) - pred) < 1e-12


def _best_partition(Wg, gamma):
    n = Wg.shape[0]
    best, best_q = None, -np.inf

    def partitions(seq):
        if not seq:
            yield []
            return
        first, rest = seq[0], seq[1:]
        for p in partitions(rest):
            for i in range(len(p)):
                yield p[:i] + [[first] + p[i]] + p[i + 1:]
            yield [[first]] + p

    for p in partitions(list(range(n))):
        z = [0] * n
        for g, blk in enumerate(p):
            for v in blk:
                z[v] = g
        q = C.modularity(Wg, z, gamma)
        if q > best_q + 1e-12:
            best, best_q = z, q
    return C._relabel(best), best_q


@pytest.mark.parametrize("seed", range(6))
def test_louvain_finds_the_optimum_of_planted_graphs(seed):
    """Tiny graphs with planted groups (strong weights inside, weak across):
    Louvain at gamma = 0.8 returns the brute-force modularity maximum."""
    rng = np.random.default_rng(10 + seed)
    n = 7
    sizes = [[3, 4], [2, 2, 3], [7], [3, 2, 2], [2, 5], [4, 3]][seed]
    z0 = np.repeat(np.arange(len(sizes)), sizes)
    rng.shuffle(z0)
    Wg = np.where(z0[:, None] == z0[None, :], rng.uniform(0.5, 1.0, (n, n)), rng.uniform(0.0, 0.05, (n, n)))
    Wg = np.triu(Wg, 1)
    Wg = Wg + Wg.T
    got = C.louvain(Wg, 0.8)
    best, best_q = _best_partition(Wg, 0.8)
    assert np.array_equal(got, best)
    assert abs(C.modularity(Wg, got, 0.8) - best_q) < 1e-12
    assert np.array_equal(got, C._relabel(z0))


def test_louvain_zero_resolution_gives_connected_components():
    """With gamma = 0 every merge along an edge raises Q, so the groups are
    the connected components of the positive-weight graph."""
    scipy = pytest.importorskip("scipy.sparse.csgraph")
    rng = np.random.default_rng(6)
    for _ in range(5):
        n = 12
        Wg = np.triu(rng.uniform(0, 1, (n, n)) * (rng.uniform(0, 1, (n, n)) < 0.15), 1)
        Wg = Wg + Wg.T
        ncomp, lab = scipy.connected_components(Wg > 0, directed=False)
        assert np.array_equal(C.louvain(Wg, 0.0), C._relabel(lab))


def test_louvain_degenerate_graphs():
    assert np.array_equal(C.louvain(np.zeros((4, 4)), 0.8), [0, 1, 2, 3])  # no edges: singletons
    assert np.array_equal(C.louvain(np.zeros((1, 1)), 0.8), [0])
    Wg = np.ones((5, 5)) - np.eye(5)  # complete graph: one group at gamma <= 1
    assert np.array_equal(C.louvain(Wg, 0.8), [0] * 5)


def test_threshold_groups_match_connected_components():
    scipy = pytest.importorskip("scipy.sparse.csgraph")
    rng = np.random.default_rng(7)
    for t in (0.5, 0.8, 0.9, 0.95):
        S = rng.uniform(0.3, 1.0, (10, 10))
        _, lab = scipy.connected_components((S + S.T) / 2 >= t, directed=False)
        assert np.array_equal(C.threshold_groups(S, t), C._relabel(lab))
    # an edge exactly at the threshold counts (s_ij >= t)
    S = np.array([[1.0, 0.9, 0.5], [0.9, 1.0, 0.89], [0.5, 0.89, 1.0]])
    assert list(C.threshold_groups(S, 0.9)) == [0, 0, 1]


# ------------------------------------------------------------------ anchor and init
def test_cka_center_anchor():
    S = np.array([[1.0, 0.6, 0.2, 0.9],
                  [0.6, 1.0, 0.7, 0.1],
                  [0.2, 0.7, 1.0, 0.3],
                  [0.9, 0.1, 0.3, 1.0]])
    # groups {0, 1, 2} and {3}: within-group sums 1.8, 2.3, 1.9 -> expert 1
    assert list(C.cka_center_anchor(S, [0, 0, 0, 1])) == [1, 3]
    # a tie goes to the lower index
    assert list(C.cka_center_anchor(np.ones((3, 3)), [0, 0, 0])) == [0]


def test_consolidation_budget_and_anchor_init():
    """r_g = sum of member ranks keeps the budget (Sec. 3.2); the anchor's
    rows start the shared adapter and the rest have B = 0, so at the
    consolidation step Delta W_g = Delta W_anchor, and all-singleton groups
    reproduce the expert-wise adapters exactly."""
    rng = np.random.default_rng(8)
    E, d_in, d_out, r = 6, 10, 7, 2
    A = [bits(rng.standard_normal((r, d_in))) for _ in range(E)]
    Bt = [bits(rng.standard_normal((r, d_out))) for _ in range(E)]
    labels = np.array([0, 1, 0, 2, 1, 0])
    anchors = np.array([2, 4, 3])
    init = rng.standard_normal((E * r, d_in))
    e2g, ro, Ag, Btg = C.consolidate(labels, [r] * E, anchors, A, Bt, init)
    assert list(np.diff(ro)) == [6, 4, 2] and ro[-1] * (d_in + d_out) == E * r * (d_in + d_out)
    f = lambda b: W.bf16_bits_to_f32(b).astype(np.float64)
    for g, a in enumerate(anchors):
        r0, r1 = ro[g], ro[g + 1]
        dWg = Btg[r0:r1].T @ Ag[r0:r1]
        assert np.allclose(dWg, f(Bt[a]).T @ f(A[a]), atol=1e-12)
        assert np.all(Btg[r0 + r:r1] == 0) and np.array_equal(Ag[r0 + r:r1], init[r0 + r:r1])
    e2g, ro, Ag, Btg = C.consolidate(np.arange(E), [r] * E, np.arange(E), A, Bt, init)
    for e in range(E):
        assert np.array_equal(Ag[r * e:r * e + r], f(A[e])) and np.array_equal(Btg[r * e:r * e + r], f(Bt[e]))


def test_end_to_end_grouping_recovers_planted_prototypes():
    """Experts whose adapters are small perturbations of a few prototypes:
    CKA on a shared probe set, the median-shifted graph and Louvain group them
    by prototype, and the fixed-threshold rule agrees."""
    rng = np.random.default_rng(9)
    E, N, d_in, d_out, r = 12, 200, 24, 16, 2
    proto = rng.integers(0, 3, E)
    PA = [rng.standard_normal((r, d_in)) for _ in range(3)]
    PB = [rng.standard_normal((r, d_out)) for _ in range(3)]
    A = [bits(PA[p] + 0.05 * rng.standard_normal((r, d_in))) for p in proto]
    Bt = [bits(PB[p] + 0.05 * rng.standard_normal((r, d_out))) for p in proto]
    X = bits(rng.standard_normal((N, d_in)))
    S = C.cka_matrix(C.adapter_outputs(X, A, Bt))
    want = C._relabel(proto)
    assert np.array_equal(C.louvain(C.similarity_graph(S), 0.8), want)
    assert np.array_equal(C.threshold_groups(S, 0.9), want)
