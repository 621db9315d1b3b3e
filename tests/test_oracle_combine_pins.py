"""Pins of the oracle's gate-weighted combine of the down projection.

The combine carries the router weight p_e(x) of Sec. 3.1's
y(x) = sum_{e in R(x)} p_e(x) (W_e h_e + B_e A_e h_e) into the sum over a
token's routed experts, with expert e using the group adapter of g(e)
(Sec. 3.3-3.4).  Each test reaches the result by a route other than the
oracle's own loops: the dense Delta W_g = B_g A_g form, the per-pair delta of
the (separately pinned) down oracle, the dedup-by-linearity rewrite that a
fused kernel uses, exact finite differences of the multilinear forward, and
the dense gradient form of Sec. 3.1.2.
"""
import numpy as np
import pytest

import oracle
from paper_2609_06072_gb300 import workloads as W


def bf(x):
    return W.bf16_bits_to_f32(x).astype(np.float64)


def layer(T=11, d=9, f=7, E=6, k=3, G=3, seed=0, ranks=None, e2g=None):
    """A hand-sized random layer with gate weights (numpy only)."""
    rng = np.random.default_rng(seed)
    idx = np.array([rng.permutation(E)[:k] for _ in range(T)], dtype=np.int32).reshape(T, k)
    if e2g is None:
        e2g = (np.arange(E) % G).astype(np.int32)
    if ranks is None:
        ranks = [2 + (g % 3) for g in range(G)]
    rank_off = np.concatenate([[0], np.cumsum(ranks)]).astype(np.int32)
    Rk = int(rank_off[-1])
    q = lambda *s: W.f32_to_bf16_bits(rng.standard_normal(s).astype(np.float32))
    logits = rng.standard_normal((T, k))
    w = (np.exp(logits) / np.exp(logits).sum(1, keepdims=True)).astype(np.float32)
    return dict(idx=idx, e2g=np.asarray(e2g, np.int32), rank_off=rank_off, G=G, T=T, k=k, E=E, d=d, f=f,
                h=q(T * k, f), w=w, A=q(Rk, f), Bt=q(Rk, d), dz=q(T, d), zin=q(T, d))


def _args(L):
    return L["idx"], L["e2g"], L["rank_off"]


def test_combine_equals_dense_delta_w():
    """z[t] = sum_j p_j s Delta W_g h_j with Delta W_g = B_g A_g materialised."""
    L = layer()
    s = 1.7
    z = oracle.combine_fwd(*_args(L), L["h"], L["w"], L["A"], L["Bt"], s)
    for t in range(L["T"]):
        ref = np.zeros(L["d"])
        for j in range(L["k"]):
            p = t * L["k"] + j
            g = L["e2g"][L["idx"][t, j]]
            r0, r1 = L["rank_off"][g], L["rank_off"][g + 1]
            dW = bf(L["Bt"][r0:r1]).T @ bf(L["A"][r0:r1])  # d x f
            ref += float(L["w"][t, j]) * s * dW @ bf(L["h"][p])
        np.testing.assert_allclose(z[t], ref, rtol=1e-12, atol=1e-12)


def test_combine_adds_base_and_selects():
    L = layer(seed=2)
    z0 = oracle.combine_fwd(*_args(L), L["h"], L["w"], L["A"], L["Bt"], 2.0)
    z1 = oracle.combine_fwd(*_args(L), L["h"], L["w"], L["A"], L["Bt"], 2.0, z_in=L["zin"])
    np.testing.assert_allclose(z1, z0 + bf(L["zin"]), rtol=0, atol=1e-12)
    sel = np.array([4, 0, 9], np.int32)
    zs = oracle.combine_fwd(*_args(L), L["h"], L["w"], L["A"], L["Bt"], 2.0, sel=sel)
    assert np.array_equal(zs, z0[sel])


def test_combine_reduces_to_per_row_down():
    """With one-hot gate weights the combine returns one pair's down delta;
    with unit weights, the sum of the token's per-pair deltas (the per-row
    down oracle, pinned on its own)."""
    L = layer(seed=3)
    s = 0.9
    y, _ = oracle.fwd(L["idx"], L["e2g"], L["rank_off"], L["h"], L["A"], L["Bt"], s, x_per_pair=True)
    T, k = L["T"], L["k"]
    ones = np.ones((T, k), np.float32)
    z = oracle.combine_fwd(*_args(L), L["h"], ones, L["A"], L["Bt"], s)
    np.testing.assert_allclose(z, y.reshape(T, k, -1).sum(1), rtol=1e-12, atol=1e-12)
    for j0 in range(k):
        onehot = np.zeros((T, k), np.float32)
        onehot[:, j0] = 1.0
        z = oracle.combine_fwd(*_args(L), L["h"], onehot, L["A"], L["Bt"], s)
        np.testing.assert_allclose(z, y.reshape(T, k, -1)[:, j0], rtol=1e-12, atol=1e-12)


def test_combine_dedup_by_linearity():
    """Within one group the weighted sum moves inside the adapter:
    sum_{e in g, R(t)} p_e B_g A_g h_e = B_g (sum p_e A_g h_e), so each unique
    (token, group) pair needs one N-side product (Sec. 3.5's reuse, applied to
    the combined output)."""
    L = layer(T=13, E=8, k=4, G=2, seed=5)  # groups of four experts: many shared pairs
    s = 1.3
    P = oracle.permute(L["idx"], L["e2g"], L["G"])
    z = oracle.combine_fwd(*_args(L), L["h"], L["w"], L["A"], L["Bt"], s)
    ref = np.zeros_like(z)
    w = L["w"].ravel().astype(np.float64)
    shared = 0
    for u in range(P["U"]):
        rows = P["uniq_rows"][P["uniq_rows_ptr"][u]:P["uniq_rows_ptr"][u + 1]]
        pairs = P["row_pair"][rows]
        shared += len(pairs) - 1
        g = int(np.searchsorted(P["uniq_off"], u, side="right") - 1)
        r0, r1 = L["rank_off"][g], L["rank_off"][g + 1]
        Hc = sum(w[p] * (bf(L["A"][r0:r1]) @ bf(L["h"][p])) for p in pairs)
        ref[P["uniq_tok"][u]] += s * bf(L["Bt"][r0:r1]).T @ Hc
    assert shared > 0
    np.testing.assert_allclose(z, ref, rtol=1e-11, atol=1e-11)


def _loss(L, h=None, w=None, A=None, Bt=None, s=1.1):
    z = oracle.combine_fwd(*_args(L), L["h"] if h is None else h, L["w"] if w is None else w,
                           L["A"] if A is None else A, L["Bt"] if Bt is None else Bt, s)
    return float(np.sum(z * bf(L["dz"])))


def _bump(arr, i, j):
    out = arr.copy()
    old = bf(arr[i:i + 1, j:j + 1])[0, 0]
    new_bits = W.f32_to_bf16_bits(np.array([[old * 1.5 + 0.25]], np.float32))
    out[i, j] = new_bits[0, 0]
    return out, bf(new_bits)[0, 0] - old


def test_combine_gradients_match_finite_differences():
    """The combine is linear in each of h, p, A, B separately, so a finite
    difference with any step is exact up to rounding."""
    L = layer(seed=13)
    s = 1.1
    dh, dw = oracle.combine_bwd_dh(*_args(L), L["dz"], L["h"], L["w"], L["A"], L["Bt"], s)
    dA, dBt = oracle.combine_bwd_w(*_args(L), L["h"], L["dz"], L["w"], L["A"], L["Bt"], s)
    base = _loss(L, s=s)
    rng = np.random.default_rng(0)
    for _ in range(10):
        i, j = rng.integers(L["h"].shape[0]), rng.integers(L["f"])
        hp, step = _bump(L["h"], i, j)
        np.testing.assert_allclose((_loss(L, h=hp, s=s) - base) / step, dh[i, j], rtol=1e-7, atol=1e-9)
        i, j = rng.integers(L["A"].shape[0]), rng.integers(L["f"])
        Ap, step = _bump(L["A"], i, j)
        np.testing.assert_allclose((_loss(L, A=Ap, s=s) - base) / step, dA[i, j], rtol=1e-7, atol=1e-9)
        i, j = rng.integers(L["Bt"].shape[0]), rng.integers(L["d"])
        Bp, step = _bump(L["Bt"], i, j)
        np.testing.assert_allclose((_loss(L, Bt=Bp, s=s) - base) / step, dBt[i, j], rtol=1e-7, atol=1e-9)
        t, j = rng.integers(L["T"]), rng.integers(L["k"])
        wp = L["w"].copy()
        wp[t, j] = np.float32(wp[t, j] + 0.375)
        step = float(wp[t, j]) - float(L["w"][t, j])
        np.testing.assert_allclose((_loss(L, w=wp, s=s) - base) / step, dw[t * L["k"] + j], rtol=1e-7,
                                   atol=1e-9)


def test_combine_gradients_against_per_row_down():
    """dh_p = p_p times the per-row down input gradient of dz_t, and the gate
    gradient is dz_t . delta_p with delta_p the pair's unweighted down delta
    (both from the per-row oracle, pinned on its own)."""
    L = layer(seed=21)
    s = 0.8
    T, k = L["T"], L["k"]
    dh, dw = oracle.combine_bwd_dh(*_args(L), L["dz"], L["h"], L["w"], L["A"], L["Bt"], s)
    dy = np.repeat(L["dz"], k, axis=0)  # dz_t on each of the token's pairs
    dh1 = oracle.bwd_dx(L["idx"], L["e2g"], L["rank_off"], dy, L["A"], L["Bt"], s, x_per_pair=True)
    np.testing.assert_allclose(dh, L["w"].reshape(-1, 1).astype(np.float64) * dh1, rtol=1e-12, atol=1e-12)
    delta, _ = oracle.fwd(L["idx"], L["e2g"], L["rank_off"], L["h"], L["A"], L["Bt"], s, x_per_pair=True)
    np.testing.assert_allclose(dw, np.sum(delta * bf(dy), axis=1), rtol=1e-11, atol=1e-12)
    dh_in = W.f32_to_bf16_bits(np.random.default_rng(4).standard_normal(dh.shape).astype(np.float32))
    dh2, _ = oracle.combine_bwd_dh(*_args(L), L["dz"], L["h"], L["w"], L["A"], L["Bt"], s, dh_in=dh_in)
    np.testing.assert_allclose(dh2, dh + bf(dh_in), rtol=0, atol=1e-12)
    sel = np.array([7, 2], np.int32)
    sh, sw = oracle.combine_bwd_dh(*_args(L), L["dz"], L["h"], L["w"], L["A"], L["Bt"], s, sel=sel)
    assert np.array_equal(sh, dh[sel]) and np.array_equal(sw, dw[sel])


def test_combine_weight_gradients_dense_form():
    """Sec. 3.1.2 / 3.4 with the gate weight: M_g = s sum_{p in g} p_p dz_t h_p^T,
    dA_g = B_g^T M_g and dB_g = M_g A_g^T."""
    L = layer(seed=17)
    s = 0.7
    dA, dBt = oracle.combine_bwd_w(*_args(L), L["h"], L["dz"], L["w"], L["A"], L["Bt"], s)
    T, k = L["T"], L["k"]
    gp = L["e2g"][L["idx"].ravel()]
    wz = bf(L["dz"])[np.arange(T * k) // k] * L["w"].reshape(-1, 1).astype(np.float64)
    for g in range(L["G"]):
        r0, r1 = L["rank_off"][g], L["rank_off"][g + 1]
        m = gp == g
        M = s * wz[m].T @ bf(L["h"])[m]  # d x f
        np.testing.assert_allclose(dA[r0:r1], bf(L["Bt"][r0:r1]) @ M, rtol=1e-11, atol=1e-11)
        np.testing.assert_allclose(dBt[r0:r1], (M @ bf(L["A"][r0:r1]).T).T, rtol=1e-11, atol=1e-11)
    sel = np.array([3, 0], np.int32)
    sA, sB = oracle.combine_bwd_w(*_args(L), L["h"], L["dz"], L["w"], L["A"], L["Bt"], s, sel=sel)
    assert np.array_equal(sA, dA[sel]) and np.array_equal(sB, dBt[sel])


def test_combine_empty_group_and_token_order():
    L = layer(E=6, G=4, e2g=[0, 0, 1, 1, 2, 2], ranks=[2, 2, 2, 3], seed=19)  # group 3 has no expert
    dA, dBt = oracle.combine_bwd_w(*_args(L), L["h"], L["dz"], L["w"], L["A"], L["Bt"], 1.0)
    r0 = L["rank_off"][3]
    assert np.all(dA[r0:] == 0) and np.all(dBt[r0:] == 0)
    # permuting tokens permutes z and dh, and leaves dA, dB unchanged
    T, k = L["T"], L["k"]
    pi = np.random.default_rng(1).permutation(T)
    pairs = (pi[:, None] * k + np.arange(k)[None, :]).ravel()
    args2 = (L["idx"][pi], L["e2g"], L["rank_off"])
    z = oracle.combine_fwd(*_args(L), L["h"], L["w"], L["A"], L["Bt"], 1.5)
    z2 = oracle.combine_fwd(*args2, L["h"][pairs], L["w"][pi], L["A"], L["Bt"], 1.5)
    np.testing.assert_array_equal(z2, z[pi])
    dh, dw = oracle.combine_bwd_dh(*_args(L), L["dz"], L["h"], L["w"], L["A"], L["Bt"], 1.5)
    dh2, dw2 = oracle.combine_bwd_dh(*args2, L["dz"][pi], L["h"][pairs], L["w"][pi], L["A"], L["Bt"], 1.5)
    np.testing.assert_array_equal(dh2, dh[pairs])
    np.testing.assert_array_equal(dw2, dw[pairs])
    dA2, dBt2 = oracle.combine_bwd_w(*args2, L["h"][pairs], L["dz"][pi], L["w"][pi], L["A"], L["Bt"], 1.0)
    np.testing.assert_allclose(dA2, dA, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(dBt2, dBt, rtol=1e-12, atol=1e-12)


def test_combine_degenerate_inputs():
    L = layer(seed=23)
    # no tokens: empty outputs, zero weight gradients
    idx0 = np.zeros((0, L["k"]), np.int32)
    h0 = np.zeros((0, L["f"]), np.uint16)
    z = oracle.combine_fwd(idx0, L["e2g"], L["rank_off"], h0, np.zeros((0, L["k"]), np.float32), L["A"], L["Bt"],
                           1.0)
    assert z.shape == (0, L["d"])
    dA, dBt = oracle.combine_bwd_w(idx0, L["e2g"], L["rank_off"], h0, np.zeros((0, L["d"]), np.uint16),
                                   np.zeros((0, L["k"]), np.float32), L["A"], L["Bt"], 1.0)
    assert np.all(dA == 0) and np.all(dBt == 0)
    # zero gate weights: no delta, no input or weight gradient, but the gate
    # gradient is still the pair's delta against dz
    zw = np.zeros_like(L["w"])
    assert np.all(oracle.combine_fwd(*_args(L), L["h"], zw, L["A"], L["Bt"], 1.0) == 0)
    dh, dw = oracle.combine_bwd_dh(*_args(L), L["dz"], L["h"], zw, L["A"], L["Bt"], 1.0)
    assert np.all(dh == 0) and np.any(dw != 0)
    with pytest.raises(ValueError):
        oracle.combine_fwd(*_args(L), L["h"], L["w"][:, :1], L["A"], L["Bt"], 1.0)
    bad = L["idx"].copy()
    bad[0, 0] = L["E"]
    with pytest.raises(oracle.OracleError):
        oracle.combine_fwd(bad, L["e2g"], L["rank_off"], L["h"], L["w"], L["A"], L["Bt"], 1.0)
