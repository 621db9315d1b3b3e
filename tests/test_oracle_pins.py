"""Pins of the fp64 oracle against what the paper and the mathematics fix.

Each test checks the oracle through a route other than its own loops:
brute-force enumeration for the permutation, the dense Delta W_g = B_g A_g
form (Sec. 3.3), the rank-consolidation identity, exact finite differences
of the (multilinear) forward, the dense gradient form of Sec. 3.1.2, token
order invariance, and the parameter percentages printed in the paper.
"""
import json
import os
import itertools

import numpy as np
import pytest

import oracle
from paper_2609_06072_gb300 import workloads as W

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def bf(x):
    return W.bf16_bits_to_f32(x).astype(np.float64)


def small_layer(T=12, d=10, f=7, E=6, k=3, G=3, seed=0, ranks=None, e2g=None):
    """A hand-sized random layer (numpy only)."""
    rng = np.random.default_rng(seed)
    idx = np.array([rng.permutation(E)[:k] for _ in range(T)], dtype=np.int32).reshape(T, k)
    if e2g is None:
        e2g = (np.arange(E) % G).astype(np.int32)
    if ranks is None:
        ranks = [2 + (g % 3) for g in range(G)]
    rank_off = np.concatenate([[0], np.cumsum(ranks)]).astype(np.int32)
    Rk = int(rank_off[-1])
    q = lambda *s: W.f32_to_bf16_bits(rng.standard_normal(s).astype(np.float32))
    return dict(idx=idx, e2g=np.asarray(e2g, np.int32), rank_off=rank_off, G=G, T=T, k=k, E=E, d=d, f=f,
                X=q(T, d), h=q(T * k, f), Ag=q(Rk, d), Btg=q(Rk, f), Ad=q(Rk, f), Btd=q(Rk, d),
                dYg=q(T * k, f), dYd=q(T * k, d), Yin=q(T * k, f))


# ---------------------------------------------------------------- permute
def brute_permutation(idx, e2g, G):
    T, k = idx.shape
    pairs = [(int(e2g[idx[t, j]]), int(idx[t, j]), t, t * k + j) for t in range(T) for j in range(k)]
    rows = sorted(pairs)  # keys are unique: a token routes to an expert at most once
    row_pair = [p for (_, _, _, p) in rows]
    uniq = sorted(set((g, t) for (g, _, t, _) in pairs))
    return rows, row_pair, uniq


@pytest.mark.parametrize("case", [
    dict(T=12, E=6, k=3, G=3), dict(T=1, E=4, k=1, G=2), dict(T=9, E=5, k=5, G=2),
    dict(T=30, E=8, k=2, G=1), dict(T=17, E=7, k=3, G=7), dict(T=0, E=4, k=2, G=2),
])
def test_permute_matches_bruteforce(case):
    L = small_layer(T=case["T"], E=case["E"], k=case["k"], G=case["G"], seed=case["T"])
    idx, e2g, G = L["idx"].reshape(case["T"], case["k"]), L["e2g"], case["G"]
    P = oracle.permute(idx, e2g, G)
    rows, row_pair, uniq = brute_permutation(idx, e2g, G)
    assert P["row_pair"].tolist() == row_pair
    assert sorted(P["pair_row"].tolist()) == list(range(len(row_pair)))
    for r, p in enumerate(row_pair):
        assert P["pair_row"][p] == r
    # group / expert segments
    for g in range(G):
        seg = [i for i, (gg, _, _, _) in enumerate(rows) if gg == g]
        assert P["group_off"][g + 1] - P["group_off"][g] == len(seg)
        if seg:
            assert P["group_off"][g] == seg[0]
    for e in range(case["E"]):
        seg = [i for i, (_, ee, _, _) in enumerate(rows) if ee == e]
        assert P["expert_cnt"][e] == len(seg)
        if seg:
            assert P["expert_off"][e] == seg[0] and seg == list(range(seg[0], seg[0] + len(seg)))
    # unique (g, t) pairs, Sec. 3.5: A(x) = {g(e) : e in R(x)}
    assert P["U"] == len(uniq)
    assert P["uniq_tok"].tolist() == [t for (_, t) in uniq]
    for g in range(G):
        assert P["uniq_off"][g + 1] - P["uniq_off"][g] == sum(1 for (gg, _) in uniq if gg == g)
    for u, (g, t) in enumerate(uniq):
        lo, hi = P["uniq_rows_ptr"][u], P["uniq_rows_ptr"][u + 1]
        expect = [i for i, (gg, _, tt, _) in enumerate(rows) if gg == g and tt == t]  # ascending e
        assert P["uniq_rows"][lo:hi].tolist() == expect
        for r in expect:
            assert P["row_uniq"][r] == u
    for t in range(case["T"]):
        expect = [u for u, (g, tt) in enumerate(uniq) if tt == t]  # ascending g
        got = [u for u in P["tok_uniq"][t].tolist() if u >= 0]
        assert got == expect
        assert all(u == -1 for u in P["tok_uniq"][t][len(expect):])


def test_permute_rejects_invalid_routing():
    idx = np.array([[0, 1], [2, 2]], np.int32)  # duplicate expert in a token
    with pytest.raises(oracle.OracleError) as ei:
        oracle.permute(idx, np.array([0, 0, 1, 1], np.int32), 2)
    assert ei.value.status == oracle.OR_ERR_INDEX
    idx = np.array([[0, 4]], np.int32)  # expert out of range
    with pytest.raises(oracle.OracleError):
        oracle.permute(idx, np.array([0, 0, 1, 1], np.int32), 2)
    with pytest.raises(oracle.OracleError):  # map out of range
        oracle.permute(np.array([[0, 1]], np.int32), np.array([0, 2, 1, 1], np.int32), 2)


def test_permute_tiny_config_invariants():
    L = W.Layer(W.get_config("tiny"), seed=1)
    P = oracle.permute(L.topk_idx, L.e2g, L.G)
    R = L.cfg.R
    assert P["group_off"][-1] == R and np.all(np.diff(P["group_off"]) >= 0)
    assert P["expert_cnt"].sum() == R
    assert np.array_equal(np.sort(P["row_pair"]), np.arange(R))
    g_of = L.e2g[L.topk_idx]
    U = sum(len(set(row)) for row in g_of.tolist())
    assert P["U"] == U and P["uniq_rows_ptr"][-1] == R


# ---------------------------------------------------------------- forward
def test_fwd_equals_dense_delta_w():
    """Sec. 3.3: the shared adapter is Delta W_g = B_g A_g; apply it densely."""
    L = small_layer()
    s = 1.7
    for proj, X, xpp, A, Bt in (("gate", L["X"], False, L["Ag"], L["Btg"]), ("down", L["h"], True, L["Ad"], L["Btd"])):
        y, H = oracle.fwd(L["idx"], L["e2g"], L["rank_off"], X, A, Bt, s, x_per_pair=xpp, want_h=True)
        for p in range(L["T"] * L["k"]):
            t = p // L["k"]
            g = L["e2g"][L["idx"].ravel()[p]]
            r0, r1 = L["rank_off"][g], L["rank_off"][g + 1]
            dW = bf(Bt[r0:r1]).T @ bf(A[r0:r1])  # d_out x d_in
            x = bf(X[p] if xpp else X[t])
            np.testing.assert_allclose(y[p], s * dW @ x, rtol=1e-12, atol=1e-12)
            np.testing.assert_allclose(H[p, : r1 - r0], bf(A[r0:r1]) @ x, rtol=1e-12, atol=1e-12)
            assert np.all(H[p, r1 - r0:] == 0)


def test_fwd_adds_base_output():
    L = small_layer(seed=3)
    y0, _ = oracle.fwd(L["idx"], L["e2g"], L["rank_off"], L["X"], L["Ag"], L["Btg"], 2.0)
    y1, _ = oracle.fwd(L["idx"], L["e2g"], L["rank_off"], L["X"], L["Ag"], L["Btg"], 2.0, y_in=L["Yin"])
    np.testing.assert_allclose(y1, y0 + bf(L["Yin"]), rtol=0, atol=1e-12)


def test_consolidated_adapter_is_sum_of_expert_adapters():
    """Rank consolidation (Sec. 3.3): stacking the experts' A_e and B_e of a
    group gives B_g A_g = sum_{e in g} B_e A_e, so the group output equals the
    sum of the expert-wise outputs (Sec. 3.1) of its members."""
    rng = np.random.default_rng(5)
    T, d, f, E, r = 10, 9, 6, 6, 3
    e2g = np.array([0, 1, 0, 2, 1, 0], np.int32)
    G = 3
    A_e = W.f32_to_bf16_bits(rng.standard_normal((E * r, d)).astype(np.float32))
    Bt_e = W.f32_to_bf16_bits(rng.standard_normal((E * r, f)).astype(np.float32))
    members = [np.flatnonzero(e2g == g) for g in range(G)]
    rows = [np.concatenate([np.arange(e * r, (e + 1) * r) for e in m]) for m in members]
    A_g = np.concatenate([A_e[rr] for rr in rows])
    Bt_g = np.concatenate([Bt_e[rr] for rr in rows])
    rank_off = np.concatenate([[0], np.cumsum([r * len(m) for m in members])]).astype(np.int32)
    X = W.f32_to_bf16_bits(rng.standard_normal((T, d)).astype(np.float32))
    ident = np.arange(E, dtype=np.int32)
    ew_off = (np.arange(E + 1) * r).astype(np.int32)
    # expert-wise delta of every expert on every token (k = 1 routing per call)
    ew = {}
    for e in range(E):
        y, _ = oracle.fwd(np.full((T, 1), e, np.int32), ident, ew_off, X, A_e, Bt_e, 1.0)
        ew[e] = y
    for g in range(G):
        e0 = members[g][0]
        yg, _ = oracle.fwd(np.full((T, 1), e0, np.int32), e2g, rank_off, X, A_g, Bt_g, 1.0)
        np.testing.assert_allclose(yg, sum(ew[e] for e in members[g]), rtol=1e-12, atol=1e-12)


def test_identity_map_is_expertwise_lora():
    """G = E with the identity map and r_g = r is expert-wise LoRA (Sec. 3.1):
    each pair uses its own expert's A_e, B_e."""
    L = small_layer(E=5, G=5, e2g=np.arange(5), ranks=[3] * 5, seed=7)
    y, _ = oracle.fwd(L["idx"], L["e2g"], L["rank_off"], L["X"], L["Ag"], L["Btg"], 0.5)
    for p in range(L["T"] * L["k"]):
        e = L["idx"].ravel()[p]
        h_e = bf(L["Ag"][3 * e:3 * e + 3]) @ bf(L["X"][p // L["k"]])
        np.testing.assert_allclose(y[p], 0.5 * bf(L["Btg"][3 * e:3 * e + 3]).T @ h_e, rtol=1e-12, atol=1e-12)


def test_shared_input_reuse_is_exact():
    """Sec. 3.5: c_g(x) is the same for every routed expert of the group, so
    pairs of one token in one group carry identical deltas."""
    L = W.Layer(W.get_config("tiny"), seed=2)
    P = oracle.permute(L.topk_idx, L.e2g, L.G)
    y, _ = oracle.fwd(L.topk_idx, L.e2g, L.rank_off, L.X(), L.A("up"), L.Bt("up"), 2.0)
    shared = 0
    for u in range(P["U"]):
        rows = P["uniq_rows"][P["uniq_rows_ptr"][u]:P["uniq_rows_ptr"][u + 1]]
        pairs = P["row_pair"][rows]
        for p in pairs[1:]:
            assert np.array_equal(y[p], y[pairs[0]])
            shared += 1
    assert shared > 0


def test_selection_matches_full():
    L = small_layer(seed=11)
    full, Hf = oracle.fwd(L["idx"], L["e2g"], L["rank_off"], L["X"], L["Ag"], L["Btg"], 2.0, want_h=True)
    sel = np.array([5, 0, 17], np.int32)
    part, Hp = oracle.fwd(L["idx"], L["e2g"], L["rank_off"], L["X"], L["Ag"], L["Btg"], 2.0, sel=sel, want_h=True)
    assert np.array_equal(part, full[sel]) and np.array_equal(Hp, Hf[sel])
    dx = oracle.bwd_dx(L["idx"], L["e2g"], L["rank_off"], L["dYg"], L["Ag"], L["Btg"], 2.0)
    sdx = oracle.bwd_dx(L["idx"], L["e2g"], L["rank_off"], L["dYg"], L["Ag"], L["Btg"], 2.0,
                        sel=np.array([3, 1], np.int32))
    assert np.array_equal(sdx, dx[[3, 1]])
    dA, dBt = oracle.bwd_w(L["idx"], L["e2g"], L["rank_off"], L["X"], L["dYg"], L["Ag"], L["Btg"], 2.0)
    sA, sB = oracle.bwd_w(L["idx"], L["e2g"], L["rank_off"], L["X"], L["dYg"], L["Ag"], L["Btg"], 2.0,
                          sel=np.array([4, 1], np.int32))
    assert np.array_equal(sA, dA[[4, 1]]) and np.array_equal(sB, dBt[[4, 1]])


# ---------------------------------------------------------------- backward
def _loss(L, proj, X=None, A=None, Bt=None, s=1.3):
    """L = sum_p dY_p . y_p for the projection (a linear functional of y)."""
    if proj == "gate":
        X = L["X"] if X is None else X
        A = L["Ag"] if A is None else A
        Bt = L["Btg"] if Bt is None else Bt
        y, _ = oracle.fwd(L["idx"], L["e2g"], L["rank_off"], X, A, Bt, s)
        return float(np.sum(y * bf(L["dYg"])))
    X = L["h"] if X is None else X
    A = L["Ad"] if A is None else A
    Bt = L["Btd"] if Bt is None else Bt
    y, _ = oracle.fwd(L["idx"], L["e2g"], L["rank_off"], X, A, Bt, s, x_per_pair=True)
    return float(np.sum(y * bf(L["dYd"])))


def _bump(arr, i, j):
    """Return a copy with element (i, j) replaced by another bf16 value, and
    the (exact) step taken."""
    out = arr.copy()
    old = bf(arr[i:i + 1, j:j + 1])[0, 0]
    new_bits = W.f32_to_bf16_bits(np.array([[old * 1.5 + 0.25]], np.float32))
    out[i, j] = new_bits[0, 0]
    return out, bf(new_bits)[0, 0] - old


@pytest.mark.parametrize("proj", ["gate", "down"])
def test_gradients_match_finite_differences(proj):
    """The forward is linear in each of X, A, B separately, so a finite
    difference with any step is exact up to rounding."""
    L = small_layer(seed=13)
    s = 1.3
    xpp = proj == "down"
    X, A, Bt, dY = (L["X"], L["Ag"], L["Btg"], L["dYg"]) if proj == "gate" else (L["h"], L["Ad"], L["Btd"], L["dYd"])
    dx = oracle.bwd_dx(L["idx"], L["e2g"], L["rank_off"], dY, A, Bt, s, x_per_pair=xpp)
    dA, dBt = oracle.bwd_w(L["idx"], L["e2g"], L["rank_off"], X, dY, A, Bt, s, x_per_pair=xpp)
    base = _loss(L, proj, s=s)
    rng = np.random.default_rng(0)
    for _ in range(12):
        i, j = rng.integers(X.shape[0]), rng.integers(X.shape[1])
        Xp, step = _bump(X, i, j)
        fd = (_loss(L, proj, X=Xp, s=s) - base) / step
        np.testing.assert_allclose(fd, dx[i, j], rtol=1e-7, atol=1e-9)
        i, j = rng.integers(A.shape[0]), rng.integers(A.shape[1])
        Ap, step = _bump(A, i, j)
        fd = (_loss(L, proj, A=Ap, s=s) - base) / step
        np.testing.assert_allclose(fd, dA[i, j], rtol=1e-7, atol=1e-9)
        i, j = rng.integers(Bt.shape[0]), rng.integers(Bt.shape[1])
        Bp, step = _bump(Bt, i, j)
        fd = (_loss(L, proj, Bt=Bp, s=s) - base) / step
        np.testing.assert_allclose(fd, dBt[i, j], rtol=1e-7, atol=1e-9)


@pytest.mark.parametrize("proj", ["gate", "down"])
def test_weight_gradients_dense_form(proj):
    """Sec. 3.1.2 / 3.4: the gradient of Delta W_g collects every pair routed
    into the group, M_g = s sum_{p in g} dy_p x_p^T; with Delta W = B A,
    dA_g = B_g^T M_g and dB_g = M_g A_g^T."""
    L = small_layer(seed=17)
    s = 0.7
    xpp = proj == "down"
    X, A, Bt, dY = (L["X"], L["Ag"], L["Btg"], L["dYg"]) if proj == "gate" else (L["h"], L["Ad"], L["Btd"], L["dYd"])
    dA, dBt = oracle.bwd_w(L["idx"], L["e2g"], L["rank_off"], X, dY, A, Bt, s, x_per_pair=xpp)
    gp = L["e2g"][L["idx"].ravel()]
    xs = bf(X) if xpp else bf(X)[np.arange(L["T"] * L["k"]) // L["k"]]
    for g in range(L["G"]):
        r0, r1 = L["rank_off"][g], L["rank_off"][g + 1]
        m = gp == g
        M = s * bf(dY)[m].T @ xs[m]  # d_out x d_in
        np.testing.assert_allclose(dA[r0:r1], bf(Bt[r0:r1]) @ M, rtol=1e-11, atol=1e-11)
        np.testing.assert_allclose(dBt[r0:r1], (M @ bf(A[r0:r1]).T).T, rtol=1e-11, atol=1e-11)


def test_empty_group_gets_zero_gradient():
    L = small_layer(E=6, G=4, e2g=[0, 0, 1, 1, 2, 2], ranks=[2, 2, 2, 3], seed=19)  # group 3 has no expert
    dA, dBt = oracle.bwd_w(L["idx"], L["e2g"], L["rank_off"], L["X"], L["dYg"], L["Ag"], L["Btg"], 1.0)
    r0 = L["rank_off"][3]
    assert np.all(dA[r0:] == 0) and np.all(dBt[r0:] == 0)


def test_token_order_invariance():
    """Permuting tokens permutes every per-token / per-pair output and leaves
    the weight gradients unchanged (Sec. 3.4: y(x) depends only on x)."""
    L = small_layer(T=14, seed=23)
    T, k = L["T"], L["k"]
    pi = np.random.default_rng(1).permutation(T)
    pairs = (pi[:, None] * k + np.arange(k)[None, :]).ravel()
    idx2 = L["idx"][pi]
    y, _ = oracle.fwd(L["idx"], L["e2g"], L["rank_off"], L["X"], L["Ag"], L["Btg"], 2.0)
    y2, _ = oracle.fwd(idx2, L["e2g"], L["rank_off"], L["X"][pi], L["Ag"], L["Btg"], 2.0)
    np.testing.assert_array_equal(y2, y[pairs])
    dx = oracle.bwd_dx(L["idx"], L["e2g"], L["rank_off"], L["dYg"], L["Ag"], L["Btg"], 2.0)
    dx2 = oracle.bwd_dx(idx2, L["e2g"], L["rank_off"], L["dYg"][pairs], L["Ag"], L["Btg"], 2.0)
    np.testing.assert_array_equal(dx2, dx[pi])
    dA, dBt = oracle.bwd_w(L["idx"], L["e2g"], L["rank_off"], L["X"], L["dYg"], L["Ag"], L["Btg"], 2.0)
    dA2, dBt2 = oracle.bwd_w(idx2, L["e2g"], L["rank_off"], L["X"][pi], L["dYg"][pairs], L["Ag"], L["Btg"], 2.0)
    np.testing.assert_allclose(dA2, dA, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(dBt2, dBt, rtol=1e-12, atol=1e-12)
    P, P2 = oracle.permute(L["idx"], L["e2g"], L["G"]), oracle.permute(idx2, L["e2g"], L["G"])
    assert P["U"] == P2["U"]
    assert np.array_equal(P["group_off"], P2["group_off"]) and np.array_equal(P["expert_cnt"], P2["expert_cnt"])


# ---------------------------------------------------------------- budget
def test_budget_equality_all_configs():
    """Sec. 3.3: sum_g (d_in + d_out) r_g = sum_e (d_in + d_out) r_e."""
    for name in W.CONFIGS:
        L = W.Layer(W.get_config(name), seed=0)
        for d_in, d_out in ((L.cfg.d, L.cfg.f), (L.cfg.f, L.cfg.d)):
            assert oracle.group_budget(L.rank_off, d_in, d_out) == oracle.expertwise_budget(
                [L.cfg.r] * L.cfg.E, d_in, d_out)
            assert oracle.uniform_rank(oracle.group_budget(L.rank_off, d_in, d_out), L.cfg.E, d_in, d_out) == L.cfg.r
        Le = W.Layer(W.get_config(name), seed=0, expertwise=True)
        assert np.array_equal(Le.rank_off, np.arange(L.cfg.E + 1) * L.cfg.r)


def test_budget_reproduces_printed_percentages():
    g = json.load(open(os.path.join(GOLDEN, "params_percent.json")))
    tol = g["implied_total_rel_tol"]
    implied = {}
    for row in g["printed"]:
        b = g["backbones"][row["model"]]
        n = oracle.model_adapter_params(b["layers"], b["E"], row["r"], b["d"], b["ff"])
        # the printed percentage is rounded to 2 decimals: the implied total
        # parameter count lies in an interval
        lo, hi = n / ((row["percent"] + 0.005) / 100), n / ((row["percent"] - 0.005) / 100)
        assert lo <= b["total_params"] * (1 + tol) and hi >= b["total_params"] * (1 - tol), row
        implied.setdefault(row["model"], []).append((lo, hi))
    # the same backbone at two ranks must admit one common total (percent is linear in r)
    for model, ivs in implied.items():
        assert max(lo for lo, _ in ivs) <= min(hi for _, hi in ivs), model
    # a plausible counting mistake (gate and up only) fails the check
    b = g["backbones"]["OLMoE"]
    n2 = 2 * b["layers"] * b["E"] * 2 * (b["d"] + b["ff"])
    assert abs(100 * n2 / b["total_params"] - 0.27) > 0.05
