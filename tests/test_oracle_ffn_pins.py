"""Pins of the expert-FFN oracle (base expert weights plus group-shared LoRA
deltas on gate, up and down, SiLU gating, gate-weighted combine): the dense
form with every Delta W_g materialised and added to W_e, reduction to the
gate/up adapter oracle when the base weights are zero, central finite
differences of the whole forward for every input and adapter tensor and the
gate weights, and token-order invariance."""
import numpy as np
import pytest

import oracle
from oracle import ffn as F
from paper_2609_06072_gb300 import workloads as W


def layer(T=5, d=7, f=6, E=5, k=2, seed=0, expertwise=False):
    rng = np.random.default_rng(seed)
    idx = np.array([rng.permutation(E)[:k] for _ in range(T)], dtype=np.int32)
    maps, A, Bt = {}, {}, {}
    for q, (di, do) in (("gate", (d, f)), ("up", (d, f)), ("down", (f, d))):
        if expertwise:
            e2g = np.arange(E, dtype=np.int32)
            ranks = [2] * E
        else:
            e2g = rng.integers(0, 3, E).astype(np.int32)
            e2g[:3] = [0, 1, 2]  # every group non-empty
            ranks = [1 + int(rng.integers(1, 4)) for _ in range(3)]
        ro = np.concatenate([[0], np.cumsum(ranks)]).astype(np.int32)
        maps[q] = (e2g, ro)
        A[q] = rng.standard_normal((ro[-1], di)) / np.sqrt(di)
        Bt[q] = rng.standard_normal((ro[-1], do)) * 0.3
    Wb = {"gate": rng.standard_normal((E, f, d)) / np.sqrt(d), "up": rng.standard_normal((E, f, d)) / np.sqrt(d),
          "down": rng.standard_normal((E, d, f)) / np.sqrt(f)}
    X = rng.standard_normal((T, d))
    w = rng.uniform(0.1, 1.0, (T, k))
    dz = rng.standard_normal((T, d))
    return dict(idx=idx, maps=maps, A=A, Bt=Bt, W=Wb, X=X, w=w, dz=dz, T=T, k=k, d=d, f=f, E=E)


def test_ffn_equals_dense_materialised_weights():
    """W_e + s B_g A_g formed explicitly per projection, then the gated FFN."""
    L = layer()
    s = 1.6
    out = F.ffn_fwd(L["idx"], L["maps"], L["X"], L["W"], L["A"], L["Bt"], s, w=L["w"])
    k = L["k"]
    z = np.zeros((L["T"], L["d"]))
    for p in range(L["T"] * k):
        t, e = p // k, L["idx"].ravel()[p]
        Weff = {}
        for q in F.PROJ:
            e2g, ro = L["maps"][q]
            g = e2g[e]
            Weff[q] = L["W"][q][e] + s * L["Bt"][q][ro[g]:ro[g + 1]].T @ L["A"][q][ro[g]:ro[g + 1]]
        u, v = Weff["up"] @ L["X"][t], Weff["gate"] @ L["X"][t]
        h = v / (1 + np.exp(-v)) * u
        y = Weff["down"] @ h
        assert np.allclose(out["u"][p], u, atol=1e-12) and np.allclose(out["v"][p], v, atol=1e-12)
        assert np.allclose(out["h"][p], h, atol=1e-12) and np.allclose(out["y"][p], y, atol=1e-12)
        z[t] += L["w"][t, p % k] * y
    assert np.allclose(out["z"], z, atol=1e-12)


def test_zero_base_weights_reduce_to_the_gate_up_adapter_oracle():
    """With W_e = 0, u and v are the shared-input adapter deltas that the
    (separately pinned) gate/up oracle computes."""
    L = layer(seed=3)
    bits = lambda a: W.f32_to_bf16_bits(np.asarray(a, np.float32))
    dec = lambda b: W.bf16_bits_to_f32(b).astype(np.float64)
    Xb = bits(L["X"])
    Ab = {q: bits(L["A"][q]) for q in F.PROJ}
    Bb = {q: bits(L["Bt"][q]) for q in F.PROJ}
    zeroW = {q: np.zeros_like(L["W"][q]) for q in F.PROJ}
    out = F.ffn_fwd(L["idx"], L["maps"], dec(Xb), zeroW, {q: dec(Ab[q]) for q in F.PROJ},
                    {q: dec(Bb[q]) for q in F.PROJ}, 2.0)
    for name, q in (("u", "up"), ("v", "gate")):
        e2g, ro = L["maps"][q]
        ref, _ = oracle.fwd(L["idx"], e2g, ro, Xb, Ab[q], Bb[q], 2.0)
        assert np.allclose(out[name], ref, rtol=1e-12, atol=1e-12)


def _loss(L, s, X=None, A=None, Bt=None, w=None):
    out = F.ffn_fwd(L["idx"], L["maps"], L["X"] if X is None else X, L["W"], L["A"] if A is None else A,
                    L["Bt"] if Bt is None else Bt, s, w=L["w"] if w is None else w)
    return float((out["z"] * L["dz"]).sum())


@pytest.mark.parametrize("expertwise", [False, True])
def test_ffn_gradients_match_central_differences(expertwise):
    L = layer(seed=7, expertwise=expertwise)
    s, eps = 1.3, 1e-6
    g = F.ffn_bwd(L["idx"], L["maps"], L["X"], L["W"], L["A"], L["Bt"], s, w=L["w"], dz=L["dz"])
    rng = np.random.default_rng(1)

    def central(fn):
        return (fn(+eps) - fn(-eps)) / (2 * eps)

    for _ in range(6):
        i, j = rng.integers(L["T"]), rng.integers(L["d"])

        def fx(h):
            X = L["X"].copy()
            X[i, j] += h
            return _loss(L, s, X=X)
        assert abs(central(fx) - g["dX"][i, j]) <= 1e-6 * max(1.0, abs(g["dX"][i, j]))
        for q in F.PROJ:
            a, b = rng.integers(L["A"][q].shape[0]), rng.integers(L["A"][q].shape[1])

            def fa(h):
                A = {k2: v.copy() for k2, v in L["A"].items()}
                A[q][a, b] += h
                return _loss(L, s, A=A)
            assert abs(central(fa) - g["dA"][q][a, b]) <= 1e-6 * max(1.0, abs(g["dA"][q][a, b]))
            a, b = rng.integers(L["Bt"][q].shape[0]), rng.integers(L["Bt"][q].shape[1])

            def fb(h):
                Bt = {k2: v.copy() for k2, v in L["Bt"].items()}
                Bt[q][a, b] += h
                return _loss(L, s, Bt=Bt)
            assert abs(central(fb) - g["dBt"][q][a, b]) <= 1e-6 * max(1.0, abs(g["dBt"][q][a, b]))
        t, jj = rng.integers(L["T"]), rng.integers(L["k"])

        def fw(h):
            w = L["w"].copy()
            w[t, jj] += h
            return _loss(L, s, w=w)
        assert abs(central(fw) - g["dp"][t * L["k"] + jj]) <= 1e-6 * max(1.0, abs(g["dp"][t * L["k"] + jj]))


def test_silu_and_its_derivative():
    v = np.linspace(-6, 6, 25)
    assert np.allclose(F.silu(v), v / (1 + np.exp(-v)), atol=1e-15)
    eps = 1e-6
    assert np.allclose(F.silu_grad(v), (F.silu(v + eps) - F.silu(v - eps)) / (2 * eps), atol=1e-8)
    assert F.silu(0.0) == 0.0 and abs(F.silu_grad(0.0) - 0.5) < 1e-15


def test_ffn_token_order_invariance():
    L = layer(T=6, seed=11)
    pi = np.random.default_rng(2).permutation(L["T"])
    k = L["k"]
    pairs = (pi[:, None] * k + np.arange(k)[None, :]).ravel()
    a = F.ffn_fwd(L["idx"], L["maps"], L["X"], L["W"], L["A"], L["Bt"], 0.9, w=L["w"])
    b = F.ffn_fwd(L["idx"][pi], L["maps"], L["X"][pi], L["W"], L["A"], L["Bt"], 0.9, w=L["w"][pi])
    assert np.allclose(b["z"], a["z"][pi], atol=1e-13) and np.allclose(b["y"], a["y"][pairs], atol=1e-13)
    ga = F.ffn_bwd(L["idx"], L["maps"], L["X"], L["W"], L["A"], L["Bt"], 0.9, w=L["w"], dz=L["dz"])
    gb = F.ffn_bwd(L["idx"][pi], L["maps"], L["X"][pi], L["W"], L["A"], L["Bt"], 0.9, w=L["w"][pi], dz=L["dz"][pi])
    assert np.allclose(gb["dX"], ga["dX"][pi], atol=1e-12)
    for q in F.PROJ:
        assert np.allclose(gb["dA"][q], ga["dA"][q], atol=1e-12) and np.allclose(gb["dBt"][q], ga["dBt"][q], atol=1e-12)
