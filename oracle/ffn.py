"""fp64 CPU oracle of the routed expert FFN with group-shared LoRA deltas:
the base expert GEMMs and the adapters together (arxiv 2609.06072).

TEST INFRASTRUCTURE ONLY, like the rest of this package.  Plain numpy in
float64, one (token, slot) pair at a time; inputs are float64 arrays (decode
bf16 before calling), so finite differences can take small steps.

For pair p = (t, j) routed to expert e (App. "Implementation and Profiling
of Grouped Adapter Execution", the gated FFN of every backbone):
    u_p = (W_e^up   + dW_g^up)   x_t
    v_p = (W_e^gate + dW_g^gate) x_t
    h_p = phi(v_p) * u_p,            phi = SiLU, phi(v) = v sigma(v)
    y_p = (W_e^down + dW_g^down) h_p
with dW_g = s B_g A_g the shared adapter of the expert's group for that
projection (Sec. 3.2-3.4; each projection may have its own map), and, with
gate weights, z_t = sum_j p_tj y_tj (Sec. 3.1's y(x)).

The backward keeps the base weights frozen (LoRA fine-tuning) and returns
the token-input gradient, the adapter gradients of the three projections
and, with gate weights, the gate-weight gradients dp_tj = dz_t . y_tj.
"""
from __future__ import annotations

from typing import Dict, Optional

import numpy as np

PROJ = ("gate", "up", "down")


def silu(v):
    return v / (1.0 + np.exp(-v))


def silu_grad(v):
    """phi'(v) = sigma(v) (1 + v (1 - sigma(v)))."""
    sg = 1.0 / (1.0 + np.exp(-v))
    return sg * (1.0 + v * (1.0 - sg))


def _adapter(maps, proj, e):
    """Rows of A / B^T holding the adapter of expert e's group for one projection."""
    e2g, rank_off = maps[proj]
    g = int(e2g[e])
    return slice(int(rank_off[g]), int(rank_off[g + 1]))


def ffn_fwd(topk_idx, maps, X, W: Dict[str, np.ndarray], A: Dict[str, np.ndarray], Bt: Dict[str, np.ndarray],
            s: float, w: Optional[np.ndarray] = None):
    """Forward over every pair.  maps[proj] = (e2g [E], rank_off [G+1]);
    W['gate'|'up'] [E, f, d], W['down'] [E, d, f]; A[proj] [sum r_g, d_in],
    Bt[proj] [sum r_g, d_out]; X [T, d]; w [T, k] gate weights or None.
    Returns dict of u, v, h [T*k, f], y [T*k, d] and, with w, z [T, d]."""
    idx = np.asarray(topk_idx)
    T, k = idx.shape
    f = W["gate"].shape[1]
    d = X.shape[1]
    out = {n: np.zeros((T * k, f)) for n in ("u", "v", "h")}
    out["y"] = np.zeros((T * k, d))
    for p in range(T * k):
        t, e = p // k, int(idx.ravel()[p])
        x = X[t]
        ru, rv, rd = (_adapter(maps, q, e) for q in ("up", "gate", "down"))
        u = W["up"][e] @ x + s * Bt["up"][ru].T @ (A["up"][ru] @ x)
        v = W["gate"][e] @ x + s * Bt["gate"][rv].T @ (A["gate"][rv] @ x)
        h = silu(v) * u
        y = W["down"][e] @ h + s * Bt["down"][rd].T @ (A["down"][rd] @ h)
        out["u"][p], out["v"][p], out["h"][p], out["y"][p] = u, v, h, y
    if w is not None:
        out["z"] = (np.asarray(w, dtype=np.float64).reshape(T, k, 1) * out["y"].reshape(T, k, d)).sum(axis=1)
    return out


def ffn_bwd(topk_idx, maps, X, W, A, Bt, s, dy=None, w=None, dz=None):
    """Backward with frozen base weights.  Either dy [T*k, d] per pair, or
    gate weights w [T, k] with a token gradient dz [T, d] (then dy_p = w_p dz_t).
    Returns dict: dX [T, d]; dA[proj], dBt[proj] (shapes of A, Bt); and, with
    w, dp [T*k] = dz_t . y_p."""
    idx = np.asarray(topk_idx)
    T, k = idx.shape
    fw = ffn_fwd(idx, maps, X, W, A, Bt, s)
    if dz is not None:
        dy = np.asarray(w, dtype=np.float64).reshape(-1, 1) * np.repeat(dz, k, axis=0)
    out = {"dX": np.zeros_like(X, dtype=np.float64)}
    out["dA"] = {q: np.zeros_like(A[q], dtype=np.float64) for q in PROJ}
    out["dBt"] = {q: np.zeros_like(Bt[q], dtype=np.float64) for q in PROJ}
    for p in range(T * k):
        t, e = p // k, int(idx.ravel()[p])
        x, h, u, v, g_out = X[t], fw["h"][p], fw["u"][p], fw["v"][p], dy[p]
        rd = _adapter(maps, "down", e)
        # y = (W_d + s B_d A_d) h
        bd = Bt["down"][rd] @ g_out                       # B_d^T dy
        dh = W["down"][e].T @ g_out + s * A["down"][rd].T @ bd
        out["dA"]["down"][rd] += s * np.outer(bd, h)
        out["dBt"]["down"][rd] += s * np.outer(A["down"][rd] @ h, g_out)
        # h = phi(v) * u
        du = dh * silu(v)
        dv = dh * u * silu_grad(v)
        for q, dq in (("up", du), ("gate", dv)):
            rq = _adapter(maps, q, e)
            bq = Bt[q][rq] @ dq                           # B_q^T dq
            out["dX"][t] += W[q][e].T @ dq + s * A[q][rq].T @ bq
            out["dA"][q][rq] += s * np.outer(bq, x)
            out["dBt"][q][rq] += s * np.outer(A[q][rq] @ x, dq)
    if dz is not None:
        out["dp"] = (np.repeat(dz, k, axis=0) * fw["y"]).sum(axis=1)
    return out
