"""fp64 CPU oracle for ACE grouped adapter execution.

TEST INFRASTRUCTURE ONLY: the test suite, the smoke check and the benchmark's
CPU-baseline / reference leg may import this package; the product library
never does, and the two share no code.  The arithmetic lives in
``ace_oracle.c`` (plain C loops in double precision, OpenMP over independent
outputs, each reduction serial in a fixed order); this module only builds it
with gcc and marshals numpy arrays through ctypes.

Functions and the passages they follow (arxiv 2609.06072):

* ``permute``  -- routing set R(x) (Sec. 3.1), active groups A(x) (Sec. 3.5);
                  rows ordered by (g(e), e, t), unique pairs by (g, t).
* ``fwd``      -- y_out = y_in + s B_g (A_g x), per pair (Sec. 3.3-3.5,
                  App. "Implementation and Profiling of Grouped Adapter
                  Execution": gate/up take x, down takes h_e).
* ``bwd_dx``   -- adjoint of ``fwd`` w.r.t. its input.
* ``bwd_w``    -- dA_g, dB_g^T: shared adapter updates (Sec. 3.4) from the
                  gradient form of Sec. 3.1.2.
* ``budget``   -- parameter budget of Sec. 3.1.1 / Sec. 3.3 (pure Python).
* ``combine_fwd``, ``combine_bwd_dh``, ``combine_bwd_w``
               -- the down projection's delta weighted by the gate p_e(x) and
                  summed over a token's routed experts (the combine of
                  Sec. 3.1's y(x)), and its adjoint: dh, the gate-weight
                  gradient, dA_g and dB_g^T.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Dict, Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ace_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lib = None

OR_OK = 0
OR_ERR_ARG = 1
OR_ERR_INDEX = 4


def build(force: bool = False) -> str:
    """Compile ace_oracle.c into liboracle.so next to it (gcc, OpenMP)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fopenmp", "-fPIC", "-shared",
               "-std=c11", _SRC, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        build()
        lib = ctypes.CDLL(_LIB_PATH)
        i32, i64, dbl, vp = ctypes.c_int32, ctypes.c_int64, ctypes.c_double, ctypes.c_void_p
        lib.oracle_version.restype = ctypes.c_int
        lib.oracle_permute.restype = ctypes.c_int
        lib.oracle_permute.argtypes = [i32, i32, i32, i32, vp, vp] + [vp] * 12
        lib.oracle_fwd.restype = ctypes.c_int
        lib.oracle_fwd.argtypes = [i32, i32, i32, i32, vp, vp, vp, i32, i32, vp, i32, vp, vp, dbl, vp, vp, vp,
                                   i32, vp, i64]
        lib.oracle_bwd_dx.restype = ctypes.c_int
        lib.oracle_bwd_dx.argtypes = [i32, i32, i32, i32, vp, vp, vp, i32, i32, i32, vp, vp, vp, dbl, vp, vp, vp,
                                      i64]
        lib.oracle_bwd_w.restype = ctypes.c_int
        lib.oracle_bwd_w.argtypes = [i32, i32, i32, i32, vp, vp, vp, i32, i32, vp, i32, vp, vp, vp, dbl, vp, vp,
                                     vp, i64]
        lib.oracle_combine_fwd.restype = ctypes.c_int
        lib.oracle_combine_fwd.argtypes = [i32, i32, i32, i32, vp, vp, vp, i32, i32, vp, vp, vp, vp, dbl, vp, vp,
                                           vp, i64]
        lib.oracle_combine_bwd_dh.restype = ctypes.c_int
        lib.oracle_combine_bwd_dh.argtypes = [i32, i32, i32, i32, vp, vp, vp, i32, i32, vp, vp, vp, vp, vp, dbl,
                                              vp, vp, vp, vp, i64]
        lib.oracle_combine_bwd_w.restype = ctypes.c_int
        lib.oracle_combine_bwd_w.argtypes = [i32, i32, i32, i32, vp, vp, vp, i32, i32, vp, vp, vp, vp, vp, dbl,
                                             vp, vp, vp, i64]
        _lib = lib
    return _lib


def _p(a: Optional[np.ndarray]):
    return None if a is None else a.ctypes.data


def _c(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


class OracleError(RuntimeError):
    def __init__(self, status: int, what: str):
        super().__init__(f"{what}: oracle status {status}")
        self.status = status


def permute(topk_idx: np.ndarray, e2g: np.ndarray, G: int) -> Dict[str, np.ndarray]:
    """Routing permutation by the plain definition (stable sort on (g, e, t))."""
    lib = _load()
    idx = _c(topk_idx, np.int32)
    T, k = idx.shape
    e2g = _c(e2g, np.int32)
    E = e2g.shape[0]
    R = T * k
    out = {
        "group_off": np.zeros(G + 1, np.int32), "expert_off": np.zeros(E, np.int32),
        "expert_cnt": np.zeros(E, np.int32), "row_pair": np.zeros(R, np.int32),
        "pair_row": np.zeros(R, np.int32), "row_uniq": np.zeros(R, np.int32),
        "uniq_off": np.zeros(G + 1, np.int32), "uniq_tok": np.zeros(max(R, 1), np.int32),
        "uniq_rows_ptr": np.zeros(R + 1, np.int32), "uniq_rows": np.zeros(R, np.int32),
        "tok_uniq": np.zeros(R, np.int32),
    }
    U = np.zeros(1, np.int32)
    st = lib.oracle_permute(T, k, E, G, _p(idx), _p(e2g), _p(out["group_off"]), _p(out["expert_off"]),
                            _p(out["expert_cnt"]), _p(out["row_pair"]), _p(out["pair_row"]),
                            _p(out["row_uniq"]), _p(out["uniq_off"]), _p(out["uniq_tok"]),
                            _p(out["uniq_rows_ptr"]), _p(out["uniq_rows"]), _p(out["tok_uniq"]), _p(U))
    if st != OR_OK:
        raise OracleError(st, "permute")
    u = int(U[0])
    out["U"] = u
    out["uniq_tok"] = out["uniq_tok"][:u].copy()
    out["uniq_rows_ptr"] = out["uniq_rows_ptr"][: u + 1].copy()
    out["tok_uniq"] = out["tok_uniq"].reshape(T, k)
    return out


def fwd(topk_idx, e2g, rank_off, X, A_all, Bt_all, s, x_per_pair=False, y_in=None, sel=None,
        want_h=False):
    """y_out[p] = y_in[p] + s B_g (A_g x_p) for every pair p (or the pairs in sel).

    Returns (y_out, H): [T*k, d_out] / [T*k, r_max] float64, or, with
    ``sel``, [len(sel), ...] with row i holding pair sel[i].
    """
    lib = _load()
    idx = _c(topk_idx, np.int32)
    T, k = idx.shape
    e2g = _c(e2g, np.int32)
    rank_off = _c(rank_off, np.int32)
    G = rank_off.shape[0] - 1
    X = _c(X, np.uint16)
    A_all = _c(A_all, np.uint16)
    Bt_all = _c(Bt_all, np.uint16)
    d_in, d_out = A_all.shape[1], Bt_all.shape[1]
    R = T * k
    sel_a = _c(sel, np.int32)
    n_out = R if sel_a is None else sel_a.shape[0]
    y_out = np.empty((n_out, d_out))
    r_max = int(np.max(np.diff(rank_off))) if G > 0 else 0
    H = np.empty((n_out, r_max)) if want_h else None
    st = lib.oracle_fwd(T, k, e2g.shape[0], G, _p(idx), _p(e2g), _p(rank_off), d_in, d_out, _p(X),
                        int(bool(x_per_pair)), _p(A_all), _p(Bt_all), float(s), _p(_c(y_in, np.uint16)),
                        _p(y_out), _p(H), r_max, _p(sel_a), 0 if sel_a is None else sel_a.shape[0])
    if st != OR_OK:
        raise OracleError(st, "fwd")
    return y_out, H


def bwd_dx(topk_idx, e2g, rank_off, dy, A_all, Bt_all, s, x_per_pair=False, dx_in=None, sel=None):
    """Input gradient: token rows [T, d_in] (gate/up) or pair rows [T*k, d_in]
    (down); with ``sel``, [len(sel), d_in] with row i holding sel[i]."""
    lib = _load()
    idx = _c(topk_idx, np.int32)
    T, k = idx.shape
    e2g = _c(e2g, np.int32)
    rank_off = _c(rank_off, np.int32)
    G = rank_off.shape[0] - 1
    A_all = _c(A_all, np.uint16)
    Bt_all = _c(Bt_all, np.uint16)
    dy = _c(dy, np.uint16)
    d_in, d_out = A_all.shape[1], Bt_all.shape[1]
    n_rows = T * k if x_per_pair else T
    sel_a = _c(sel, np.int32)
    dx = np.empty((n_rows if sel_a is None else sel_a.shape[0], d_in))
    st = lib.oracle_bwd_dx(T, k, e2g.shape[0], G, _p(idx), _p(e2g), _p(rank_off), d_in, d_out,
                           int(bool(x_per_pair)), _p(dy), _p(A_all), _p(Bt_all), float(s),
                           _p(_c(dx_in, np.uint16)), _p(dx), _p(sel_a), 0 if sel_a is None else sel_a.shape[0])
    if st != OR_OK:
        raise OracleError(st, "bwd_dx")
    return dx


def bwd_w(topk_idx, e2g, rank_off, X, dy, A_all, Bt_all, s, x_per_pair=False, sel=None):
    """(dA [sum r_g, d_in], dBt [sum r_g, d_out]) in float64; with ``sel``,
    [len(sel), ...] with row i holding rank row sel[i]."""
    lib = _load()
    idx = _c(topk_idx, np.int32)
    T, k = idx.shape
    e2g = _c(e2g, np.int32)
    rank_off = _c(rank_off, np.int32)
    G = rank_off.shape[0] - 1
    X = _c(X, np.uint16)
    dy = _c(dy, np.uint16)
    A_all = _c(A_all, np.uint16)
    Bt_all = _c(Bt_all, np.uint16)
    d_in, d_out = A_all.shape[1], Bt_all.shape[1]
    n_rank = int(rank_off[-1])
    sel_a = _c(sel, np.int32)
    n_out = n_rank if sel_a is None else sel_a.shape[0]
    dA = np.empty((n_out, d_in))
    dBt = np.empty((n_out, d_out))
    st = lib.oracle_bwd_w(T, k, e2g.shape[0], G, _p(idx), _p(e2g), _p(rank_off), d_in, d_out, _p(X),
                          int(bool(x_per_pair)), _p(dy), _p(A_all), _p(Bt_all), float(s), _p(dA), _p(dBt),
                          _p(sel_a), 0 if sel_a is None else sel_a.shape[0])
    if st != OR_OK:
        raise OracleError(st, "bwd_w")
    return dA, dBt


def _combine_args(topk_idx, e2g, rank_off, w, A_all, Bt_all):
    idx = _c(topk_idx, np.int32)
    e2g = _c(e2g, np.int32)
    rank_off = _c(rank_off, np.int32)
    A_all = _c(A_all, np.uint16)
    Bt_all = _c(Bt_all, np.uint16)
    w = _c(np.asarray(w).reshape(-1), np.float32)
    if w.shape[0] != idx.size:
        raise ValueError("gate weights must hold one value per (token, slot) pair")
    return idx, e2g, rank_off, w, A_all, Bt_all


def combine_fwd(topk_idx, e2g, rank_off, h, w, A_all, Bt_all, s, z_in=None, sel=None):
    """z_out[t] = z_in[t] + sum_j w[t,j] s B_g (A_g h_{t*k+j}): token rows
    [T, d_out] float64 (or [len(sel), d_out], row i holding token sel[i])."""
    lib = _load()
    idx, e2g, rank_off, w, A_all, Bt_all = _combine_args(topk_idx, e2g, rank_off, w, A_all, Bt_all)
    T, k = idx.shape
    G = rank_off.shape[0] - 1
    h = _c(h, np.uint16)
    d_in, d_out = A_all.shape[1], Bt_all.shape[1]
    sel_a = _c(sel, np.int32)
    z = np.empty((T if sel_a is None else sel_a.shape[0], d_out))
    st = lib.oracle_combine_fwd(T, k, e2g.shape[0], G, _p(idx), _p(e2g), _p(rank_off), d_in, d_out, _p(h), _p(w),
                                _p(A_all), _p(Bt_all), float(s), _p(_c(z_in, np.uint16)), _p(z), _p(sel_a),
                                0 if sel_a is None else sel_a.shape[0])
    if st != OR_OK:
        raise OracleError(st, "combine_fwd")
    return z


def combine_bwd_dh(topk_idx, e2g, rank_off, dz, h, w, A_all, Bt_all, s, dh_in=None, sel=None):
    """(dh [T*k, d_in], dw [T*k]) in float64 for the token-space gradient dz
    [T, d_out]; with ``sel``, row i holds pair sel[i]."""
    lib = _load()
    idx, e2g, rank_off, w, A_all, Bt_all = _combine_args(topk_idx, e2g, rank_off, w, A_all, Bt_all)
    T, k = idx.shape
    G = rank_off.shape[0] - 1
    dz = _c(dz, np.uint16)
    h = _c(h, np.uint16)
    d_in, d_out = A_all.shape[1], Bt_all.shape[1]
    sel_a = _c(sel, np.int32)
    n = T * k if sel_a is None else sel_a.shape[0]
    dh = np.empty((n, d_in))
    dw = np.empty(n)
    st = lib.oracle_combine_bwd_dh(T, k, e2g.shape[0], G, _p(idx), _p(e2g), _p(rank_off), d_in, d_out, _p(dz),
                                   _p(h), _p(w), _p(A_all), _p(Bt_all), float(s), _p(_c(dh_in, np.uint16)), _p(dh),
                                   _p(dw), _p(sel_a), 0 if sel_a is None else sel_a.shape[0])
    if st != OR_OK:
        raise OracleError(st, "combine_bwd_dh")
    return dh, dw


def combine_bwd_w(topk_idx, e2g, rank_off, h, dz, w, A_all, Bt_all, s, sel=None):
    """(dA [sum r_g, d_in], dBt [sum r_g, d_out]) in float64 for the combine;
    with ``sel``, row i holds rank row sel[i]."""
    lib = _load()
    idx, e2g, rank_off, w, A_all, Bt_all = _combine_args(topk_idx, e2g, rank_off, w, A_all, Bt_all)
    T, k = idx.shape
    G = rank_off.shape[0] - 1
    h = _c(h, np.uint16)
    dz = _c(dz, np.uint16)
    d_in, d_out = A_all.shape[1], Bt_all.shape[1]
    n_rank = int(rank_off[-1])
    sel_a = _c(sel, np.int32)
    n = n_rank if sel_a is None else sel_a.shape[0]
    dA = np.empty((n, d_in))
    dBt = np.empty((n, d_out))
    st = lib.oracle_combine_bwd_w(T, k, e2g.shape[0], G, _p(idx), _p(e2g), _p(rank_off), d_in, d_out, _p(h),
                                  _p(dz), _p(w), _p(A_all), _p(Bt_all), float(s), _p(dA), _p(dBt), _p(sel_a),
                                  0 if sel_a is None else sel_a.shape[0])
    if st != OR_OK:
        raise OracleError(st, "combine_bwd_w")
    return dA, dBt


# ------------------------------------------------------------------ budget
def expertwise_budget(ranks_per_expert, d_in: int, d_out: int) -> int:
    """B = sum_e (d_in + d_out) r_e  (Sec. 3.1.1)."""
    return int(sum((d_in + d_out) * int(r) for r in ranks_per_expert))


def group_budget(rank_off, d_in: int, d_out: int) -> int:
    """sum_g (d_in + d_out) r_g with r_g = rank_off[g+1] - rank_off[g]  (Sec. 3.3)."""
    ro = np.asarray(rank_off, dtype=np.int64)
    return int(((d_in + d_out) * np.diff(ro)).sum())


def uniform_rank(budget: int, E: int, d_in: int, d_out: int) -> float:
    """r_e = B / (E (d_in + d_out))  (Sec. 3.1.1)."""
    return budget / (E * (d_in + d_out))


def model_adapter_params(layers: int, E: int, r: int, d: int, f: int) -> int:
    """Trainable LoRA parameters of a backbone: gate, up (d->f) and down (f->d)
    of every routed expert in every MoE layer, rank r each."""
    return layers * E * 3 * r * (d + f)
