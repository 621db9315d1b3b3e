"""Thin ctypes binding of the ACE C ABI (include/ace.h).

Argument marshalling only: every step of the hot path runs in the CUDA
kernels of libace.so.  PyTorch supplies device memory and streams.  There is
no fallback: if libace.so is missing or the device is not sm_103, calls raise.

Functions keep the C names (``ace_permute``, ``ace_fwd_shared``, ...); the
``Plan`` class is a convenience holder for one layer description.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import torch

from . import _build

ACE_OK = 0
ACE_ERR_ARG = 1
ACE_ERR_SHAPE = 2
ACE_ERR_WORKSPACE = 3
ACE_ERR_INDEX = 4
ACE_ERR_UNSUPPORTED = 5
ACE_ERR_CUDA = 6
ACE_ERR_DEVICE_TIMEOUT = 7
ACE_ERR_CHECK = 8  # libace_checks.so: an index or a tile outside its range
ACE_FLAG_DETERMINISTIC = 1
ACE_FLAG_TEST_WAIT_EXPIRY = 2  # test only: makes the down forward's bounded flag wait give up

STATUS_NAMES = {0: "ACE_OK", 1: "ACE_ERR_ARG", 2: "ACE_ERR_SHAPE", 3: "ACE_ERR_WORKSPACE", 4: "ACE_ERR_INDEX",
                5: "ACE_ERR_UNSUPPORTED", 6: "ACE_ERR_CUDA", 7: "ACE_ERR_DEVICE_TIMEOUT",
                8: "ACE_ERR_CHECK"}

EXPORTED = ["ace_version", "ace_last_error_message", "ace_plan_create", "ace_plan_destroy", "ace_plan_rank_max",
            "ace_workspace_size", "ace_permute", "ace_fwd_shared", "ace_fwd_shared_noalloc", "ace_fwd_row",
            "ace_bwd_shared", "ace_bwd_row", "ace_plan_rank_cols", "ace_fwd_combine", "ace_bwd_combine",
            "ace_group_experts", "ace_ffn_workspace_size", "ace_ffn_fwd", "ace_ffn_bwd", "ace_cka_workspace_size", "ace_cka", "ace_consolidate_adapters",
            "ace_gather_rows", "ace_scatter_rows", "ace_get_error", "ace_build_checks"]


class AceError(RuntimeError):
    def __init__(self, status: int, what: str, msg: str = ""):
        super().__init__(f"{what}: {STATUS_NAMES.get(status, status)} {msg}".strip())
        self.status = status


class ace_layer_desc(ctypes.Structure):
    _fields_ = [("T_max", ctypes.c_int32), ("k", ctypes.c_int32), ("E", ctypes.c_int32), ("G", ctypes.c_int32),
                ("e2g", ctypes.POINTER(ctypes.c_int32)), ("rank_off", ctypes.POINTER(ctypes.c_int32)),
                ("d", ctypes.c_int32), ("f", ctypes.c_int32), ("flags", ctypes.c_uint32)]


class ace_perm(ctypes.Structure):
    _fields_ = [("T", ctypes.c_int32), ("R", ctypes.c_int32), ("counts", ctypes.c_void_p),
                ("group_off", ctypes.c_void_p), ("expert_off", ctypes.c_void_p), ("expert_cnt", ctypes.c_void_p),
                ("row_pair", ctypes.c_void_p), ("pair_row", ctypes.c_void_p), ("uniq_off", ctypes.c_void_p),
                ("uniq_tok", ctypes.c_void_p), ("tok_uniq", ctypes.c_void_p), ("row_uniq", ctypes.c_void_p),
                ("ws", ctypes.c_void_p)]


_libs = {}


def lib_path(checks: bool = False) -> str:
    return _build.lib_path(checks)


def load(build_if_missing: bool = False, checks: bool = False) -> ctypes.CDLL:
    """Load libace.so (in-tree), or with checks=True its range-checked debug
    build libace_checks.so.  Raises if it has not been built."""
    if checks in _libs:
        return _libs[checks]
    path = _build.lib_path(checks)
    if not os.path.exists(path):
        if build_if_missing:
            _build.build(checks=checks)
        else:
            raise RuntimeError(f"ACE CUDA library not built ({path}); run __graft_entry__.build()")
    lib = ctypes.CDLL(path)
    vp, i32, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    lib.ace_version.restype = i32
    lib.ace_last_error_message.restype = ctypes.c_char_p
    lib.ace_plan_create.restype = i32
    lib.ace_plan_create.argtypes = [ctypes.POINTER(vp), ctypes.POINTER(ace_layer_desc)]
    lib.ace_plan_destroy.restype = None
    lib.ace_plan_destroy.argtypes = [vp]
    lib.ace_plan_rank_max.restype = i32
    lib.ace_plan_rank_max.argtypes = [vp]
    lib.ace_plan_rank_cols.restype = i32
    lib.ace_plan_rank_cols.argtypes = [vp]
    lib.ace_workspace_size.restype = i32
    lib.ace_workspace_size.argtypes = [vp, i32, ctypes.POINTER(sz), ctypes.POINTER(sz), ctypes.POINTER(sz)]
    lib.ace_permute.restype = i32
    lib.ace_permute.argtypes = [vp, vp, i32, vp, sz, ctypes.POINTER(ace_perm), vp]
    lib.ace_fwd_shared.restype = i32
    lib.ace_fwd_shared.argtypes = [vp, ctypes.POINTER(ace_perm), vp, i32, vp, vp, ctypes.c_float, vp, vp, vp, sz, vp]
    lib.ace_fwd_shared_noalloc.restype = i32
    lib.ace_fwd_shared_noalloc.argtypes = [vp, ctypes.POINTER(ace_perm), vp, i32, vp, vp, ctypes.c_float, vp, vp]
    lib.ace_fwd_row.restype = i32
    lib.ace_fwd_row.argtypes = [vp, ctypes.POINTER(ace_perm), vp, vp, vp, ctypes.c_float, vp, vp, vp, sz, vp]
    lib.ace_bwd_shared.restype = i32
    lib.ace_bwd_shared.argtypes = [vp, ctypes.POINTER(ace_perm), i32, vp, vp, vp, vp, vp, ctypes.c_float, vp, vp, vp,
                                   vp, sz, vp]
    lib.ace_bwd_row.restype = i32
    lib.ace_bwd_row.argtypes = [vp, ctypes.POINTER(ace_perm), vp, vp, vp, vp, vp, ctypes.c_float, vp, vp, vp, vp, sz,
                                vp]
    lib.ace_fwd_combine.restype = i32
    lib.ace_fwd_combine.argtypes = [vp, ctypes.POINTER(ace_perm), vp, vp, vp, vp, ctypes.c_float, vp, vp, vp, vp]
    lib.ace_bwd_combine.restype = i32
    lib.ace_bwd_combine.argtypes = [vp, ctypes.POINTER(ace_perm), vp, vp, vp, vp, vp, vp, vp, ctypes.c_float, vp, vp,
                                    vp, vp, vp, sz, vp]
    lib.ace_cka_workspace_size.restype = i32
    lib.ace_cka_workspace_size.argtypes = [i32, i32, i32, i32, i32, ctypes.POINTER(sz)]
    lib.ace_cka.restype = i32
    lib.ace_cka.argtypes = [i32, i32, i32, i32, i32, vp, vp, vp, i32, vp, vp, sz, vp]
    lib.ace_consolidate_adapters.restype = i32
    lib.ace_consolidate_adapters.argtypes = [i32, i32, i32, i32, vp, vp, i32, vp, vp, vp, vp, vp, vp, vp]
    lib.ace_ffn_workspace_size.restype = i32
    lib.ace_ffn_workspace_size.argtypes = [vp, i32, ctypes.POINTER(sz)]
    lib.ace_ffn_fwd.restype = i32
    lib.ace_ffn_fwd.argtypes = [vp, ctypes.POINTER(ace_perm), vp, vp, vp, vp, vp, vp, ctypes.c_float, vp, vp, vp, vp,
                                vp, vp, vp, sz, vp]
    lib.ace_ffn_bwd.restype = i32
    lib.ace_ffn_bwd.argtypes = [vp, ctypes.POINTER(ace_perm), vp, vp, vp, vp, vp, vp, vp, ctypes.c_float, vp, vp, vp,
                                vp, vp, vp, vp, vp, vp, sz, vp, sz, vp]
    lib.ace_group_experts.restype = i32
    lib.ace_group_experts.argtypes = [vp, i32, i32, ctypes.c_double, vp, vp, vp]
    lib.ace_gather_rows.restype = i32
    lib.ace_gather_rows.argtypes = [ctypes.POINTER(ace_perm), vp, vp, i32, vp]
    lib.ace_scatter_rows.restype = i32
    lib.ace_scatter_rows.argtypes = [ctypes.POINTER(ace_perm), vp, vp, i32, vp]
    lib.ace_get_error.restype = i32
    lib.ace_get_error.argtypes = [ctypes.POINTER(ace_perm), vp]
    lib.ace_build_checks.restype = i32
    want = 1 if checks else 0
    if lib.ace_build_checks() != want:
        raise RuntimeError(f"{path} reports ace_build_checks() = {lib.ace_build_checks()}, expected {want}")
    _libs[checks] = lib
    return lib


def _check(st: int, what: str, lib=None):
    if st != ACE_OK:
        msg = (lib or load()).ace_last_error_message()
        raise AceError(st, what, msg.decode() if msg else "")


def _ptr(t: Optional[torch.Tensor], dtype=None, name: str = "tensor") -> Optional[int]:
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    return t.data_ptr()


def _arr(ptrs: Sequence[Optional[int]]):
    return (ctypes.c_void_p * len(ptrs))(*[p or 0 for p in ptrs])


def _stream(stream) -> int:
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


class Perm:
    """Device views filled by ace_permute (the workspace tensor is kept alive)."""

    def __init__(self, c: ace_perm, ws: torch.Tensor):
        self.c = c
        self.ws = ws

    @property
    def T(self):
        return self.c.T

    @property
    def R(self):
        return self.c.R


class Plan:
    """One layer description (ace_plan) on the current CUDA device."""

    def __init__(self, T_max: int, k: int, E: int, G: int, e2g, rank_off, d: int, f: int, deterministic=False,
                 flags=0, checks=False):
        # checks=True: every call of this plan goes to libace_checks.so
        self.lib = load(checks=checks)
        self._e2g = (ctypes.c_int32 * E)(*[int(x) for x in e2g])
        self._ro = (ctypes.c_int32 * (G + 1))(*[int(x) for x in rank_off])
        desc = ace_layer_desc(int(T_max), int(k), int(E), int(G), self._e2g, self._ro, int(d), int(f),
                              (ACE_FLAG_DETERMINISTIC if deterministic else 0) | int(flags))
        h = ctypes.c_void_p()
        self._check(self.lib.ace_plan_create(ctypes.byref(h), ctypes.byref(desc)), "ace_plan_create")
        self.h = h
        self.T_max, self.k, self.E, self.G, self.d, self.f = T_max, k, E, G, d, f
        self.rank_max = self.lib.ace_plan_rank_max(h)
        self.n_rank = int(rank_off[-1])

    def _check(self, st: int, what: str):
        _check(st, what, self.lib)

    def __del__(self):
        h = getattr(self, "h", None)
        if h is not None and h.value:
            self.lib.ace_plan_destroy(h)
            self.h = None

    def workspace_size(self, T: int):
        p, fw, bw = ctypes.c_size_t(), ctypes.c_size_t(), ctypes.c_size_t()
        self._check(self.lib.ace_workspace_size(self.h, int(T), ctypes.byref(p), ctypes.byref(fw), ctypes.byref(bw)),
               "ace_workspace_size")
        return p.value, fw.value, bw.value

    def alloc_workspaces(self, T: int, device="cuda"):
        p, fw, bw = self.workspace_size(T)
        mk = lambda n: torch.empty(max(n, 16), dtype=torch.uint8, device=device)
        return mk(p), mk(fw), mk(bw)

    def permute(self, topk_idx: torch.Tensor, perm_ws: torch.Tensor, stream=None) -> Perm:
        T = int(topk_idx.shape[0]) if topk_idx.numel() else 0
        c = ace_perm()
        self._check(self.lib.ace_permute(self.h, _ptr(topk_idx, torch.int32, "topk_idx"), T, _ptr(perm_ws),
                                    perm_ws.numel(), ctypes.byref(c), _stream(stream)), "ace_permute")
        return Perm(c, perm_ws)

    def fwd_shared(self, perm: Perm, X, A, Bt, s, Y, H=None, ws=None, stream=None):
        n = len(A)
        Hp = _arr([_ptr(h, torch.float32, "H") for h in H]) if H is not None else None
        self._check(self.lib.ace_fwd_shared(self.h, ctypes.byref(perm.c), _ptr(X, torch.bfloat16, "X"), n,
                                       _arr([_ptr(a, torch.bfloat16, "A") for a in A]),
                                       _arr([_ptr(b, torch.bfloat16, "Bt") for b in Bt]), float(s),
                                       _arr([_ptr(y, torch.bfloat16, "Y") for y in Y]), Hp,
                                       _ptr(ws) if ws is not None else None, 0 if ws is None else ws.numel(),
                                       _stream(stream)), "ace_fwd_shared")

    def fwd_shared_noalloc(self, perm: Perm, X, A, Bt, s, Y, stream=None):
        """ace_fwd_shared_noalloc: no H output, scratch inside the library."""
        self._check(self.lib.ace_fwd_shared_noalloc(self.h, ctypes.byref(perm.c), _ptr(X, torch.bfloat16, "X"), len(A),
                                               _arr([_ptr(a, torch.bfloat16, "A") for a in A]),
                                               _arr([_ptr(b, torch.bfloat16, "Bt") for b in Bt]), float(s),
                                               _arr([_ptr(y, torch.bfloat16, "Y") for y in Y]), _stream(stream)),
               "ace_fwd_shared_noalloc")

    def fwd_row(self, perm: Perm, Hin, A, Bt, s, Y, H=None, ws=None, stream=None):
        self._check(self.lib.ace_fwd_row(self.h, ctypes.byref(perm.c), _ptr(Hin, torch.bfloat16, "Hin"),
                                    _ptr(A, torch.bfloat16, "A"), _ptr(Bt, torch.bfloat16, "Bt"), float(s),
                                    _ptr(Y, torch.bfloat16, "Y"), _ptr(H, torch.float32, "H"),
                                    _ptr(ws) if ws is not None else None, 0 if ws is None else ws.numel(),
                                    _stream(stream)), "ace_fwd_row")

    def bwd_shared(self, perm: Perm, dY, X, H, A, Bt, s, dX, dA, dBt, ws, stream=None):
        n = len(dY)
        self._check(self.lib.ace_bwd_shared(self.h, ctypes.byref(perm.c), n,
                                       _arr([_ptr(t, torch.bfloat16, "dY") for t in dY]),
                                       _ptr(X, torch.bfloat16, "X"), _arr([_ptr(t, torch.float32, "H") for t in H]),
                                       _arr([_ptr(t, torch.bfloat16, "A") for t in A]),
                                       _arr([_ptr(t, torch.bfloat16, "Bt") for t in Bt]), float(s),
                                       _ptr(dX, torch.bfloat16, "dX"), _arr([_ptr(t, torch.float32, "dA") for t in dA]),
                                       _arr([_ptr(t, torch.float32, "dBt") for t in dBt]), _ptr(ws), ws.numel(),
                                       _stream(stream)), "ace_bwd_shared")

    def bwd_row(self, perm: Perm, dY, Hin, H, A, Bt, s, dHin, dA, dBt, ws, stream=None):
        self._check(self.lib.ace_bwd_row(self.h, ctypes.byref(perm.c), _ptr(dY, torch.bfloat16, "dY"),
                                    _ptr(Hin, torch.bfloat16, "Hin"), _ptr(H, torch.float32, "H"),
                                    _ptr(A, torch.bfloat16, "A"), _ptr(Bt, torch.bfloat16, "Bt"), float(s),
                                    _ptr(dHin, torch.bfloat16, "dHin"), _ptr(dA, torch.float32, "dA"),
                                    _ptr(dBt, torch.float32, "dBt"), _ptr(ws), ws.numel(), _stream(stream)),
               "ace_bwd_row")

    def ffn_workspace(self, T: int, device="cuda"):
        n = ctypes.c_size_t()
        self._check(self.lib.ace_ffn_workspace_size(self.h, int(T), ctypes.byref(n)), "ace_ffn_workspace_size")
        return torch.empty(max(n.value, 16), dtype=torch.uint8, device=device)

    def ffn_fwd(self, perm: Perm, X, W_gate, W_up, W_down, A, Bt, s, U, V, Hh, Y, Hgu, Hd, ws, stream=None):
        """ace_ffn_fwd: A / Bt are (gate, up, down); Hgu is (gate, up)."""
        self._check(self.lib.ace_ffn_fwd(self.h, ctypes.byref(perm.c), _ptr(X, torch.bfloat16, "X"),
                                    _ptr(W_gate, torch.bfloat16, "W_gate"), _ptr(W_up, torch.bfloat16, "W_up"),
                                    _ptr(W_down, torch.bfloat16, "W_down"),
                                    _arr([_ptr(t, torch.bfloat16, "A") for t in A]),
                                    _arr([_ptr(t, torch.bfloat16, "Bt") for t in Bt]), float(s),
                                    _ptr(U, torch.bfloat16, "U"), _ptr(V, torch.bfloat16, "V"),
                                    _ptr(Hh, torch.bfloat16, "Hh"), _ptr(Y, torch.bfloat16, "Y"),
                                    _arr([_ptr(t, torch.float32, "Hgu") for t in Hgu]), _ptr(Hd, torch.float32, "Hd"),
                                    _ptr(ws), ws.numel(), _stream(stream)), "ace_ffn_fwd")

    def ffn_bwd(self, perm: Perm, dY, X, W_gate, W_up, W_down, A, Bt, s, U, V, Hh, Hgu, Hd, dX, dA, dBt, ws, bws,
                stream=None):
        """ace_ffn_bwd: A / Bt / dA / dBt are (gate, up, down); Hgu is (gate, up)."""
        self._check(self.lib.ace_ffn_bwd(self.h, ctypes.byref(perm.c), _ptr(dY, torch.bfloat16, "dY"),
                                    _ptr(X, torch.bfloat16, "X"), _ptr(W_gate, torch.bfloat16, "W_gate"),
                                    _ptr(W_up, torch.bfloat16, "W_up"), _ptr(W_down, torch.bfloat16, "W_down"),
                                    _arr([_ptr(t, torch.bfloat16, "A") for t in A]),
                                    _arr([_ptr(t, torch.bfloat16, "Bt") for t in Bt]), float(s),
                                    _ptr(U, torch.bfloat16, "U"), _ptr(V, torch.bfloat16, "V"),
                                    _ptr(Hh, torch.bfloat16, "Hh"),
                                    _arr([_ptr(t, torch.float32, "Hgu") for t in Hgu]), _ptr(Hd, torch.float32, "Hd"),
                                    _ptr(dX, torch.bfloat16, "dX"), _arr([_ptr(t, torch.float32, "dA") for t in dA]),
                                    _arr([_ptr(t, torch.float32, "dBt") for t in dBt]), _ptr(ws), ws.numel(),
                                    _ptr(bws), bws.numel(), _stream(stream)), "ace_ffn_bwd")

    @property
    def rank_cols(self) -> int:
        """Row stride of the token-major combined H (stacked ranks rounded up to 64)."""
        return int(self.lib.ace_plan_rank_cols(self.h))

    def fwd_combine(self, perm: Perm, Hin, topk_w, A, Bt, s, Z, H, Hx, stream=None):
        self._check(self.lib.ace_fwd_combine(self.h, ctypes.byref(perm.c), _ptr(Hin, torch.bfloat16, "Hin"),
                                        _ptr(topk_w, torch.float32, "topk_w"), _ptr(A, torch.bfloat16, "A"),
                                        _ptr(Bt, torch.bfloat16, "Bt"), float(s), _ptr(Z, torch.bfloat16, "Z"),
                                        _ptr(H, torch.float32, "H"), _ptr(Hx, torch.bfloat16, "Hx"),
                                        _stream(stream)), "ace_fwd_combine")

    def bwd_combine(self, perm: Perm, dZ, Hin, topk_w, H, Hx, A, Bt, s, dHin, dtopk_w, dA, dBt, ws, stream=None):
        self._check(self.lib.ace_bwd_combine(self.h, ctypes.byref(perm.c), _ptr(dZ, torch.bfloat16, "dZ"),
                                        _ptr(Hin, torch.bfloat16, "Hin"), _ptr(topk_w, torch.float32, "topk_w"),
                                        _ptr(H, torch.float32, "H"), _ptr(Hx, torch.bfloat16, "Hx"),
                                        _ptr(A, torch.bfloat16, "A"), _ptr(Bt, torch.bfloat16, "Bt"), float(s),
                                        _ptr(dHin, torch.bfloat16, "dHin"), _ptr(dtopk_w, torch.float32, "dtopk_w"),
                                        _ptr(dA, torch.float32, "dA"), _ptr(dBt, torch.float32, "dBt"), _ptr(ws),
                                        ws.numel(), _stream(stream)), "ace_bwd_combine")

    def gather_rows(self, perm: Perm, src_pairs, dst_rows, stream=None):
        self._check(self.lib.ace_gather_rows(ctypes.byref(perm.c), _ptr(src_pairs), _ptr(dst_rows),
                                        int(src_pairs.shape[-1]), _stream(stream)), "ace_gather_rows")

    def scatter_rows(self, perm: Perm, src_rows, dst_pairs, stream=None):
        self._check(self.lib.ace_scatter_rows(ctypes.byref(perm.c), _ptr(src_rows), _ptr(dst_pairs),
                                         int(src_rows.shape[-1]), _stream(stream)), "ace_scatter_rows")

    def get_error(self, perm: Perm, stream=None) -> int:
        """Synchronise, read and clear the device flag; returns the status code."""
        return self.lib.ace_get_error(ctypes.byref(perm.c), _stream(stream))


GROUP_LOUVAIN, GROUP_THRESHOLD = 0, 1


def cka(X, A, Bt, E: int, r: int, center: bool = True, S=None, ws=None, stream=None):
    """ace_cka: the E x E linear-CKA matrix of expert adapters (A [E*r, d_in],
    Bt [E*r, d_out], bf16) on the probe inputs X [N, d_in] (bf16), all on the
    GPU.  Returns S (fp32 [E, E], allocated when not given)."""
    lib = load()
    N, d_in = int(X.shape[0]), int(X.shape[1])
    d_out = int(Bt.shape[1])
    if ws is None:
        nb = ctypes.c_size_t()
        _check(lib.ace_cka_workspace_size(N, d_in, d_out, int(E), int(r), ctypes.byref(nb)), "ace_cka_workspace_size")
        ws = torch.empty(max(nb.value, 16), dtype=torch.uint8, device=X.device)
    if S is None:
        S = torch.empty(E, E, dtype=torch.float32, device=X.device)
    _check(lib.ace_cka(N, d_in, d_out, int(E), int(r), _ptr(X, torch.bfloat16, "X"), _ptr(A, torch.bfloat16, "A"),
                       _ptr(Bt, torch.bfloat16, "Bt"), int(bool(center)), _ptr(S, torch.float32, "S"), _ptr(ws),
                       ws.numel(), _stream(stream)), "ace_cka")
    return S


def group_experts(S, method: int = GROUP_LOUVAIN, param: float = 0.8):
    """ace_group_experts on a host [E, E] similarity matrix: returns
    (e2g [E] int32, anchors [G] int32, G).  No GPU work."""
    import numpy as np
    S = np.ascontiguousarray(S, dtype=np.float32)
    if S.ndim != 2 or S.shape[0] != S.shape[1]:
        raise ValueError("S must be a square matrix")
    E = S.shape[0]
    e2g = np.empty(E, np.int32)
    anchors = np.empty(E, np.int32)
    G = ctypes.c_int32()
    _check(load().ace_group_experts(S.ctypes.data, E, int(method), float(param), e2g.ctypes.data,
                                    anchors.ctypes.data, ctypes.byref(G)), "ace_group_experts")
    return e2g, anchors[: G.value].copy(), G.value


def consolidate_adapters(e2g, anchors, A_e, Bt_e, A_init, r: int, stream=None):
    """ace_consolidate_adapters: the groups' shared adapters (bf16, on the
    device of A_e) and the plan's rank offsets (numpy) from expert-wise
    adapters of rank r, a grouping and its anchors."""
    import numpy as np
    e2g = np.ascontiguousarray(e2g, dtype=np.int32)
    anchors = np.ascontiguousarray(anchors, dtype=np.int32)
    E, G = int(e2g.shape[0]), int(anchors.shape[0])
    d_in, d_out = int(A_e.shape[1]), int(Bt_e.shape[1])
    A_g = torch.empty_like(A_e)
    Bt_g = torch.empty_like(Bt_e)
    rank_off = np.empty(G + 1, np.int32)
    _check(load().ace_consolidate_adapters(E, int(r), d_in, d_out, e2g.ctypes.data, anchors.ctypes.data, G,
                                           _ptr(A_e, torch.bfloat16, "A_e"), _ptr(Bt_e, torch.bfloat16, "Bt_e"),
                                           _ptr(A_init, torch.bfloat16, "A_init"), _ptr(A_g), _ptr(Bt_g),
                                           rank_off.ctypes.data, _stream(stream)), "ace_consolidate_adapters")
    return A_g, Bt_g, rank_off


def consolidate(X_probe, A_e, Bt_e, E: int, r: int, A_init, method: int = 0, param: float = 0.8,
                center: bool = True, stream=None):
    """Rank consolidation of one layer and projection (Sec. 3.2): CKA of the
    expert-wise adapters on the probe (GPU), grouping and anchors (host),
    then the shared adapters.  Returns (e2g, rank_off, A_g, Bt_g, S) ready
    for a group plan."""
    S = cka(X_probe, A_e, Bt_e, E, r, center=center, stream=stream)
    S_host = S.cpu().numpy()  # synchronises the stream
    e2g, anchors, _ = group_experts(S_host, method, param)
    A_g, Bt_g, rank_off = consolidate_adapters(e2g, anchors, A_e, Bt_e, A_init, r, stream=stream)
    return e2g, rank_off, A_g, Bt_g, S_host


def perm_arrays(plan: Plan, perm: Perm) -> dict:
    """Copy the permutation views to host numpy arrays (synchronises)."""
    import numpy as np
    T, R, E, G, k = perm.T, perm.R, plan.E, plan.G, plan.k
    ws = perm.ws
    base = ws.data_ptr()

    def view(ptr, n):
        if n == 0:
            return np.zeros(0, np.int32)
        off = ptr - base
        return ws[off: off + 4 * n].view(torch.int32).cpu().numpy().copy()

    c = perm.c
    counts = view(c.counts, 8)
    U = int(counts[0])
    return {"U": U, "rows": int(counts[1]), "group_off": view(c.group_off, G + 1),
            "expert_off": view(c.expert_off, E), "expert_cnt": view(c.expert_cnt, E),
            "row_pair": view(c.row_pair, R), "pair_row": view(c.pair_row, R), "uniq_off": view(c.uniq_off, G + 1),
            "uniq_tok": view(c.uniq_tok, U), "tok_uniq": view(c.tok_uniq, R).reshape(T, k),
            "row_uniq": view(c.row_uniq, R)}
