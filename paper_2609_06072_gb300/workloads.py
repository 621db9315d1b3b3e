"""Seeded synthetic MoE-layer inputs for the grouped-adapter hot path.

This module only draws random inputs; it holds none of the method's
arithmetic (no adapter products, no routing permutation, no gradients), so
both the CUDA path and the CPU oracle can consume exactly the same bytes.

Shapes follow the paper's backbones (Tab. "model_configs": OLMoE-1B-7B
d=2048/ff=1024/E=64/top-8, Qwen1.5-MoE d=2048/ff=1408/E=60/top-4, the
Moonlight-style DeepSeek layer d=2048/ff=1408/E=64/top-6, Kimi-Linear
d=2304/ff=1024/E=256/top-8) plus a Mixtral-shaped layer and a tiny
oracle-scale layer.  The "paperlike" grouping mimics the group statistics
of the Louvain-resolution study (one large group of 43 experts, mid-size
groups and unmerged singletons per 64 experts), at the paper's OLMoE rank
r = 2, so r_g runs from 2 to 86.  Nothing here comes from
any dataset; routing is synthetic:

* router logits l_{t,e} = log w_e + Gumbel(0,1) (tiny layer: l ~ N(0,1)),
  the top-k experts by logit (ties toward the lower expert id), slot j in
  descending-logit order, gate weights = softmax over the k selected logits;
* expert load weights w: uniform, Zipf(alpha) over a seeded permutation of
  the experts, or Dirichlet(alpha * 1_E).

Tensors: activations X, h and upstream gradients dY ~ N(0,1); A_g ~
U(-1/sqrt(d_in), +1/sqrt(d_in)); B_g ~ N(0, 0.02^2) (stored transposed as
Bt_g = B_g^T, rank-major like A_g).  Every bf16 tensor is drawn in float32
and rounded to bf16 (round-to-nearest-even); it is returned as its raw
uint16 bit pattern.  Each array has its own child seed, so any subset can be
drawn without drawing the rest.

Pair p = t*k + j indexes the routed (token, slot) pairs; per-pair tensors
(h, dY) are in pair order.
"""
from __future__ import annotations

import dataclasses
import zlib
from typing import Dict, List, Optional

import numpy as np

__all__ = ["LayerConfig", "CONFIGS", "get_config", "Layer", "f32_to_bf16_bits", "bf16_bits_to_f32"]


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """float32 -> bf16 bit pattern, round-to-nearest-even (inputs are finite)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


@dataclasses.dataclass(frozen=True)
class LayerConfig:
    name: str
    T: int          # tokens
    d: int          # hidden size (gate/up d_in, down d_out)
    f: int          # expert intermediate size (gate/up d_out, down d_in)
    E: int          # routed experts
    k: int          # top-k
    r: int          # expert-wise LoRA rank
    routing: str    # "normal" | "uniform" | "zipf" | "dirichlet"
    alpha: float    # Zipf exponent or Dirichlet concentration
    groups: str     # "contiguous4" | "pairs" | "uneven16" | "all8" | "identity" | "halves"
    s: float = 2.0  # LoRA scale

    @property
    def R(self) -> int:
        return self.T * self.k


CONFIGS: Dict[str, LayerConfig] = {
    # tiny oracle-scale layer: 2 groups of 4 experts (0-3, 4-7), r=4 -> r_g=16
    "tiny": LayerConfig("tiny", 256, 256, 128, 8, 2, 4, "normal", 0.0, "halves"),
    # OLMoE-shaped: T=4x2048, Zipf(1.0), 16 groups of 4 contiguous ids, r=8 -> 32
    "olmoe": LayerConfig("olmoe", 8192, 2048, 1024, 64, 8, 8, "zipf", 1.0, "contiguous4"),
    # Qwen1.5-MoE-shaped: uniform routing, 15 groups of 4, r=16 -> 64
    "qwen": LayerConfig("qwen", 16384, 2048, 1408, 60, 4, 16, "uniform", 0.0, "contiguous4"),
    # Mixtral-shaped: Dirichlet(2) load, 2 groups of 4, r=8 -> 32
    "mixtral": LayerConfig("mixtral", 16384, 4096, 14336, 8, 2, 8, "dirichlet", 2.0, "contiguous4"),
    # DeepSeek/Moonlight-shaped grouping sweep, Zipf(1.2), expert-wise r=8
    "deepseek_g32": LayerConfig("deepseek_g32", 16384, 2048, 1408, 64, 6, 8, "zipf", 1.2, "pairs"),
    "deepseek_g16": LayerConfig("deepseek_g16", 16384, 2048, 1408, 64, 6, 8, "zipf", 1.2, "uneven16"),
    "deepseek_g8": LayerConfig("deepseek_g8", 16384, 2048, 1408, 64, 6, 8, "zipf", 1.2, "all8"),
    # paper-like uneven groups at r = 2: OLMoE-shaped, and a Kimi-Linear-shaped layer (many small segments)
    "olmoe_uneven": LayerConfig("olmoe_uneven", 8192, 2048, 1024, 64, 8, 2, "zipf", 1.0, "paperlike"),
    "kimi": LayerConfig("kimi", 8192, 2304, 1024, 256, 8, 2, "zipf", 1.0, "paperlike"),
}


def get_config(name: str, **overrides) -> LayerConfig:
    """A named config, optionally with fields replaced (e.g. T for a sample)."""
    base = CONFIGS[name]
    return dataclasses.replace(base, **overrides) if overrides else base


# admissible size mixes (a, b, c) of groups of sizes 2, 4, 8 with 16 groups
# covering 64 experts, the all-4 mix excluded
_UNEVEN16_MIXES = [(2, 13, 1), (4, 10, 2), (6, 7, 3), (8, 4, 4), (10, 1, 5)]
# group sizes per block of 64 experts for the "paperlike" grouping
_PAPERLIKE64 = [43, 9, 5, 3, 1, 1, 1, 1]


class Layer:
    """Lazily drawn, seeded inputs of one MoE layer.

    ``expertwise=True`` gives the matched-budget expert-wise layout of the
    same layer: identity expert->group map, rank r per expert.
    """

    def __init__(self, cfg: LayerConfig, seed: int = 0, expertwise: bool = False):
        self.cfg = cfg
        self.seed = int(seed)
        self.expertwise = bool(expertwise)
        self._cache: Dict[str, np.ndarray] = {}

    # -- seeding ---------------------------------------------------------
    def _rng(self, name: str) -> np.random.Generator:
        key = zlib.crc32(f"{self.cfg.name}/{name}".encode())
        return np.random.Generator(np.random.PCG64(np.random.SeedSequence([self.seed, key])))

    def _get(self, name, fn):
        if name not in self._cache:
            self._cache[name] = fn()
        return self._cache[name]

    # -- grouping (an input of the hot path) -----------------------------
    def group_sizes_and_map(self):
        c = self.cfg
        if self.expertwise or c.groups == "identity":
            return np.arange(c.E, dtype=np.int32), np.ones(c.E, dtype=np.int64)
        if c.groups == "halves":
            sizes = [c.E // 2, c.E - c.E // 2]
            e2g = np.repeat(np.arange(2), sizes).astype(np.int32)
            return e2g, np.array(sizes, dtype=np.int64)
        if c.groups == "contiguous4":
            assert c.E % 4 == 0
            return (np.arange(c.E) // 4).astype(np.int32), np.full(c.E // 4, 4, dtype=np.int64)
        if c.groups == "pairs":
            return (np.arange(c.E) // 2).astype(np.int32), np.full(c.E // 2, 2, dtype=np.int64)
        if c.groups == "all8":
            return (np.arange(c.E) // 8).astype(np.int32), np.full(c.E // 8, 8, dtype=np.int64)
        if c.groups in ("uneven16", "paperlike"):
            rng = self._rng("groups")
            if c.groups == "uneven16":
                a, b, cc = _UNEVEN16_MIXES[int(rng.integers(len(_UNEVEN16_MIXES)))]
                sizes = np.array([2] * a + [4] * b + [8] * cc, dtype=np.int64)
            else:
                assert c.E % 64 == 0
                sizes = np.array(_PAPERLIKE64 * (c.E // 64), dtype=np.int64)
            rng.shuffle(sizes)
            perm = rng.permutation(c.E)
            e2g = np.empty(c.E, dtype=np.int32)
            start = 0
            for g, sz in enumerate(sizes):
                e2g[perm[start:start + sz]] = g
                start += sz
            return e2g, sizes
        raise ValueError(c.groups)

    @property
    def e2g(self) -> np.ndarray:
        return self._get("e2g", lambda: self.group_sizes_and_map()[0])

    @property
    def G(self) -> int:
        return int(self.e2g.max()) + 1

    @property
    def rank_off(self) -> np.ndarray:
        """rank_off[g] = sum_{g' < g} r * |G_g'|  (r_g = r |G_g|, Sec. 3.3)."""
        def mk():
            sizes = np.bincount(self.e2g, minlength=self.G).astype(np.int64)
            return np.concatenate([[0], np.cumsum(sizes * self.cfg.r)]).astype(np.int32)
        return self._get("rank_off", mk)

    # -- routing ---------------------------------------------------------
    def load_weights(self) -> Optional[np.ndarray]:
        c = self.cfg
        rng = self._rng("load")
        if c.routing == "uniform":
            return np.full(c.E, 1.0 / c.E)
        if c.routing == "zipf":
            perm = rng.permutation(c.E)
            w = np.empty(c.E)
            w[perm] = (np.arange(1, c.E + 1, dtype=np.float64)) ** (-c.alpha)
            return w / w.sum()
        if c.routing == "dirichlet":
            return rng.dirichlet(np.full(c.E, c.alpha))
        if c.routing == "normal":
            return None
        raise ValueError(c.routing)

    def _routing(self):
        c = self.cfg
        rng = self._rng("routing")
        w = self.load_weights()
        out_idx = np.empty((c.T, c.k), dtype=np.int32)
        out_w = np.empty((c.T, c.k), dtype=np.float32)
        chunk = 4096
        for t0 in range(0, c.T, chunk):
            t1 = min(c.T, t0 + chunk)
            if w is None:
                logits = rng.standard_normal((t1 - t0, c.E))
            else:
                logits = np.log(w)[None, :] + rng.gumbel(size=(t1 - t0, c.E))
            order = np.argsort(-logits, axis=1, kind="stable")[:, : c.k]
            sel = np.take_along_axis(logits, order, axis=1)
            z = np.exp(sel - sel[:, :1])
            out_idx[t0:t1] = order
            out_w[t0:t1] = (z / z.sum(axis=1, keepdims=True)).astype(np.float32)
        return out_idx, out_w

    @property
    def topk_idx(self) -> np.ndarray:
        return self._get("topk_idx", lambda: self._routing()[0])

    @property
    def topk_w(self) -> np.ndarray:
        return self._get("topk_w", lambda: self._routing()[1])

    # -- dense tensors (bf16 bit patterns) --------------------------------
    def _normal_bf16(self, name, shape, std=1.0):
        def mk():
            rng = self._rng(name)
            x = rng.standard_normal(shape, dtype=np.float32)
            if std != 1.0:
                x *= np.float32(std)
            return f32_to_bf16_bits(x)
        return self._get(name, mk)

    def _uniform_bf16(self, name, shape, bound):
        def mk():
            rng = self._rng(name)
            x = rng.uniform(-bound, bound, size=shape).astype(np.float32)
            return f32_to_bf16_bits(x)
        return self._get(name, mk)

    def dims(self, proj: str):
        """(d_in, d_out) of a projection."""
        c = self.cfg
        return (c.d, c.f) if proj in ("gate", "up") else (c.f, c.d)

    def X(self) -> np.ndarray:
        """Token activations entering gate/up, [T, d]."""
        return self._normal_bf16("X", (self.cfg.T, self.cfg.d))

    def h(self) -> np.ndarray:
        """Expert-specific down-projection input per pair, [T*k, f]."""
        return self._normal_bf16("h", (self.cfg.R, self.cfg.f))

    def A(self, proj: str) -> np.ndarray:
        d_in, _ = self.dims(proj)
        tag = "ew" if self.expertwise else "grp"
        return self._uniform_bf16(f"A_{proj}_{tag}", (int(self.rank_off[-1]), d_in), 1.0 / np.sqrt(d_in))

    def Bt(self, proj: str) -> np.ndarray:
        _, d_out = self.dims(proj)
        tag = "ew" if self.expertwise else "grp"
        return self._normal_bf16(f"Bt_{proj}_{tag}", (int(self.rank_off[-1]), d_out), 0.02)

    def dY(self, proj: str) -> np.ndarray:
        """Upstream gradient of the projection output per pair, [T*k, d_out]."""
        _, d_out = self.dims(proj)
        return self._normal_bf16(f"dY_{proj}", (self.cfg.R, d_out))

    def Y_base(self, proj: str) -> np.ndarray:
        """Base-path projection output per pair (nonzero Y_in), [T*k, d_out]."""
        _, d_out = self.dims(proj)
        return self._normal_bf16(f"Ybase_{proj}", (self.cfg.R, d_out))

    def dX_base(self) -> np.ndarray:
        return self._normal_bf16("dXbase", (self.cfg.T, self.cfg.d))

    def dh_base(self) -> np.ndarray:
        return self._normal_bf16("dhbase", (self.cfg.R, self.cfg.f))

    def W_base(self, proj: str) -> np.ndarray:
        """Frozen base expert weights: gate / up [E, f, d], down [E, d, f],
        N(0, 1/fan_in) in bf16."""
        c = self.cfg
        d_in, d_out = self.dims(proj)
        return self._normal_bf16(f"Wbase_{proj}", (c.E, d_out, d_in), 1.0 / np.sqrt(d_in))

    def dZ(self) -> np.ndarray:
        """Upstream gradient of the gate-weighted combined down output, [T, d]."""
        return self._normal_bf16("dZ", (self.cfg.T, self.cfg.d))

    def Z_base(self) -> np.ndarray:
        """Base-path combined output (nonzero z_in), [T, d]."""
        return self._normal_bf16("Zbase", (self.cfg.T, self.cfg.d))

    # -- descriptors -----------------------------------------------------
    def describe(self) -> Dict[str, float]:
        """Realised routing statistics (workload descriptors only)."""
        c = self.cfg
        idx = self.topk_idx
        load = np.bincount(idx.ravel(), minlength=c.E).astype(np.float64)
        p = load / max(1.0, load.sum())
        ent = float(-(p[p > 0] * np.log(p[p > 0])).sum())
        return {"R": c.R, "max_load": float(load.max()), "min_load": float(load.min()),
                "load_entropy": ent, "load_entropy_max": float(np.log(c.E))}

def all_config_names() -> List[str]:
    return list(CONFIGS)
