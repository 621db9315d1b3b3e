"""Benchmark of the grouped adapter execution hot path (one MoE layer).

One step = route-permute + fused gate/up forward (shared input, dedup) +
down forward (per row) + down backward + gate/up backward (incl. dX), i.e. the
forward and backward passes of the group-shared LoRA deltas on all three
expert projections of one layer.  Metric: routed rows (T*k) per second.

Default workload: the OLMoE-shaped layer (T=8192, d=2048, ff=1024, E=64,
top-8, Zipf(1.0) routing, 16 groups of 4, rank 8 -> 32, s=2), synthetic
seeded inputs.  Inputs are resident in HBM for ``value``; ``e2e`` also moves
the step's inputs from pinned host memory and reads the weight gradients back.

    python bench.py [--gpus N --steps K --warmup W] [--impl reference]
                    [--config olmoe] [--expertwise] [--det] [--no-cpu]
Multi-GPU (torchrun, one rank per GPU): independent replicas, weak scaling.
"""
from __future__ import annotations

import argparse
import hashlib
import glob
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "grouped-LoRA fwd+bwd routed rows/s per MoE layer"
UNIT = "rows/s"


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def reduce_max(x, device):
    """Max of x over the ranks of the default process group (x itself when
    there is none): timed regions are reported as the slowest rank's."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(x)
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"hbm_gbs": float(d["hbm_gbs"]), "bf16_tflops": float(d["bf16_tflops"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}


def csrc_sha():
    """Hash of the kernel sources with comments and blank space taken out, so
    that a comment edit does not orphan counters taken from the same code."""
    import re
    h = hashlib.sha256()
    for p in sorted(glob.glob(os.path.join(ROOT, "paper_2609_06072_gb300", "csrc", "*"))):
        src = open(p, encoding="utf-8").read()
        src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
        src = re.sub(r"//[^\n]*", " ", src)
        h.update(" ".join(src.split()).encode())
    return h.hexdigest()[:16]


# ------------------------------------------------------------------ byte model
def model(T, k, d, f, rank_off, U_g, R_g, nproj_shared=2):
    """Algorithmic bytes / flops per call (each distinct tensor counted once)."""
    r_g = np.diff(np.asarray(rank_off, np.int64))
    Pw = int(r_g.sum()) * (d + f)
    R = T * k
    U = int(np.sum(U_g))
    sUr = int(np.sum(np.asarray(U_g) * r_g))
    sRr = int(np.sum(np.asarray(R_g) * r_g))
    npj = nproj_shared
    b = {
        "permute": 4 * R + 16 * R + 4 * U,
        "fwd_shared": 2 * T * d + npj * 4 * R * f + npj * 4 * sUr + npj * 2 * Pw,
        "fwd_row": 2 * R * f + 4 * R * d + 4 * sRr + 2 * Pw,
        "bwd_row": 2 * R * d + 2 * R * f + 4 * sRr + 4 * R * f + 6 * Pw,
        "bwd_shared": npj * 2 * R * f + 2 * T * d + npj * 4 * sUr + 4 * T * d + npj * 6 * Pw,
    }
    fl = {
        "permute": 0,
        "fwd_shared": npj * 2 * sUr * (d + f),
        "fwd_row": 2 * sRr * (d + f),
        "bwd_row": 4 * sRr * (d + f),
        "bwd_shared": npj * 4 * sUr * (d + f),
    }
    return b, fl


# ------------------------------------------------------------------ clocks
class ClockSampler:
    """nvidia-smi clock samples during the timed region, into `path` (a temp
    file unless --clocks-csv names one; {rank} in it becomes the rank)."""

    def __init__(self, index: int, path: str = ""):
        self.index = index
        self.proc = None
        import tempfile
        self.path = (path.format(rank=index) if path else
                     os.path.join(tempfile.gettempdir(), f"ace_clocks_{os.getpid()}_{index}.csv"))

    def start(self):
        q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.index), f"--query-gpu={q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"], stdout=self.fh,
                                         stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.fh.close()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ------------------------------------------------------------------ GPU arm
class Layer:
    """Device-resident tensors of one layer plus the plan and workspaces."""

    def __init__(self, cfg_name, seed, expertwise, det, T=None, combine=False):
        import torch
        from paper_2609_06072_gb300 import ace, workloads as W
        over = {"T": T} if T else {}
        self.L = W.Layer(W.get_config(cfg_name, **over), seed=seed, expertwise=expertwise)
        c = self.L.cfg
        self.c = c
        self.plan = ace.Plan(c.T, c.k, c.E, self.L.G, self.L.e2g, self.L.rank_off, c.d, c.f, deterministic=det)
        self.det = det
        dev = "cuda"
        self.pws, _, self.bws = self.plan.alloc_workspaces(c.T)
        gen = torch.Generator().manual_seed(1000 + seed)

        def randn(*shape, std=1.0):
            return (torch.randn(*shape, generator=gen) * std).to(torch.bfloat16)

        def unif(*shape, bound):
            return ((torch.rand(*shape, generator=gen) * 2 - 1) * bound).to(torch.bfloat16)

        R, d, f, nr = c.R, c.d, c.f, self.plan.n_rank
        # host (pinned) inputs of a step: routing, activations, upstream gradients
        self.h_topk = torch.from_numpy(self.L.topk_idx).pin_memory()
        self.h_X = randn(c.T, d).pin_memory()
        self.h_hin = randn(R, f).pin_memory()
        self.h_dY = [randn(R, f).pin_memory(), randn(R, f).pin_memory(), randn(R, d).pin_memory()]
        self.topk = self.h_topk.to(dev)
        self.X = self.h_X.to(dev)
        self.hin = self.h_hin.to(dev)
        self.dY = [t.to(dev) for t in self.h_dY]
        # adapters (rank-major A_g, B_g^T), three projections
        self.A = [unif(nr, d, bound=d ** -0.5).to(dev), unif(nr, d, bound=d ** -0.5).to(dev),
                  unif(nr, f, bound=f ** -0.5).to(dev)]
        self.Bt = [randn(nr, f, std=0.02).to(dev), randn(nr, f, std=0.02).to(dev), randn(nr, d, std=0.02).to(dev)]
        # base-path outputs / input gradients that the deltas accumulate onto
        self.Y = [randn(R, f).to(dev), randn(R, f).to(dev), randn(R, d).to(dev)]
        self.dX = randn(c.T, d).to(dev)
        self.dh = randn(R, f).to(dev)
        self.H = [torch.empty(R, self.plan.rank_max, device=dev) for _ in range(3)]
        self.dA = [torch.empty(nr, d, device=dev), torch.empty(nr, d, device=dev), torch.empty(nr, f, device=dev)]
        self.dBt = [torch.empty(nr, f, device=dev), torch.empty(nr, f, device=dev), torch.empty(nr, d, device=dev)]
        self.h_grads = [torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in self.dA + self.dBt]
        self.perm = None
        self._randn = randn
        # down through the gate-weighted combine: token-space output and gradient
        self.combine = combine
        if combine:
            self.w = torch.from_numpy(np.ascontiguousarray(self.L.topk_w, dtype=np.float32)).to(dev)
            self.Z = randn(c.T, d).to(dev)
            self.dZ = randn(c.T, d).to(dev)
            self.Hx = torch.empty(c.T, self.plan.rank_cols, dtype=torch.bfloat16, device=dev)
            self.dw = torch.empty(c.T, c.k, device=dev)

    def kernels_per_step(self):
        # permute 3, fwd_shared 2 (H per unique pair, row stream), fwd_row 1,
        # bwd_row 2 (zeroing, row stream), bwd_shared 4 (zeroing, row stream, dX, dA);
        # deterministic mode: bwd_row has nothing to zero and adds a dB^T and a dA reduce,
        # bwd_shared adds the fixed-order dH_u sum and one dB^T reduce per projection.
        # With the combine, down is fwd_combine 3 (H per row, combined H, output GEMM)
        # and bwd_combine 4 (B^T dz per unique pair, zeroing, row stream, dB^T GEMM),
        # plus a dA reduce in deterministic mode
        return (16 if self.combine else 12) + (4 if self.det else 0)

    def step(self, ev=None, only=None):
        """One pass of the hot path.  ev: 6 CUDA events or None at the call
        boundaries (before permute, ..., after bwd_shared); None entries are
        not recorded.  only: a set of call names to run (the permutation
        always runs), or None for all."""
        c, p = self.c, self.plan
        ev = ev or [None] * 6
        run = lambda n: only is None or n in only

        def mark(j):
            if ev[j] is not None:
                ev[j].record()
        mark(0)
        self.perm = p.permute(self.topk, self.pws)
        mark(1)
        if run("fwd_shared"):
            p.fwd_shared(self.perm, self.X, self.A[:2], self.Bt[:2], c.s, self.Y[:2], self.H[:2])
        mark(2)
        if self.combine:
            if run("fwd_row"):
                p.fwd_combine(self.perm, self.hin, self.w, self.A[2], self.Bt[2], c.s, self.Z, self.H[2], self.Hx)
            mark(3)
            if run("bwd_row"):
                p.bwd_combine(self.perm, self.dZ, self.hin, self.w, self.H[2], self.Hx, self.A[2], self.Bt[2], c.s,
                              self.dh, self.dw, self.dA[2], self.dBt[2], self.bws)
        else:
            if run("fwd_row"):
                p.fwd_row(self.perm, self.hin, self.A[2], self.Bt[2], c.s, self.Y[2], self.H[2])
            mark(3)
            if run("bwd_row"):
                p.bwd_row(self.perm, self.dY[2], self.hin, self.H[2], self.A[2], self.Bt[2], c.s, self.dh,
                          self.dA[2], self.dBt[2], self.bws)
        mark(4)
        if run("bwd_shared"):
            p.bwd_shared(self.perm, self.dY[:2], self.X, self.H[:2], self.A[:2], self.Bt[:2], c.s, self.dX,
                         self.dA[:2], self.dBt[:2], self.bws)
        mark(5)

    # ---- end to end: every input of a step comes from pinned host memory and
    # every result goes back, through two device sets so that one step's
    # copies overlap the other's compute
    _IN = ("topk", "X", "hin", "dY", "Y", "dX", "dh")   # routing, activations, upstream gradients, base outputs
    _OUT = ("Y", "dX", "dh", "dA", "dBt")               # outputs with the deltas added, input and weight gradients

    def e2e_setup(self):
        import torch
        dev = "cuda"
        # host copies of the base outputs / input gradients the deltas accumulate onto, and of every result
        self.h_Y = [self._randn(*t.shape).pin_memory() for t in self.Y]
        self.h_dX = self._randn(*self.dX.shape).pin_memory()
        self.h_dh = self._randn(*self.dh.shape).pin_memory()
        self.h_out = {"Y": [torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in self.Y],
                      "dX": torch.empty(self.dX.shape, dtype=self.dX.dtype).pin_memory(),
                      "dh": torch.empty(self.dh.shape, dtype=self.dh.dtype).pin_memory(),
                      "dA": [torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in self.dA],
                      "dBt": [torch.empty(t.shape, dtype=t.dtype).pin_memory() for t in self.dBt]}
        mk = lambda t: torch.empty(t.shape, dtype=t.dtype, device=dev)
        self.sets = []
        for _ in range(2):
            st = {n: ([mk(x) for x in getattr(self, n)] if isinstance(getattr(self, n), list) else mk(getattr(self, n)))
                  for n in set(self._IN) | set(self._OUT)}
            self.sets.append(st)
        self.h_in = {"topk": self.h_topk, "X": self.h_X, "hin": self.h_hin, "dY": self.h_dY, "Y": self.h_Y,
                     "dX": self.h_dX, "dh": self.h_dh}

    def use_set(self, st):
        for n, v in st.items():
            setattr(self, n, v)

    def e2e_h2d(self, st):
        for n in self._IN:
            d, h = st[n], self.h_in[n]
            for a, b in (zip(d, h) if isinstance(d, list) else [(d, h)]):
                a.copy_(b, non_blocking=True)

    def e2e_d2h(self, st):
        for n in self._OUT:
            d, h = st[n], self.h_out[n]
            for a, b in (zip(h, d) if isinstance(d, list) else [(h, d)]):
                a.copy_(b, non_blocking=True)

    def e2e_bytes(self):
        nb = lambda t: sum(x.numel() * x.element_size() for x in (t if isinstance(t, list) else [t]))
        return sum(nb(self.h_in[n]) for n in self._IN), sum(nb(self.h_out[n]) for n in self._OUT)

    def h2d_inputs(self):
        self.topk.copy_(self.h_topk, non_blocking=True)
        self.X.copy_(self.h_X, non_blocking=True)
        self.hin.copy_(self.h_hin, non_blocking=True)
        for dst, src in zip(self.dY, self.h_dY):
            dst.copy_(src, non_blocking=True)

    def d2h_result(self):
        for dst, src in zip(self.h_grads, self.dA + self.dBt):
            dst.copy_(src, non_blocking=True)

    def h2d_bytes(self):
        return sum(t.numel() * t.element_size() for t in [self.h_topk, self.h_X, self.h_hin] + self.h_dY)

    def d2h_bytes(self):
        return sum(t.numel() * t.element_size() for t in self.h_grads)


class NvmlSampler:
    """Reads the SM clock and the clock-event reasons of one GPU through NVML
    every few milliseconds on a host thread (read-only queries), so that a
    short timed region still gets many samples.  Silently inactive when the
    NVML library or the device cannot be found."""
    # nvmlClocksEventReasons bits (nvml.h)
    BITS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown", 0x40: "hw_thermal_slowdown",
            0x80: "hw_power_brake_slowdown"}

    def __init__(self, props, period_s=0.002):
        import ctypes
        import threading
        self.ct, self.period, self.samples, self.stop_ev = ctypes, period_s, [], threading.Event()
        self.thread, self.lib, self.dev, self.max_mhz = None, None, None, None
        try:
            lib = ctypes.CDLL("libnvidia-ml.so.1")
            if lib.nvmlInit_v2() != 0:
                return
            dev = ctypes.c_void_p()
            bus = f"{props.pci_domain_id:08x}:{props.pci_bus_id:02x}:{props.pci_device_id:02x}.0".encode()
            if lib.nvmlDeviceGetHandleByUUID(("GPU-" + str(props.uuid)).encode(), ctypes.byref(dev)) != 0 and \
                    lib.nvmlDeviceGetHandleByPciBusId_v2(bus, ctypes.byref(dev)) != 0:
                return
            mx = ctypes.c_uint()
            if lib.nvmlDeviceGetMaxClockInfo(dev, 1, ctypes.byref(mx)) == 0:  # 1 = NVML_CLOCK_SM
                self.max_mhz = float(mx.value)
            self.reasons_fn = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                getattr(lib, "nvmlDeviceGetCurrentClocksThrottleReasons")
            self.lib, self.dev = lib, dev
        except (OSError, AttributeError):
            self.lib = None

    def _run(self):
        ct = self.ct
        mhz, mask = ct.c_uint(), ct.c_ulonglong()
        while not self.stop_ev.is_set():
            if self.lib.nvmlDeviceGetClockInfo(self.dev, 1, ct.byref(mhz)) == 0 and \
                    self.reasons_fn(self.dev, ct.byref(mask)) == 0:
                self.samples.append((float(mhz.value), int(mask.value)))
            self.stop_ev.wait(self.period)

    def start(self):
        import threading
        if self.lib is not None:
            self.thread = threading.Thread(target=self._run, daemon=True)
            self.thread.start()

    def stop(self):
        if self.thread is None:
            return None
        self.stop_ev.set()
        self.thread.join()
        if not self.samples:
            return None
        reasons = sorted({n for _, m in self.samples for bit, n in self.BITS.items() if m & bit})
        return {"sm_mhz": statistics.median(v for v, _ in self.samples), "sm_max_mhz": self.max_mhz,
                "reasons": reasons, "samples": len(self.samples), "source": "nvml"}


def merge_clocks(nvml, smi):
    """NVML samples (many) when present, nvidia-smi ones otherwise; reasons of both."""
    if nvml is None and smi is None:
        return None
    out = dict(nvml or smi)
    if nvml and smi:
        out["reasons"] = sorted(set(nvml["reasons"]) | set(smi["reasons"]))
        out["nvidia_smi"] = {k: smi[k] for k in ("sm_mhz", "sm_max_mhz", "samples")}
    out.setdefault("source", "nvidia-smi")
    return out


CALLS = ["permute", "fwd_shared", "fwd_row", "bwd_row", "bwd_shared"]
# the calls whose time is one row kernel of ours: fwd_row launches only
# k_fwd_rows<down>; bwd_row launches k_bwd_rows<down> after one zeroing launch
# of its atomic targets (a few microseconds, inside its event span, so its
# achieved rate is a slight underestimate).  The roofline object reports the
# larger of the two, the dominant kernel of the step.
SINGLE_KERNEL = {"fwd_row": "k_fwd_rows<down>", "bwd_row": "k_bwd_rows<down>"}
SINGLE_KERNEL_NOTE = {"fwd_row": "the call's only launch",
                      "bwd_row": "timed with its call, which also runs one zeroing launch before it"}


class L2Flush:
    """Leaves L2 cold and clean between timed steps: a 256 MB write (evicts
    the step's lines) followed by a 256 MB read (evicts the write's dirty
    lines, so their write-back is not charged to the next timed step).  Both
    run on the stream outside the event pair."""

    def __init__(self):
        import torch
        n = 256 * 1024 * 1024  # each > L2 (~126 MB)
        self.w = torch.empty(n, dtype=torch.uint8, device="cuda")
        self.r = torch.ones(n // 4, dtype=torch.float32, device="cuda")
        self.out = torch.empty((), dtype=torch.float32, device="cuda")

    def __call__(self):
        import torch
        self.w.zero_()
        torch.sum(self.r, dim=0, out=self.out)


def load_stats(expert_cnt, R, U):
    """Realised routing of the step: rows per unique (token, group) pair and
    the expert load spread (max / min rows, entropy of the load in bits and
    its ratio to the uniform log2 E)."""
    cnt = np.asarray(expert_cnt, dtype=np.float64)
    p = cnt / max(1.0, cnt.sum())
    nz = p[p > 0]
    h = float(-(nz * np.log2(nz)).sum())
    return {"R_over_U": R / max(1, U), "expert_rows_max": int(cnt.max()), "expert_rows_min": int(cnt.min()),
            "load_entropy_bits": h, "load_entropy_ratio": float(h / np.log2(len(cnt))) if len(cnt) > 1 else 1.0}


def workload_config(args, L, U, expert_cnt, world, l2):
    """The `config` object of both arms: the workload's shape, grouping and
    realised routing (U and the expert loads), plus how L2 was handled."""
    c = L.cfg
    return {"workload": f"{args.config}-shaped MoE layer"
                        f"{' (expert-wise, matched budget)' if args.expertwise else ' (grouped)'}",
            "T": c.T, "d": c.d, "f": c.f, "E": c.E, "k": c.k, "G": L.G, "r": c.r,
            "rank_g": int(np.max(np.diff(L.rank_off))), "s": c.s, "routing": f"{c.routing}({c.alpha})",
            "rows_per_step": c.R, "U": int(U), **load_stats(expert_cnt, c.R, int(U)),
            "deterministic": bool(args.det), "l2": l2, "parallelism": f"replicas x{world}"}


def time_steps(lay, steps, warmup, flush, bracket=None):
    """Mean step time (ms) of `steps` steps, events at the step boundaries and,
    with bracket = j, around call j as in the main timed region (so a variant
    is timed under the same events as the main line); flush: an L2Flush run
    before each step, or None."""
    import torch
    for _ in range(warmup):
        lay.step()
    torch.cuda.synchronize()
    ev = lambda: torch.cuda.Event(enable_timing=True)
    evs = []
    for _ in range(steps):
        e = [ev(), None, None, None, None, ev()]
        if bracket is not None:
            e[bracket], e[bracket + 1] = ev(), ev()
        evs.append(e)
    for e in evs:
        if flush is not None:
            flush()
        lay.step(e)
    torch.cuda.synchronize()
    assert lay.plan.get_error(lay.perm) == 0
    return float(np.mean([e[0].elapsed_time(e[5]) for e in evs]))


def time_expert_ffn(args, lay, flush):
    """Opt-in (--ffn): the routed expert FFN with frozen base weights and the
    group-shared adapters, forward and backward (ace_ffn_fwd / ace_ffn_bwd), on
    the main layer's routing and adapters, with synthetic base weights."""
    import torch
    c, p = lay.c, lay.plan
    gen = torch.Generator().manual_seed(2000 + args.seed)
    w = lambda *s_, fan: (torch.randn(*s_, generator=gen) / fan ** 0.5).to(torch.bfloat16).cuda()
    Wg, Wu, Wd = w(c.E, c.f, c.d, fan=c.d), w(c.E, c.f, c.d, fan=c.d), w(c.E, c.d, c.f, fan=c.f)
    bf = lambda *s_: torch.empty(*s_, dtype=torch.bfloat16, device="cuda")
    U, V, Hh, Y = bf(c.R, c.f), bf(c.R, c.f), bf(c.R, c.f), bf(c.R, c.d)
    Hgu = [torch.empty(c.R, p.rank_max, device="cuda") for _ in range(2)]
    Hd = torch.empty(c.R, p.rank_max, device="cuda")
    dX = bf(c.T, c.d)
    ws = p.ffn_workspace(c.T)
    A, Bt = lay.A, lay.Bt  # gate, up, down

    def fwd():
        p.ffn_fwd(lay.perm, lay.X, Wg, Wu, Wd, A, Bt, c.s, U, V, Hh, Y, Hgu, Hd, ws)

    def step():
        lay.perm = p.permute(lay.topk, lay.pws)
        fwd()
        p.ffn_bwd(lay.perm, lay.dY[2], lay.X, Wg, Wu, Wd, A, Bt, c.s, U, V, Hh, Hgu, Hd, dX, lay.dA, lay.dBt, ws,
                  lay.bws)

    def timed(fn):
        for _ in range(args.warmup):
            fn()
        torch.cuda.synchronize()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.steps)]
        for e0, e1 in ev:
            flush()
            e0.record()
            fn()
            e1.record()
        torch.cuda.synchronize()
        assert p.get_error(lay.perm) == 0
        return float(np.mean([a.elapsed_time(b) for a, b in ev]))
    ms = timed(step)
    ms_fwd = timed(fwd)
    base_fwd = 2 * c.R * c.d * 2 * c.f + 2 * c.R * c.f * c.d  # u, v and y base GEMMs
    flops = 2 * base_fwd  # forward + the input gradients through the frozen weights
    peaks = load_peaks()
    fwd_tf = base_fwd / (ms_fwd * 1e-3) / 1e12
    return {"ms_per_step": ms, "value": c.R / (ms * 1e-3), "unit": UNIT,
            "base_tflops": flops / (ms * 1e-3) / 1e12,
            "forward": {"ms": ms_fwd, "rows_per_s": c.R / (ms_fwd * 1e-3), "base_tflops": fwd_tf,
                        "peak_tflops": peaks["bf16_tflops_sustained"],
                        "frac_of_sustained_bf16": fwd_tf / peaks["bf16_tflops_sustained"],
                        "kernels": "k_ffn_fused (gate/up: base + adapter + SiLU gating; down: base + adapter), "
                                   "the gate/up H kernel and the down H kernel"},
            "note": "forward fused (base GEMMs with the adapter K steps and the SiLU gating in one kernel per "
                    "projection pair), backward composed"}


def time_cka(args, lay):
    """Opt-in (--cka): rank consolidation of the gate projection -- the CKA
    matrix of the expert-wise adapters (rank r each) on a 10 000-token probe
    (ace_cka), then the grouping on the host (ace_group_experts)."""
    import time as _time
    import torch
    from paper_2609_06072_gb300 import ace
    c = lay.c
    gen = torch.Generator().manual_seed(3000 + args.seed)
    N = 10000
    X = torch.randn(N, c.d, generator=gen).to(torch.bfloat16).cuda()
    A = ((torch.rand(c.E * c.r, c.d, generator=gen) * 2 - 1) / c.d ** 0.5).to(torch.bfloat16).cuda()
    Bt = (torch.randn(c.E * c.r, c.f, generator=gen) * 0.02).to(torch.bfloat16).cuda()
    S = torch.empty(c.E, c.E, device="cuda")
    nb = ace.ctypes.c_size_t()
    ace._check(ace.load().ace_cka_workspace_size(N, c.d, c.f, c.E, c.r, ace.ctypes.byref(nb)), "workspace")
    ws = torch.empty(nb.value, dtype=torch.uint8, device="cuda")
    for _ in range(args.warmup):
        ace.cka(X, A, Bt, c.E, c.r, S=S, ws=ws)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.steps):
        ace.cka(X, A, Bt, c.E, c.r, S=S, ws=ws)
    e1.record()
    torch.cuda.synchronize()
    cka_ms = e0.elapsed_time(e1) / args.steps
    S_host = S.cpu().numpy()
    t0 = _time.perf_counter()
    _, _, G = ace.group_experts(S_host, ace.GROUP_LOUVAIN, 0.8)
    group_ms = (_time.perf_counter() - t0) * 1e3
    return {"cka_ms": cka_ms, "grouping_ms_host": group_ms, "groups": int(G), "probe_tokens": N,
            "experts": c.E, "rank": c.r, "d_in": c.d, "d_out": c.f}


def e2e_pipeline(args, lay, world):
    """End-to-end rows/s through pinned host buffers (see run_gpu): host to
    device copies on one stream, device to host on another (both directions of
    the link at once), compute on the current stream."""
    import torch
    lay.e2e_setup()
    main = torch.cuda.current_stream()
    up, down = torch.cuda.Stream(), torch.cuda.Stream()
    ev = lambda: torch.cuda.Event()
    in_ready, done, freed = [ev(), ev()], [ev(), ev()], [ev(), ev()]
    started = [False, False]

    def run(n):
        for i in range(n + 1):
            if i < n:  # inputs of step i into set i % 2, once that set's previous results are back
                b = i % 2
                with torch.cuda.stream(up):
                    if started[b]:
                        up.wait_event(freed[b])
                    lay.e2e_h2d(lay.sets[b])
                    in_ready[b].record(up)
            if i >= 1:  # compute step i - 1, then read its results back
                b = (i - 1) % 2
                main.wait_event(in_ready[b])
                lay.use_set(lay.sets[b])
                lay.step()
                done[b].record(main)
                with torch.cuda.stream(down):
                    down.wait_event(done[b])
                    lay.e2e_d2h(lay.sets[b])
                    freed[b].record(down)
                started[b] = True
        main.wait_stream(up)
        main.wait_stream(down)

    run(2)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(main)
    run(args.steps)
    e1.record(main)
    torch.cuda.synchronize()
    assert lay.plan.get_error(lay.perm) == 0
    ms = e0.elapsed_time(e1)
    if world > 1:
        ms = reduce_max(ms, "cuda")
    h2d, d2h = lay.e2e_bytes()
    return world * lay.c.R * args.steps / (ms * 1e-3), h2d, d2h


def run_variants(args, flush, main_layer, bracket=None):
    """The other timings of the same workload: the expert-wise layout at the
    matched adapter budget, the deterministic split-K mode, and no L2 flush,
    each timed under the main timed region's events (bracket: the index of
    the call it brackets)."""
    out = {}
    c_rows = main_layer.c.R
    for name, ew, det in (("expertwise_matched_budget", not args.expertwise, args.det),
                          ("deterministic" if not args.det else "fast_atomics", args.expertwise, not args.det)):
        lay = Layer(args.config, args.seed, ew, det)
        ms = time_steps(lay, args.steps, args.warmup, flush, bracket)
        out[name] = {"value": c_rows / (ms * 1e-3), "ms_per_step": ms, "expertwise": ew, "deterministic": det}
        del lay
    ms = time_steps(main_layer, args.steps, args.warmup, None, bracket)
    out["unflushed"] = {"value": c_rows / (ms * 1e-3), "ms_per_step": ms}
    if args.combine:
        # down through the gate-weighted combine (token-space output) in place
        # of the per-row down forward and backward
        lay = Layer(args.config, args.seed, args.expertwise, args.det, combine=True)
        ms = time_steps(lay, args.steps, args.warmup, flush, bracket)
        out["down_via_gate_weighted_combine"] = {"value": c_rows / (ms * 1e-3), "ms_per_step": ms,
                                                 "kernels_per_step": lay.kernels_per_step()}
        del lay
        if not args.no_cpu:
            # the oracle of the same step on a bounded sample, beside it
            os.environ.setdefault("OMP_NUM_THREADS", str(cpu_cores()))
            f1, f2 = 1.0 / 1024, 1.0 / 256
            t1, _ = combine_oracle_sample(args.config, args.seed, f1)
            t2, _ = combine_oracle_sample(args.config, args.seed, f2)
            slope = max((t2 - t1) / (f2 - f1), 1e-6)
            frac = float(min(1.0, max(f1, (min(args.cpu_seconds, 10.0) - max(t1 - slope * f1, 0.0)) / slope)))
            dt, rows = combine_oracle_sample(args.config, args.seed, frac)
            out["down_via_gate_weighted_combine"]["cpu_baseline"] = {
                "value": rows / dt, "unit": UNIT, "cores": int(os.environ["OMP_NUM_THREADS"]), "kind": "oracle",
                "sample": f"permutation plus {frac:.4f} of the pairs, tokens and rank rows; {dt:.1f} s"}
    return out


def run_gpu(args, rank, world, local):
    import torch
    torch.cuda.set_device(local)
    from paper_2609_06072_gb300 import ace
    ace.load()
    lay = Layer(args.config, args.seed, args.expertwise, args.det)
    c = lay.c
    flush = L2Flush()
    # warm-up steps (untimed); they carry events at every call boundary, which
    # pick the dominant row kernel whose call the timed region brackets
    warm_evs = []
    for _ in range(max(args.warmup, 1)):
        e = [torch.cuda.Event(enable_timing=True) for _ in range(6)]
        flush()
        lay.step(e)
        warm_evs.append(e)
    torch.cuda.synchronize()
    assert lay.plan.get_error(lay.perm) == 0
    P = ace.perm_arrays(lay.plan, lay.perm)
    U_g = np.diff(P["uniq_off"])
    R_g = np.diff(P["group_off"])
    bytes_, flops = model(c.T, c.k, c.d, c.f, lay.L.rank_off, U_g, R_g)

    # ---- device-resident timed region: events at the step boundaries and
    # around the dominant row kernel's call only (an event between two calls
    # ends the early launch of the next one, a few microseconds each), so the
    # other calls' kernels follow one another as they do without a profiler
    def new_ev():
        return torch.cuda.Event(enable_timing=True)
    jw = {n: CALLS.index(n) for n in SINGLE_KERNEL}
    warm_ms = {n: float(np.mean([e[j].elapsed_time(e[j + 1]) for e in warm_evs[1:] or warm_evs]))
               for n, j in jw.items()}
    dom = max(warm_ms, key=warm_ms.get)
    evs = []
    for _ in range(args.steps):
        e = [new_ev(), None, None, None, None, new_ev()]
        e[jw[dom]], e[jw[dom] + 1] = new_ev(), new_ev()
        evs.append(e)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    clk = ClockSampler(local, args.clocks_csv)
    nv = NvmlSampler(torch.cuda.get_device_properties(local))
    clk.start()
    nv.start()
    t_wall0 = time.perf_counter()
    for i in range(args.steps):
        flush()  # L2 flush between timed steps (outside the event pair)
        lay.step(evs[i])
    torch.cuda.synchronize()
    t_wall = time.perf_counter() - t_wall0
    clocks = merge_clocks(nv.stop(), clk.stop())
    step_ms = [e[0].elapsed_time(e[5]) for e in evs]
    kern_ms = float(np.mean([e[jw[dom]].elapsed_time(e[jw[dom] + 1]) for e in evs]))
    ms = float(np.sum(step_ms))
    step_stats = {"median_ms": float(np.median(step_ms)), "mean_ms": float(np.mean(step_ms)),
                  "std_ms": float(np.std(step_ms)), "min_ms": float(np.min(step_ms))}
    # per-call breakdown (diagnostic, not part of `value`): a second pass with
    # events at every call boundary
    evs_b = [[new_ev() for _ in range(6)] for _ in range(args.steps)]
    for i in range(args.steps):
        flush()
        lay.step(evs_b[i])
    torch.cuda.synchronize()
    per_call = {n: [e[j].elapsed_time(e[j + 1]) for e in evs_b] for j, n in enumerate(CALLS)}
    if world > 1:
        ms = reduce_max(ms, "cuda")
        torch.distributed.barrier()
    ms_per_step = ms / args.steps
    value = world * c.R / (ms_per_step * 1e-3)

    # ---- end to end through host buffers: every step copies all of its inputs
    # in from pinned host memory (routing, X, h, the three dY, the three base
    # outputs and the base dX / dh that the deltas accumulate onto) and reads all
    # of its results back (the three outputs, dX, dh, the six weight
    # gradients); two device sets, the copies on a second stream, so step i's
    # copies overlap step i - 1's compute
    e2e_value, e2e_h2d, e2e_d2h = e2e_pipeline(args, lay, world)

    peaks = load_peaks()
    call_ms = {n: float(np.mean(v)) for n, v in per_call.items()}
    # dominant kernel: the longer of the two row kernels in the warm-up steps,
    # timed in the timed region (the launch list under profiles/ gives the
    # shares)
    achieved = bytes_[dom] / (kern_ms * 1e-3) / 1e9
    traffic = None
    traffic_sha = None  # kernel sources the stored counters were taken from
    sources_sha = csrc_sha()
    tf = os.path.join(ROOT, "profiles", "traffic.json")
    if os.path.exists(tf):
        tj = json.load(open(tf))
        traffic_sha = tj.get("csrc_sha")
        ent = tj.get(f"{args.config}{'_ew' if args.expertwise else ''}{'_det' if args.det else ''}", {}).get(dom)
        if ent and traffic_sha == sources_sha:
            traffic = ent
    total_bytes = sum(bytes_.values())
    total_flops = sum(flops.values())
    out = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": workload_config(args, lay.L, P["U"], P["expert_cnt"], world,
                                  "flushed between timed steps (256 MB write, then 256 MB read so no dirty line "
                                  "is left; outside the event pair)"),
        "roofline": {"bound": "hbm", "kernel": SINGLE_KERNEL[dom], "call": dom, "achieved": achieved,
                     "launch_ms": kern_ms, "timing": SINGLE_KERNEL_NOTE[dom], "peak": peaks["hbm_gbs"],
                     "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"], "traffic": traffic,
                     "traffic_counters_csrc_sha": traffic_sha, "csrc_sha": sources_sha,
                     "algorithmic_bytes": bytes_[dom], "peak_source": peaks["source"]},
        "step_roofline": {"algorithmic_bytes": total_bytes, "algorithmic_flops": total_flops,
                          "achieved_GBps": total_bytes / (ms_per_step * 1e-3) / 1e9,
                          "frac_hbm": total_bytes / (ms_per_step * 1e-3) / 1e9 / peaks["hbm_gbs"],
                          "tensor_TFLOPs": total_flops / (ms_per_step * 1e-3) / 1e12},
        "step_ms_stats": step_stats,
        "per_call_ms": call_ms,
        "per_call_frac_hbm": {n: bytes_[n] / (call_ms[n] * 1e-3) / 1e9 / peaks["hbm_gbs"] for n in CALLS},
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": e2e_h2d, "d2h_bytes_per_step": e2e_d2h,
                "overlap": "two device sets; H2D on one stream, D2H on another, beside the compute of the "
                           "neighbouring steps"},
        "gpu_launches": lay.kernels_per_step() * args.steps,
        "clocks": clocks,
        "wall_s_timed": t_wall,
    }
    if not args.no_variants:
        out["variants"] = run_variants(args, flush, lay, jw[dom])
    if args.ffn:
        ffn = time_expert_ffn(args, lay, flush)
        if not args.no_cpu:
            dt, rows = ffn_oracle_sample(args.config, args.seed, 4)
            ffn["cpu_baseline"] = {"value": rows / dt, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
                                   "sample": f"4 tokens ({int(rows)} rows), forward and backward; {dt:.1f} s"}
        out.setdefault("variants", {})["expert_ffn"] = ffn
    if args.cka:
        cons = time_cka(args, lay)
        if not args.no_cpu:
            n = 4
            dt, _ = cka_oracle_sample(args.config, args.seed, n)
            cons["cpu_baseline"] = {"value": dt / n * lay.c.E ** 2 * 1e3, "unit": "ms per CKA matrix (estimated)",
                                    "cores": cpu_cores(), "kind": "oracle",
                                    "sample": f"{n} expert pairs by the definition on the 10k probe, "
                                              f"scaled to {lay.c.E}^2 pairs; {dt:.1f} s"}
        out["consolidation"] = cons
    return out, lay


# ------------------------------------------------------------------ CPU oracle
def combine_oracle_sample(cfg_name, seed, frac, rng_seed=0):
    """The oracle on a sample of the step with down through the gate-weighted
    combine: gate/up as in oracle_sample, and for down the combined output of
    a fraction of the tokens, dh and the gate-weight gradient of that fraction
    of the pairs and dA / dB^T of that fraction of the rank rows.  Returns
    (seconds, sampled rows)."""
    import oracle
    from paper_2609_06072_gb300 import workloads as W
    L = W.Layer(W.get_config(cfg_name), seed=seed)
    c = L.cfg
    rng = np.random.default_rng(rng_seed)
    n_p = max(1, int(round(frac * c.R)))
    n_t = max(1, int(round(frac * c.T)))
    n_r = max(1, int(round(frac * int(L.rank_off[-1]))))
    sel_p = np.sort(rng.choice(c.R, n_p, replace=False)).astype(np.int32)
    sel_t = np.sort(rng.choice(c.T, n_t, replace=False)).astype(np.int32)
    sel_r = np.sort(rng.choice(int(L.rank_off[-1]), n_r, replace=False)).astype(np.int32)
    X, h, w, dZ = L.X(), L.h(), L.topk_w, L.dZ()
    A = {p: L.A(p) for p in ("gate", "up", "down")}
    Bt = {p: L.Bt(p) for p in ("gate", "up", "down")}
    dY = {p: L.dY(p) for p in ("gate", "up")}
    t0 = time.perf_counter()
    oracle.permute(L.topk_idx, L.e2g, L.G)
    for p in ("gate", "up"):
        oracle.fwd(L.topk_idx, L.e2g, L.rank_off, X, A[p], Bt[p], c.s, sel=sel_p)
        oracle.bwd_dx(L.topk_idx, L.e2g, L.rank_off, dY[p], A[p], Bt[p], c.s, sel=sel_t)
        oracle.bwd_w(L.topk_idx, L.e2g, L.rank_off, X, dY[p], A[p], Bt[p], c.s, sel=sel_r)
    oracle.combine_fwd(L.topk_idx, L.e2g, L.rank_off, h, w, A["down"], Bt["down"], c.s, sel=sel_t)
    oracle.combine_bwd_dh(L.topk_idx, L.e2g, L.rank_off, dZ, h, w, A["down"], Bt["down"], c.s, sel=sel_p)
    oracle.combine_bwd_w(L.topk_idx, L.e2g, L.rank_off, h, dZ, w, A["down"], Bt["down"], c.s, sel=sel_r)
    return time.perf_counter() - t0, frac * c.R


def ffn_oracle_sample(cfg_name, seed, n_tokens, rng_seed=0):
    """The expert-FFN oracle (forward and backward, frozen base weights) on
    n_tokens sampled tokens of the layer (all their pairs).  Returns
    (seconds, sampled rows)."""
    from oracle import ffn as F
    from paper_2609_06072_gb300 import workloads as W
    L = W.Layer(W.get_config(cfg_name), seed=seed)
    c = L.cfg
    rng = np.random.default_rng(rng_seed)
    toks = np.sort(rng.choice(c.T, n_tokens, replace=False))
    dec = lambda b: W.bf16_bits_to_f32(b).astype(np.float64)
    projs = ("gate", "up", "down")
    # only the experts the sampled tokens route to, renumbered compactly, with
    # base weights of the same distribution drawn for them alone (the timing
    # does not depend on their values)
    used, idx = np.unique(L.topk_idx[toks], return_inverse=True)
    idx = idx.reshape(n_tokens, c.k).astype(np.int32)
    maps = {q: (L.e2g[used], L.rank_off) for q in projs}
    shapes = {"gate": (c.f, c.d), "up": (c.f, c.d), "down": (c.d, c.f)}
    Wb = {q: rng.standard_normal((len(used),) + shapes[q]) / np.sqrt(shapes[q][1]) for q in projs}
    A = {q: dec(L.A(q)) for q in projs}
    Bt = {q: dec(L.Bt(q)) for q in projs}
    X = dec(L.X())[toks]
    dy = dec(L.dY("down")).reshape(c.T, c.k, c.d)[toks].reshape(-1, c.d)
    t0 = time.perf_counter()
    F.ffn_fwd(idx, maps, X, Wb, A, Bt, c.s)
    F.ffn_bwd(idx, maps, X, Wb, A, Bt, c.s, dy=dy)
    return time.perf_counter() - t0, n_tokens * c.k


def cka_oracle_sample(cfg_name, seed, n_pairs, rng_seed=0):
    """Linear CKA by its definition (explicit representation matrices on a
    10 000-token probe) for n_pairs sampled expert pairs of the gate
    projection.  Returns (seconds, pairs)."""
    from oracle import consolidation as C
    from paper_2609_06072_gb300 import workloads as W
    L = W.Layer(W.get_config(cfg_name), seed=seed, expertwise=True)
    c = L.cfg
    rng = np.random.default_rng(rng_seed)
    X = W.f32_to_bf16_bits(rng.standard_normal((10000, c.d)).astype(np.float32))
    A, Bt = L.A("gate"), L.Bt("gate")
    pairs = rng.integers(0, c.E, (n_pairs, 2))
    t0 = time.perf_counter()
    for i, j in pairs:
        Zi, Zj = C.adapter_outputs(X, [A[i * c.r:(i + 1) * c.r], A[j * c.r:(j + 1) * c.r]],
                                   [Bt[i * c.r:(i + 1) * c.r], Bt[j * c.r:(j + 1) * c.r]])
        C.cka(Zi, Zj)
    return time.perf_counter() - t0, n_pairs


def oracle_sample(cfg_name, seed, expertwise, frac, rng_seed=0):
    """Time the fp64 oracle on a sample of one step: the full permutation, the
    forward of a fraction `frac` of the pairs, input gradients of the same
    fraction of tokens / pairs and weight gradients of that fraction of the
    rank rows, for all three projections.  Returns (seconds, sampled rows)."""
    import oracle
    from paper_2609_06072_gb300 import workloads as W
    L = W.Layer(W.get_config(cfg_name), seed=seed, expertwise=expertwise)
    c = L.cfg
    rng = np.random.default_rng(rng_seed)
    n_p = max(1, int(round(frac * c.R)))
    n_t = max(1, int(round(frac * c.T)))
    n_r = max(1, int(round(frac * int(L.rank_off[-1]))))
    sel_p = np.sort(rng.choice(c.R, n_p, replace=False)).astype(np.int32)
    sel_t = np.sort(rng.choice(c.T, n_t, replace=False)).astype(np.int32)
    sel_r = np.sort(rng.choice(int(L.rank_off[-1]), n_r, replace=False)).astype(np.int32)
    _ = (L.topk_idx, L.e2g, L.G)
    ins = {"X": L.X(), "h": L.h(), "dY": {p: L.dY(p) for p in ("gate", "up", "down")},
           "A": {p: L.A(p) for p in ("gate", "up", "down")}, "Bt": {p: L.Bt(p) for p in ("gate", "up", "down")}}
    t0 = time.perf_counter()
    oracle.permute(L.topk_idx, L.e2g, L.G)
    for p in ("gate", "up"):
        oracle.fwd(L.topk_idx, L.e2g, L.rank_off, ins["X"], ins["A"][p], ins["Bt"][p], c.s, sel=sel_p)
        oracle.bwd_dx(L.topk_idx, L.e2g, L.rank_off, ins["dY"][p], ins["A"][p], ins["Bt"][p], c.s, sel=sel_t)
        oracle.bwd_w(L.topk_idx, L.e2g, L.rank_off, ins["X"], ins["dY"][p], ins["A"][p], ins["Bt"][p], c.s,
                     sel=sel_r)
    p = "down"
    oracle.fwd(L.topk_idx, L.e2g, L.rank_off, ins["h"], ins["A"][p], ins["Bt"][p], c.s, x_per_pair=True, sel=sel_p)
    oracle.bwd_dx(L.topk_idx, L.e2g, L.rank_off, ins["dY"][p], ins["A"][p], ins["Bt"][p], c.s, x_per_pair=True,
                  sel=sel_p)
    oracle.bwd_w(L.topk_idx, L.e2g, L.rank_off, ins["h"], ins["dY"][p], ins["A"][p], ins["Bt"][p], c.s,
                 x_per_pair=True, sel=sel_r)
    dt = time.perf_counter() - t0
    return dt, frac * c.R


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def calibrate_fraction(cfg_name, seed, expertwise, target_s):
    """Sample fraction whose oracle time is about target_s: the time of a
    sample is a fixed part (permutations, per-call setup) plus a part linear
    in the fraction, so two short probes fix both."""
    f1, f2 = 1.0 / 1024, 1.0 / 256
    t1, _ = oracle_sample(cfg_name, seed, expertwise, f1)
    t2, _ = oracle_sample(cfg_name, seed, expertwise, f2)
    slope = max((t2 - t1) / (f2 - f1), 1e-6)
    fixed = max(t1 - slope * f1, 0.0)
    return float(min(1.0, max(f1, (target_s - fixed) / slope)))


def cpu_baseline(cfg_name, seed, expertwise, target_s):
    """Calibrate a sample fraction to ~target_s seconds of oracle work, then time it."""
    os.environ.setdefault("OMP_NUM_THREADS", str(cpu_cores()))
    frac = calibrate_fraction(cfg_name, seed, expertwise, target_s)
    dt, rows = oracle_sample(cfg_name, seed, expertwise, frac)
    reps = 1
    while frac >= 1.0 and dt < 0.75 * target_s and reps < 16:  # whole steps are short: time several
        t, r = oracle_sample(cfg_name, seed, expertwise, frac, rng_seed=reps)
        dt, rows, reps = dt + t, rows + r, reps + 1
    what = (f"{reps} whole step(s) (permutation, forward, dX/dh, dA, dB^T of all 3 projections)" if frac >= 1.0 else
            f"one step's permutation plus {frac:.4f} of its pairs (forward, dX/dh) and of its rank rows "
            f"(dA, dB^T), all 3 projections")
    return {"value": rows / dt, "unit": UNIT, "cores": int(os.environ["OMP_NUM_THREADS"]), "kind": "oracle",
            "sample": f"{what}; {dt:.1f} s", "seconds": dt}


def oracle_single_thread(seed, expertwise):
    """The oracle on one host core (a child process with OMP_NUM_THREADS=1):
    whole steps of the tiny layer, and a ~3 s sample of the OLMoE-shaped one."""
    code = ("import json, sys; sys.path.insert(0, %r); import bench\n"
            "out = {}\n"
            "t = r = 0.0; n = 0\n"
            "while t < 1.0 and n < 100:\n"
            "    dt, dr = bench.oracle_sample('tiny', %d, %r, 1.0, rng_seed=n); t += dt; r += dr; n += 1\n"
            "out['tiny'] = {'value': r / t, 'sample': '%%d whole steps' %% n, 'seconds': t}\n"
            "f = bench.calibrate_fraction('olmoe', %d, %r, 3.0)\n"
            "t, r = bench.oracle_sample('olmoe', %d, %r, f)\n"
            "out['olmoe'] = {'value': r / t, 'sample': 'permutation plus %%.5f of one step' %% f, 'seconds': t}\n"
            "print(json.dumps(out))\n") % (ROOT, seed, expertwise, seed, expertwise, seed, expertwise)
    env = dict(os.environ, OMP_NUM_THREADS="1")
    r = subprocess.run([sys.executable, "-c", code], env=env, capture_output=True, text=True, timeout=300)
    if r.returncode != 0:
        return {"error": r.stderr.strip().splitlines()[-1] if r.stderr.strip() else "failed"}
    res = json.loads(r.stdout.strip().splitlines()[-1])
    return {"cores": 1, "unit": UNIT, **res}


def run_reference(args, rank, world):
    if rank != 0:
        return None
    from paper_2609_06072_gb300 import workloads as W
    os.environ.setdefault("OMP_NUM_THREADS", str(cpu_cores()))
    L = W.Layer(W.get_config(args.config), seed=args.seed, expertwise=args.expertwise)
    c = L.cfg
    # realised routing, for the config object: distinct (token, group) pairs
    U = len(np.unique(np.arange(c.T)[:, None] * L.G + np.asarray(L.e2g)[L.topk_idx]))
    # per step: a bounded sample sized so that warmup + steps end within minutes
    per_step_s = max(2.0, min(20.0, 120.0 / max(1, args.steps + args.warmup)))
    frac = calibrate_fraction(args.config, args.seed, args.expertwise, per_step_s)
    for _ in range(args.warmup):
        oracle_sample(args.config, args.seed, args.expertwise, frac)
    times, rows = [], 0.0
    for i in range(args.steps):
        dt, r = oracle_sample(args.config, args.seed, args.expertwise, frac, rng_seed=i + 1)
        times.append(dt)
        rows += r
    total = float(np.sum(times))
    value = rows / total
    cores = int(os.environ["OMP_NUM_THREADS"])
    return {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": 1e3 * c.R / value, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": workload_config(args, L, U, np.bincount(L.topk_idx.ravel(), minlength=c.E), world,
                                  "not applicable: the fp64 CPU oracle on host cores"),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                         "sample": f"per step: permutation plus {frac:.4f} of the pairs and rank rows of one step"},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }


def run_once(args):
    """--once: the calls of one layer step, each run --repeat times in step
    order with no timing (the launch pattern a profiler captures); with --ffn
    the expert FFN forward (base GEMMs with the adapters fused in) follows."""
    import torch
    from paper_2609_06072_gb300 import ace
    ace.load()
    lay = Layer(args.config, args.seed, args.expertwise, args.det, combine=args.combine)
    only = set(args.only.split(",")) if args.only else None
    for _ in range(args.repeat):
        lay.step(only=only)
    if args.ffn:
        import torch as _t
        c, p = lay.c, lay.plan
        gen = _t.Generator().manual_seed(2000 + args.seed)
        w = lambda *s_, fan: (_t.randn(*s_, generator=gen) / fan ** 0.5).to(_t.bfloat16).cuda()
        Wg, Wu, Wd = w(c.E, c.f, c.d, fan=c.d), w(c.E, c.f, c.d, fan=c.d), w(c.E, c.d, c.f, fan=c.f)
        bf = lambda *s_: _t.empty(*s_, dtype=_t.bfloat16, device="cuda")
        U, V, Hh, Y = bf(c.R, c.f), bf(c.R, c.f), bf(c.R, c.f), bf(c.R, c.d)
        Hgu = [_t.empty(c.R, p.rank_max, device="cuda") for _ in range(2)]
        Hd = _t.empty(c.R, p.rank_max, device="cuda")
        ws = p.ffn_workspace(c.T)
        for _ in range(args.repeat):
            p.ffn_fwd(lay.perm, lay.X, Wg, Wu, Wd, lay.A, lay.Bt, c.s, U, V, Hh, Y, Hgu, Hd, ws)
    torch.cuda.synchronize()
    assert lay.plan.get_error(lay.perm) == 0
    print(json.dumps({"mode": "once", "config": args.config, "repeat": args.repeat, "only": args.only,
                      "deterministic": bool(args.det), "combine": bool(args.combine), "ffn": bool(args.ffn)}))


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--clocks-csv", default="",
                    help="keep the nvidia-smi clock samples of the timed region in this file ({rank} = rank)")
    ap.add_argument("--impl", default="ace", choices=["ace", "reference"])
    ap.add_argument("--config", default="olmoe")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--expertwise", action="store_true", help="matched-budget expert-wise layout (G=E, rank r)")
    ap.add_argument("--det", action="store_true", help="deterministic two-stage split-K for dA / dB^T")
    ap.add_argument("--no-cpu", action="store_true", help="skip the CPU-oracle baseline leg")
    ap.add_argument("--combine", action="store_true",
                    help="also time the step with down through the gate-weighted combine (a variant)")
    ap.add_argument("--ffn", action="store_true",
                    help="also time the routed expert FFN with base weights and adapters, forward and backward")
    ap.add_argument("--cka", action="store_true",
                    help="also time rank consolidation: the CKA matrix on a 10k-token probe and the grouping")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--once", action="store_true",
                    help="untimed: run the step's calls --repeat times and exit (for profilers)")
    ap.add_argument("--repeat", type=int, default=1)
    ap.add_argument("--only", default="", help="with --once: comma-separated calls to run after the permutation")
    ap.add_argument("--no-variants", action="store_true",
                    help="skip the expert-wise, deterministic-mode and unflushed timings")
    args = ap.parse_args()
    if args.once:
        run_once(args)
        return
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    rank, world, local = dist_env()
    if args.impl == "reference":
        out = run_reference(args, rank, world)
        if out is not None:
            print(json.dumps(out))
        return
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    out, _ = run_gpu(args, rank, world, local)
    if rank == 0:
        if world == 1 and not args.no_cpu:
            out["cpu_baseline"] = cpu_baseline(args.config, args.seed, args.expertwise, args.cpu_seconds)
            out["cpu_baseline"]["single_thread"] = oracle_single_thread(args.seed, args.expertwise)
        print(json.dumps(out))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
