"""Helpers shared by the GPU parity tests: moving seeded bf16 inputs to the
device, mapping row order <-> pair order with the (verified) permutation, and
the tolerance check for bf16-input / fp32-accumulate outputs."""
import numpy as np

from paper_2609_06072_gb300 import workloads as W

# per-tensor bar for floating-point outputs: max|err| <= 2e-2 * max|ref| and
# relative Frobenius error <= 5e-3
MAX_REL = 2e-2
FRO_REL = 5e-3


def dev_bf16(bits, device="cuda"):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(device)


def host_f64(t):
    import torch
    if t.dtype == torch.bfloat16:
        bits = t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
        return W.bf16_bits_to_f32(bits).astype(np.float64)
    return t.detach().cpu().numpy().astype(np.float64)


def check_close(got, ref, name, max_rel=MAX_REL, fro_rel=FRO_REL):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert got.shape == ref.shape, (name, got.shape, ref.shape)
    assert np.all(np.isfinite(got)), f"{name}: non-finite output"
    if ref.size == 0:
        return 0.0, 0.0
    err = np.abs(got - ref)
    mref = float(np.abs(ref).max())
    fro = float(np.linalg.norm(got - ref) / max(np.linalg.norm(ref), 1e-300))
    if mref == 0.0:
        assert float(err.max()) == 0.0, f"{name}: expected exact zeros, max err {err.max()}"
        return 0.0, 0.0
    me = float(err.max()) / mref
    assert me <= max_rel and fro <= fro_rel, f"{name}: max|err|/max|ref|={me:.3e} (<= {max_rel}), rel_fro={fro:.3e} (<= {fro_rel})"
    return me, fro
