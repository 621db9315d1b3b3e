"""GPU parity of the fused backward (both split-K modes) against the oracle,
plus determinism, empty groups and the expert-wise configuration."""
import numpy as np
import pytest

import oracle
from paper_2609_06072_gb300 import workloads as W
from ace_testlib import check_close, dev_bf16, host_f64
from test_gpu_fwd import compare_perm, make_plan, run_perm

pytestmark = pytest.mark.gpu


def _shared_case(L, deterministic, with_base=False, nproj=2, topk=None):
    import torch
    c = L.cfg
    idx = L.topk_idx if topk is None else topk
    plan = make_plan(L, deterministic=deterministic)
    pws, _, bws = plan.alloc_workspaces(c.T)
    perm = plan.permute(torch.from_numpy(idx).cuda(), pws)
    O = oracle.permute(idx, L.e2g, L.G)
    from paper_2609_06072_gb300 import ace
    compare_perm(ace.perm_arrays(plan, perm), O)
    rp = O["row_pair"]
    projs = ["gate", "up"][:nproj]
    X = dev_bf16(L.X())
    A = [dev_bf16(L.A(p)) for p in projs]
    Bt = [dev_bf16(L.Bt(p)) for p in projs]
    Y = [torch.zeros(c.R, c.f, dtype=torch.bfloat16, device="cuda") for _ in projs]
    H = [torch.zeros(c.R, plan.rank_max, device="cuda") for _ in projs]
    plan.fwd_shared(perm, X, A, Bt, c.s, Y, H)
    dY = [dev_bf16(L.dY(p)[rp]) for p in projs]
    dXb = L.dX_base() if with_base else np.zeros((c.T, c.d), np.uint16)
    dX = dev_bf16(dXb)
    dA = [torch.full((plan.n_rank, c.d), float("nan"), device="cuda") for _ in projs]
    dBt = [torch.full((plan.n_rank, c.f), float("nan"), device="cuda") for _ in projs]
    plan.bwd_shared(perm, dY, X, H, A, Bt, c.s, dX, dA, dBt, bws)
    assert plan.get_error(perm) == 0
    ref_dx = sum(oracle.bwd_dx(idx, L.e2g, L.rank_off, L.dY(p), L.A(p), L.Bt(p), c.s) for p in projs)
    if with_base:
        ref_dx = ref_dx + W.bf16_bits_to_f32(dXb).astype(np.float64)
    check_close(host_f64(dX), ref_dx, "dX")
    out = {"dX": host_f64(dX)}
    for j, p in enumerate(projs):
        rdA, rdBt = oracle.bwd_w(idx, L.e2g, L.rank_off, L.X(), L.dY(p), L.A(p), L.Bt(p), c.s)
        check_close(host_f64(dA[j]), rdA, f"dA_{p}")
        check_close(host_f64(dBt[j]), rdBt, f"dBt_{p}")
        out[f"dA_{p}"] = host_f64(dA[j])
        out[f"dBt_{p}"] = host_f64(dBt[j])
    return out


def _row_case(L, deterministic, with_base=False):
    import torch
    c = L.cfg
    plan = make_plan(L, deterministic=deterministic)
    perm, P = run_perm(L, plan)
    O = oracle.permute(L.topk_idx, L.e2g, L.G)
    compare_perm(P, O)
    rp = O["row_pair"]
    hin = dev_bf16(L.h()[rp])
    A, Bt = dev_bf16(L.A("down")), dev_bf16(L.Bt("down"))
    Y = torch.zeros(c.R, c.d, dtype=torch.bfloat16, device="cuda")
    H = torch.zeros(c.R, plan.rank_max, device="cuda")
    plan.fwd_row(perm, hin, A, Bt, c.s, Y, H)
    _, _, bws = plan.alloc_workspaces(c.T)
    dY = dev_bf16(L.dY("down")[rp])
    dhb = L.dh_base() if with_base else np.zeros((c.R, c.f), np.uint16)
    dh = dev_bf16(dhb[rp])
    dA = torch.full((plan.n_rank, c.f), float("nan"), device="cuda")
    dBt = torch.full((plan.n_rank, c.d), float("nan"), device="cuda")
    plan.bwd_row(perm, dY, hin, H, A, Bt, c.s, dh, dA, dBt, bws)
    assert plan.get_error(perm) == 0
    ref_dh = oracle.bwd_dx(L.topk_idx, L.e2g, L.rank_off, L.dY("down"), L.A("down"), L.Bt("down"), c.s,
                           x_per_pair=True, dx_in=dhb if with_base else None)
    got = np.empty((c.R, c.f))
    got[rp] = host_f64(dh)
    check_close(got, ref_dh, "dh")
    rdA, rdBt = oracle.bwd_w(L.topk_idx, L.e2g, L.rank_off, L.h(), L.dY("down"), L.A("down"), L.Bt("down"), c.s,
                             x_per_pair=True)
    check_close(host_f64(dA), rdA, "dA_down")
    check_close(host_f64(dBt), rdBt, "dBt_down")
    return {"dh": got, "dA": host_f64(dA), "dBt": host_f64(dBt)}


CASES = [("tiny", 0, {}), ("tiny", 1, {"T": 300}), ("olmoe", 0, {"T": 1024}), ("qwen", 0, {"T": 1024}),
         ("deepseek_g16", 0, {"T": 1024}),
         # r_g = 12: rank offsets that are not multiples of 8 (unaligned dH_u columns)
         ("tiny", 4, {"r": 3}),
         # paper-like uneven groups, r_g from 2 to 86 (128-wide rank tiles), and E = 256
         ("olmoe_uneven", 0, {"T": 512}), ("kimi", 0, {"T": 256}),
         # the grouping sweep's uniform points (r_g = 16 and r_g = 64)
         ("deepseek_g32", 0, {"T": 1024}), ("deepseek_g8", 0, {"T": 1024}),
         # full Mixtral widths (d = 4096, f = 14336) at a reduced token count
         ("mixtral", 0, {"T": 256})]


@pytest.mark.parametrize("det", [True, False])
@pytest.mark.parametrize("name,seed,over", CASES)
def test_bwd_shared_parity(name, seed, over, det):
    _shared_case(W.Layer(W.get_config(name, **over), seed=seed), det)


@pytest.mark.parametrize("det", [True, False])
@pytest.mark.parametrize("name,seed,over", CASES)
def test_bwd_row_parity(name, seed, over, det):
    _row_case(W.Layer(W.get_config(name, **over), seed=seed), det)


def test_bwd_nonzero_base_and_single_projection():
    L = W.Layer(W.get_config("tiny"), seed=6)
    _shared_case(L, True, with_base=True)
    _shared_case(L, False, nproj=1)
    _row_case(L, True, with_base=True)


def test_bwd_expertwise_padded_rank():
    L = W.Layer(W.get_config("olmoe", T=512), seed=0, expertwise=True)
    _shared_case(L, True)
    _row_case(L, False)


def test_bwd_deterministic_mode_is_bitwise_reproducible():
    L = W.Layer(W.get_config("olmoe", T=1024), seed=1)
    a = _shared_case(L, True)
    b = _shared_case(L, True)
    for key in a:
        assert np.array_equal(a[key], b[key]), key
    a = _row_case(L, True)
    b = _row_case(L, True)
    for key in a:
        assert np.array_equal(a[key], b[key]), key


def test_bwd_empty_groups_get_zero_gradients():
    L = W.Layer(W.get_config("tiny"), seed=0)
    rng = np.random.default_rng(0)
    topk = np.stack([rng.permutation(4)[:2] for _ in range(L.cfg.T)]).astype(np.int32)  # only group 0 routed
    for det in (True, False):
        out = _shared_case(L, det, topk=topk)
        r0 = L.rank_off[1]
        assert np.all(out["dA_gate"][r0:] == 0) and np.all(out["dBt_up"][r0:] == 0)
