"""GPU parity of the gate-weighted combine of down (forward and backward,
both split-K modes) against the oracle's combine functions, with the
intermediate H per row and token-major combined H, nonzero base outputs,
the expert-wise configuration and run-to-run determinism."""
import numpy as np
import pytest

import oracle
from paper_2609_06072_gb300 import workloads as W
from ace_testlib import check_close, dev_bf16, host_f64
from test_gpu_fwd import compare_perm, make_plan, run_perm

pytestmark = pytest.mark.gpu


def _combine_case(L, deterministic, with_base=False):
    import torch
    c = L.cfg
    idx, e2g, ro = L.topk_idx, L.e2g, L.rank_off
    plan = make_plan(L, deterministic=deterministic)
    perm, P = run_perm(L, plan)
    O = oracle.permute(idx, e2g, L.G)
    compare_perm(P, O)
    rp = O["row_pair"]
    hin = dev_bf16(L.h()[rp])
    w = torch.from_numpy(np.ascontiguousarray(L.topk_w, dtype=np.float32)).cuda()
    A, Bt = dev_bf16(L.A("down")), dev_bf16(L.Bt("down"))
    zb = L.Z_base() if with_base else np.zeros((c.T, c.d), np.uint16)
    Z = dev_bf16(zb)
    H = torch.full((c.R, plan.rank_max), float("nan"), device="cuda")
    Hx = torch.full((c.T, plan.rank_cols), float("nan"), dtype=torch.bfloat16, device="cuda")
    plan.fwd_combine(perm, hin, w, A, Bt, c.s, Z, H, Hx)
    assert plan.get_error(perm) == 0
    ref_z = oracle.combine_fwd(idx, e2g, ro, L.h(), L.topk_w, L.A("down"), L.Bt("down"), c.s,
                               z_in=zb if with_base else None)
    check_close(host_f64(Z), ref_z, "z")
    _, ref_H = oracle.fwd(idx, e2g, ro, L.h(), L.A("down"), L.Bt("down"), c.s, x_per_pair=True, want_h=True)
    got_H = np.empty_like(ref_H)
    got_H[rp] = host_f64(H)
    check_close(got_H, ref_H, "H")
    # the combined H, from the oracle's H: s sum_j p_j H_p in the group's columns
    ref_Hx = np.zeros((c.T, plan.rank_cols))
    gp = e2g[idx.ravel()]
    for p in range(c.R):
        g = gp[p]
        ref_Hx[p // c.k, ro[g]:ro[g + 1]] += c.s * float(L.topk_w.ravel()[p]) * ref_H[p, : ro[g + 1] - ro[g]]
    check_close(host_f64(Hx), ref_Hx, "Hx")

    _, _, bws = plan.alloc_workspaces(c.T)
    dZ = dev_bf16(L.dZ())
    dhb = L.dh_base() if with_base else np.zeros((c.R, c.f), np.uint16)
    dh = dev_bf16(dhb[rp])
    dw = torch.full((c.T, c.k), float("nan"), device="cuda")
    dA = torch.full((plan.n_rank, c.f), float("nan"), device="cuda")
    dBt = torch.full((plan.n_rank, c.d), float("nan"), device="cuda")
    plan.bwd_combine(perm, dZ, hin, w, H, Hx, A, Bt, c.s, dh, dw, dA, dBt, bws)
    assert plan.get_error(perm) == 0
    ref_dh, ref_dw = oracle.combine_bwd_dh(idx, e2g, ro, L.dZ(), L.h(), L.topk_w, L.A("down"), L.Bt("down"), c.s,
                                           dh_in=dhb if with_base else None)
    got_dh = np.empty((c.R, c.f))
    got_dh[rp] = host_f64(dh)
    check_close(got_dh, ref_dh, "dh")
    check_close(host_f64(dw).ravel(), ref_dw, "dp")
    rdA, rdBt = oracle.combine_bwd_w(idx, e2g, ro, L.h(), L.dZ(), L.topk_w, L.A("down"), L.Bt("down"), c.s)
    check_close(host_f64(dA), rdA, "dA_down")
    check_close(host_f64(dBt), rdBt, "dBt_down")
    return {"z": host_f64(Z), "dh": got_dh, "dp": host_f64(dw), "dA": host_f64(dA), "dBt": host_f64(dBt)}


CASES = [("tiny", 0, {}), ("tiny", 1, {"T": 300}), ("tiny", 2, {"T": 1}), ("olmoe", 0, {"T": 1024}),
         # 960 stacked ranks: B^T dz per unique pair by the gathering H kernel
         ("qwen", 0, {"T": 1024}),
         # r_g = 12: rank offsets that are not multiples of 8
         ("tiny", 4, {"r": 3}),
         # paper-like uneven groups (r_g up to 86, 128-wide rank tiles) and E = 256
         ("olmoe_uneven", 0, {"T": 512}), ("kimi", 0, {"T": 256})]


@pytest.mark.parametrize("det", [True, False])
@pytest.mark.parametrize("name,seed,over", CASES)
def test_combine_parity(name, seed, over, det):
    _combine_case(W.Layer(W.get_config(name, **over), seed=seed), det)


def test_combine_nonzero_base_and_expertwise():
    _combine_case(W.Layer(W.get_config("tiny"), seed=6), True, with_base=True)
    _combine_case(W.Layer(W.get_config("olmoe", T=512), seed=0, expertwise=True), False)


def test_combine_deterministic_mode_is_bitwise_reproducible():
    L = W.Layer(W.get_config("olmoe", T=1024), seed=1)
    a = _combine_case(L, True)
    b = _combine_case(L, True)
    for key in a:
        assert np.array_equal(a[key], b[key]), key


def test_combine_flags_non_finite_gate_weights():
    """A non-finite gate weight is reported through the device flag (read and
    cleared by ace_get_error) instead of passing silently."""
    import torch
    from paper_2609_06072_gb300 import ace
    L = W.Layer(W.get_config("tiny"), seed=0)
    c = L.cfg
    plan = make_plan(L)
    perm, P = run_perm(L, plan)
    rp = P["row_pair"]
    hin = dev_bf16(L.h()[rp])
    A, Bt = dev_bf16(L.A("down")), dev_bf16(L.Bt("down"))
    w = torch.from_numpy(np.ascontiguousarray(L.topk_w, dtype=np.float32)).cuda()
    w[3, 1] = float("inf")
    Z = torch.zeros(c.T, c.d, dtype=torch.bfloat16, device="cuda")
    H = torch.empty(c.R, plan.rank_max, device="cuda")
    Hx = torch.empty(c.T, plan.rank_cols, dtype=torch.bfloat16, device="cuda")
    plan.fwd_combine(perm, hin, w, A, Bt, c.s, Z, H, Hx)
    assert plan.get_error(perm) == ace.ACE_ERR_ARG
    assert plan.get_error(perm) == ace.ACE_OK
