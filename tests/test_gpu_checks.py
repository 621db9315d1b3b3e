"""The range-checked debug build (libace_checks.so: the same sources compiled
with ACE_CHECKS).

* Same results: one deterministic-mode step (permute, both forwards, both
  backwards, and the gate-weighted combine's forward and backward) through a
  plan of the checked library gives bit-identical outputs to the same step
  through libace.so and reports no violation, on a layout with the dense
  token-major H, one with the gathering H kernel and one at rank_pad 128.
* A violation is reported instead of faulting: after the permutation, one
  entry of an index array is overwritten with a value outside its range that
  still addresses allocated memory (the tensors that entry indexes have room
  for it, so even a read that the checks missed would stay in bounds); the
  next call through the checked library then returns ACE_ERR_CHECK from
  ace_get_error, and the context stays usable."""
import numpy as np
import pytest

import oracle
from paper_2609_06072_gb300 import workloads as W
from ace_testlib import dev_bf16
from test_gpu_fwd import compare_perm

pytestmark = pytest.mark.gpu


def _plan(L, checks, det=True):
    from paper_2609_06072_gb300 import ace
    c = L.cfg
    return ace.Plan(c.T, c.k, c.E, L.G, L.e2g, L.rank_off, c.d, c.f, deterministic=det, checks=checks)


def _step(L, plan):
    """Every call of one layer step plus the combine; returns the outputs."""
    import torch
    c = L.cfg
    pws, _, bws = plan.alloc_workspaces(c.T)
    perm = plan.permute(torch.from_numpy(L.topk_idx).cuda(), pws)
    s = c.s
    rp = oracle.permute(L.topk_idx, L.e2g, L.G)["row_pair"]
    X = dev_bf16(L.X())
    A = {p: dev_bf16(L.A(p)) for p in ("gate", "up", "down")}
    Bt = {p: dev_bf16(L.Bt(p)) for p in ("gate", "up", "down")}
    out = {}
    Y = [dev_bf16(L.Y_base(p)[rp]) for p in ("gate", "up")]
    H = [torch.zeros(c.R, plan.rank_max, device="cuda") for _ in range(3)]
    plan.fwd_shared(perm, X, [A["gate"], A["up"]], [Bt["gate"], Bt["up"]], s, Y, H[:2])
    hin = dev_bf16(L.h()[rp])
    Yd = dev_bf16(L.Y_base("down")[rp])
    plan.fwd_row(perm, hin, A["down"], Bt["down"], s, Yd, H[2])
    out.update(Y_gate=Y[0], Y_up=Y[1], Y_down=Yd, H_gate=H[0], H_up=H[1], H_down=H[2])
    n_rank = plan.n_rank
    dh = torch.zeros(c.R, c.f, dtype=torch.bfloat16, device="cuda")
    dA = [torch.zeros(n_rank, c.d, device="cuda"), torch.zeros(n_rank, c.d, device="cuda"),
          torch.zeros(n_rank, c.f, device="cuda")]
    dBt = [torch.zeros(n_rank, c.f, device="cuda"), torch.zeros(n_rank, c.f, device="cuda"),
           torch.zeros(n_rank, c.d, device="cuda")]
    plan.bwd_row(perm, dev_bf16(L.dY("down")[rp]), hin, H[2], A["down"], Bt["down"], s, dh, dA[2], dBt[2], bws)
    dX = torch.zeros(c.T, c.d, dtype=torch.bfloat16, device="cuda")
    plan.bwd_shared(perm, [dev_bf16(L.dY(p)[rp]) for p in ("gate", "up")], X, H[:2], [A["gate"], A["up"]],
                    [Bt["gate"], Bt["up"]], s, dX, dA[:2], dBt[:2], bws)
    out.update(dh=dh, dX=dX, dA_gate=dA[0], dA_up=dA[1], dA_down=dA[2], dBt_gate=dBt[0], dBt_up=dBt[1],
               dBt_down=dBt[2])
    # the gate-weighted combine of down, forward and backward
    w = torch.from_numpy(np.ascontiguousarray(L.topk_w, dtype=np.float32)).cuda()
    Z = torch.zeros(c.T, c.d, dtype=torch.bfloat16, device="cuda")
    Hc = torch.zeros(c.R, plan.rank_max, device="cuda")
    Hx = torch.zeros(c.T, plan.rank_cols, dtype=torch.bfloat16, device="cuda")
    plan.fwd_combine(perm, hin, w, A["down"], Bt["down"], s, Z, Hc, Hx)
    dhc = torch.zeros(c.R, c.f, dtype=torch.bfloat16, device="cuda")
    dw = torch.zeros(c.T * c.k, device="cuda")
    dAc = torch.zeros(n_rank, c.f, device="cuda")
    dBc = torch.zeros(n_rank, c.d, device="cuda")
    plan.bwd_combine(perm, dev_bf16(L.dZ()), hin, w, Hc, Hx, A["down"], Bt["down"], s, dhc, dw, dAc, dBc, bws)
    out.update(Z=Z, dh_comb=dhc, dw=dw, dA_comb=dAc, dBt_comb=dBc)
    return perm, out


@pytest.mark.parametrize("name,over", [("olmoe", {"T": 1024}),  # dense token-major H
                                       ("qwen", {"T": 512}),  # gathering H kernel (960 stacked ranks)
                                       ("olmoe_uneven", {"T": 512})])  # rank_pad 128
def test_checked_build_gives_identical_results(name, over):
    import torch
    from paper_2609_06072_gb300 import ace
    L = W.Layer(W.get_config(name, **over), seed=5)
    pc = _plan(L, checks=True)
    assert pc.lib.ace_build_checks() == 1
    pn = _plan(L, checks=False)
    assert pn.lib.ace_build_checks() == 0
    perm_c, got = _step(L, pc)
    assert pc.get_error(perm_c) == ace.ACE_OK
    compare_perm(ace.perm_arrays(pc, perm_c), oracle.permute(L.topk_idx, L.e2g, L.G))
    perm_n, ref = _step(L, pn)
    assert pn.get_error(perm_n) == ace.ACE_OK
    for k in ref:
        assert got[k].dtype == ref[k].dtype and got[k].shape == ref[k].shape, k
        bits = torch.int16 if ref[k].dtype == torch.bfloat16 else torch.int32
        a, b = got[k].contiguous().view(bits), ref[k].contiguous().view(bits)
        assert torch.equal(a, b), f"{name}: {k} differs between the checked and the normal build"


def _poke(perm, field, index, value):
    """Overwrite entry `index` of the int32 permutation view `field`."""
    import torch
    base = perm.ws.data_ptr()
    off = getattr(perm.c, field) - base
    assert off >= 0 and off % 4 == 0
    perm.ws.view(torch.int32)[off // 4 + index] = int(value)


def _counts(perm):
    import torch
    off = (perm.c.counts - perm.ws.data_ptr()) // 4
    return perm.ws.view(torch.int32)[off:off + 8].cpu().numpy()


@pytest.mark.parametrize("name,field,what", [
    ("olmoe", "tok_uniq", "unique pair of a token past U (dense H GEMM)"),
    ("qwen", "uniq_tok", "token of a unique pair past T (gathering H kernel)"),
    ("olmoe", "row_uniq", "unique pair of a row past U (row kernel's H staging)"),
])
def test_checked_build_reports_an_out_of_range_index(name, field, what):
    import torch
    from paper_2609_06072_gb300 import ace
    L = W.Layer(W.get_config(name, T=512), seed=6)
    c = L.cfg
    plan = _plan(L, checks=True, det=False)
    pws, _, _ = plan.alloc_workspaces(c.T)
    perm = plan.permute(torch.from_numpy(L.topk_idx).cuda(), pws)
    assert plan.get_error(perm) == ace.ACE_OK
    U = int(_counts(perm)[0])
    assert U + 8 <= c.R  # the bad values below still index allocated rows
    if field == "uniq_tok":
        _poke(perm, "uniq_tok", 0, c.T + 5)
    else:
        _poke(perm, field, 3, U + 5)
    # X has T + 8 rows and H has R rows, so every entry set above still addresses allocated memory
    X = torch.zeros(c.T + 8, c.d, dtype=torch.bfloat16, device="cuda")
    X.copy_(torch.cat([dev_bf16(L.X()), torch.zeros(8, c.d, dtype=torch.bfloat16, device="cuda")]))
    A = [dev_bf16(L.A(p)) for p in ("gate", "up")]
    Bt = [dev_bf16(L.Bt(p)) for p in ("gate", "up")]
    Y = [torch.zeros(c.R, c.f, dtype=torch.bfloat16, device="cuda") for _ in range(2)]
    H = [torch.zeros(c.R, plan.rank_max, device="cuda") for _ in range(2)]
    plan.fwd_shared(perm, X[:c.T], A, Bt, c.s, Y, H)
    st = plan.get_error(perm)
    assert st == ace.ACE_ERR_CHECK, (what, ace.STATUS_NAMES.get(st, st))
    assert plan.get_error(perm) == ace.ACE_OK  # the read cleared the flag
    # the context stays usable: a fresh permutation and forward run clean
    perm2 = plan.permute(torch.from_numpy(L.topk_idx).cuda(), pws)
    plan.fwd_shared(perm2, X[:c.T], A, Bt, c.s, Y, H)
    assert plan.get_error(perm2) == ace.ACE_OK

