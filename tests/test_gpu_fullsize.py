"""Full-size parity: the workloads at their full token counts, run through the
same calls and launch configuration as the benchmark (fast split-K mode; one
case per workload family also in the deterministic mode), with
sampled outputs checked one by one against the oracle (which computes just
the sampled pairs, tokens and rank rows)."""
import numpy as np
import pytest

import oracle
from paper_2609_06072_gb300 import workloads as W
from ace_testlib import check_close, dev_bf16, host_f64
from test_gpu_fwd import compare_perm, make_plan, run_perm

pytestmark = pytest.mark.gpu

N_PAIRS, N_TOK, N_RANK = 256, 96, 48


def _full_case(name, seed, det=False):
    import torch
    L = W.Layer(W.get_config(name), seed=seed)
    c = L.cfg
    plan = make_plan(L, deterministic=det)
    perm, P = run_perm(L, plan)
    O = oracle.permute(L.topk_idx, L.e2g, L.G)
    compare_perm(P, O)
    rp, pr = O["row_pair"], O["pair_row"]
    rng = np.random.default_rng(1234 + seed)
    sel_p = np.sort(rng.choice(c.R, N_PAIRS, replace=False)).astype(np.int32)
    sel_t = np.sort(rng.choice(c.T, N_TOK, replace=False)).astype(np.int32)
    n_rank = int(L.rank_off[-1])
    sel_r = np.sort(rng.choice(n_rank, min(N_RANK, n_rank), replace=False)).astype(np.int32)
    s = c.s

    # ---- forward: gate/up (shared input) and down (per row)
    X = dev_bf16(L.X())
    A = {p: dev_bf16(L.A(p)) for p in ("gate", "up", "down")}
    Bt = {p: dev_bf16(L.Bt(p)) for p in ("gate", "up", "down")}
    Y = [torch.zeros(c.R, c.f, dtype=torch.bfloat16, device="cuda") for _ in range(2)]
    H = [torch.zeros(c.R, plan.rank_max, device="cuda") for _ in range(3)]
    plan.fwd_shared(perm, X, [A["gate"], A["up"]], [Bt["gate"], Bt["up"]], s, Y, H[:2])
    hin = dev_bf16(L.h()[rp])
    Yd = torch.zeros(c.R, c.d, dtype=torch.bfloat16, device="cuda")
    plan.fwd_row(perm, hin, A["down"], Bt["down"], s, Yd, H[2])
    assert plan.get_error(perm) == 0
    rows = pr[sel_p]
    for j, p in enumerate(("gate", "up")):
        ref, _ = oracle.fwd(L.topk_idx, L.e2g, L.rank_off, L.X(), L.A(p), L.Bt(p), s, sel=sel_p)
        check_close(host_f64(Y[j][torch.from_numpy(rows).long().cuda()]), ref, f"Y_{p}[sampled]")
    ref, _ = oracle.fwd(L.topk_idx, L.e2g, L.rank_off, L.h(), L.A("down"), L.Bt("down"), s, x_per_pair=True,
                        sel=sel_p)
    check_close(host_f64(Yd[torch.from_numpy(rows).long().cuda()]), ref, "Y_down[sampled]")
    del Y, Yd

    # ---- backward: down (per row), then gate/up (shared input, with dX)
    _, _, bws = plan.alloc_workspaces(c.T)
    dYd = dev_bf16(L.dY("down")[rp])
    dh = torch.zeros(c.R, c.f, dtype=torch.bfloat16, device="cuda")
    dA = {p: torch.full((n_rank, c.f if p == "down" else c.d), float("nan"), device="cuda")
          for p in ("gate", "up", "down")}
    dBt = {p: torch.full((n_rank, c.d if p == "down" else c.f), float("nan"), device="cuda")
           for p in ("gate", "up", "down")}
    plan.bwd_row(perm, dYd, hin, H[2], A["down"], Bt["down"], s, dh, dA["down"], dBt["down"], bws)
    dY = [dev_bf16(L.dY(p)[rp]) for p in ("gate", "up")]
    dX = torch.zeros(c.T, c.d, dtype=torch.bfloat16, device="cuda")
    plan.bwd_shared(perm, dY, X, H[:2], [A["gate"], A["up"]], [Bt["gate"], Bt["up"]], s, dX,
                    [dA["gate"], dA["up"]], [dBt["gate"], dBt["up"]], bws)
    assert plan.get_error(perm) == 0

    ref = oracle.bwd_dx(L.topk_idx, L.e2g, L.rank_off, L.dY("down"), L.A("down"), L.Bt("down"), s,
                        x_per_pair=True, sel=sel_p)
    check_close(host_f64(dh[torch.from_numpy(rows).long().cuda()]), ref, "dh[sampled]")
    ref = sum(oracle.bwd_dx(L.topk_idx, L.e2g, L.rank_off, L.dY(p), L.A(p), L.Bt(p), s, sel=sel_t)
              for p in ("gate", "up"))
    check_close(host_f64(dX[torch.from_numpy(sel_t).long().cuda()]), ref, "dX[sampled]")
    ri = torch.from_numpy(sel_r).long().cuda()
    for p in ("gate", "up", "down"):
        xin, per_pair = (L.h(), True) if p == "down" else (L.X(), False)
        rdA, rdBt = oracle.bwd_w(L.topk_idx, L.e2g, L.rank_off, xin, L.dY(p), L.A(p), L.Bt(p), s,
                                 x_per_pair=per_pair, sel=sel_r)
        check_close(host_f64(dA[p][ri]), rdA, f"dA_{p}[sampled]")
        check_close(host_f64(dBt[p][ri]), rdBt, f"dBt_{p}[sampled]")


@pytest.mark.parametrize("name", ["olmoe", "qwen", "deepseek_g16", "deepseek_g32", "deepseek_g8", "olmoe_uneven",
                                  "kimi", "mixtral"])
def test_full_size_sampled_parity(name):
    _full_case(name, 0)


@pytest.mark.parametrize("name", ["olmoe", "olmoe_uneven"])
def test_full_size_sampled_parity_deterministic(name):
    """The deterministic two-stage split-K mode at full size."""
    _full_case(name, 1, det=True)
