"""The allocation-free forward entry point (for callers that cannot allocate
device memory, e.g. a serving process whose device memory is all reserved by
its own pool) must give the same result as the regular entry point, on two
calls in a row (the second call finds the previous call's scratch contents).
Kept in a file collected last."""
import numpy as np
import pytest

from paper_2609_06072_gb300 import workloads as W
from ace_testlib import check_close, dev_bf16, host_f64

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("name,over", [("tiny", {}), ("olmoe", {"T": 1024})])
def test_fwd_shared_noalloc_matches_workspace_entry_point(name, over):
    import torch
    from paper_2609_06072_gb300 import ace
    L = W.Layer(W.get_config(name, **over), seed=3)
    c = L.cfg
    plan = ace.Plan(c.T, c.k, c.E, L.G, L.e2g, L.rank_off, c.d, c.f)
    pws, _, _ = plan.alloc_workspaces(c.T)
    perm = plan.permute(torch.from_numpy(L.topk_idx).cuda(), pws)
    X = dev_bf16(L.X())
    A = [dev_bf16(L.A(p)) for p in ("gate", "up")]
    Bt = [dev_bf16(L.Bt(p)) for p in ("gate", "up")]
    base = [dev_bf16(L.Y_base(p)) for p in ("gate", "up")]
    ref = [b.clone() for b in base]
    H = [torch.empty(c.R, plan.rank_max, device="cuda") for _ in range(2)]
    plan.fwd_shared(perm, X, A, Bt, c.s, ref, H)
    for _ in range(2):
        got = [b.clone() for b in base]
        plan.fwd_shared_noalloc(perm, X, A, Bt, c.s, got)
        assert plan.get_error(perm) == 0
        for g_, r_ in zip(got, ref):
            check_close(host_f64(g_), host_f64(r_), "Y noalloc vs workspace entry point")


def test_fwd_shared_noalloc_rejects_oversize():
    import torch
    from paper_2609_06072_gb300 import ace
    # T*k*rank_max*4*2 bytes > 32 MiB: 65536*8*32*8 = 128 MiB
    L = W.Layer(W.get_config("olmoe", T=65536), seed=0)
    c = L.cfg
    plan = ace.Plan(c.T, c.k, c.E, L.G, L.e2g, L.rank_off, c.d, c.f)
    pws, _, _ = plan.alloc_workspaces(c.T)
    perm = plan.permute(torch.from_numpy(L.topk_idx).cuda(), pws)
    X = torch.zeros(c.T, c.d, dtype=torch.bfloat16, device="cuda")
    A = [torch.zeros(plan.n_rank, c.d, dtype=torch.bfloat16, device="cuda") for _ in range(2)]
    Bt = [torch.zeros(plan.n_rank, c.f, dtype=torch.bfloat16, device="cuda") for _ in range(2)]
    Y = [torch.zeros(8, c.f, dtype=torch.bfloat16, device="cuda") for _ in range(2)]  # never touched
    with pytest.raises(ace.AceError) as ei:
        plan.fwd_shared_noalloc(perm, X, A, Bt, c.s, Y)
    assert ei.value.status == ace.ACE_ERR_WORKSPACE
