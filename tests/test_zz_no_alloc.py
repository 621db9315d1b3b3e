"""The allocation-free forward entry point, for callers that cannot allocate
device memory (a serving process or plug-in host whose device memory is all
reserved by its own pool, with no allocator or workspace handed to the
plug-in).  It must give exactly the result of the regular entry point: both
launch the same kernels on the same inputs and the forward has no atomics, so
the outputs are compared bit for bit, on two calls in a row (the second call
finds the previous call's contents in the library's scratch array).  One case
is also checked against the fp64 oracle.  Kept in a file collected last."""
import numpy as np
import pytest

import oracle
from paper_2609_06072_gb300 import workloads as W
from ace_testlib import check_close, dev_bf16, host_f64

pytestmark = pytest.mark.gpu

# tiny and OLMoE stack <= 512 ranks per projection (token-major H GEMM);
# the Qwen shape stacks 15 x 64 = 960, so H is gathered per unique pair and
# the scratch's H is read back by the row kernel from a gathered layout.
CASES = [("tiny", {}), ("olmoe", {"T": 1024}), ("qwen", {"T": 512})]


@pytest.mark.parametrize("name,over", CASES)
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
    assert plan.get_error(perm) == 0
    for _ in range(2):
        got = [b.clone() for b in base]
        plan.fwd_shared_noalloc(perm, X, A, Bt, c.s, got)
        assert plan.get_error(perm) == 0
        for g_, r_ in zip(got, ref):
            assert torch.equal(g_, r_), "Y of the allocation-free call differs from the workspace entry point"


def test_fwd_shared_noalloc_matches_oracle():
    import torch
    from paper_2609_06072_gb300 import ace
    L = W.Layer(W.get_config("tiny"), seed=5)
    c = L.cfg
    plan = ace.Plan(c.T, c.k, c.E, L.G, L.e2g, L.rank_off, c.d, c.f)
    pws, _, _ = plan.alloc_workspaces(c.T)
    perm = plan.permute(torch.from_numpy(L.topk_idx).cuda(), pws)
    O = oracle.permute(L.topk_idx, L.e2g, L.G)
    Y = [dev_bf16(np.zeros((c.R, c.f), np.uint16)) for _ in range(2)]
    plan.fwd_shared_noalloc(perm, dev_bf16(L.X()), [dev_bf16(L.A(p)) for p in ("gate", "up")],
                            [dev_bf16(L.Bt(p)) for p in ("gate", "up")], c.s, Y)
    assert plan.get_error(perm) == 0
    for j, pj in enumerate(("gate", "up")):
        ref, _ = oracle.fwd(L.topk_idx, L.e2g, L.rank_off, L.X(), L.A(pj), L.Bt(pj), c.s)
        got = np.empty((c.R, c.f))
        got[O["row_pair"]] = host_f64(Y[j])
        check_close(got, ref, f"Y_{pj} (allocation-free entry point)")


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
