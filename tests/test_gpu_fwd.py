"""GPU parity of the route-permute and the fused forward against the oracle.

Permutation arrays must be bit-exact; forward outputs must meet the per-tensor
bar of tests/ace_testlib.py.  Every call goes through the C ABI."""
import numpy as np
import pytest

import oracle
from paper_2609_06072_gb300 import workloads as W
from ace_testlib import check_close, dev_bf16, host_f64

pytestmark = pytest.mark.gpu

# H = A_g x is accumulated in fp32 from exact bf16 products over K <= 16384
# terms: sqrt(K) * 2^-24 ~ 8e-6 relative; a 10x / 2.5x margin.
H_MAX_REL = 1e-4
H_FRO_REL = 2e-5


def make_plan(L, deterministic=False, T_max=None):
    from paper_2609_06072_gb300 import ace
    c = L.cfg
    return ace.Plan(T_max or c.T, c.k, c.E, L.G, L.e2g, L.rank_off, c.d, c.f, deterministic=deterministic)


def run_perm(L, plan):
    import torch
    from paper_2609_06072_gb300 import ace
    pws, _, _ = plan.alloc_workspaces(L.cfg.T)
    idx = torch.from_numpy(L.topk_idx).cuda()
    perm = plan.permute(idx, pws)
    perm._idx = idx
    return perm, ace.perm_arrays(plan, perm)


def compare_perm(G_arr, O):
    assert G_arr["U"] == O["U"]
    for key in ("group_off", "expert_off", "expert_cnt", "row_pair", "pair_row", "uniq_off", "uniq_tok", "tok_uniq",
                "row_uniq"):
        assert np.array_equal(G_arr[key], O[key]), key


PERM_CASES = [("tiny", 0, {}), ("tiny", 1, {}), ("olmoe", 0, {}), ("qwen", 0, {"T": 4096}),
              ("deepseek_g16", 0, {"T": 4096}), ("mixtral", 0, {"T": 2048}), ("tiny", 2, {"T": 1}),
              ("tiny", 3, {"T": 300}), ("olmoe_uneven", 0, {"T": 2048}), ("kimi", 0, {"T": 1024})]


@pytest.mark.parametrize("name,seed,over", PERM_CASES)
def test_permute_bit_exact(name, seed, over):
    L = W.Layer(W.get_config(name, **over), seed=seed)
    plan = make_plan(L)
    perm, got = run_perm(L, plan)
    O = oracle.permute(L.topk_idx, L.e2g, L.G)
    compare_perm(got, O)
    assert plan.get_error(perm) == 0
    # deterministic: a second run gives identical bytes
    perm2, got2 = run_perm(L, plan)
    for k in got:
        assert np.array_equal(np.asarray(got[k]), np.asarray(got2[k])), k


def test_permute_expertwise_identity():
    L = W.Layer(W.get_config("olmoe"), seed=0, expertwise=True)
    plan = make_plan(L)
    perm, got = run_perm(L, plan)
    O = oracle.permute(L.topk_idx, L.e2g, L.G)
    compare_perm(got, O)
    assert got["U"] == L.cfg.R  # dedup degenerates: every pair is its own (g, t)


def test_permute_flags_invalid_routing():
    import torch
    from paper_2609_06072_gb300 import ace
    L = W.Layer(W.get_config("tiny"), seed=0)
    plan = make_plan(L)
    pws, _, _ = plan.alloc_workspaces(L.cfg.T)
    bad = L.topk_idx.copy()
    bad[5, 1] = bad[5, 0]          # repeated expert
    bad[9, 0] = L.cfg.E + 3        # out of range
    perm = plan.permute(torch.from_numpy(bad).cuda(), pws)
    assert plan.get_error(perm) == ace.ACE_ERR_INDEX
    assert plan.get_error(perm) == ace.ACE_OK  # cleared by the read


def _fwd_shared_case(L, s, with_base, nproj=2):
    import torch
    c = L.cfg
    plan = make_plan(L)
    perm, P = run_perm(L, plan)
    O = oracle.permute(L.topk_idx, L.e2g, L.G)
    compare_perm(P, O)
    projs = ["gate", "up"][:nproj]
    R, f = c.R, c.f
    Y, H, ybase = [], [], []
    for pj in projs:
        yb = L.Y_base(pj) if with_base else np.zeros((R, f), np.uint16)
        ybase.append(yb)
        Y.append(dev_bf16(yb[O["row_pair"]]))
        H.append(torch.full((R, plan.rank_max), float("nan"), device="cuda"))
    X = dev_bf16(L.X())
    plan.fwd_shared(perm, X, [dev_bf16(L.A(p)) for p in projs], [dev_bf16(L.Bt(p)) for p in projs], s, Y, H)
    assert plan.get_error(perm) == 0
    U = O["U"]
    lead_pair = O["row_pair"][O["uniq_rows"][O["uniq_rows_ptr"][:-1]]]
    for j, pj in enumerate(projs):
        ref, Href = oracle.fwd(L.topk_idx, L.e2g, L.rank_off, L.X(), L.A(pj), L.Bt(pj), s,
                               y_in=ybase[j] if with_base else None, want_h=True)
        got_rows = host_f64(Y[j])
        got = np.empty_like(got_rows)
        got[O["row_pair"]] = got_rows
        if with_base:
            check_close(got, ref, f"Y_{pj}")
        else:
            check_close(got, ref, f"Y_{pj}")
        Hg = host_f64(H[j])[:U]
        check_close(Hg, Href[lead_pair][:, : plan.rank_max], f"H_{pj}", max_rel=H_MAX_REL, fro_rel=H_FRO_REL)


@pytest.mark.parametrize("name,seed,over", [("tiny", 0, {}), ("tiny", 1, {"T": 300}), ("olmoe", 0, {"T": 1024}),
                                            ("olmoe", 2, {"T": 4096}), ("qwen", 0, {"T": 1024}),
                                            ("deepseek_g16", 0, {"T": 1024}), ("tiny", 4, {"r": 3}),
                                            ("olmoe_uneven", 0, {"T": 512}), ("kimi", 0, {"T": 256}),
                                            ("deepseek_g32", 0, {"T": 1024}), ("deepseek_g8", 0, {"T": 1024}),
                                            # full Mixtral widths: 224 column chunks of f, a 64-step K loop
                                            ("mixtral", 0, {"T": 256})])
def test_fwd_shared_parity(name, seed, over):
    L = W.Layer(W.get_config(name, **over), seed=seed)
    _fwd_shared_case(L, L.cfg.s, with_base=False)


def test_fwd_shared_nonzero_base_and_single_projection():
    L = W.Layer(W.get_config("tiny"), seed=4)
    _fwd_shared_case(L, 2.0, with_base=True)
    _fwd_shared_case(L, 0.5, with_base=False, nproj=1)


def test_fwd_shared_expertwise_padded_rank():
    L = W.Layer(W.get_config("olmoe", T=512), seed=0, expertwise=True)  # r = 8 -> MMA N padded to 16
    _fwd_shared_case(L, 2.0, with_base=False)


def _fwd_row_case(L, s, with_base):
    import torch
    c = L.cfg
    plan = make_plan(L)
    perm, P = run_perm(L, plan)
    O = oracle.permute(L.topk_idx, L.e2g, L.G)
    compare_perm(P, O)
    R, d = c.R, c.d
    yb = L.Y_base("down") if with_base else np.zeros((R, d), np.uint16)
    Y = dev_bf16(yb[O["row_pair"]])
    H = torch.full((R, plan.rank_max), float("nan"), device="cuda")
    hin = dev_bf16(L.h()[O["row_pair"]])
    plan.fwd_row(perm, hin, dev_bf16(L.A("down")), dev_bf16(L.Bt("down")), s, Y, H)
    assert plan.get_error(perm) == 0
    ref, Href = oracle.fwd(L.topk_idx, L.e2g, L.rank_off, L.h(), L.A("down"), L.Bt("down"), s, x_per_pair=True,
                           y_in=yb if with_base else None, want_h=True)
    got_rows = host_f64(Y)
    got = np.empty_like(got_rows)
    got[O["row_pair"]] = got_rows
    check_close(got, ref, "Y_down")
    check_close(host_f64(H), Href[O["row_pair"]][:, : plan.rank_max], "H_down", max_rel=H_MAX_REL, fro_rel=H_FRO_REL)


@pytest.mark.parametrize("with_ws", [False, True])
def test_fwd_row_without_saved_h(with_ws):
    """No H to save: with forward scratch the last wave's tiles get their H up
    front in the scratch and run in column parts; without it they run whole.
    Y is the same either way."""
    import torch
    L = W.Layer(W.get_config("olmoe", T=4096), seed=3)
    c = L.cfg
    plan = make_plan(L)
    perm, P = run_perm(L, plan)
    O = oracle.permute(L.topk_idx, L.e2g, L.G)
    Y = dev_bf16(np.zeros((c.R, c.d), np.uint16))
    ws = None
    if with_ws:
        _, fwd_bytes, _ = plan.workspace_size(c.T)
        ws = torch.empty(fwd_bytes, dtype=torch.uint8, device="cuda")
    plan.fwd_row(perm, dev_bf16(L.h()[O["row_pair"]]), dev_bf16(L.A("down")), dev_bf16(L.Bt("down")), c.s, Y,
                 None, ws)
    assert plan.get_error(perm) == 0
    ref, _ = oracle.fwd(L.topk_idx, L.e2g, L.rank_off, L.h(), L.A("down"), L.Bt("down"), c.s, x_per_pair=True)
    got = np.empty((c.R, c.d))
    got[O["row_pair"]] = host_f64(Y)
    check_close(got, ref, "Y_down")


@pytest.mark.parametrize("name,seed,over,base", [("tiny", 0, {}, False), ("tiny", 5, {"T": 77}, True),
                                                 ("olmoe", 0, {"T": 512}, False), ("olmoe", 2, {"T": 4096}, True),
                                                 ("qwen", 1, {"T": 512}, False),
                                                 ("deepseek_g16", 0, {"T": 512}, True), ("tiny", 4, {"r": 3}, False),
                                                 ("olmoe_uneven", 0, {"T": 512}, True), ("kimi", 0, {"T": 256}, False),
                                                 ("deepseek_g32", 0, {"T": 1024}, False),
                                                 ("deepseek_g8", 0, {"T": 1024}, True),
                                                 # full Mixtral widths: a 224-step K loop over f, 64 chunks of d
                                                 ("mixtral", 0, {"T": 256}, True)])
def test_fwd_row_parity(name, seed, over, base):
    L = W.Layer(W.get_config(name, **over), seed=seed)
    _fwd_row_case(L, L.cfg.s, with_base=base)


def test_no_tokens():
    """T = 0: every call succeeds with empty (null) token and row tensors,
    launches no row work, and leaves exact-zero weight gradients."""
    import torch
    L = W.Layer(W.get_config("tiny"), seed=0)
    c = L.cfg
    plan = make_plan(L)
    pws, _, bws = plan.alloc_workspaces(0)
    perm = plan.permute(torch.zeros(0, c.k, dtype=torch.int32, device="cuda"), pws)
    assert perm.T == 0 and perm.R == 0
    bf = lambda *s: torch.empty(*s, dtype=torch.bfloat16, device="cuda")
    f32 = lambda *s: torch.empty(*s, dtype=torch.float32, device="cuda")
    rm = plan.rank_max
    A = [dev_bf16(L.A(p)) for p in ("gate", "up", "down")]
    Bt = [dev_bf16(L.Bt(p)) for p in ("gate", "up", "down")]
    plan.fwd_shared(perm, bf(0, c.d), A[:2], Bt[:2], c.s, [bf(0, c.f), bf(0, c.f)], [f32(0, rm), f32(0, rm)])
    plan.fwd_row(perm, bf(0, c.f), A[2], Bt[2], c.s, bf(0, c.d), f32(0, rm))
    nan = lambda *s: torch.full(s, float("nan"), device="cuda")
    dA = [nan(plan.n_rank, c.d), nan(plan.n_rank, c.d), nan(plan.n_rank, c.f)]
    dBt = [nan(plan.n_rank, c.f), nan(plan.n_rank, c.f), nan(plan.n_rank, c.d)]
    plan.bwd_shared(perm, [bf(0, c.f), bf(0, c.f)], bf(0, c.d), [f32(0, rm), f32(0, rm)], A[:2], Bt[:2], c.s,
                    bf(0, c.d), dA[:2], dBt[:2], bws)
    plan.bwd_row(perm, bf(0, c.d), bf(0, c.f), f32(0, rm), A[2], Bt[2], c.s, bf(0, c.f), dA[2], dBt[2], bws)
    dAc, dBc = nan(plan.n_rank, c.f), nan(plan.n_rank, c.d)
    plan.fwd_combine(perm, bf(0, c.f), f32(0, c.k), A[2], Bt[2], c.s, bf(0, c.d), f32(0, rm), bf(0, plan.rank_cols))
    plan.bwd_combine(perm, bf(0, c.d), bf(0, c.f), f32(0, c.k), f32(0, rm), bf(0, plan.rank_cols), A[2], Bt[2], c.s,
                     bf(0, c.f), f32(0, c.k), dAc, dBc, bws)
    assert plan.get_error(perm) == 0
    for t in dA + dBt + [dAc, dBc]:
        assert bool((t == 0).all())
