"""Failure paths and boundary helpers on the GPU.

* A bounded device wait that runs out: with the test-only plan flag
  ACE_FLAG_TEST_WAIT_EXPIRY the down forward never raises the ready flags of
  its split row tiles' up-front H, so the row kernel's flag wait gives up
  (after 2 ms), every CTA winds down through its own bounded waits, frees its
  tensor memory and returns; ace_get_error reports ACE_ERR_DEVICE_TIMEOUT and
  the context stays usable.  Nothing faults, traps or hangs.
* ace_gather_rows / ace_scatter_rows move bf16 rows between pair order and
  row order bit for bit."""
import time

import numpy as np
import pytest

import oracle
from paper_2609_06072_gb300 import workloads as W
from ace_testlib import dev_bf16
from test_gpu_fwd import _fwd_row_case, compare_perm, run_perm

pytestmark = pytest.mark.gpu


def test_bounded_wait_expiry_reports_timeout_and_context_survives():
    import torch
    from paper_2609_06072_gb300 import ace
    L = W.Layer(W.get_config("olmoe", T=4096), seed=3)
    c = L.cfg
    plan = ace.Plan(c.T, c.k, c.E, L.G, L.e2g, L.rank_off, c.d, c.f, flags=ace.ACE_FLAG_TEST_WAIT_EXPIRY)
    perm, P = run_perm(L, plan)
    compare_perm(P, oracle.permute(L.topk_idx, L.e2g, L.G))
    assert plan.get_error(perm) == ace.ACE_OK
    hin = dev_bf16(L.h()[P["row_pair"]])
    Y = torch.zeros(c.R, c.d, dtype=torch.bfloat16, device="cuda")
    H = torch.zeros(c.R, plan.rank_max, device="cuda")  # a saved H: the split tiles get an up-front H
    t0 = time.perf_counter()
    plan.fwd_row(perm, hin, dev_bf16(L.A("down")), dev_bf16(L.Bt("down")), c.s, Y, H)
    st = plan.get_error(perm)  # synchronises
    dt = time.perf_counter() - t0
    assert st == ace.ACE_ERR_DEVICE_TIMEOUT, ace.STATUS_NAMES.get(st, st)
    assert dt < 20.0, dt  # every wait is bounded (1 s each at most, 2 ms for the flag)
    assert plan.get_error(perm) == ace.ACE_OK  # the read cleared the flag
    # the same permutation workspace and device context still give correct results
    ok = ace.Plan(c.T, c.k, c.E, L.G, L.e2g, L.rank_off, c.d, c.f)
    perm2, _ = run_perm(L, ok)
    Y2 = torch.zeros(c.R, c.d, dtype=torch.bfloat16, device="cuda")
    ok.fwd_row(perm2, hin, dev_bf16(L.A("down")), dev_bf16(L.Bt("down")), c.s, Y2, H)
    assert ok.get_error(perm2) == ace.ACE_OK
    _fwd_row_case(L, c.s, with_base=False)


@pytest.mark.parametrize("name,over,cols", [("tiny", {}, 256), ("olmoe", {"T": 2048}, 1024),
                                            ("kimi", {"T": 300}, 72), ("tiny", {"T": 1}, 8)])
def test_gather_scatter_rows_bit_exact(name, over, cols):
    import torch
    from paper_2609_06072_gb300 import ace
    L = W.Layer(W.get_config(name, **over), seed=2)
    c = L.cfg
    plan = ace.Plan(c.T, c.k, c.E, L.G, L.e2g, L.rank_off, c.d, c.f)
    perm, P = run_perm(L, plan)
    rp = P["row_pair"]
    rng = np.random.default_rng(7)
    src = rng.integers(0, 1 << 16, size=(c.R, cols), dtype=np.uint16)  # arbitrary bit patterns, NaNs included
    src_d = torch.from_numpy(src.view(np.int16)).cuda()
    rows = torch.empty_like(src_d)
    plan.gather_rows(perm, src_d, rows)
    got = rows.cpu().numpy().view(np.uint16)
    assert np.array_equal(got, src[rp])  # dst[row] = src[row_pair[row]]
    back = torch.empty_like(src_d)
    plan.scatter_rows(perm, rows, back)
    assert np.array_equal(back.cpu().numpy().view(np.uint16), src)  # dst[row_pair[row]] = src[row]
