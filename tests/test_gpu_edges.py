"""Edge cases of the scope table on the GPU, through the same parity checks
as the main cases: top-1 routing, every token routed to every expert (k = E,
so every token is active in every group), hidden and expert sizes that are
not multiples of the 64-column tiles (and too small for the last wave's
column parts), and a ragged token count."""
import pytest

from paper_2609_06072_gb300 import workloads as W
from test_gpu_bwd import _row_case, _shared_case
from test_gpu_fwd import _fwd_row_case, _fwd_shared_case

pytestmark = pytest.mark.gpu

EDGES = [("tiny", 8, {"k": 1}), ("tiny", 9, {"k": 8}), ("tiny", 10, {"d": 136, "f": 72}),
         ("tiny", 11, {"d": 200, "f": 120, "T": 77})]


@pytest.mark.parametrize("name,seed,over", EDGES)
def test_edge_forward(name, seed, over):
    L = W.Layer(W.get_config(name, **over), seed=seed)
    _fwd_shared_case(L, L.cfg.s, with_base=False)
    _fwd_row_case(L, L.cfg.s, with_base=False)


@pytest.mark.parametrize("det", [True, False])
@pytest.mark.parametrize("name,seed,over", EDGES)
def test_edge_backward(name, seed, over, det):
    L = W.Layer(W.get_config(name, **over), seed=seed)
    _shared_case(L, det)
    _row_case(L, det)
