"""The C oracle sums every output element serially in a fixed order, so its
results must not depend on the OpenMP thread count: one thread and all
threads give bit-identical outputs."""
import os
import subprocess
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SCRIPT = r"""
import sys
import numpy as np
sys.path.insert(0, ROOT)
import oracle
from paper_2609_06072_gb300 import workloads as W
L = W.Layer(W.get_config("tiny", T=96), seed=3)
c = L.cfg
out = {}
y, H = oracle.fwd(L.topk_idx, L.e2g, L.rank_off, L.X(), L.A("up"), L.Bt("up"), c.s, want_h=True)
out["y"], out["H"] = y, H
out["dx"] = oracle.bwd_dx(L.topk_idx, L.e2g, L.rank_off, L.dY("up"), L.A("up"), L.Bt("up"), c.s)
dA, dBt = oracle.bwd_w(L.topk_idx, L.e2g, L.rank_off, L.X(), L.dY("up"), L.A("up"), L.Bt("up"), c.s)
out["dA"], out["dBt"] = dA, dBt
out["z"] = oracle.combine_fwd(L.topk_idx, L.e2g, L.rank_off, L.h(), L.topk_w, L.A("down"), L.Bt("down"), c.s)
dh, dw = oracle.combine_bwd_dh(L.topk_idx, L.e2g, L.rank_off, L.dZ(), L.h(), L.topk_w, L.A("down"), L.Bt("down"), c.s)
out["dh"], out["dw"] = dh, dw
cA, cB = oracle.combine_bwd_w(L.topk_idx, L.e2g, L.rank_off, L.h(), L.dZ(), L.topk_w, L.A("down"), L.Bt("down"), c.s)
out["cA"], out["cB"] = cA, cB
np.savez(sys.argv[1], **out)
""".replace("ROOT", repr(ROOT))


def _run(tmp_path, threads, tag):
    path = str(tmp_path / f"{tag}.npz")
    env = dict(os.environ, OMP_NUM_THREADS=str(threads))
    subprocess.run([sys.executable, "-c", SCRIPT, path], check=True, env=env, cwd=ROOT)
    return np.load(path)


def test_oracle_is_bitwise_independent_of_thread_count(tmp_path):
    one = _run(tmp_path, 1, "one")
    many = _run(tmp_path, max(2, os.cpu_count() or 2), "many")
    for key in one.files:
        assert np.array_equal(one[key], many[key]), key
