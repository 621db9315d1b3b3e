"""Host-side logic that needs no GPU: the seeded groupings of the workloads,
the benchmark's routing statistics and byte model, and the kernel-source hash
that ties stored ncu counters to the code they were taken from."""
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2609_06072_gb300 import workloads as W  # noqa: E402


def test_paperlike_grouping_sizes_and_budget():
    for name in ("olmoe_uneven", "kimi"):
        L = W.Layer(W.get_config(name), seed=0)
        c = L.cfg
        sizes = np.bincount(L.e2g, minlength=L.G)
        # per block of 64 experts: one group of 43, mid-size groups, four singletons
        assert sizes.sum() == c.E and sizes.min() >= 1
        assert sorted(sizes.tolist(), reverse=True)[: c.E // 64] == [43] * (c.E // 64)
        assert (sizes == 1).sum() == 4 * (c.E // 64)
        # matched budget: sum_g r_g = E * r
        assert int(L.rank_off[-1]) == c.E * c.r
        assert np.array_equal(np.diff(L.rank_off), sizes * c.r)
        # seeded: the same grouping on every draw, another seed another shuffle
        assert np.array_equal(L.e2g, W.Layer(W.get_config(name), seed=0).e2g)
        assert not np.array_equal(L.e2g, W.Layer(W.get_config(name), seed=1).e2g)


def test_load_stats():
    st = bench.load_stats([5, 0, 10, 20], 35, 30)
    assert st["expert_rows_max"] == 20 and st["expert_rows_min"] == 0
    assert abs(st["R_over_U"] - 35 / 30) < 1e-12
    p = np.array([5, 10, 20]) / 35
    assert abs(st["load_entropy_bits"] - float(-(p * np.log2(p)).sum())) < 1e-12
    uni = bench.load_stats([7] * 8, 56, 56)
    assert abs(uni["load_entropy_ratio"] - 1.0) < 1e-12


def test_byte_model_counts_each_tensor_once():
    # two groups, equal ranks: bytes of the forward per row call follow the
    # stated formula term by term
    T, k, d, f = 64, 2, 32, 16
    rank_off = [0, 8, 16]
    U_g, R_g = np.array([40, 30]), np.array([64, 64])
    b, fl = bench.model(T, k, d, f, rank_off, U_g, R_g)
    R, Pw = T * k, 16 * (d + f)
    assert b["fwd_row"] == 2 * R * f + 4 * R * d + 4 * int((R_g * 8).sum()) + 2 * Pw
    assert fl["fwd_row"] == 2 * int((R_g * 8).sum()) * (d + f)
    assert b["bwd_row"] == 2 * R * d + 2 * R * f + 4 * int((R_g * 8).sum()) + 4 * R * f + 6 * Pw


def test_olmoe_byte_model_is_the_reported_one():
    # the algorithmic bytes the benchmark's roofline divides by, for the
    # OLMoE-shaped layer at seed 0 (the bench's default), from the realised
    # routing: per-group row and unique-pair counts of the oracle permutation
    import oracle
    L = W.Layer(W.get_config("olmoe"), seed=0)
    c = L.cfg
    O = oracle.permute(L.topk_idx, L.e2g, L.G)
    b, fl = bench.model(c.T, c.k, c.d, c.f, L.rank_off, np.diff(O["uniq_off"]), np.diff(O["group_off"]))
    assert b["fwd_row"] == 682622976
    assert b["bwd_row"] == 688914432
    # every routed row moves its Y / dY / h / dh bytes once: the row traffic
    # alone is most of each down call
    R = c.T * c.k
    assert 2 * R * c.f + 4 * R * c.d > 0.95 * b["fwd_row"]


def test_source_hash_ignores_comments(tmp_path, monkeypatch):
    src = tmp_path / "paper_2609_06072_gb300" / "csrc"
    src.mkdir(parents=True)
    (src / "a.cu").write_text("int f() {  // one\n  return 1; /* two */ }\n")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    h0 = bench.csrc_sha()
    (src / "a.cu").write_text("// header\nint f() {\n  return 1;\n}\n")
    assert bench.csrc_sha() == h0
    (src / "a.cu").write_text("int f() { return 2; }\n")
    assert bench.csrc_sha() != h0


def test_combine_oracle_sample_runs_on_cpu():
    """The CPU baseline beside the combine variant: every oracle call of the
    sample accepts its selections (no GPU needed)."""
    dt, rows = bench.combine_oracle_sample("tiny", 0, 0.25)
    c = W.get_config("tiny")
    assert dt > 0 and abs(rows - 0.25 * c.R) < 1e-9


def test_ffn_and_cka_oracle_samples_run_on_cpu():
    dt, rows = bench.ffn_oracle_sample("tiny", 0, 4)
    assert dt > 0 and rows == 4 * W.get_config("tiny").k
    dt, n = bench.cka_oracle_sample("tiny", 0, 2)
    assert dt > 0 and n == 2
