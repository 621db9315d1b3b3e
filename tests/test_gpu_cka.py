"""GPU parity of the CKA similarity matrix (Sec. 3.2) against the
consolidation oracle: every pair at small sizes, sampled pairs at the
OLMoE-shaped probe size, both centering variants, and the grouping that
follows from it."""
import numpy as np
import pytest

from oracle import consolidation as C
from paper_2609_06072_gb300 import workloads as W
from ace_testlib import dev_bf16

pytestmark = pytest.mark.gpu


def bits(x):
    return W.f32_to_bf16_bits(np.asarray(x, dtype=np.float32))


def planted(rng, E, N, d_in, d_out, r, n_proto, noise):
    proto = rng.integers(0, n_proto, E)
    PA = [rng.standard_normal((r, d_in)) for _ in range(n_proto)]
    PB = [rng.standard_normal((r, d_out)) for _ in range(n_proto)]
    A = np.concatenate([bits(PA[p] + noise * rng.standard_normal((r, d_in))) for p in proto])
    Bt = np.concatenate([bits(PB[p] + noise * rng.standard_normal((r, d_out))) for p in proto])
    X = bits(rng.standard_normal((N, d_in)) + 0.5)  # a nonzero mean: centering matters
    return X, A, Bt, proto


@pytest.mark.parametrize("center", [True, False])
@pytest.mark.parametrize("E,N,d_in,d_out,r", [(16, 2000, 256, 128, 4), (12, 777, 192, 72, 3), (8, 64, 64, 40, 32)])
def test_cka_matrix_parity(E, N, d_in, d_out, r, center):
    from paper_2609_06072_gb300 import ace
    rng = np.random.default_rng(E + N)
    X, A, Bt, proto = planted(rng, E, N, d_in, d_out, r, 3, 0.3)
    S = ace.cka(dev_bf16(X), dev_bf16(A), dev_bf16(Bt), E, r, center=center).cpu().numpy().astype(np.float64)
    Z = C.adapter_outputs(X, [A[e * r:(e + 1) * r] for e in range(E)], [Bt[e * r:(e + 1) * r] for e in range(E)])
    ref = C.cka_matrix(Z, center=center)
    assert np.all(np.isfinite(S))
    assert np.abs(S - ref).max() <= 2e-3, np.abs(S - ref).max()
    # the grouping decided on the GPU's similarities equals the oracle's
    g_gpu = ace.group_experts(S.astype(np.float32), ace.GROUP_LOUVAIN, 0.8)[0]
    g_ref = C.louvain(C.similarity_graph(ref), 0.8)
    assert np.array_equal(g_gpu, g_ref)


@pytest.mark.parametrize("mean", [16.0, 64.0])
def test_cka_probe_with_a_large_mean(mean):
    """Probe activations whose mean dwarfs their spread: centring must not
    cancel (the covariance of the centred probe, not X^T X minus a rank-one
    correction)."""
    from paper_2609_06072_gb300 import ace
    rng = np.random.default_rng(int(mean))
    E, N, d_in, d_out, r = 12, 1500, 128, 96, 4
    X, A, Bt, proto = planted(rng, E, N, d_in, d_out, r, 3, 0.3)
    X = bits(W.bf16_bits_to_f32(X).astype(np.float64) + mean)
    S = ace.cka(dev_bf16(X), dev_bf16(A), dev_bf16(Bt), E, r, center=True).cpu().numpy().astype(np.float64)
    Z = C.adapter_outputs(X, [A[e * r:(e + 1) * r] for e in range(E)], [Bt[e * r:(e + 1) * r] for e in range(E)])
    ref = C.cka_matrix(Z, center=True)
    assert np.all(np.isfinite(S))
    assert np.abs(S - ref).max() <= 2e-3, np.abs(S - ref).max()


def test_cka_olmoe_probe_sampled_pairs():
    """OLMoE gate shapes (d 2048 -> f 1024, 64 experts of rank 8) on the
    paper's 10k-token probe: sampled pairs against the oracle's definition."""
    from paper_2609_06072_gb300 import ace
    rng = np.random.default_rng(0)
    E, N, d_in, d_out, r = 64, 10000, 2048, 1024, 8
    X, A, Bt, proto = planted(rng, E, N, d_in, d_out, r, 8, 0.5)
    S = ace.cka(dev_bf16(X), dev_bf16(A), dev_bf16(Bt), E, r).cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(S)) and np.allclose(np.diag(S), 1.0, atol=2e-3)
    for i, j in [(0, 1), (5, 40), (63, 62), (17, 17), (30, 2)]:
        Zi, Zj = C.adapter_outputs(X, [A[i * r:(i + 1) * r], A[j * r:(j + 1) * r]],
                                   [Bt[i * r:(i + 1) * r], Bt[j * r:(j + 1) * r]])
        assert abs(S[i, j] - C.cka(Zi, Zj)) <= 2e-3, (i, j)


def test_consolidation_pipeline_against_oracle():
    """Probe -> CKA -> Louvain groups and anchors -> shared adapters: the
    library's result equals the oracle's consolidation of the same grouping
    bit for bit (a copy), with the budget kept."""
    import torch
    from paper_2609_06072_gb300 import ace
    rng = np.random.default_rng(5)
    E, N, d_in, d_out, r = 16, 1500, 128, 96, 4
    X, A, Bt, proto = planted(rng, E, N, d_in, d_out, r, 4, 0.2)
    A_init = bits(rng.standard_normal((E * r, d_in)) / np.sqrt(d_in))
    e2g, rank_off, A_g, Bt_g, S = ace.consolidate(dev_bf16(X), dev_bf16(A), dev_bf16(Bt), E, r, dev_bf16(A_init))
    torch.cuda.synchronize()
    Sd = S.astype(np.float64)
    labels = C.louvain(C.similarity_graph(Sd), 0.8)
    assert np.array_equal(e2g, labels) and np.array_equal(labels, C._relabel(proto))
    anchors = C.cka_center_anchor(Sd, labels)
    _, ro, rA, rB = C.consolidate(labels, [r] * E, anchors, [A[e * r:(e + 1) * r] for e in range(E)],
                                  [Bt[e * r:(e + 1) * r] for e in range(E)],
                                  W.bf16_bits_to_f32(A_init).astype(np.float64))
    assert np.array_equal(rank_off, ro) and rank_off[-1] == E * r
    got_A = W.bf16_bits_to_f32(A_g.view(torch.int16).cpu().numpy().view(np.uint16)).astype(np.float64)
    got_B = W.bf16_bits_to_f32(Bt_g.view(torch.int16).cpu().numpy().view(np.uint16)).astype(np.float64)
    assert np.array_equal(got_A, rA) and np.array_equal(got_B, rB)
