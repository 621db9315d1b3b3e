"""The library's expert grouping (host code, no GPU) against the
consolidation oracle: Louvain on the median-shifted similarity graph, the
fixed-threshold rule and the CKA-centre anchors, label for label."""
import numpy as np
import pytest

from oracle import consolidation as C


@pytest.fixture(scope="module")
def ace():
    from paper_2609_06072_gb300 import _build, ace
    _build.build()
    return ace


def planted_similarity(rng, E, n_groups, noise):
    """A symmetric similarity matrix with planted blocks (fp32-representable)."""
    z = rng.integers(0, n_groups, E)
    base = np.where(z[:, None] == z[None, :], 0.85, 0.35)
    S = base + noise * rng.standard_normal((E, E))
    S = np.clip(0.5 * (S + S.T), 0.0, 1.0)
    np.fill_diagonal(S, 1.0)
    return S.astype(np.float32)


@pytest.mark.parametrize("E,groups,noise,seed", [(8, 2, 0.05, 0), (16, 4, 0.1, 1), (64, 16, 0.1, 2),
                                                 (64, 5, 0.2, 3), (256, 24, 0.15, 4), (7, 3, 0.3, 5)])
def test_louvain_matches_oracle(ace, E, groups, noise, seed):
    rng = np.random.default_rng(seed)
    S = planted_similarity(rng, E, groups, noise)
    Sd = S.astype(np.float64)
    want = C.louvain(C.similarity_graph(Sd), 0.8)
    e2g, anchors, G = ace.group_experts(S, ace.GROUP_LOUVAIN, 0.8)
    assert np.array_equal(e2g, want) and G == int(want.max()) + 1
    assert np.array_equal(anchors, C.cka_center_anchor(Sd, want))


@pytest.mark.parametrize("t", [0.5, 0.7, 0.9])
def test_threshold_matches_oracle(ace, t):
    rng = np.random.default_rng(11)
    S = planted_similarity(rng, 40, 6, 0.2)
    want = C.threshold_groups(S.astype(np.float64), t)
    e2g, anchors, G = ace.group_experts(S, ace.GROUP_THRESHOLD, t)
    assert np.array_equal(e2g, want)
    assert np.array_equal(anchors, C.cka_center_anchor(S.astype(np.float64), want))


def test_asymmetric_input_and_resolution_sweep(ace):
    """S is symmetrised before use; other resolutions follow the oracle too."""
    rng = np.random.default_rng(12)
    S = planted_similarity(rng, 32, 5, 0.1)
    S = (S + np.float32(0.02) * rng.standard_normal(S.shape).astype(np.float32)).astype(np.float32)
    for gamma in (0.0, 0.5, 0.8, 1.0, 1.5):
        want = C.louvain(C.similarity_graph(S.astype(np.float64)), gamma)
        e2g, _, _ = ace.group_experts(S, ace.GROUP_LOUVAIN, gamma)
        assert np.array_equal(e2g, want), gamma


def test_grouping_degenerate_and_invalid(ace):
    e2g, anchors, G = ace.group_experts(np.eye(5, dtype=np.float32), ace.GROUP_LOUVAIN, 0.8)
    assert list(e2g) == [0, 1, 2, 3, 4] and list(anchors) == [0, 1, 2, 3, 4] and G == 5
    e2g, anchors, G = ace.group_experts(np.ones((1, 1), np.float32), ace.GROUP_LOUVAIN, 0.8)
    assert list(e2g) == [0] and G == 1
    bad = np.ones((3, 3), np.float32)
    bad[0, 1] = np.nan
    with pytest.raises(ace.AceError):
        ace.group_experts(bad, ace.GROUP_LOUVAIN, 0.8)
    with pytest.raises(ace.AceError):
        ace.group_experts(np.ones((3, 3), np.float32), 7, 0.8)
    with pytest.raises(ace.AceError):
        ace.group_experts(np.ones((3, 3), np.float32), ace.GROUP_LOUVAIN, -1.0)
