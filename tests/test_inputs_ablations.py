"""Structural-ablation pattern recipes (Sec. 4.5 ablation study, App. B): each
keeps what the paper says it keeps and removes what it removes, at matched
physical retention. CPU only."""
import numpy as np
import pytest

from paper_2609_32663_gb300 import inputs as I

WL = I.WORKLOADS["llama8b-128k"]
G, Hkv, D = WL.G, WL.Hkv, WL.D


def union_by_group(M):
    L, H, _ = M.shape
    return M.reshape(L, H // G, G, D).max(axis=2)  # [l][g][d]


@pytest.fixture(scope="module")
def base():
    return I.make_pattern(WL)


def ablated(kind):
    return I.make_pattern(I.WORKLOADS["llama8b-128k-" + kind.replace("_", "-")])


@pytest.mark.parametrize("kind", I.ABLATIONS)
def test_binary_shape_and_deterministic(kind, base):
    M = ablated(kind)
    assert M.shape == base.shape and M.dtype == np.uint8 and set(np.unique(M)) <= {0, 1}
    assert np.array_equal(M, ablated(kind))
    assert not np.array_equal(M, base)


def test_distance_shuffled_keeps_head_counts_and_group_unions(base):
    M = ablated("distance_shuffled")
    assert np.array_equal(M.sum(axis=2), base.sum(axis=2))  # per query head
    assert np.array_equal(union_by_group(M).sum(axis=2), union_by_group(base).sum(axis=2))  # per KV head
    # the same permutation for all heads of a group: the group's columns are a permutation of the base's
    L, H, _ = M.shape
    for l in range(0, L, 7):
        for g in range(H // G):
            cols = lambda X: sorted(map(tuple, X[l, g * G:(g + 1) * G].T.tolist()))
            assert cols(M) == cols(base)


def test_fully_shuffled_keeps_totals_only(base):
    M = ablated("fully_shuffled")
    assert M.sum() == base.sum()
    assert union_by_group(M).sum() == union_by_group(base).sum()
    # columns keep their number of heads on (a permutation of columns, heads permuted within)
    col_sums = lambda X: np.sort(X.reshape(X.shape[0], -1, G, D).sum(axis=2).reshape(-1))
    assert np.array_equal(col_sums(M), col_sums(base))
    assert not np.array_equal(M.sum(axis=2), base.sum(axis=2))  # per-head counts are not kept


def test_head_only_decides_whole_heads_at_matched_physical(base):
    M = ablated("head_only")
    rows = M.sum(axis=2)
    assert set(np.unique(rows)) <= {0, D}  # every head keeps all of its bins or none
    target = int(union_by_group(base).sum())
    assert abs(int(union_by_group(M).sum()) - target) <= D // 2


def test_distance_only_shares_decisions_across_heads_at_matched_physical(base):
    M = ablated("distance_only")
    assert (M == M[:, :1, :]).all()  # one decision per (layer, bin)
    target = int(union_by_group(base).sum())
    assert abs(int(union_by_group(M).sum()) - target) <= Hkv // 2


def test_recipes_on_a_small_pattern_by_hand():
    rng = np.random.default_rng(0)
    M = (rng.random((2, 4, 6)) < 0.4).astype(np.uint8)  # L=2, H=4, G=2, D=6
    U = int(M.reshape(2, 2, 2, 6).max(axis=2).sum())
    ho = I.ablate_head_only(M, 2)
    assert int(ho.reshape(2, 2, 2, 6).max(axis=2).sum()) == 6 * int(np.floor(U / 6 + 0.5))
    do = I.ablate_distance_only(M, 2)
    assert int(do.reshape(2, 2, 2, 6).max(axis=2).sum()) == 2 * int(np.floor(U / 2 + 0.5))
