"""Pins of the oracle's tree-attention inputs (mask, positions, root-to-leaf
paths of the pruned tree).

The paper runs its target model on the tree inside its code base (Sec. 5.1)
and prints no such arrays, so the oracle's definitions are pinned against
independent constructions: the transitive closure of the parent relation by
boolean matrix products, ancestor counts, the set of nodes that are nobody's
parent, and a hand-built tree whose arrays are written out below.
"""
import numpy as np
import pytest

import oracle


def _closure(parent: np.ndarray) -> np.ndarray:
    """reach[i, j] = 1 iff j is i or an ancestor of i (fixpoint of R <- R or R.A)."""
    n = len(parent)
    A = np.zeros((n, n), dtype=np.int64)
    for i, p in enumerate(parent):
        if p >= 0:
            A[i, p] = 1
    R = np.eye(n, dtype=np.int64)
    while True:
        R2 = ((R + R @ A) > 0).astype(np.int64)
        if np.array_equal(R2, R):
            return R.astype(np.uint8)
        R = R2


def _oracle_tree(V, K, m, S, D, N, B=3, seed=7, T=0.8):
    rng = np.random.default_rng(seed)
    cfg = oracle.Config(B=B, V=V, K=K, m=m, S=S, D=D, N=N, eps=1e-6)
    tree = oracle.Tree(cfg)
    Ts = np.full(B, T, np.float32)
    seeds = rng.integers(1, 2**63, size=B, dtype=np.uint64)
    offs = np.zeros(B, np.uint64)
    for d in range(1, D + 1):
        rows = rng.normal(size=(B, cfg.rows_at(d), V)).astype(np.float32) * 2.0
        oracle.expand(cfg, d, rows, Ts, seeds, offs, tree)
    return cfg, oracle.prune(cfg, tree)


CASES = [
    # V, K, m, S, D, N
    (40, 3, 1, 12, 3, 9),
    (64, 4, 2, 20, 4, 25),
    (30, 2, 0, 10, 4, 1),          # budget 1: a single child of the root
    (50, 3, 1, 12, 3, 3 + 1 + 2 * 3 * 4),  # every generated node kept
    (20, 0, 0, 5, 1, 1),           # K = 0
    (200, 6, 1, 40, 5, 60),
]


@pytest.mark.parametrize("V,K,m,S,D,N", CASES)
def test_tree_attention_against_closure_and_paths(V, K, m, S, D, N):
    cfg, pr = _oracle_tree(V, K, m, S, D, N)
    ta = oracle.tree_attention(cfg, pr)
    NP, W = N + 1, D + 1
    for b in range(cfg.B):
        parent = pr.parent[b]
        R = _closure(parent)
        np.testing.assert_array_equal(ta.mask[b], R)
        # depth = number of strict ancestors
        np.testing.assert_array_equal(ta.position[b], R.sum(axis=1) - 1)
        np.testing.assert_array_equal(ta.position[b], pr.depth[b])
        leaves = sorted(set(range(NP)) - set(int(p) for p in parent if p >= 0))
        assert ta.n_leaves[b] == len(leaves)
        for r, leaf in enumerate(leaves):
            row = ta.retrieve[b, r]
            path = [int(x) for x in row if x >= 0]
            assert np.all(row[len(path):] == -1)
            assert path[0] == 0 and path[-1] == leaf and len(path) == pr.depth[b, leaf] + 1
            for k in range(1, len(path)):
                assert parent[path[k]] == path[k - 1]
            # the path is exactly the leaf's mask row
            assert sorted(path) == list(np.nonzero(R[leaf])[0])
        assert np.all(ta.retrieve[b, len(leaves):] == -1)
        assert ta.retrieve.shape == (cfg.B, NP, W)


def test_hand_built_tree():
    """Root 0 with children 1, 2; node 1 with children 3, 4; node 2 with child 5."""
    cfg = oracle.Config(B=1, V=16, K=2, m=1, S=8, D=3, N=5, eps=1e-6)
    pr = oracle.Pruned(cfg)
    pr.parent[0] = [-1, 0, 0, 1, 1, 2]
    pr.depth[0] = [0, 1, 1, 2, 2, 2]
    pr.n_child[0] = [2, 2, 1, 0, 0, 0]
    pr.first_child[0] = [1, 3, 5, -1, -1, -1]
    ta = oracle.tree_attention(cfg, pr)
    want = np.array([[1, 0, 0, 0, 0, 0],
                     [1, 1, 0, 0, 0, 0],
                     [1, 0, 1, 0, 0, 0],
                     [1, 1, 0, 1, 0, 0],
                     [1, 1, 0, 0, 1, 0],
                     [1, 0, 1, 0, 0, 1]], np.uint8)
    np.testing.assert_array_equal(ta.mask[0], want)
    np.testing.assert_array_equal(ta.position[0], [0, 1, 1, 2, 2, 2])
    assert ta.n_leaves[0] == 3
    np.testing.assert_array_equal(ta.retrieve[0, :3], [[0, 1, 3, -1], [0, 1, 4, -1], [0, 2, 5, -1]])
    assert np.all(ta.retrieve[0, 3:] == -1)


def test_inconsistent_depth_is_rejected():
    cfg = oracle.Config(B=1, V=16, K=2, m=1, S=8, D=3, N=2, eps=1e-6)
    pr = oracle.Pruned(cfg)
    pr.parent[0] = [-1, 0, 1]
    pr.depth[0] = [0, 1, 1]  # node 2 sits at depth 2
    pr.n_child[0] = [1, 1, 0]
    with pytest.raises(oracle.OracleError):
        oracle.tree_attention(cfg, pr)
