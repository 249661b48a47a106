"""Pins of the oracle's full-support mode (S = V; App. B, Table tab:sparse_support,
row Full): the sampled token is drawn from the tempered draft distribution over
the whole vocabulary minus the leads, with draw index = token id.

Pinned against scipy's softmax, the law of Y (chi-square over seeds), and the
exhaustive enumeration of brute_force.py, whose law of trees with S = V does
not depend on how the uniforms are indexed: the acceptance and the emitted
two-token law of the oracle's Monte-Carlo runs must match it.
"""
import math

import numpy as np
import pytest
from scipy import special, stats

import brute_force as bf
import oracle


def _chisq_p(obs, exp):
    keep = exp >= 5
    o = np.append(obs[keep], obs[~keep].sum())
    e = np.append(exp[keep], exp[~keep].sum())
    if e[-1] == 0:
        o, e = o[:-1], e[:-1]
    return stats.chisquare(o, e * o.sum() / e.sum()).pvalue


def test_tail_distribution_and_lse_against_scipy():
    rng = np.random.default_rng(3)
    V, K, m, B, T = 300, 4, 2, 3, 0.8
    cfg = oracle.Config(B=B, V=V, K=K, m=m, S=0, D=1, N=K + 1)
    tree = oracle.Tree(cfg)
    rows = (rng.normal(size=(B, 1, V)) * 2).astype(np.float32)
    oracle.expand(cfg, 1, rows, np.full(B, T, np.float32), rng.integers(1, 2**62, size=B, dtype=np.uint64),
                  np.zeros(B, np.uint64), tree)
    for b in range(B):
        l = rows[b, 0].astype(np.float64)
        order = np.lexsort((np.arange(V), -rows[b, 0]))
        tail = order[m:]
        np.testing.assert_array_equal(tree.tail_ids[b, 0], tail)
        tau = (rows[b, 0][tail] / np.float32(T)).astype(np.float64)
        np.testing.assert_allclose(tree.tail_q[b, 0], special.softmax(tau), rtol=2e-6, atol=1e-12)
        assert abs(tree.lse_tail[b, 0] - special.logsumexp(tau)) < 2e-6
        assert abs(tree.lse1[b, 0] - special.logsumexp(l)) < 2e-6


def test_sampled_token_law():
    V, K, m, T, n = 16, 2, 1, 0.9, 40000
    rng = np.random.default_rng(9)
    row = (rng.normal(size=V) * 1.5).astype(np.float32)
    cfg = oracle.Config(B=n, V=V, K=K, m=m, S=0, D=1, N=K + 1)
    tree = oracle.Tree(cfg)
    rows = np.broadcast_to(row, (n, 1, V)).copy()
    seeds = np.arange(1, n + 1, dtype=np.uint64) * np.uint64(2654435761)
    oracle.expand(cfg, 1, rows, np.full(n, T, np.float32), seeds, np.zeros(n, np.uint64), tree)
    ys = tree.token[:, 1 + m]  # slot m of the root's children (gen ids 1..K+1)
    order = np.lexsort((np.arange(V), -row))
    q = np.zeros(V)
    q[order[m:]] = special.softmax((row[order[m:]] / np.float32(T)).astype(np.float64))
    assert _chisq_p(np.bincount(ys, minlength=V), q * n) > 0.01


@pytest.mark.parametrize("K,m,T,D,N", [(2, 1, 1.0, 1, 3), (3, 0, 0.7, 2, 6), (2, 2, 1.2, 2, 5)])
def test_monte_carlo_against_enumeration(K, m, T, D, N):
    V, n = 12, 200000
    rng = np.random.default_rng(40 + K + m)
    dr, tg = bf.random_tables(rng, V, D)
    cfg = oracle.Config(B=1, V=V, K=K, m=m, S=0, D=D, N=N)
    st, acc = oracle.run_prefix_lm(cfg, dr, tg, D, n, T, 31337, 2)
    en = bf.Enumerator(V, K, m, V, D, N, T, dr, tg)
    _, accl = en.stream_distribution(2)
    ea = np.array([accl.get(i, 0.0) for i in range(D + 1)])
    assert _chisq_p(np.bincount(acc, minlength=D + 1), ea * n) > 0.01
    tl = en.target_law(2)
    p2 = np.zeros(V * V)
    for (a, b), pr in tl.items():
        p2[a * V + b] += pr
    assert _chisq_p(np.bincount(st[:, 0] * V + st[:, 1], minlength=V * V), p2 * n) > 0.01


def _two_stage_draws(V, m, T, n, row, plant=0):
    cfg = oracle.Config(B=n, V=V, K=2, m=m, S=0, D=1, N=3, plant_mode=plant)
    tree = oracle.Tree(cfg)
    rows = np.broadcast_to(row, (n, 1, V)).copy()
    seeds = np.arange(1, n + 1, dtype=np.uint64) * np.uint64(0x9E3779B97F4A7C15 % (2**61))
    oracle.expand(cfg, 1, rows, np.full(n, T, np.float32), seeds, np.zeros(n, np.uint64), tree)
    return tree.token[:, 1 + m]


def _tail_law(row, m, T):
    V = row.size
    order = np.lexsort((np.arange(V), -row))
    q = np.zeros(V)
    q[order[m:]] = special.softmax((row[order[m:]] / np.float32(T)).astype(np.float64))
    return q


@pytest.mark.parametrize("m,T", [(1, 0.8), (0, 1.3)])
def test_two_stage_draw_law_across_blocks(m, T):
    """V = 700 spans three blocks of 256 token ids (the last one partial): the
    block of Y follows the blocks' tail masses and Y the tail law q~."""
    V, n = 700, 60000
    rng = np.random.default_rng(71 + m)
    row = (rng.normal(size=V) * 1.2).astype(np.float32)
    row[300:330] += 2.0  # a heavier stretch inside the second block
    ys = _two_stage_draws(V, m, T, n, row)
    q = _tail_law(row, m, T)
    blocks = np.array([q[0:256].sum(), q[256:512].sum(), q[512:].sum()])
    assert _chisq_p(np.bincount(ys // 256, minlength=3), blocks * n) > 0.01
    assert _chisq_p(np.bincount(ys, minlength=V), q * n) > 0.01


def test_two_stage_draw_detects_unweighted_blocks():
    """A planted mistake (blocks chosen without their mass) fails the same law
    test: the pin has teeth."""
    V, n = 700, 60000
    rng = np.random.default_rng(72)
    row = (rng.normal(size=V) * 1.2).astype(np.float32)
    row[300:330] += 2.0
    q = _tail_law(row, 1, 0.8)
    blocks = np.array([q[0:256].sum(), q[256:512].sum(), q[512:].sum()])
    ys = _two_stage_draws(V, 1, 0.8, n, row, plant=oracle.PLANT_BLOCK_UNWEIGHTED)
    assert _chisq_p(np.bincount(ys // 256, minlength=3), blocks * n) < 1e-6


@pytest.mark.parametrize("V", [256, 257, 512])
def test_two_stage_draw_block_edges(V):
    """V a multiple of the block (256, 512) and one past it (257: the last
    block holds a single token, here given the row's largest logit after the
    lead so that its block carries real mass)."""
    n = 40000
    rng = np.random.default_rng(300 + V)
    row = (rng.normal(size=V) * 1.0).astype(np.float32)
    row[0] = row.max() + 1.0      # the lead (m = 1)
    row[V - 1] = row[0] - 0.5     # the last token, alone in its block when V = 257
    ys = _two_stage_draws(V, 1, 1.0, n, row)
    q = _tail_law(row, 1, 1.0)
    assert np.all(ys != 0)  # the lead is never the sampled token
    assert _chisq_p(np.bincount(ys, minlength=V), q * n) > 0.01
    nb = (V + 255) // 256
    if nb == 1:
        assert np.all(ys < 256)
    else:
        blocks = np.array([q[256 * k:256 * (k + 1)].sum() for k in range(nb)])
        assert _chisq_p(np.bincount(ys // 256, minlength=nb), blocks * n) > 0.01
