"""Pins of the oracle's verification variants (RRSw and vanilla one-hot).

App. A compares RheoVerification with recursive rejection sampling without
replacement (RRSw) on the same hybrid pool and with vanilla verification of a
top-K tree; App. D.2 derives RRSw's single-layer acceptance in closed form
(eq. rrsw-acc).  The variants are pinned against:
  * exhaustive enumeration of every tree and sample path (the independent
    fp64 restatement in brute_force.py): all three rules are lossless;
  * the closed form of App. D.2 for RRSw at depth 1, and E_Y[sum of p over the
    pool] for one-hot verification at depth 1;
  * Monte-Carlo runs of the oracle itself against those exact values.
"""
import math

import numpy as np
import pytest
from scipy import stats

import brute_force as bf
import oracle

VARIANTS = {"rrsw": oracle.VERIFY_RRSW, "onehot": oracle.VERIFY_ONEHOT}

LOSSLESS_CASES = [
    # V, K, m, S, D, N, T
    (5, 2, 1, 5, 1, 2, 1.0),
    (6, 3, 0, 6, 1, 3, 0.5),
    (6, 2, 1, 6, 2, 3, 1.0),
    (7, 2, 2, 7, 2, 5, 0.5),
    (8, 2, 0, 5, 2, 4, 1.0),
    (8, 3, 1, 8, 2, 1, 1.0),
    (6, 2, 1, 6, 2, 9, 1.0),
]


@pytest.mark.parametrize("variant", list(VARIANTS))
@pytest.mark.parametrize("V,K,m,S,D,N,T", LOSSLESS_CASES)
def test_variants_are_lossless_by_enumeration(variant, V, K, m, S, D, N, T):
    rng = np.random.default_rng(V * 100 + K * 10 + m + D)
    dr, tg = bf.random_tables(rng, V, D)
    en = bf.Enumerator(V, K, m, S, D, N, T, dr, tg, verify=variant)
    law, _ = en.stream_distribution(D + 1)
    tl = en.target_law(D + 1)
    assert abs(sum(law.values()) - 1.0) < 1e-12
    assert max(abs(law.get(k, 0.0) - tl[k]) for k in tl) < 1e-12


def _single_layer(V, K, m, T, seed):
    rng = np.random.default_rng(seed)
    dr, tg = bf.random_tables(rng, V, 1, spread=1.2)
    p = bf.softmax64(tg[0].astype(np.float64) / T)
    row = dr[0].astype(np.float64)
    order = sorted(range(V), key=lambda v: (-row[v], v))
    qt = np.zeros(V)
    qt[order[m:]] = bf.softmax64(row[order[m:]] / T)
    return dr, tg, p, order, qt


def _rrsw_closed_form(p, order, qt, m, n):
    """App. D.2, eq. rrsw-acc: pool = Top_m leads, Y ~ q~, fills up to n slots."""
    A = sum(p[v] for v in order[:m])
    ptil = p.copy()
    ptil[order[:m]] = 0.0
    ptil /= ptil.sum()
    r = np.maximum(0.0, ptil - qt)
    r /= r.sum()
    top = order[: n - 1]
    rest = [v for v in range(len(p)) if v not in top]
    return (sum(p[v] for v in top) + sum(min(p[v], (1 - A) * qt[v]) for v in rest)
            + (1 - A) * r[order[n - 1]] * sum(max(0.0, qt[v] - ptil[v]) for v in top))


def _onehot_closed_form(p, order, qt, m, K):
    """E over Y ~ q~ of the target mass of the pool {Top_m, Y, K-m fills}."""
    total = 0.0
    for y in order[m:]:
        fills = [v for v in order[m:] if v != y][: K - m]
        total += qt[y] * (sum(p[v] for v in order[:m]) + p[y] + sum(p[v] for v in fills))
    return total


SINGLE = [(8, 2, 1, 1.0), (9, 3, 1, 0.7), (8, 3, 2, 1.0), (7, 2, 0, 1.3), (10, 4, 1, 0.8)]


@pytest.mark.parametrize("V,K,m,T", SINGLE)
def test_single_layer_closed_forms(V, K, m, T):
    dr, tg, p, order, qt = _single_layer(V, K, m, T, seed=V * 11 + K)
    en = bf.Enumerator(V, K, m, V, 1, K + 1, T, dr, tg, verify="rrsw")
    _, acc = en.stream_distribution(1)
    assert abs(acc[1] - _rrsw_closed_form(p, order, qt, m, K + 1)) < 1e-12
    en = bf.Enumerator(V, K, m, V, 1, K + 1, T, dr, tg, verify="onehot")
    _, acc = en.stream_distribution(1)
    assert abs(acc[1] - _onehot_closed_form(p, order, qt, m, K)) < 1e-12


@pytest.mark.parametrize("variant", list(VARIANTS))
@pytest.mark.parametrize("V,K,m,T", SINGLE[:3])
def test_oracle_single_layer_acceptance(variant, V, K, m, T):
    dr, tg, p, order, qt = _single_layer(V, K, m, T, seed=V * 11 + K)
    en = bf.Enumerator(V, K, m, V, 1, K + 1, T, dr, tg, verify=variant)
    _, acc = en.stream_distribution(1)
    want = acc[1]
    cfg = oracle.Config(B=1, V=V, K=K, m=m, D=1, N=K + 1, verify_mode=VARIANTS[variant])
    n = 200000
    _, a = oracle.run_prefix_lm(cfg, dr, tg, 1, n, T, 4242, 1)
    assert abs(a.mean() - want) <= 5 * math.sqrt(want * (1 - want) / n) + 1e-12


def _chisq_p(obs, exp):
    keep = exp >= 5
    o = np.append(obs[keep], obs[~keep].sum())
    e = np.append(exp[keep], exp[~keep].sum())
    if e[-1] == 0:
        o, e = o[:-1], e[:-1]
    return stats.chisquare(o, e * o.sum() / e.sum()).pvalue


@pytest.mark.parametrize("variant", list(VARIANTS))
def test_oracle_variants_monte_carlo_vocab16(variant):
    V, K, m, D, N, T, n = 16, 2, 1, 2, 4, 1.0, 300_000
    rng = np.random.default_rng(1616)
    dr, tg = bf.random_tables(rng, V, D)
    cfg = oracle.Config(B=1, V=V, K=K, m=m, D=D, N=N, verify_mode=VARIANTS[variant])
    st, acc = oracle.run_prefix_lm(cfg, dr, tg, D, n, T, 777, 2)
    en = bf.Enumerator(V, K, m, V, D, N, T, dr, tg, verify=variant)
    tl = en.target_law(2)
    p2 = np.zeros(V * V)
    for (a, b), pr in tl.items():
        p2[a * V + b] += pr
    assert _chisq_p(np.bincount(st[:, 0] * V + st[:, 1], minlength=V * V), p2 * n) > 0.01
    _, accl = en.stream_distribution(2)
    ea = np.array([accl.get(i, 0.0) for i in range(D + 1)])
    assert _chisq_p(np.bincount(acc, minlength=D + 1), ea * n) > 0.01
