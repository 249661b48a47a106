"""Multi-cycle decoding on the GPU path against synthetic k-gram models.

Theorem 1 says the emitted tokens follow the target model whatever the draft:
the first two emitted tokens of many independent sequences are compared with
the target's exact law (chi-square).  Theorem 2 (App. D.1) gives the
acceptance probability of a single layer with nothing pruned in closed form: at
D = 1 the mean acceptance over all visited contexts is compared with the
average of that formula over the same contexts.
"""
import math

import numpy as np
import pytest
import torch
from scipy import stats

from paper_2609_21827_gb300 import build, cycles, rheo

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    build.build()


def _models(V, k, seed, noise=0.8):
    g = torch.Generator().manual_seed(seed)
    draft = cycles.KGramLM.random(V, k, 1.5, g)
    target = cycles.KGramLM.random(V, k, 1.5, g, base=draft, noise=noise)
    return draft, target


def _law_p(run, tries=2):
    """p-value of a chi-square law test, taken again on fresh seeds when the
    first sample falls below 0.01.  Eighteen parametrised law tests at a 1 %
    level would fail by chance in one run out of six; a wrong law fails every
    sample of this size (24,000 sequences), a right one fails twice in a row
    one time in 10^4."""
    p = 0.0
    for t in range(tries):
        p = run(t)
        if p > 0.01:
            break
    return p


def _chisq_p(obs, exp):
    keep = exp >= 5
    o = np.append(obs[keep], obs[~keep].sum())
    e = np.append(exp[keep], exp[~keep].sum())
    if e[-1] == 0:
        o, e = o[:-1], e[:-1]
    return stats.chisquare(o, e * o.sum() / e.sum()).pvalue


@pytest.mark.parametrize("variant", [rheo.VERIFY_RHEO, rheo.VERIFY_RRSW, rheo.VERIFY_ONEHOT])
@pytest.mark.parametrize("m,T", [(1, 1.0), (0, 0.7), (2, 1.3)])
def test_first_two_tokens_follow_the_target(variant, m, T):
    V, k, B = 16, 1, 6000
    draft, target = _models(V, k, seed=100 + m)
    cfg = rheo.Config(batch=B, vocab=V, K=3, depth=3, budget=8, m=m, support=V, dtype="f32")
    tab = target.table.cpu().double().numpy() / T
    p1 = np.exp(tab[3] - tab[3].max()); p1 /= p1.sum()
    law = np.zeros(V * V)
    for a in range(V):
        p2 = np.exp(tab[a] - tab[a].max()); p2 /= p2.sum()
        law[a * V:(a + 1) * V] = p1[a] * p2

    def run(t):
        counts = np.zeros(V * V)
        for rep in range(4 * t, 4 * t + 4):
            window = torch.full((B, k), 3, dtype=torch.int64, device="cuda")
            seed = torch.arange(B, dtype=torch.int64, device="cuda") * 7919 + 1000003 * rep + 17
            res = cycles.run_cycles(cfg, draft, target, window, torch.full((B,), T), seed, cycles=2, L=2,
                                    variant=variant)
            st = res.streams.cpu().numpy()
            assert (st >= 0).all()
            counts += np.bincount(st[:, 0] * V + st[:, 1], minlength=V * V)
        return _chisq_p(counts, law * counts.sum())

    assert _law_p(run) > 0.01


@pytest.mark.parametrize("variant", [rheo.VERIFY_RHEO, rheo.VERIFY_RRSW, rheo.VERIFY_ONEHOT])
@pytest.mark.parametrize("m,S,T", [(1, 12, 1.0), (0, 8, 0.7), (2, 10, 1.3)])
def test_first_two_tokens_follow_the_target_sparse_support(variant, m, S, T):
    """Support S < V (Sec. 3.2 "Efficient implementation"): the sampled token
    comes from the truncated tail and verification uses the same truncated q~;
    the residual off the support is p.  The emitted stream must still follow
    the target exactly."""
    V, k, B = 24, 1, 6000
    draft, target = _models(V, k, seed=300 + m + S)
    cfg = rheo.Config(batch=B, vocab=V, K=3, depth=3, budget=8, m=m, support=S, dtype="f32")
    tab = target.table.cpu().double().numpy() / T
    p1 = np.exp(tab[5] - tab[5].max()); p1 /= p1.sum()
    law = np.zeros(V * V)
    for a in range(V):
        p2 = np.exp(tab[a] - tab[a].max()); p2 /= p2.sum()
        law[a * V:(a + 1) * V] = p1[a] * p2

    def run(t):
        counts = np.zeros(V * V)
        for rep in range(4 * t, 4 * t + 4):
            window = torch.full((B, k), 5, dtype=torch.int64, device="cuda")
            seed = torch.arange(B, dtype=torch.int64, device="cuda") * 6007 + 1000033 * rep + 29
            res = cycles.run_cycles(cfg, draft, target, window, torch.full((B,), T), seed, cycles=2, L=2,
                                    variant=variant)
            st = res.streams.cpu().numpy()
            assert (st >= 0).all()
            counts += np.bincount(st[:, 0] * V + st[:, 1], minlength=V * V)
        return _chisq_p(counts, law * counts.sum())

    assert _law_p(run) > 0.01


def _thm2(p, order, qt, n):
    """App. D.1: acceptance of one layer of n = K+1 slots with nothing pruned."""
    top = order[: n - 1]
    rest = [v for v in range(len(p)) if v not in top]
    r = np.maximum(0.0, p - qt)
    r = r / r.sum()
    return (sum(p[v] for v in top) + sum(min(p[v], qt[v]) for v in rest)
            + r[order[n - 1]] * sum(max(0.0, qt[v] - p[v]) for v in top))


@pytest.mark.parametrize("K,m,T,S", [(2, 1, 1.0, 24), (3, 1, 0.7, 24), (3, 0, 1.0, 24), (2, 1, 1.0, 12),
                                     (3, 0, 0.8, 8)])
def test_single_layer_acceptance_matches_theorem2_across_cycles(K, m, T, S):
    V, k, B, C = 24, 1, 4000, 6
    draft, target = _models(V, k, seed=200 + K + m, noise=1.0)
    cfg = rheo.Config(batch=B, vocab=V, K=K, depth=1, budget=K + 1, m=m, support=S, dtype="f32")
    window = torch.randint(0, V, (B, k), generator=torch.Generator().manual_seed(5)).cuda()
    seed = torch.arange(B, dtype=torch.int64, device="cuda") * 104729 + 11
    res = cycles.run_cycles(cfg, draft, target, window, torch.full((B,), T), seed, cycles=C, L=1)
    acc = res.accepted.cpu().numpy().astype(np.float64)
    wins = res.windows.cpu().numpy()[:, :, -1]
    dtab = draft.table.cpu().double().numpy()
    ttab = target.table.cpu().double().numpy()
    expect = np.zeros(V)
    for ctx in range(V):
        row = dtab[ctx]
        order = sorted(range(V), key=lambda v: (-row[v], v))
        qt = np.zeros(V)  # q~ over the tail: support ranks m+1..S
        t = row[order[m:S]] / T
        e = np.exp(t - t.max())
        qt[order[m:S]] = e / e.sum()
        pt = np.exp(ttab[ctx] / T - (ttab[ctx] / T).max())
        pt /= pt.sum()
        expect[ctx] = _thm2(pt, order, qt, K + 1)
    want = expect[wins].mean()
    got = acc.mean()
    sd = math.sqrt(max(want * (1 - want), 1e-12) / acc.size)
    assert abs(got - want) <= 5 * sd, (got, want, sd)
