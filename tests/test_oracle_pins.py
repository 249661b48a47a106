"""Pins of the CPU oracle against what the paper and the mathematics fix.

Each test checks the oracle against something other than itself: a library
routine (cuRAND's Philox stream, numpy sorting, scipy log-sum-exp), the worked
example of Table tab:proxy, Lemma 1 / Lemma 2, exhaustive enumeration of
Theorem 1, the closed form of Theorem 2, textbook special cases, and
Monte-Carlo chi-square tests of the emitted-token law.
"""
import ctypes
import ctypes.util
import json
import math
import os

import numpy as np
import pytest
from scipy import special, stats

import brute_force as bf

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# --------------------------------------------------------------------------
# Philox4x32-10 and the uniform conversion
# --------------------------------------------------------------------------

def _curand():
    for name in ("/usr/local/cuda/lib64/libcurand.so", ctypes.util.find_library("curand")):
        if name and os.path.exists(name) if name.startswith("/") else name:
            try:
                return ctypes.CDLL(name)
            except OSError:
                continue
    return None


def _curand_host_philox(lib, seed, offset, n):
    gen = ctypes.c_void_p()
    assert lib.curandCreateGeneratorHost(ctypes.byref(gen), 161) == 0  # PHILOX4_32_10
    assert lib.curandSetPseudoRandomGeneratorSeed(gen, ctypes.c_ulonglong(seed)) == 0
    assert lib.curandSetGeneratorOffset(gen, ctypes.c_ulonglong(offset)) == 0
    out = (ctypes.c_uint32 * n)()
    assert lib.curandGenerate(gen, out, ctypes.c_size_t(n)) == 0
    lib.curandDestroyGenerator(gen)
    return np.array(out, dtype=np.uint32)


@pytest.mark.parametrize("seed", [0, 1, 0x0123456789ABCDEF, 0xFFFFFFFFFFFFFFFF])
def test_philox_matches_curand_host_generator(orc, seed):
    """Philox4x32-10 (Salmon et al., SC'11) against cuRAND's host generator.

    cuRAND's host PHILOX4_32_10 stream places output block b at counter
    (lo32(b >> 16), lo32(b >> 48), b & 0xffff, 0) under key (lo32, hi32) of the
    seed; offsets reach every counter word the oracle's layout uses.
    """
    lib = _curand()
    if lib is None:
        pytest.skip("libcurand not available")
    key = [seed & 0xFFFFFFFF, seed >> 32]
    for offset in (0, 4 * 77, 4 * ((5 << 16) + 9), 4 * ((3 << 48) + (11 << 16) + 2)):
        got = _curand_host_philox(lib, seed, offset, 64)
        for blk in range(16):
            b = offset // 4 + blk
            ctr = [(b >> 16) & 0xFFFFFFFF, (b >> 48) & 0xFFFFFFFF, b & 0xFFFF, 0]
            np.testing.assert_array_equal(orc.philox(ctr, key), got[4 * blk: 4 * blk + 4])


def test_uniform_conversion_and_counter_layout(orc):
    """u = ((w >> 9) + 0.5) 2^-23 from word draw&3 of counter
    (draw>>2, lo32 offset, 4 node + tag, hi32 offset): exact, inside (0, 1)."""
    rng = np.random.default_rng(3)
    for _ in range(200):
        seed = int(rng.integers(0, 2**63))
        offset = int(rng.integers(0, 2**40))
        tag = int(rng.integers(0, 4))
        node = int(rng.integers(0, 16384))
        draw = int(rng.integers(0, 200000))
        ctr = [draw >> 2, offset & 0xFFFFFFFF, 4 * node + tag, offset >> 32]
        w = int(orc.philox(ctr, [seed & 0xFFFFFFFF, seed >> 32])[draw & 3])
        want = ((w >> 9) + 0.5) / 2**23
        u = orc.uniform(seed, offset, tag, node, draw)
        assert u == want and 0.0 < u < 1.0
        assert np.float32(u) == u  # exactly representable
    assert (0 + 0.5) / 2**23 == 2.0**-24 and ((2**23 - 1) + 0.5) / 2**23 == 1 - 2.0**-24


def test_uniforms_are_uniform(orc):
    us = np.array([orc.uniform(5, 9, 3, 17, v) for v in range(20000)])
    assert stats.kstest(us, "uniform").pvalue > 0.01


# --------------------------------------------------------------------------
# sparse support, log-partition, tempered tail
# --------------------------------------------------------------------------

@pytest.mark.parametrize("V,S", [(7, 7), (50, 5), (1000, 128), (4096, 128)])
def test_topk_matches_lexsort_with_ties(orc, V, S):
    rng = np.random.default_rng(V)
    for kind in ("normal", "integer", "bf16"):
        if kind == "normal":
            row = rng.normal(size=V).astype(np.float32)
        elif kind == "integer":
            row = rng.integers(-3, 3, size=V).astype(np.float32)  # massive ties
        else:
            x = rng.normal(size=V).astype(np.float32)
            row = (x.view(np.uint32) & 0xFFFF0000).view(np.float32)  # bf16-truncated values
        ids = np.arange(V)
        want = np.lexsort((ids, -row.astype(np.float64)))[:S]
        np.testing.assert_array_equal(orc.topk_row(row, S), want)


def test_expand_support_lse_and_tail_against_scipy(orc):
    """Sec. 3.2 sparse draft: support = top-S logits; tail q~ = softmax(l/T)
    over ranks m+1..S; construction probabilities use the full-vocabulary,
    untempered softmax (Sec. 5.4)."""
    rng = np.random.default_rng(11)
    for (V, K, m, T) in [(300, 4, 1, 0.7), (300, 6, 0, 1.0), (129, 3, 2, 1.3)]:
        cfg = orc.Config(B=3, V=V, K=K, m=m, D=1, N=K + 1)
        rows = rng.normal(0, 2, size=(3, 1, V)).astype(np.float32)
        tree = orc.Tree(cfg)
        orc.expand(cfg, 1, rows, T, [1, 2, 3], [0, 0, 0], tree)
        for b in range(3):
            l = rows[b, 0].astype(np.float64)
            lse = special.logsumexp(l)
            assert abs(tree.lse1[b, 0] - lse) <= 2e-6 * max(1, abs(lse))
            order = np.lexsort((np.arange(V), -l))[: cfg.S]
            np.testing.assert_array_equal(tree.tail_ids[b, 0], order[m:])
            qt = special.softmax(l[order[m:]] / T)
            np.testing.assert_allclose(tree.tail_q[b, 0], qt, rtol=1e-6, atol=1e-9)
            kids = range(1, K + 2)
            for j, g in enumerate(kids):
                if tree.slot[b, g] != orc.SLOT_SAMPLED:
                    tok = tree.token[b, g]
                    assert abs(tree.log_proxy[b, g] - (l[tok] - lse)) < 5e-6 * max(1, abs(l[tok] - lse))
            # leads are the top-m ranks, in order
            np.testing.assert_array_equal(tree.token[b, 1:1 + m], order[:m])


# --------------------------------------------------------------------------
# the worked example of Table tab:proxy
# --------------------------------------------------------------------------

def _worked_example_run(orc, proxy_mode, fixed, seeds):
    g = json.load(open(os.path.join(GOLDEN, "worked_example_proxy.json")))
    q = np.array(g["draft_q"])
    cfg = orc.Config(B=len(seeds), V=3, K=g["deterministic_slots_K"], m=g["m"], D=1,
                     N=g["prune_budget_R"], proxy_mode=proxy_mode, fixed_log_proxy=fixed)
    rows = np.tile(np.log(q).astype(np.float32), (len(seeds), 1, 1))
    tree = orc.Tree(cfg)
    orc.expand(cfg, 1, rows, 1.0, seeds, 0, tree)
    pr = orc.prune(cfg, tree)
    return g, tree, pr


def test_worked_example_rheo_proxy(orc):
    names = ["A", "B", "C"]
    seeds = list(range(4000))
    g, tree, pr = _worked_example_run(orc, 0, 0.0, seeds)
    ys = []
    for b in range(len(seeds)):
        y = names[tree.token[b, 2]]
        assert tree.slot[b, 2] == orc.SLOT_SAMPLED and tree.token[b, 1] == 0
        assert math.isclose(math.exp(tree.log_proxy[b, 2]), g["rheo_proxy"], rel_tol=1e-6)
        assert math.isclose(tree.qtilde[b, 2], g["qtilde"][y], rel_tol=1e-6)
        assert names[tree.token[b, 3]] == g["rheo_fill"][f"Y={y}"]
        kept = [int(x) for x in pr.gen_id[b, 1:]]
        surv = ["Y" if tree.slot[b, k] == orc.SLOT_SAMPLED else names[tree.token[b, k]] for k in kept]
        assert surv == g["rheo_survivors"][f"Y={y}"]
        ys.append(y)
    frac_b = ys.count("B") / len(ys)
    assert abs(frac_b - g["qtilde"]["B"]) < 4 * math.sqrt(0.24 / len(ys))


def test_worked_example_adhoc_proxy_drops_sampled_slot(orc):
    names = ["A", "B", "C"]
    seeds = list(range(2000))
    g, tree, pr = _worked_example_run(orc, 1, math.log(0.25), seeds)
    for b in range(len(seeds)):
        y = names[tree.token[b, 2]]
        kept = [int(x) for x in pr.gen_id[b, 1:]]
        surv = ["Y" if tree.slot[b, k] == orc.SLOT_SAMPLED else names[tree.token[b, k]] for k in kept]
        assert surv == g["adhoc_survivors"][f"Y={y}"]


# --------------------------------------------------------------------------
# Lemma 1 (local rank), Lemma 2 (ancestor monotonicity), closure
# --------------------------------------------------------------------------

@pytest.mark.parametrize("m", [0, 1, 2, 3])
def test_lemma1_lemma2_and_closure(orc, m):
    rng = np.random.default_rng(100 + m)
    V, K, D = 200, 5, 4
    cfg = orc.Config(B=6, V=V, K=K, m=m, D=D, N=20)
    rows = [rng.normal(0, 1 + 2 * rng.random(), size=(6, cfg.rows_at(d), V)).astype(np.float32)
            for d in range(1, D + 1)]
    tree = orc.Tree(cfg)
    for d in range(1, D + 1):
        orc.expand(cfg, d, rows[d - 1], 0.9, np.arange(6) + 40, 3, tree)
    pr = orc.prune(cfg, tree)  # raises if not ancestor-closed
    for b in range(6):
        for g in range(1, cfg.G1):
            par = tree.parent[b, g]
            assert tree.score[b, g] <= tree.score[b, par]            # Lemma 2
            assert tree.log_proxy[b, g] <= 0.0
        for first in range(1, cfg.G1, K + 1):
            pool = list(range(first, first + K + 1))
            ys = [g for g in pool if tree.slot[b, g] == orc.SLOT_SAMPLED]
            assert len(ys) == 1 and ys[0] == first + m                # slot m+1 (1-based)
            for g in pool[m + 1:]:
                assert tree.log_proxy[b, g] <= tree.log_proxy[b, ys[0]]  # Lemma 1
        for i in range(1, cfg.N + 1):
            assert pr.parent[b, i] < i


# --------------------------------------------------------------------------
# Theorem 1 by exhaustive enumeration; negative control
# --------------------------------------------------------------------------

ENUM_CASES = [
    # V, K, m, S, D, N, T
    (5, 2, 1, 5, 1, 2, 1.0),
    (6, 3, 0, 6, 1, 3, 0.5),
    (6, 2, 1, 6, 2, 3, 1.0),
    (7, 2, 2, 7, 2, 5, 0.5),
    (8, 2, 0, 5, 2, 4, 1.0),    # sparse support S < V
    (8, 2, 1, 5, 2, 6, 0.5),
    (8, 3, 1, 8, 2, 1, 1.0),
    (6, 2, 1, 6, 2, 9, 1.0),    # N = G: nothing pruned
]


@pytest.mark.parametrize("V,K,m,S,D,N,T", ENUM_CASES)
def test_theorem1_exact_enumeration(V, K, m, S, D, N, T):
    rng = np.random.default_rng(V * 100 + K * 10 + m + D)
    dr, tg = bf.random_tables(rng, V, D)
    en = bf.Enumerator(V, K, m, S, D, N, T, dr, tg)
    law, _ = en.stream_distribution(D + 1)
    tl = en.target_law(D + 1)
    err = max(abs(law.get(k, 0.0) - tl[k]) for k in tl)
    assert abs(sum(law.values()) - 1.0) < 1e-12
    assert err < 1e-12, err


def test_theorem1_every_budget():
    rng = np.random.default_rng(5)
    V, K, m, D = 6, 2, 1, 2
    dr, tg = bf.random_tables(rng, V, D)
    G = (K + 1) + (D - 1) * K * (K + 1)
    for N in range(1, G + 1):
        en = bf.Enumerator(V, K, m, V, D, N, 1.0, dr, tg)
        law, _ = en.stream_distribution(D + 1)
        tl = en.target_law(D + 1)
        assert max(abs(law.get(k, 0.0) - tl[k]) for k in tl) < 1e-12, N


def test_negative_control_adhoc_proxy_breaks_losslessness():
    """Sec. 4: a proxy below q(x_{m+1}) makes survival depend on Y."""
    q = np.log(np.array([0.5, 0.3, 0.2], dtype=np.float32))
    p = np.log(np.array([0.2, 0.2, 0.6], dtype=np.float32))
    V, D = 3, 1
    dr = np.tile(q, (bf.table_rows(V, D + 1), 1))
    tg = np.tile(p, (bf.table_rows(V, D + 1), 1))
    good = bf.Enumerator(V, 2, 1, 3, D, 2, 1.0, dr, tg)
    bad = bf.Enumerator(V, 2, 1, 3, D, 2, 1.0, dr, tg, proxy=0.25)
    tl = good.target_law(1)
    lg, _ = good.stream_distribution(1)
    lb, _ = bad.stream_distribution(1)
    assert max(abs(lg[k] - tl[k]) for k in tl) < 1e-12
    assert max(abs(lb[k] - tl[k]) for k in tl) > 1e-2


# --------------------------------------------------------------------------
# oracle trees against the enumerator, under the oracle's own draws
# --------------------------------------------------------------------------

@pytest.mark.parametrize("V,K,m,S,D,N,T", [(12, 3, 1, 12, 3, 7, 0.8), (16, 2, 0, 10, 3, 6, 1.0),
                                           (10, 4, 2, 9, 2, 9, 1.2)])
def test_oracle_tree_matches_enumerator(orc, V, K, m, S, D, N, T):
    rng = np.random.default_rng(V + K + m)
    dr, tg = bf.random_tables(rng, V, D)
    en = bf.Enumerator(V, K, m, S, D, N, T, dr, tg)
    cfg = orc.Config(B=1, V=V, K=K, m=m, S=S, D=D, N=N)
    for seed in range(60):
        tree = orc.Tree(cfg)
        for d in range(1, D + 1):
            F = cfg.rows_at(d)
            parents = [0] if d == 1 else list(tree.frontier[0, :K])
            rows = np.stack([dr[bf.prefix_row(_path(tree, g), V)] for g in parents])[None]
            orc.expand(cfg, d, rows, T, seed, 0, tree)
        ys = {int(tree.parent[0, g]): int(tree.token[0, g])
              for g in range(1, cfg.G1) if tree.slot[0, g] == orc.SLOT_SAMPLED}
        nodes = en.tree_for(ys)
        assert sorted(nodes) == list(range(cfg.G1))
        for g in range(1, cfg.G1):
            n = nodes[g]
            assert (n.token, n.parent) == (tree.token[0, g], tree.parent[0, g]), (seed, g)
            assert abs(n.score - tree.score[0, g]) < 1e-5 * max(1.0, abs(n.score))
        pr = orc.prune(cfg, tree)
        assert set(pr.gen_id[0].tolist()) == en.prune(nodes)


def _path(tree, g):
    out = []
    while g != 0:
        out.append(int(tree.token[0, g]))
        g = int(tree.parent[0, g])
    return tuple(reversed(out))


# --------------------------------------------------------------------------
# Theorem 2 and textbook special cases (single layer)
# --------------------------------------------------------------------------

def _single_layer(V, K, m, N, T, seed, S=None):
    rng = np.random.default_rng(seed)
    dr, tg = bf.random_tables(rng, V, 1, spread=1.2)
    S = V if S is None else S
    en = bf.Enumerator(V, K, m, S, 1, N, T, dr, tg)
    p = bf.softmax64(tg[0].astype(np.float64) / T)
    row = dr[0].astype(np.float64)
    order = sorted(range(V), key=lambda v: (-row[v], v))
    qt = np.zeros(V)
    qt[order[m:S]] = bf.softmax64(row[order[m:S]] / T)
    return dr, tg, en, p, order, qt


def _thm2(p, order, qt, n):
    top_nm1 = order[: n - 1]
    rest = [v for v in range(len(p)) if v not in top_nm1]
    r = np.maximum(0.0, p - qt)
    r = r / r.sum()
    return (sum(p[v] for v in top_nm1) + sum(min(p[v], qt[v]) for v in rest)
            + r[order[n - 1]] * sum(max(0.0, qt[v] - p[v]) for v in top_nm1))


@pytest.mark.parametrize("V,K,m,T,S", [(8, 2, 1, 1.0, 8), (9, 3, 1, 0.7, 9), (8, 3, 2, 1.0, 8), (7, 2, 0, 1.3, 7),
                                       (8, 2, 1, 1.0, 5), (10, 2, 1, 0.8, 4), (7, 2, 0, 1.3, 4)])
def test_theorem2_single_layer_acceptance(orc, V, K, m, T, S):
    """App. D.1 closed form (q~ truncated to the support when S < V) against
    the enumerator and 2*10^5 oracle cycles."""
    dr, tg, en, p, order, qt = _single_layer(V, K, m, K + 1, T, seed=V * 7 + K, S=S)
    want = _thm2(p, order, qt, K + 1)
    _, acc = en.stream_distribution(1)
    assert abs(acc[1] - want) < 1e-12
    upper = sum(p[v] for v in order[: K + 1]) + sum(min(p[v], qt[v]) for v in order[K + 1:])
    assert want <= upper + 1e-15
    cfg = orc.Config(B=1, V=V, K=K, m=m, S=S, D=1, N=K + 1)
    n = 200000
    _, a = orc.run_prefix_lm(cfg, dr, tg, 1, n, T, 999, 1)
    assert abs(a.mean() - want) <= 5 * math.sqrt(want * (1 - want) / n) + 1e-12


def test_special_case_single_sampled_slot_is_speculative_sampling(orc):
    """m = 0 and a pool of one sampled token: acceptance sum_x min(p, q) (Sec. 2.2)."""
    V, T = 10, 1.0
    dr, tg, en, p, order, qt = _single_layer(V, 0, 0, 1, T, seed=21)
    want = float(np.minimum(p, qt).sum())
    _, acc = en.stream_distribution(1)
    assert abs(acc[1] - want) < 1e-12
    cfg = orc.Config(B=1, V=V, K=0, m=0, D=1, N=1)
    n = 200000
    st, a = orc.run_prefix_lm(cfg, dr, tg, 1, n, T, 5, 1)
    assert abs(a.mean() - want) <= 5 * math.sqrt(want * (1 - want) / n) + 1e-12
    freq = np.bincount(st[:, 0], minlength=V)
    assert stats.chisquare(freq, p * n).pvalue > 0.01


def test_special_case_sampled_slot_pruned_is_topk(orc):
    """s = -1 (only the m leads survive): acceptance = sum over Top_m of p (Theorem 2)."""
    V, K, m, T = 9, 3, 2, 1.0
    dr, tg, en, p, order, qt = _single_layer(V, K, m, m, T, seed=33)
    want = sum(p[v] for v in order[:m])
    _, acc = en.stream_distribution(1)
    assert abs(acc[1] - want) < 1e-12
    cfg = orc.Config(B=1, V=V, K=K, m=m, D=1, N=m)
    n = 200000
    _, a = orc.run_prefix_lm(cfg, dr, tg, 1, n, T, 77, 1)
    assert abs(a.mean() - want) <= 5 * math.sqrt(want * (1 - want) / n) + 1e-12


# --------------------------------------------------------------------------
# Monte-Carlo losslessness at vocab 16 (10^6 cycles)
# --------------------------------------------------------------------------

def _chisq_p(obs, exp):
    keep = exp >= 5
    o = np.append(obs[keep], obs[~keep].sum())
    e = np.append(exp[keep], exp[~keep].sum())
    if e[-1] == 0:
        o, e = o[:-1], e[:-1]
    return stats.chisquare(o, e * o.sum() / e.sum()).pvalue


@pytest.mark.parametrize("K,m,N,T", [(2, 1, 4, 1.0), (3, 0, 7, 0.7)])
def test_monte_carlo_losslessness_vocab16(orc, K, m, N, T):
    V, D, n = 16, 2, 1_000_000
    rng = np.random.default_rng(1600 + K)
    dr, tg = bf.random_tables(rng, V, D)
    cfg = orc.Config(B=1, V=V, K=K, m=m, D=D, N=N)
    st, acc = orc.run_prefix_lm(cfg, dr, tg, D, n, T, 12345, 2)
    en = bf.Enumerator(V, K, m, V, D, N, T, dr, tg)
    tl = en.target_law(2)
    p1 = np.zeros(V)
    p2 = np.zeros(V * V)
    for (a, b), pr in tl.items():
        p1[a] += pr
        p2[a * V + b] += pr
    f1 = np.bincount(st[:, 0], minlength=V)
    f2 = np.bincount(st[:, 0] * V + st[:, 1], minlength=V * V)
    assert _chisq_p(f1, p1 * n) > 0.01
    assert _chisq_p(f2, p2 * n) > 0.01
    _, accl = en.stream_distribution(2)
    ea = np.array([accl.get(i, 0.0) for i in range(D + 1)])
    fa = np.bincount(acc, minlength=D + 1)
    assert _chisq_p(fa, ea * n) > 0.01


def test_monte_carlo_detects_planted_proxy_mistake(orc):
    """The same chi-square test rejects the oracle run with the ad hoc proxy
    (a planted mistake): the pins have teeth."""
    q = np.log(np.array([0.5, 0.3, 0.2], dtype=np.float32))
    p = np.log(np.array([0.2, 0.2, 0.6], dtype=np.float32))
    V, D, n = 3, 1, 200000
    dr = np.tile(q, (bf.table_rows(V, 1), 1))
    tg = np.tile(p, (bf.table_rows(V, 1), 1))
    pt = np.exp(p.astype(np.float64)) / np.exp(p.astype(np.float64)).sum()
    good = orc.Config(B=1, V=3, K=2, m=1, D=1, N=2)
    st, _ = orc.run_prefix_lm(good, dr, tg, 1, n, 1.0, 1, 1)
    assert _chisq_p(np.bincount(st[:, 0], minlength=3), pt * n) > 0.01
    bad = orc.Config(B=1, V=3, K=2, m=1, D=1, N=2, proxy_mode=1, fixed_log_proxy=math.log(0.25))
    st, _ = orc.run_prefix_lm(bad, dr, tg, 1, n, 1.0, 1, 1)
    assert _chisq_p(np.bincount(st[:, 0], minlength=3), pt * n) < 1e-6


# --------------------------------------------------------------------------
# sparse support S < V (Sec. 3.2 "Efficient implementation": verification with
# the same truncated q~ stays lossless).  Only here does the residual off the
# support (r^ = p there) and the mass M = 1 - sum_tail min(p, q~) take part.
# --------------------------------------------------------------------------

def _sparse_laws(V, K, m, S, D, N, T, seed):
    rng = np.random.default_rng(seed)
    dr, tg = bf.random_tables(rng, V, D)
    en = bf.Enumerator(V, K, m, S, D, N, T, dr, tg)
    tl = en.target_law(2)
    p1 = np.zeros(V)
    p2 = np.zeros(V * V)
    for (a, b), pr in tl.items():
        p1[a] += pr
        p2[a * V + b] += pr
    _, accl = en.stream_distribution(2)
    return dr, tg, p1, p2, np.array([accl.get(i, 0.0) for i in range(D + 1)])


SPARSE_MC = [(8, 0), (8, 1), (8, 2), (12, 0), (12, 1), (12, 2)]


@pytest.mark.parametrize("S,m", SPARSE_MC)
def test_monte_carlo_losslessness_sparse_support(orc, S, m):
    """10^6 oracle cycles at V = 16 with support S < V: the first emitted token
    and the first two follow the target (Theorem 1), and the accepted length
    follows the enumerator's exact law, which forms the residual as
    max(0, p - q~) over the whole vocabulary (q~ = 0 off the tail)."""
    V, K, D, N, T, n = 16, 2, 2, 5, 0.9, 1_000_000
    dr, tg, p1, p2, ea = _sparse_laws(V, K, m, S, D, N, T, seed=1700 + 10 * S + m)
    cfg = orc.Config(B=1, V=V, K=K, m=m, S=S, D=D, N=N)
    st, acc = orc.run_prefix_lm(cfg, dr, tg, D, n, T, 4242 + S + m, 2)
    assert _chisq_p(np.bincount(st[:, 0], minlength=V), p1 * n) > 0.01
    assert _chisq_p(np.bincount(st[:, 0] * V + st[:, 1], minlength=V * V), p2 * n) > 0.01
    assert _chisq_p(np.bincount(acc, minlength=D + 1), ea * n) > 0.01


@pytest.mark.parametrize("plant", ["residual_on_support", "mass_on_support"])
def test_monte_carlo_detects_planted_sparse_support_mistakes(orc, plant):
    """Two plausible mistakes planted in the oracle (restricting the final draw
    to the expansion's support; summing the residual mass over the support
    only) are invisible at S = V, where the support is the whole vocabulary,
    and the chi-square tests above reject each of them at S < V."""
    mode = {"residual_on_support": orc.PLANT_RESIDUAL_ON_SUPPORT, "mass_on_support": orc.PLANT_MASS_ON_SUPPORT}[plant]
    V, K, m, D, N, T, n = 16, 2, 1, 2, 5, 0.9, 400_000
    for S, must_pass in ((V, True), (8, False)):
        dr, tg, p1, p2, ea = _sparse_laws(V, K, m, S, D, N, T, seed=1900 + S)
        clean = orc.Config(B=1, V=V, K=K, m=m, S=S, D=D, N=N)
        bad = orc.Config(B=1, V=V, K=K, m=m, S=S, D=D, N=N, plant_mode=mode)
        st0, acc0 = orc.run_prefix_lm(clean, dr, tg, D, n, T, 99, 2)
        st1, acc1 = orc.run_prefix_lm(bad, dr, tg, D, n, T, 99, 2)
        pv = min(_chisq_p(np.bincount(st1[:, 0] * V + st1[:, 1], minlength=V * V), p2 * n),
                 _chisq_p(np.bincount(acc1, minlength=D + 1), ea * n))
        if must_pass:
            # same draws, and the planted branch is never taken differently
            np.testing.assert_array_equal(st0, st1)
            np.testing.assert_array_equal(acc0, acc1)
        else:
            assert _chisq_p(np.bincount(st0[:, 0] * V + st0[:, 1], minlength=V * V), p2 * n) > 0.01
            assert pv < 1e-6, (plant, pv)


# --------------------------------------------------------------------------
# temperature degeneracy (Sec. 5.4), validation, replay
# --------------------------------------------------------------------------

def test_low_temperature_degeneracy(orc):
    """T -> 0: m = 0 collapses to the top-(K+1) tree (dual degeneracy); m = 1
    samples x_2 but keeps the proxy min{q(x_1), z} in the scores (single)."""
    rng = np.random.default_rng(8)
    V, K, D = 64, 3, 3
    rows = [rng.normal(0, 2, size=(4, 1 if d == 1 else K, V)).astype(np.float32) for d in range(1, D + 1)]
    for m in (0, 1):
        cfg = orc.Config(B=4, V=V, K=K, m=m, D=D, N=10)
        tree = orc.Tree(cfg)
        for d in range(1, D + 1):
            orc.expand(cfg, d, rows[d - 1], 1e-4, np.arange(4), 0, tree)
        for b in range(4):
            for first in range(1, cfg.G1, K + 1):
                par = tree.parent[b, first]
                toks = tree.token[b, first:first + K + 1]
                depth = 1 if first == 1 else 2 + (first - (K + 2)) // (K * (K + 1))
                f = 0 if first == 1 else ((first - (K + 2)) % (K * (K + 1))) // (K + 1)
                row = rows[depth - 1][b, f].astype(np.float64)
                order = np.lexsort((np.arange(V), -row))
                np.testing.assert_array_equal(toks, order[:K + 1])
                y = first + m
                if m == 1:
                    lq = row - special.logsumexp(row)
                    want = min(lq[order[0]], math.log1p(-math.exp(lq[order[0]])))
                    assert abs(tree.log_proxy[b, y] - want) < 1e-5


def test_config_validation(orc):
    ok = dict(B=1, V=100, K=4, m=1, D=3, N=10)
    assert orc.Config(**ok).valid()
    for bad in (dict(m=5), dict(S=4), dict(S=101), dict(N=0), dict(N=10**4), dict(D=0),
                dict(K=0, D=2), dict(m=0, eps=0.0)):
        assert not orc.Config(**{**ok, **bad}).valid(), bad


def test_bad_rows_are_rejected(orc):
    cfg = orc.Config(B=1, V=20, K=2, m=1, D=1, N=2)
    for bad in (np.nan, np.inf):
        rows = np.zeros((1, 1, 20), np.float32)
        rows[0, 0, 7] = bad
        with pytest.raises(orc.OracleError):
            orc.expand(cfg, 1, rows, 1.0, 0, 0, orc.Tree(cfg))
    rows = np.full((1, 1, 20), -np.inf, np.float32)
    rows[0, 0, 3] = 0.0  # only one finite logit, m + 1 = 2 needed
    with pytest.raises(orc.OracleError):
        orc.expand(cfg, 1, rows, 1.0, 0, 0, orc.Tree(cfg))


def test_replay_is_bit_exact_and_offset_changes_draws(orc):
    rng = np.random.default_rng(2)
    cfg = orc.Config(B=3, V=500, K=4, m=1, D=3, N=12)
    rows = [rng.normal(0, 1.5, size=(3, cfg.rows_at(d), 500)).astype(np.float32) for d in (1, 2, 3)]
    tgt = rng.normal(0, 1.5, size=(3, 13, 500)).astype(np.float32)
    a = orc.run_step(cfg, rows, tgt, 1.0, [1, 2, 3], [7, 7, 7])
    b = orc.run_step(cfg, rows, tgt, 1.0, [1, 2, 3], [7, 7, 7])
    c = orc.run_step(cfg, rows, tgt, 1.0, [1, 2, 3], [8, 8, 8])
    np.testing.assert_array_equal(a[0].token, b[0].token)
    np.testing.assert_array_equal(a[2].bonus_token, b[2].bonus_token)
    assert not np.array_equal(a[0].token, c[0].token)
