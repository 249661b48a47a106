"""Exhaustive enumeration of RheoSampling trees and verification paths.

An independent fp64 restatement of the method used to pin the oracle: for a
tiny vocabulary it enumerates every joint realisation of the sampled tokens
(one per expanded node, each drawn with probability q~), builds the pruned tree
for each, and integrates Algorithm 1 analytically (acceptance probabilities
instead of coins).  Theorem 1 then says the probability of every emitted
stream equals its probability under autoregressive sampling from the target.

Language models are tables indexed by token prefix, the same layout the oracle
uses: the row of prefix x_1..x_j is sum_{i<j} V^i + (x_1..x_j read in base V).
"""
from __future__ import annotations

import itertools
import math
from collections import defaultdict
from dataclasses import dataclass

import numpy as np


def prefix_row(prefix, V):
    base = sum(V ** i for i in range(len(prefix)))
    val = 0
    for x in prefix:
        val = val * V + x
    return base + val


def table_rows(V, depth):
    return sum(V ** i for i in range(depth + 1))


def softmax64(x):
    x = np.asarray(x, dtype=np.float64)
    m = np.max(x)
    e = np.exp(x - m)
    return e / e.sum()


@dataclass
class Node:
    gen: int
    token: int
    parent: int
    depth: int
    slot: int          # position in its pool
    kind: str          # 'root' | 'lead' | 'sampled' | 'fill'
    score: float       # log path score (fp64)
    qtilde: float = 0.0
    tail: dict | None = None   # for expanded nodes: token -> q~ over the tail


class Enumerator:
    """Brute force over all sampled-token realisations (Theorem 1, App. C)."""

    def __init__(self, V, K, m, S, D, N, T, draft_table, target_table, eps=1e-6,
                 proxy=None, verify="rheo"):
        self.V, self.K, self.m, self.S, self.D, self.N, self.T = V, K, m, S, D, N, T
        self.draft = np.asarray(draft_table, dtype=np.float64)
        self.target = np.asarray(target_table, dtype=np.float64)
        self.eps = eps
        self.proxy = proxy  # None: the paper's proxy; a float: a fixed (ad hoc) proxy probability
        # "rheo": Algorithm 1; "rrsw": recursive rejection, leads first, then the
        # sampled child, then fills (App. D.2); "onehot": every child a one-hot
        # candidate in slot order, residual from p (vanilla top-K, App. A)
        self.verify = verify

    # -- one pool (Sec. 3.2, App. C.1) ------------------------------------
    def support(self, row):
        order = sorted(range(self.V), key=lambda v: (-row[v], v))
        return order[: self.S]

    def pool(self, prefix):
        """Returns (ranked support, q0, tail q~ dict, proxy) for a parent prefix."""
        row = self.draft[prefix_row(prefix, self.V)]
        q0 = softmax64(row)                     # untempered, full vocabulary (Sec. 5.4)
        sup = self.support(row)
        tail = sup[self.m:]
        qt = softmax64(row[tail] / self.T)       # tempered, truncated, renormalised tail
        qtail = {v: float(qt[i]) for i, v in enumerate(tail)}
        if self.proxy is not None:
            proxy = self.proxy
        elif self.m >= 1:
            z = 1.0 - sum(q0[x] for x in sup[: self.m])
            proxy = min(q0[sup[self.m - 1]], z)
        else:
            proxy = min(1.0, q0[sup[0]] + self.eps)
        return sup, q0, qtail, proxy

    def children(self, parent: Node, prefix, y, gen0):
        sup, q0, qtail, proxy = self.pool(prefix)
        kids = []
        for j in range(self.m):
            x = sup[j]
            kids.append(Node(gen0 + j, x, parent.gen, parent.depth + 1, j, "lead",
                             parent.score + math.log(q0[x])))
        kids.append(Node(gen0 + self.m, y, parent.gen, parent.depth + 1, self.m, "sampled",
                         parent.score + math.log(proxy) if proxy > 0 else -math.inf,
                         qtilde=qtail[y]))
        rest = [x for x in sup[self.m:] if x != y]
        for j in range(self.K - self.m):
            x = rest[j]
            kids.append(Node(gen0 + self.m + 1 + j, x, parent.gen, parent.depth + 1,
                             self.m + 1 + j, "fill", parent.score + math.log(q0[x])))
        parent.tail = qtail
        return kids

    # -- tree for one realisation ----------------------------------------
    def path(self, nodes, g):
        out = []
        while g != 0:
            out.append(nodes[g].token)
            g = nodes[g].parent
        return tuple(reversed(out))

    def realisations(self):
        """Yields (probability, nodes dict) over every joint choice of sampled tokens."""
        root = Node(0, -1, -1, 0, 0, "root", 0.0)
        yield from self._expand_depth({0: root}, 1, [0], 1.0)

    def _expand_depth(self, nodes, d, frontier, prob):
        K = self.K
        prefixes = [self.path(nodes, g) for g in frontier]
        tails = [self.pool(pf)[2] for pf in prefixes]
        base = 1 if d == 1 else 1 + (K + 1) + (d - 2) * K * (K + 1)
        for ys in itertools.product(*[list(t.keys()) for t in tails]):
            pr = prob
            for t, y in zip(tails, ys):
                pr *= t[y]
            if pr == 0.0:
                continue
            new = {g: Node(**vars(n)) for g, n in nodes.items()}
            made = []
            for f, (g, y) in enumerate(zip(frontier, ys)):
                kids = self.children(new[g], prefixes[f], y, base + f * (K + 1))
                for kd in kids:
                    new[kd.gen] = kd
                made += kids
            if d == self.D:
                yield pr, new
            else:
                ranked = sorted(made, key=lambda n: (-n.score, n.gen))
                nxt = sorted(n.gen for n in ranked[:K])
                yield from self._expand_depth(new, d + 1, nxt, pr)

    def prune(self, nodes):
        cand = sorted((n for g, n in nodes.items() if g != 0), key=lambda n: (-n.score, n.gen))
        keep = {0} | {n.gen for n in cand[: self.N]}
        for g in keep:
            if g != 0:
                assert nodes[g].parent in keep, "pruned tree not ancestor-closed"
        return keep

    # -- Algorithm 1, integrated analytically -----------------------------
    def p_of(self, prefix):
        return softmax64(self.target[prefix_row(prefix, self.V)] / self.T)

    def continue_to(self, prefix, L, weight, out):
        if weight == 0.0:
            return
        if len(prefix) >= L:
            out[prefix[:L]] += weight
            return
        p = self.p_of(prefix)
        for v in range(self.V):
            if p[v] > 0:
                self.continue_to(prefix + (v,), L, weight * p[v], out)

    def walk(self, nodes, keep, g, prefix, L, weight, out, acc, depth=0):
        if weight == 0.0:
            return
        p = self.p_of(prefix)
        kids = sorted((n for n in nodes.values() if n.parent == g and n.gen in keep),
                      key=lambda n: n.gen)
        if not kids:
            acc[depth] += weight
            for v in range(self.V):
                self.continue_to(prefix + (v,), L, weight * p[v], out)
            return
        s = next((n for n in kids if n.kind == "sampled"), None)
        reach = weight
        if self.verify == "onehot":
            s = None
        qt = np.zeros(self.V)
        if s is not None:
            for v, q in nodes[g].tail.items():
                qt[v] = q
        rhat = p.copy()
        M = rhat.sum()

        def one_hot(c):  # accept c with probability r^(c) / M, else drop it from r^
            nonlocal reach, M
            a = rhat[c.token] / M if M > 0 else 1.0
            self.walk(nodes, keep, c.gen, prefix + (c.token,), L, reach * a, out, acc, depth + 1)
            reach *= 1.0 - a
            M -= rhat[c.token]
            rhat[c.token] = 0.0

        if self.verify == "rrsw":
            for c in kids:
                if c.kind == "lead":
                    one_hot(c)
            if s is not None:
                a = min(1.0, (rhat[s.token] / M) / s.qtilde) if M > 0 else 1.0
                self.walk(nodes, keep, s.gen, prefix + (s.token,), L, reach * a, out, acc, depth + 1)
                reach *= 1.0 - a
                rhat = np.maximum(0.0, rhat - M * qt)
                M = rhat.sum()
            for c in kids:
                if c.kind == "fill":
                    one_hot(c)
        else:
            if s is not None:
                a = min(1.0, p[s.token] / s.qtilde)
                self.walk(nodes, keep, s.gen, prefix + (s.token,), L, reach * a, out, acc, depth + 1)
                reach *= 1.0 - a
                rhat = np.maximum(0.0, p - qt)
                M = rhat.sum()
            for c in kids:
                if c is not s:
                    one_hot(c)
        acc[depth] += reach
        for c in kids:
            rhat[c.token] = 0.0
        tot = rhat.sum()
        if tot > 0 and reach > 0:
            for v in range(self.V):
                if rhat[v] > 0:
                    self.continue_to(prefix + (v,), L, reach * rhat[v] / tot, out)

    def stream_distribution(self, L):
        """Exact law of the first L emitted tokens, plus the law of the accepted length."""
        out = defaultdict(float)
        acc = defaultdict(float)
        for pr, nodes in self.realisations():
            keep = self.prune(nodes)
            self.walk(nodes, keep, 0, (), L, pr, out, acc)
        return out, acc

    def target_law(self, L):
        out = defaultdict(float)
        self.continue_to((), L, 1.0, out)
        return out

    def tree_for(self, ys_by_parent):
        """Tree built with forced sampled tokens: ys_by_parent maps parent gen -> Y."""
        root = Node(0, -1, -1, 0, 0, "root", 0.0)
        nodes = {0: root}
        frontier = [0]
        K = self.K
        for d in range(1, self.D + 1):
            base = 1 if d == 1 else 1 + (K + 1) + (d - 2) * K * (K + 1)
            made = []
            for f, g in enumerate(frontier):
                kids = self.children(nodes[g], self.path(nodes, g), ys_by_parent[g], base + f * (K + 1))
                for kd in kids:
                    nodes[kd.gen] = kd
                made += kids
            if d < self.D:
                ranked = sorted(made, key=lambda n: (-n.score, n.gen))
                frontier = sorted(n.gen for n in ranked[:K])
        return nodes


def random_tables(rng, V, depth, spread=1.5):
    """Draft/target tables over all prefixes up to `depth`, target = draft + noise."""
    n = table_rows(V, depth)
    draft = rng.normal(0.0, spread, size=(n, V)).astype(np.float32)
    target = (draft + rng.normal(0.0, 0.8, size=(n, V))).astype(np.float32)
    return draft, target
