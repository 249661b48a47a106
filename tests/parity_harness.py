"""Runs one decoding cycle through the CUDA library and through the CPU oracle
on the same seeded inputs and compares them.

Bar (the benchmark specification): token ids, parents, slots, frontiers,
pruned trees, accepted lengths/tokens/nodes and bonus tokens bit-exact; fp32
values (log proxies, path scores, q~, log-partitions) within 1e-5 relative /
1e-7 absolute.  A mismatch of an integer result counts as an explained near-tie
flip when the oracle's relative gap at the first divergent decision is below
GAP; the request is then left out of later comparisons.  Anything else fails.

Target rows are built by the seeded generator from each side's OWN tree, so no
oracle input ever comes from the CUDA path.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch

import oracle
from paper_2609_21827_gb300 import rheo, synth

RTOL, ATOL, GAP = 1e-5, 1e-7, 1e-6
# Log-domain values (log q0 = l - lse1, path scores, log-partitions) come out
# of an fp32 subtraction with an operand of magnitude up to ~32, so they carry
# an absolute rounding of up to 2 ulp(32) = 3.8e-6 on either side.
LOG_ATOL = 4e-6
LOG_FIELDS = ("score", "log_proxy", "lse1", "row_lse")


def u64(t: torch.Tensor) -> np.ndarray:
    return t.cpu().numpy().view(np.uint64)


@dataclass
class Side:
    token: np.ndarray
    parent: np.ndarray
    slot: np.ndarray
    score: np.ndarray
    log_proxy: np.ndarray
    qtilde: np.ndarray
    tail_ids: np.ndarray
    tail_q: np.ndarray
    lse1: np.ndarray
    frontiers: list
    pruned: dict
    acc_len: np.ndarray
    acc_tok: np.ndarray
    acc_node: np.ndarray
    bonus: np.ndarray
    row_lse: np.ndarray
    status: int = 0
    gaps: dict = field(default_factory=dict)


def run_gpu(w: synth.Workload, draft: synth.DraftInputs, cfg: rheo.Config, target_override=None,
            row_stride_pad: int = 0, variant: int = 0) -> Side:
    tree = rheo.Tree(cfg)
    pr = rheo.Pruned(cfg)
    out = rheo.VerifyOut(cfg)
    ws = rheo.Workspace(cfg)
    frontiers = []
    for d in range(1, cfg.depth + 1):
        x = draft.rows[d - 1]
        if row_stride_pad:
            B, F, V = x.shape
            padded = torch.zeros((B, F, V + row_stride_pad), dtype=x.dtype, device=x.device)
            padded[..., :V] = x
            x = padded[..., :V]
        rheo.expand(cfg, d, x, draft.temperature, draft.seed, draft.offset, tree, ws)
        if d < cfg.depth:
            frontiers.append(tree.frontier.clone())
    rheo.prune(cfg, tree, pr, ws)
    tgt = target_override(pr.gen_id) if target_override else synth.target_rows(w, draft, frontiers, pr.gen_id)
    if row_stride_pad:
        B, NP, V = tgt.shape
        padded = torch.zeros((B, NP, V + row_stride_pad), dtype=tgt.dtype, device=tgt.device)
        padded[..., :V] = tgt
        tgt = padded[..., :V]
    if variant:
        rheo.verify_variant(cfg, variant, tgt, draft.temperature, draft.seed, draft.offset, tree, pr, out, ws)
    else:
        rheo.verify(cfg, tgt, draft.temperature, draft.seed, draft.offset, tree, pr, out, ws)
    st = rheo.status(cfg, ws)
    c = lambda t: t.cpu().numpy()
    return Side(c(tree.token), c(tree.parent), c(tree.slot), c(tree.score), c(tree.log_proxy), c(tree.qtilde),
                c(tree.tail_ids), c(tree.tail_q), c(tree.lse1), [c(f) for f in frontiers],
                {k: c(getattr(pr, k)) for k in ("gen_id", "token", "parent", "depth", "first_child", "n_child",
                                                  "sampled_child")},
                c(out.accepted_len), c(out.accepted_tokens), c(out.accepted_nodes), c(out.bonus_token),
                c(out.row_lse), st)


def run_oracle(w: synth.Workload, draft: synth.DraftInputs, cfg: rheo.Config, reqs, target_override=None,
               variant: int = 0) -> Side:
    """The oracle on requests `reqs` (a sub-batch of the same inputs)."""
    reqs = list(reqs)
    ocfg = oracle.Config(B=len(reqs), V=cfg.vocab, K=cfg.K, m=cfg.m, S=cfg.support, D=cfg.depth, N=cfg.budget,
                         eps=cfg.eps, verify_mode=variant)
    T = draft.temperature.cpu().numpy()[reqs]
    seed = u64(draft.seed)[reqs]
    off = u64(draft.offset)[reqs]
    tree = oracle.Tree(ocfg)
    frontiers = []
    for d in range(1, cfg.depth + 1):
        rows = draft.rows[d - 1][reqs].float().cpu().numpy()
        oracle.expand(ocfg, d, rows, T, seed, off, tree)
        if d < cfg.depth:
            frontiers.append(tree.frontier.copy())
    pr = oracle.prune(ocfg, tree)
    gids = torch.from_numpy(pr.gen_id.copy())
    if target_override:
        tgt = target_override(gids, reqs)
    else:
        sub = synth.DraftInputs(w, [r[reqs] for r in draft.rows], draft.temperature[reqs], draft.seed[reqs],
                                draft.offset[reqs])
        tgt = synth.target_rows(w, sub, [torch.from_numpy(f) for f in frontiers], gids,
                                device=draft.rows[0].device, noise_seed=None, request_ids=reqs)
    out = oracle.verify(ocfg, tgt.float().cpu().numpy(), T, seed, off, tree, pr)
    side = Side(tree.token, tree.parent, tree.slot, tree.score, tree.log_proxy, tree.qtilde, tree.tail_ids,
                tree.tail_q, tree.lse1, frontiers,
                {k: getattr(pr, k) for k in ("gen_id", "token", "parent", "depth", "first_child", "n_child",
                                             "sampled_child")},
                out.accepted_len, out.accepted_tokens, out.accepted_nodes, out.bonus_token, out.row_lse)
    side.gaps = {"sample": tree.gap_sample, "frontier": tree.gap_frontier, "prune": pr.gap_prune,
                 "level": out.gap_level}
    return side


@dataclass
class Report:
    requests: int = 0
    exact: int = 0
    verified: int = 0  # requests whose verification outputs were compared (trees identical)
    explained: list = field(default_factory=list)
    unexplained: list = field(default_factory=list)
    fp_fail: list = field(default_factory=list)

    def ok(self) -> bool:
        return not self.unexplained and not self.fp_fail

    def __str__(self):
        return (f"requests={self.requests} exact={self.exact} verified={self.verified} "
                f"explained_flips={len(self.explained)} {self.explained[:5]} "
                f"unexplained={self.unexplained[:5]} fp_fail={self.fp_fail[:5]}")


def _close(a, b, atol=ATOL):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    both_inf = np.isinf(a) & np.isinf(b) & (np.sign(a) == np.sign(b))
    ok = both_inf | (np.abs(a - b) <= atol + RTOL * np.abs(b))
    return bool(ok.all())


def compare(cfg: rheo.Config, g: Side, o: Side, reqs) -> Report:
    rep = Report()
    K, D = cfg.K, cfg.depth
    for j, b in enumerate(reqs):
        rep.requests += 1
        why = None  # (kind, gap)
        # expansion, depth by depth
        for d in range(1, D + 1):
            F = 1 if d == 1 else K
            base = 1 if d == 1 else 1 + (K + 1) + (d - 2) * K * (K + 1)
            sl = slice(base, base + F * (K + 1))
            same = (np.array_equal(g.token[b, sl], o.token[j, sl]) and np.array_equal(g.parent[b, sl], o.parent[j, sl])
                    and np.array_equal(g.slot[b, sl], o.slot[j, sl]))
            if not same:
                for f in range(F):
                    ps = slice(base + f * (K + 1), base + (f + 1) * (K + 1))
                    if not np.array_equal(g.token[b, ps], o.token[j, ps]):
                        e = 0 if d == 1 else 1 + (d - 2) * K + f
                        why = ("sample", o.gaps["sample"][j, e])
                        break
                if why is None:
                    # same tokens, other parents or slots: the frontiers were
                    # compared equal already, so no decision margin can explain it
                    why = ("pool", 1.0)
                break
            if d < D and not np.array_equal(g.frontiers[d - 1][b], o.frontiers[d - 1][j]):
                why = ("frontier", o.gaps["frontier"][j, d - 1])
                break
        if why is None and not np.array_equal(g.pruned["gen_id"][b], o.pruned["gen_id"][j]):
            why = ("prune", o.gaps["prune"][j])
        if why is None:
            for k in ("token", "parent", "depth", "first_child", "n_child", "sampled_child"):
                if not np.array_equal(g.pruned[k][b], o.pruned[k][j]):
                    why = (f"pruned.{k}", 1.0)
                    break
        if why is None:
            # fp values of a structurally identical tree
            bad = [k for k in ("score", "log_proxy", "qtilde", "tail_q", "lse1", "row_lse")
                   if not _close(getattr(g, k)[b], getattr(o, k)[j], LOG_ATOL if k in LOG_FIELDS else ATOL)]
            if not np.array_equal(g.tail_ids[b], o.tail_ids[j]):
                bad.append("tail_ids")
            if bad:
                errs = {k: float(np.nanmax(np.abs(np.asarray(getattr(g, k)[b], np.float64)
                                                  - np.asarray(getattr(o, k)[j], np.float64)))) for k in bad
                        if k != "tail_ids"}
                rep.fp_fail.append((b, bad, errs))
                continue
            # verification
            rep.verified += 1
            n = int(o.acc_len[j])
            lvl = None
            for i in range(D):
                if g.acc_node[b, i] != o.acc_node[j, i] or g.acc_tok[b, i] != o.acc_tok[j, i]:
                    lvl = i
                    break
            if lvl is None and (g.acc_len[b] != o.acc_len[j] or g.bonus[b] != o.bonus[j]):
                lvl = min(n, int(g.acc_len[b]))
            if lvl is not None:
                why = ("verify", o.gaps["level"][j, lvl])
        if why is None:
            rep.exact += 1
        elif why[1] < GAP:
            rep.explained.append((b, why[0], float(why[1])))
        else:
            rep.unexplained.append((b, why[0], float(why[1])))
    return rep
