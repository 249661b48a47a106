"""Multi-cycle speculative decoding against synthetic order-k language models.

A driver around the C-ABI path (expand x D, prune, verify) for the synthetic
analogue of the paper's decoding experiments (Sec. 5.3, Sec. 5.4): B
independent sequences advance cycle by cycle; each cycle builds the draft tree
from a draft model, prunes it, verifies it against a target model and appends
the accepted tokens plus the bonus token.  The models are tables of logits
indexed by the last k tokens of the context (a k-gram model: row = the last k
tokens read in base V), so the law of every emitted stream under the target is
known exactly and the losslessness of Theorem 1 can be checked on the GPU path
over many cycles.

Every step of the method runs in the library's kernels; this module only
gathers the rows of the tables for the frontier and pruned nodes (torch
indexing) and keeps the contexts.
"""
from __future__ import annotations

from dataclasses import dataclass

import torch

from . import rheo


@dataclass
class KGramLM:
    """Logits [V**k, V] of a k-gram model (row = last k tokens in base V, oldest first)."""

    table: torch.Tensor
    V: int
    k: int

    @staticmethod
    def random(V: int, k: int, spread: float, gen: torch.Generator, device="cuda", base=None, noise=0.0):
        """Gaussian logits (scale `spread`); with `base`, base.table + N(0, noise) (a correlated target)."""
        if base is not None:
            t = base.table.float().cpu() + noise * torch.randn(base.table.shape, generator=gen)
        else:
            t = spread * torch.randn((V ** k, V), generator=gen)
        return KGramLM(t.to(device=device, dtype=torch.float32), V, k)

    def rows(self, ctx: torch.Tensor) -> torch.Tensor:
        """Logit rows for contexts ctx [..., k] (int64 tokens)."""
        idx = torch.zeros(ctx.shape[:-1], dtype=torch.int64, device=ctx.device)
        for j in range(self.k):
            idx = idx * self.V + ctx[..., j]
        return self.table[idx]


def _paths(tok: torch.Tensor, par: torch.Tensor, nodes: torch.Tensor, depth: int) -> torch.Tensor:
    """Tokens on the path root -> node for nodes [B, n] (gen ids or pruned indices,
    parents in `par`): [B, n, depth], right-aligned, 0 before the path starts;
    also the path lengths."""
    B, n = nodes.shape
    out = torch.zeros((B, n, depth), dtype=torch.int64, device=nodes.device)
    length = torch.zeros((B, n), dtype=torch.int64, device=nodes.device)
    cur = nodes.long()
    for i in range(depth):
        alive = cur > 0
        t = torch.gather(tok.long(), 1, cur.clamp(min=0))
        out[:, :, depth - 1 - i] = torch.where(alive, t, torch.zeros_like(t))
        length += alive.long()
        cur = torch.where(alive, torch.gather(par.long(), 1, cur.clamp(min=0)), torch.full_like(cur, -1))
    return out, length


def _contexts(window: torch.Tensor, path: torch.Tensor, length: torch.Tensor, k: int) -> torch.Tensor:
    """Last k tokens of (window, path[:length]) for every node: [B, n, k]."""
    B, n, depth = path.shape
    full = torch.cat([window[:, None, :].expand(B, n, k), path], dim=2)  # [B, n, k + depth]
    # the path is right-aligned (its l tokens are the last l columns), so position
    # c >= k of the sequence window ++ path reads column c + (depth - l)
    shift = (depth - length)[:, :, None]
    col = torch.arange(k + depth, device=window.device)[None, None, :].expand(B, n, k + depth)
    src = torch.where(col < k, col, col + shift)
    seq = torch.gather(full, 2, src.clamp(0, k + depth - 1))
    total = k + length  # valid length of the virtual sequence
    take = total[:, :, None] - k + torch.arange(k, device=window.device)[None, None, :]
    return torch.gather(seq, 2, take)


@dataclass
class CycleResult:
    streams: torch.Tensor      # [B, L] first L emitted tokens of every sequence (-1 if fewer)
    accepted: torch.Tensor     # [B, cycles] accepted draft tokens per cycle
    windows: torch.Tensor      # [B, cycles, k] the last k context tokens at the start of each cycle
    cycles: int


def run_cycles(cfg: rheo.Config, draft_lm: KGramLM, target_lm: KGramLM, window: torch.Tensor,
               temperature: torch.Tensor, seed: torch.Tensor, cycles: int, L: int,
               variant: int = rheo.VERIFY_RHEO, stream=None) -> CycleResult:
    """`cycles` decoding cycles for the cfg.batch sequences whose last k tokens are
    `window` [B, k]; Philox offset = cycle index.  Returns the first L emitted
    tokens and the accepted lengths."""
    B, D, K, V, k = cfg.batch, cfg.depth, cfg.K, cfg.vocab, draft_lm.k
    dev = window.device
    tree, pr, out, ws = rheo.Tree(cfg, dev), rheo.Pruned(cfg, dev), rheo.VerifyOut(cfg, row_lse=False, device=dev), \
        rheo.Workspace(cfg, dev)
    win = window.long().clone()
    emitted = torch.full((B, L), -1, dtype=torch.int64, device=dev)
    n_emit = torch.zeros(B, dtype=torch.int64, device=dev)
    acc_hist = torch.zeros((B, cycles), dtype=torch.int32, device=dev)
    win_hist = torch.zeros((B, cycles, k), dtype=torch.int64, device=dev)
    T = temperature.float().to(dev)
    for c in range(cycles):
        offset = torch.full((B,), c, dtype=torch.int64, device=dev)
        win_hist[:, c] = win
        for d in range(1, D + 1):
            if d == 1:
                ctx = win[:, None, :]
            else:
                fr = tree.frontier.long()  # [B, K] gen ids
                path, length = _paths(tree.token, tree.parent, fr, d - 1)
                ctx = _contexts(win, path, length, k)
            rows = draft_lm.rows(ctx).contiguous()  # [B, F_d, V]
            rheo.expand(cfg, d, rows, T, seed, offset, tree, ws, stream)
        rheo.prune(cfg, tree, pr, ws, stream)
        nodes = torch.arange(cfg.budget + 1, device=dev)[None, :].expand(B, -1)
        path, length = _paths(pr.token, pr.parent, nodes, D)
        tgt = target_lm.rows(_contexts(win, path, length, k)).contiguous()  # [B, N+1, V]
        rheo.verify_variant(cfg, variant, tgt, T, seed, offset, tree, pr, out, ws, stream)
        a = out.accepted_len.long()
        acc_hist[:, c] = out.accepted_len
        toks = torch.cat([out.accepted_tokens.long(), torch.zeros((B, 1), dtype=torch.int64, device=dev)], dim=1)
        toks.scatter_(1, a[:, None], out.bonus_token.long()[:, None])
        # append to the emitted streams and slide the k-token windows
        for j in range(D + 1):
            live = j <= a
            pos = n_emit + j
            put = live & (pos < L)
            emitted[put, pos[put]] = toks[put, j]
        n_emit += a + 1
        full = torch.cat([win, toks], dim=1)  # [B, k + D + 1]
        take = (a + 1)[:, None] + torch.arange(k, device=dev)[None, :]
        win = torch.gather(full, 1, take)
    if rheo.status(cfg, ws, stream) != 0:
        raise rheo.RheoError("device status set during the cycles")
    return CycleResult(emitted, acc_hist, win_hist, cycles)
