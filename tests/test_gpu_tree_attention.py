"""GPU parity of rheo_tree_attention (ancestor mask, positions, root-to-leaf
paths of the pruned tree) against the oracle.

Both sides build their own trees from the same seeded draft logits (expansion
and prune on each side), then derive the tree-attention arrays; every request
whose pruned tree agrees must give byte-identical arrays.
"""
import dataclasses

import numpy as np
import pytest
import torch

from paper_2609_21827_gb300 import build, rheo, synth
import parity_harness as ph

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    build.build()
    import oracle
    oracle.build()


def _W(name, **kw):
    base = dict(name=name, batch=4, vocab=1000, depth=3, K=4, budget=12, dtype="f32", zipf_s=1.1,
                sigma_draft=0.5, sigma_target=0.5, temperatures=(1.0,), seed=777)
    base.update(kw)
    return synth.Workload(**base)


CASES = [
    _W("small"),
    _W("budget1", K=3, budget=1, batch=6),
    _W("every_node", vocab=700, K=3, depth=3, budget=(3 + 1) + 2 * 3 * (3 + 1), batch=6),
    _W("k0", vocab=300, K=0, m=0, depth=1, budget=1, batch=8),
    _W("wide_bf16", vocab=5000, K=8, depth=5, budget=200, dtype="bf16", batch=5),
    dataclasses.replace(synth.WORKLOADS["qwen3_batch"], name="qwen3_batch_4req"),
]


@pytest.mark.parametrize("w", CASES, ids=[w.name for w in CASES])
def test_tree_attention_matches_oracle(w):
    import oracle

    reqs = list(range(min(w.batch, 4)))
    cfg = rheo.Config(batch=w.batch, vocab=w.vocab, K=w.K, depth=w.depth, budget=w.budget, m=w.m,
                      support=min(w.support, w.vocab), dtype=w.dtype)
    draft = synth.make_draft_inputs(w, device="cuda")
    tree, pr, ws = rheo.Tree(cfg), rheo.Pruned(cfg), rheo.Workspace(cfg)
    for d in range(1, cfg.depth + 1):
        rheo.expand(cfg, d, draft.rows[d - 1], draft.temperature, draft.seed, draft.offset, tree, ws)
    rheo.prune(cfg, tree, pr, ws)
    ta = rheo.TreeAttn(cfg)
    rheo.tree_attention(cfg, pr, ta, ws)
    assert rheo.status(cfg, ws) == 0

    ocfg = oracle.Config(B=len(reqs), V=cfg.vocab, K=cfg.K, m=cfg.m, S=cfg.support, D=cfg.depth, N=cfg.budget,
                         eps=cfg.eps)
    otree = oracle.Tree(ocfg)
    T = draft.temperature.cpu().numpy()[reqs]
    seed, off = ph.u64(draft.seed)[reqs], ph.u64(draft.offset)[reqs]
    for d in range(1, cfg.depth + 1):
        oracle.expand(ocfg, d, draft.rows[d - 1][reqs].float().cpu().numpy(), T, seed, off, otree)
    opr = oracle.prune(ocfg, otree)
    ota = oracle.tree_attention(ocfg, opr)

    gid = pr.gen_id.cpu().numpy()
    same = [j for j, b in enumerate(reqs) if np.array_equal(gid[b], opr.gen_id[j])]
    assert len(same) >= max(1, len(reqs) - 1), "pruned trees differ beyond a near-tie flip"
    for j in same:
        b = reqs[j]
        np.testing.assert_array_equal(ta.mask[b].cpu().numpy(), ota.mask[j], err_msg=f"mask {w.name} {b}")
        np.testing.assert_array_equal(ta.position[b].cpu().numpy(), ota.position[j])
        np.testing.assert_array_equal(ta.retrieve[b].cpu().numpy(), ota.retrieve[j])
        assert int(ta.n_leaves[b]) == int(ota.n_leaves[j])


def test_null_outputs_are_skipped_and_large_budgets_rejected():
    w = CASES[0]
    cfg = rheo.Config(batch=w.batch, vocab=w.vocab, K=w.K, depth=w.depth, budget=w.budget, m=w.m, dtype=w.dtype)
    draft = synth.make_draft_inputs(w, device="cuda")
    tree, pr, ws = rheo.Tree(cfg), rheo.Pruned(cfg), rheo.Workspace(cfg)
    for d in range(1, cfg.depth + 1):
        rheo.expand(cfg, d, draft.rows[d - 1], draft.temperature, draft.seed, draft.offset, tree, ws)
    rheo.prune(cfg, tree, pr, ws)
    full = rheo.TreeAttn(cfg)
    rheo.tree_attention(cfg, pr, full, ws)
    only = rheo.TreeAttn(cfg)
    only.mask.fill_(7)
    only.retrieve.fill_(7)
    c = only.c()
    c.mask = None
    c.retrieve = None
    import ctypes
    rc = rheo.lib().rheo_tree_attention(ctypes.byref(cfg.c()), ctypes.byref(pr.c()), ctypes.byref(c), ws.ptr(), None)
    assert rc == 0
    torch.cuda.synchronize()
    assert torch.equal(only.position, full.position) and torch.equal(only.n_leaves, full.n_leaves)
    assert int(only.mask.max()) == 7 and int(only.retrieve.max()) == 7  # untouched
    big = rheo.Config(batch=1, vocab=100000, K=16, depth=20, budget=5000, m=1)
    rc = rheo.lib().rheo_tree_attention(ctypes.byref(big.c()), ctypes.byref(pr.c()), ctypes.byref(full.c()),
                                        ws.ptr(), None)
    assert rc == rheo.RHEO_EINVAL
