"""rheo_verify_static: verification for callers that may not allocate.

Some callers cannot allocate device memory when they verify (code given only
fixed buffers by a host framework, runtimes whose device memory is partitioned
up front, loops that must avoid cudaMalloc's implicit synchronisation).  For
them the library keeps the scratch state of verification in a static device
array instead of a caller workspace.  These tests call that entry point through
the C ABI and check it against rheo_verify on the same tree and target logits,
for two calls in a row with different configurations (so the second call runs
on the array as the first one left it).  The file is named to be collected
last, and passes alone in a fresh process or after the rest of the suite.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2609_21827_gb300 import build, rheo, synth
import parity_harness as ph


def _cfg(w: synth.Workload) -> rheo.Config:
    return rheo.Config(batch=w.batch, vocab=w.vocab, K=w.K, depth=w.depth, budget=w.budget, m=w.m,
                       support=min(w.support, w.vocab), dtype=w.dtype)


def _W(name, **kw):
    base = dict(name=name, batch=4, vocab=1000, depth=3, K=4, budget=12, dtype="f32", zipf_s=1.1,
                sigma_draft=0.5, sigma_target=0.5, temperatures=(1.0,), seed=4242)
    base.update(kw)
    return synth.Workload(**base)


def _tree_and_targets(w):
    """Expansion and prune through the workspace entry points, then the target rows."""
    cfg = _cfg(w)
    draft = synth.make_draft_inputs(w, device="cuda")
    tree, pr, ws = rheo.Tree(cfg), rheo.Pruned(cfg), rheo.Workspace(cfg)
    frontiers = []
    for d in range(1, cfg.depth + 1):
        rheo.expand(cfg, d, draft.rows[d - 1], draft.temperature, draft.seed, draft.offset, tree, ws)
        if d < cfg.depth:
            frontiers.append(tree.frontier.clone())
    rheo.prune(cfg, tree, pr, ws)
    tgt = synth.target_rows(w, draft, frontiers, pr.gen_id)
    assert rheo.status(cfg, ws) == 0
    return cfg, draft, tree, pr, ws, tgt


def _same(cfg, ref: rheo.VerifyOut, got: rheo.VerifyOut):
    for k in ("accepted_len", "accepted_tokens", "accepted_nodes", "bonus_token"):
        np.testing.assert_array_equal(getattr(got, k).cpu().numpy(), getattr(ref, k).cpu().numpy(), err_msg=k)
    a = got.row_lse.cpu().numpy().astype(np.float64)
    b = ref.row_lse.cpu().numpy().astype(np.float64)
    assert np.all(np.abs(a - b) <= ph.LOG_ATOL + ph.RTOL * np.abs(b)), "row_lse"


@pytest.mark.gpu
def test_verify_static_matches_workspace_entry_point_twice():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    build.build()
    cases = [
        _W("static_bf16_chunks", vocab=50000, K=6, depth=4, budget=20, dtype="bf16", batch=8,
           temperatures=(0.5, 0.8, 1.0)),
        _W("static_f32_small", vocab=1001, K=3, m=0, support=40, depth=3, budget=9, batch=5,
           temperatures=(0.7, 1.3)),
    ]
    for w in cases:
        cfg, draft, tree, pr, ws, tgt = _tree_and_targets(w)
        ref = rheo.VerifyOut(cfg)
        rheo.verify(cfg, tgt, draft.temperature, draft.seed, draft.offset, tree, pr, ref, ws)
        assert rheo.status(cfg, ws) == 0
        got = rheo.VerifyOut(cfg)
        st = torch.full((1,), -1, dtype=torch.int32, device="cuda")
        rheo.verify_static(cfg, tgt, draft.temperature, draft.seed, draft.offset, tree, pr, got, status=st)
        torch.cuda.synchronize()
        assert int(st.item()) == 0, w.name
        _same(cfg, ref, got)


def test_verify_static_rejects_configurations_beyond_the_array():
    """A configuration whose scratch exceeds RHEO_STATIC_SCRATCH_BYTES is refused
    on the host, before any device work, with RHEO_ETOOLARGE."""
    L = rheo.lib()
    big = rheo.Config(batch=64, vocab=262144, K=8, depth=8, budget=200, m=1, support=128, dtype="bf16")
    fake = 256  # never dereferenced: the size check comes first
    vals = [fake] * 10
    tree = rheo._Tree(*vals)
    pr = rheo._Pruned(*[fake] * 7)
    out = rheo._VerifyOut(*[fake] * 5)
    rc = L.rheo_verify_static(ctypes.byref(big.c()), fake, big.vocab, fake, fake, fake, ctypes.byref(tree),
                              ctypes.byref(pr), ctypes.byref(out), None, None)
    assert rc == rheo.RHEO_ETOOLARGE
