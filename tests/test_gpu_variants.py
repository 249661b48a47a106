"""GPU parity of the verification variants (RRSw, vanilla one-hot; App. A and
App. D.2) against the oracle, on the same seeded trees and target rows.

The expansion and prune are the same kernels as for Algorithm 1; only the
per-node rule differs, so every case checks accepted lengths, tokens, nodes and
bonus tokens bit for bit (near-tie flips of a decision counted as for
Algorithm 1).
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
    base = dict(name=name, batch=8, vocab=1000, depth=3, K=4, budget=12, dtype="f32", zipf_s=1.1,
                sigma_draft=0.5, sigma_target=0.5, temperatures=(1.0,), seed=5151)
    base.update(kw)
    return synth.Workload(**base)


CASES = [
    _W("small_m1"),
    _W("m0", vocab=64, support=64, K=3, m=0, depth=2, budget=6, batch=32),
    _W("m2_bf16", vocab=500, K=5, m=2, depth=3, budget=14, dtype="bf16", batch=16, temperatures=(0.6, 1.2)),
    _W("chunks_bf16", vocab=50000, K=6, depth=4, budget=20, dtype="bf16", temperatures=(0.5, 0.8, 1.0)),
    _W("every_node", vocab=700, K=3, depth=3, budget=(3 + 1) + 2 * 3 * (3 + 1), batch=6),
    _W("budget1", vocab=700, K=3, depth=3, budget=1, batch=6),
]
VARIANTS = {"rrsw": rheo.VERIFY_RRSW, "onehot": rheo.VERIFY_ONEHOT}


def _cfg(w):
    return rheo.Config(batch=w.batch, vocab=w.vocab, K=w.K, depth=w.depth, budget=w.budget, m=w.m,
                       support=min(w.support, w.vocab), dtype=w.dtype)


@pytest.mark.parametrize("variant", list(VARIANTS))
@pytest.mark.parametrize("w", CASES, ids=[w.name for w in CASES])
def test_variant_parity(w, variant):
    v = VARIANTS[variant]
    cfg = _cfg(w)
    draft = synth.make_draft_inputs(w, device="cuda")
    g = ph.run_gpu(w, draft, cfg, variant=v)
    assert g.status == 0
    reqs = list(range(w.batch))
    o = ph.run_oracle(w, draft, cfg, reqs, variant=v)
    rep = ph.compare(cfg, g, o, reqs)
    print(w.name, variant, rep)
    assert rep.ok(), str(rep)
    assert len(rep.explained) <= max(1, len(reqs) // 20), str(rep)


@pytest.mark.parametrize("variant", list(VARIANTS))
def test_variant_parity_full_size_qwen3(variant):
    w = synth.WORKLOADS["qwen3_batch"]
    cfg = _cfg(w)
    draft = synth.make_draft_inputs(w, device="cuda")
    g = ph.run_gpu(w, draft, cfg, variant=VARIANTS[variant])
    assert g.status == 0
    reqs = [2, 9]
    o = ph.run_oracle(w, draft, cfg, reqs, variant=VARIANTS[variant])
    rep = ph.compare(cfg, g, o, reqs)
    assert rep.ok(), str(rep)


def test_rheo_variant_equals_rheo_verify():
    w = CASES[2]
    cfg = _cfg(w)
    draft = synth.make_draft_inputs(w, device="cuda")
    a = ph.run_gpu(w, draft, cfg)
    b = ph.run_gpu(w, draft, cfg, variant=rheo.VERIFY_RHEO)
    for k in ("acc_len", "acc_tok", "acc_node", "bonus"):
        np.testing.assert_array_equal(getattr(a, k), getattr(b, k))


def test_unknown_variant_rejected():
    import ctypes
    cfg = _cfg(CASES[0])
    rc = rheo.lib().rheo_verify_variant(ctypes.byref(cfg.c()), 7, None, 0, None, None, None, None, None, None,
                                        None, None)
    assert rc == rheo.RHEO_EINVAL
