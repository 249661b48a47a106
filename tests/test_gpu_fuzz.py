"""Seeded random configurations, GPU against the oracle: sparse support through
the parity harness, full support (App. B, row Full) through the full-support
comparison.  Each case draws the vocabulary size (log-uniform, 40..30,000),
the logit type, K, m, the support, the depth, the budget, the temperature
and the batch from a fixed seed, so a failure names a reproducible case."""
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


def _nodes(K, D):
    return 1 + (K + 1) + (D - 1) * K * (K + 1) if D > 1 else 1 + (K + 1)


def _case(i, full):
    rng = np.random.default_rng(90210 + 97 * i + (5000 if full else 0))
    V = int(np.exp(rng.uniform(np.log(40), np.log(30000))))
    K = int(rng.integers(1, 9))
    K = min(K, V - 1)
    m = int(rng.integers(0, min(K, 1 if full else 2) + 1))
    D = int(rng.integers(1, 5))
    G1 = _nodes(K, D)
    N = int(rng.integers(1, min(G1 - 1, 40) + 1))
    S = 0 if full else int(rng.integers(K + 1, min(V, 128) + 1))
    T = float(np.round(rng.choice([0.3, 0.6, 0.8, 1.0, 1.5]), 2))
    B = int(rng.integers(2, 7))
    dtype = "bf16" if rng.random() < 0.5 else "f32"
    name = f"{'full' if full else 'sparse'}{i}_V{V}_K{K}_m{m}_S{S}_D{D}_N{N}_{dtype}"
    return synth.Workload(name=name, batch=B, vocab=V, depth=D, K=K, budget=N, dtype=dtype, zipf_s=1.1,
                          sigma_draft=0.6, sigma_target=0.6, temperatures=(T,), m=m, support=S,
                          seed=1000 + i)


SPARSE = [_case(i, False) for i in range(24)]
FULL = [_case(i, True) for i in range(16)]


@pytest.mark.parametrize("w", SPARSE, ids=[w.name for w in SPARSE])
def test_fuzz_sparse(w):
    cfg = rheo.Config(batch=w.batch, vocab=w.vocab, K=w.K, depth=w.depth, budget=w.budget, m=w.m,
                      support=min(w.support, w.vocab), dtype=w.dtype)
    draft = synth.make_draft_inputs(w, device="cuda")
    g = ph.run_gpu(w, draft, cfg)
    assert g.status == 0, f"device status {g.status}"
    reqs = list(range(w.batch))
    o = ph.run_oracle(w, draft, cfg, reqs)
    rep = ph.compare(cfg, g, o, reqs)
    assert rep.ok(), str(rep)
    assert len(rep.explained) <= 1, str(rep)


@pytest.mark.parametrize("w", FULL, ids=[w.name for w in FULL])
def test_fuzz_full_support(w):
    import test_gpu_full_support as fs
    reqs = list(range(w.batch))
    assert fs._run(w, reqs) <= 1
    assert fs._cycle(w, reqs) <= 1
