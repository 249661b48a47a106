"""GPU parity of full support (support = 0: the sampled token over the whole
vocabulary; App. B, Table tab:sparse_support, row Full) against the oracle.

Expansion and prune on both sides from the same seeded draft rows: tokens,
parents, slots, frontiers and pruned trees bit-exact, scores / log proxies /
lse1 / lse_tail within the log-domain tolerance, q~(Y) within rtol 1e-5; a
request whose first difference sits at a Gumbel or frontier decision with an
oracle margin below 1e-6 counts as an explained near-tie flip.
"""
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
    base = dict(name=name, batch=6, vocab=3000, depth=3, K=4, budget=12, dtype="f32", zipf_s=1.1,
                sigma_draft=0.5, sigma_target=0.5, temperatures=(1.0,), seed=8181)
    base.update(kw)
    return synth.Workload(**base)


CASES = [
    _W("small"),
    _W("v40_m0", vocab=40, K=3, m=0, depth=2, budget=6, batch=16),
    _W("m1_bf16", vocab=5000, K=5, m=1, depth=3, budget=14, dtype="bf16", temperatures=(0.6, 1.3)),
    _W("ragged", vocab=20011, K=6, m=1, depth=3, budget=20, dtype="bf16", temperatures=(0.8,)),
    _W("low_T", vocab=2000, K=4, depth=3, budget=10, temperatures=(0.05,)),
    # rows cut into segments over the SMs (a segment per tile), merged by the
    # row's last CTA: m = 0 (no lead left out), and T = 0.05 over five fp32 tiles
    _W("seg_m0", vocab=20011, K=5, m=0, depth=3, budget=12, dtype="bf16", temperatures=(0.9,)),
    _W("seg_low_T", vocab=40000, K=4, m=1, depth=3, budget=10, temperatures=(0.05,)),
    # a one-token last block of the two-stage draw (V = 257), in both dtypes
    _W("v257_bf16", vocab=257, K=4, m=1, depth=3, budget=10, dtype="bf16", batch=8),
    _W("v257_f32_m0", vocab=257, K=4, m=0, depth=3, budget=10, batch=8, temperatures=(1.3,)),
    # the largest vocabulary the library accepts: 1024 blocks, 2048 fp32 groups a row
    _W("max_vocab_bf16", vocab=262144, K=4, m=1, depth=2, budget=8, batch=2, dtype="bf16", temperatures=(0.8,)),
    _W("max_vocab_f32", vocab=262144, K=4, m=0, depth=2, budget=8, batch=2, temperatures=(0.6,)),
]


def _cfg(w):
    return rheo.Config(batch=w.batch, vocab=w.vocab, K=w.K, depth=w.depth, budget=w.budget, m=w.m, support=0,
                       dtype=w.dtype)


def _masked(draft):
    """Most logits of every draft row set to -inf (a masked vocabulary), a few
    finite ones kept at the start and the end of the row."""
    g = torch.Generator(device="cuda")
    g.manual_seed(11)
    for r in draft.rows:
        mask = torch.rand(r.shape, generator=g, device=r.device) < 0.9
        mask[..., :16] = False
        mask[..., -16:] = False
        r.masked_fill_(mask, float("-inf"))


def _run(w, reqs, transform=None):
    import oracle
    cfg = _cfg(w)
    draft = synth.make_draft_inputs(w, device="cuda")
    if transform:
        transform(draft)
    tree, pr, ws = rheo.Tree(cfg), rheo.Pruned(cfg), rheo.Workspace(cfg)
    for d in range(1, cfg.depth + 1):
        rheo.expand(cfg, d, draft.rows[d - 1], draft.temperature, draft.seed, draft.offset, tree, ws)
    rheo.prune(cfg, tree, pr, ws)
    assert rheo.status(cfg, ws) == 0
    ocfg = oracle.Config(B=len(reqs), V=w.vocab, K=w.K, m=w.m, S=0, D=w.depth, N=w.budget, eps=cfg.eps)
    ot = oracle.Tree(ocfg)
    T = draft.temperature.cpu().numpy()[reqs]
    seed, off = ph.u64(draft.seed)[reqs], ph.u64(draft.offset)[reqs]
    for d in range(1, w.depth + 1):
        oracle.expand(ocfg, d, draft.rows[d - 1][reqs].float().cpu().numpy(), T, seed, off, ot)
    op = oracle.prune(ocfg, ot)
    g = {k: getattr(tree, k).cpu().numpy() for k in ("token", "parent", "slot", "score", "log_proxy", "qtilde",
                                                      "lse1", "lse_tail")}
    gp = {k: getattr(pr, k).cpu().numpy() for k in ("gen_id", "parent", "first_child", "n_child", "sampled_child")}
    explained = 0
    for j, b in enumerate(reqs):
        same = (np.array_equal(g["token"][b], ot.token[j]) and np.array_equal(g["parent"][b], ot.parent[j])
                and np.array_equal(g["slot"][b], ot.slot[j]) and np.array_equal(gp["gen_id"][b], op.gen_id[j]))
        if not same:
            gap = min(float(np.min(ot.gap_sample[j])), float(np.min(ot.gap_frontier[j])), float(op.gap_prune[j]))
            assert gap < ph.GAP, f"{w.name} request {b}: trees differ, oracle margin {gap}"
            explained += 1
            continue
        for k in ("parent", "first_child", "n_child", "sampled_child"):
            np.testing.assert_array_equal(gp[k][b], getattr(op, k)[j], err_msg=k)
        for k in ("score", "log_proxy", "lse1", "lse_tail"):
            a, o = g[k][b].astype(np.float64), getattr(ot, k)[j].astype(np.float64)
            assert np.all(np.abs(a - o) <= ph.LOG_ATOL + ph.RTOL * np.abs(o)), (w.name, b, k)
        a, o = g["qtilde"][b].astype(np.float64), ot.qtilde[j].astype(np.float64)
        assert np.all(np.abs(a - o) <= ph.ATOL + ph.RTOL * np.abs(o)), (w.name, b, "qtilde")
    return explained


@pytest.mark.parametrize("w", CASES, ids=[w.name for w in CASES])
def test_full_support_tree_parity(w):
    reqs = list(range(w.batch))
    assert _run(w, reqs) <= 1


def test_full_support_requires_m_at_most_one():
    import ctypes
    cfg = rheo.Config(batch=2, vocab=1000, K=4, depth=2, budget=8, m=2, support=0, dtype="f32")
    sz = ctypes.c_size_t()
    assert rheo.lib().rheo_sizes(ctypes.byref(cfg.c()), None, None, ctypes.byref(sz)) == rheo.RHEO_EINVAL


def test_full_support_tree_parity_qwen3_size():
    w = synth.WORKLOADS["qwen3_batch"]
    assert _run(w, [1, 12]) <= 1


def _cycle(w, reqs, transform=None):
    """Full cycle with full support on both sides; returns (explained flips, requests compared)."""
    import oracle
    cfg = _cfg(w)
    draft = synth.make_draft_inputs(w, device="cuda")
    if transform:
        transform(draft)
    tree, pr, ws, out = rheo.Tree(cfg), rheo.Pruned(cfg), rheo.Workspace(cfg), rheo.VerifyOut(cfg)
    frontiers = []
    for d in range(1, cfg.depth + 1):
        rheo.expand(cfg, d, draft.rows[d - 1], draft.temperature, draft.seed, draft.offset, tree, ws)
        if d < cfg.depth:
            frontiers.append(tree.frontier.clone())
    rheo.prune(cfg, tree, pr, ws)
    tgt = synth.target_rows(w, draft, frontiers, pr.gen_id)
    rheo.verify_full(cfg, tgt, draft.rows, draft.temperature, draft.seed, draft.offset, tree, pr, out, ws)
    assert rheo.status(cfg, ws) == 0
    ocfg = oracle.Config(B=len(reqs), V=w.vocab, K=w.K, m=w.m, S=0, D=w.depth, N=w.budget, eps=cfg.eps)
    ot = oracle.Tree(ocfg)
    T = draft.temperature.cpu().numpy()[reqs]
    seed, off = ph.u64(draft.seed)[reqs], ph.u64(draft.offset)[reqs]
    ofr = []
    for d in range(1, w.depth + 1):
        oracle.expand(ocfg, d, draft.rows[d - 1][reqs].float().cpu().numpy(), T, seed, off, ot)
        if d < w.depth:
            ofr.append(ot.frontier.copy())
    op = oracle.prune(ocfg, ot)
    sub = synth.DraftInputs(w, [r_[reqs] for r_ in draft.rows], draft.temperature[reqs], draft.seed[reqs],
                            draft.offset[reqs])
    otg = synth.target_rows(w, sub, [torch.from_numpy(f) for f in ofr], torch.from_numpy(op.gen_id.copy()),
                            device=draft.rows[0].device, request_ids=reqs)
    oo = oracle.verify(ocfg, otg.float().cpu().numpy(), T, seed, off, ot, op)
    explained = 0
    gl, gt, gb = out.accepted_len.cpu().numpy(), out.accepted_tokens.cpu().numpy(), out.bonus_token.cpu().numpy()
    for j, b in enumerate(reqs):
        same = (gl[b] == oo.accepted_len[j] and np.array_equal(gt[b], oo.accepted_tokens[j])
                and gb[b] == oo.bonus_token[j])
        if not same:
            gap = min(float(np.min(ot.gap_sample[j])), float(np.min(ot.gap_frontier[j])), float(op.gap_prune[j]),
                      float(np.min(oo.gap_level[j])))
            assert gap < ph.GAP, f"{w.name} request {b}: verification differs, oracle margin {gap}"
            explained += 1
    return explained


@pytest.mark.parametrize("w", CASES, ids=[w.name for w in CASES])
def test_full_support_verification_parity(w):
    assert _cycle(w, list(range(w.batch))) <= 1


def test_full_support_verification_parity_qwen3_size():
    w = synth.WORKLOADS["qwen3_batch"]
    assert _cycle(w, [4, 13]) <= 1


def test_sparse_entry_points_reject_full_support():
    import ctypes
    cfg = _cfg(CASES[0])
    rc = rheo.lib().rheo_verify_variant(ctypes.byref(cfg.c()), 0, None, 0, None, None, None, None, None, None,
                                        None, None)
    assert rc == rheo.RHEO_EINVAL


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_full_support_masked_vocab(dtype):
    """90 % of every draft row at -inf, rows cut into segments (V = 20011): the
    group sums, the block masses and both draws skip the masked tokens."""
    w = _W(f"masked_full_{dtype}", vocab=20011, K=4, m=1, depth=3, budget=10, dtype=dtype, temperatures=(0.8,))
    assert _run(w, list(range(w.batch)), transform=_masked) <= 1
    assert _cycle(w, list(range(w.batch)), transform=_masked) <= 1
