"""Seeded synthetic workloads: Zipf-shaped draft and target logits.

Stand-ins for the LM heads of the paper's experiments (EAGLE-3 drafts of
Llama-3.1-8B / Vicuna-13B / DeepSeek-R1-Distill-8B on six benchmarks, Sec. 5.1),
whose weights and data are not available here.  A row is built from a random
permutation pi of the ranks 1..V:  l(v) = -s * ln(pi(v)) + N(0, sigma).  A
target row for a node whose draft row is known is that row plus N(0, sigma_t);
otherwise it is a fresh Zipf row plus the same noise.

This module holds no arithmetic of the method; both the CUDA path and the CPU
oracle receive the very tensors it produces.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import torch


@dataclass(frozen=True)
class Workload:
    name: str
    batch: int
    vocab: int
    depth: int
    K: int
    budget: int
    dtype: str              # "f32" | "bf16"
    zipf_s: float
    sigma_draft: float
    sigma_target: float
    temperatures: tuple     # per-request T values to draw from
    uniform_frac: float = 0.0   # rows replaced by near-uniform N(0, 0.1) logits
    m: int = 1
    support: int = 128
    seed: int = 1234


# The five workloads of the benchmark specification (tiny, Llama-3-8B-shaped,
# Qwen3-shaped batch, serving mix, stress).
WORKLOADS = {
    "tiny": Workload("tiny", 1, 1024, 3, 4, 16, "f32", 1.1, 0.5, 0.5, (1.0,), seed=1235),
    "llama8b": Workload("llama8b", 1, 128256, 6, 10, 60, "bf16", 1.1, 0.5, 0.7, (1.0,), seed=1236),
    "qwen3_batch": Workload("qwen3_batch", 16, 151936, 8, 8, 48, "bf16", 1.2, 0.5, 0.7, (0.7,), seed=1237),
    "serving_mix": Workload("serving_mix", 64, 128256, 6, 10, 60, "bf16", 1.1, 0.5, 0.7, (0.5, 0.8, 1.0), seed=1238),
    "stress": Workload("stress", 256, 151936, 10, 16, 128, "f32", 1.0, 0.5, 1.0, (1.0,), uniform_frac=0.01,
                       seed=1239),
}


def torch_dtype(w: Workload):
    return torch.bfloat16 if w.dtype == "bf16" else torch.float32


def rows_at(w: Workload, d: int) -> int:
    return 1 if d == 1 else w.K


def zipf_rows(gen: torch.Generator, n_rows: int, vocab: int, s: float, sigma: float, device,
              uniform_frac: float = 0.0, chunk_rows: int = 256) -> torch.Tensor:
    """[n_rows, vocab] float32 Zipf-shaped logits over random rank permutations."""
    out = torch.empty((n_rows, vocab), dtype=torch.float32, device=device)
    lnr = torch.log(torch.arange(1, vocab + 1, dtype=torch.float32, device=device))
    for r0 in range(0, n_rows, chunk_rows):
        r1 = min(n_rows, r0 + chunk_rows)
        perm = torch.argsort(torch.rand((r1 - r0, vocab), generator=gen, device=device), dim=1)
        rows = -s * lnr[perm]
        rows += sigma * torch.randn((r1 - r0, vocab), generator=gen, device=device)
        out[r0:r1] = rows
    if uniform_frac > 0:
        pick = torch.rand(n_rows, generator=gen, device=device) < uniform_frac
        k = int(pick.sum().item())
        if k:
            out[pick] = 0.1 * torch.randn((k, vocab), generator=gen, device=device)
    return out


@dataclass
class DraftInputs:
    workload: Workload
    rows: list                      # rows[d-1]: [B, F_d, V] tensor of the workload dtype
    temperature: torch.Tensor       # [B] float32
    seed: torch.Tensor              # [B] int64 (bit pattern of the uint64 Philox key)
    offset: torch.Tensor            # [B] int64
    extra: dict = field(default_factory=dict)


def splitmix64(x: int) -> int:
    x = (x + 0x9E3779B97F4A7C15) & 0xFFFFFFFFFFFFFFFF
    z = x
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & 0xFFFFFFFFFFFFFFFF
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & 0xFFFFFFFFFFFFFFFF
    return z ^ (z >> 31)


def as_int64(u: int) -> int:
    return u - (1 << 64) if u >= (1 << 63) else u


def make_draft_inputs(w: Workload, device="cpu", batch: int | None = None, gen_device=None) -> DraftInputs:
    """Draft rows for every depth, per-request temperatures, Philox seeds and offsets."""
    B = w.batch if batch is None else batch
    gdev = device if gen_device is None else gen_device
    gen = torch.Generator(device=gdev)
    gen.manual_seed(w.seed)
    dt = torch_dtype(w)
    rows = []
    for d in range(1, w.depth + 1):
        F = rows_at(w, d)
        r = zipf_rows(gen, B * F, w.vocab, w.zipf_s, w.sigma_draft, gdev, w.uniform_frac)
        rows.append(r.to(dt).reshape(B, F, w.vocab).to(device))
    tg = torch.Generator(device="cpu")
    tg.manual_seed(w.seed + 17)
    Ts = torch.tensor(w.temperatures, dtype=torch.float32)
    T = Ts[torch.randint(0, len(w.temperatures), (B,), generator=tg)].to(device)
    seed = torch.tensor([as_int64(splitmix64(w.seed ^ b)) for b in range(B)], dtype=torch.int64, device=device)
    offset = torch.zeros(B, dtype=torch.int64, device=device)
    return DraftInputs(w, rows, T, seed, offset)


def target_rows(w: Workload, draft: DraftInputs, frontiers: list, pruned_gen_ids: torch.Tensor,
                device=None, noise_seed: int | None = None, request_ids=None) -> torch.Tensor:
    """Target logits [B, N+1, V] in pruned order.

    frontiers[d-1] ([B, K] gen ids) are the nodes whose rows were fed at depth
    d+1; together with the root (row of depth 1) they identify the expanded
    nodes, whose target row is their draft row plus N(0, sigma_t).  Noise and
    fresh rows are keyed by (request id, gen id), so two trees that agree get
    the same target tensor.  request_ids[b] names request b of this batch (for
    sub-batches of a larger workload).
    """
    device = draft.rows[0].device if device is None else device
    B, NP = pruned_gen_ids.shape
    V = w.vocab
    ids = list(range(B)) if request_ids is None else [int(x) for x in request_ids]
    base = w.seed * 1000003 if noise_seed is None else noise_seed
    gids = pruned_gen_ids.cpu()
    src = {}
    for b in range(B):
        src[(b, 0)] = (0, 0)
        for d, fr in enumerate(frontiers, start=2):
            for f, g in enumerate(fr[b].cpu().tolist()):
                src[(b, int(g))] = (d - 1, f)
    out = torch.empty((B, NP, V), dtype=torch_dtype(w), device=device)
    for b in range(B):
        for i in range(NP):
            g = int(gids[b, i])
            gen = torch.Generator(device=device)
            gen.manual_seed(base + ids[b] * 65537 + g)
            noise = w.sigma_target * torch.randn(V, generator=gen, device=device)
            if (b, g) in src:
                d0, f = src[(b, g)]
                row = draft.rows[d0][b, f].to(device).float() + noise
            else:
                row = zipf_rows(gen, 1, V, w.zipf_s, w.sigma_draft, device)[0] + noise
            out[b, i] = row.to(out.dtype)
    return out
