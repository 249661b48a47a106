"""Benchmark: tree-steps/s of the RheoSampling hot path (expand x D + prune + verify).

One step = D rheo_expand calls, one rheo_prune and one rheo_verify for all B
requests of the Qwen3-shaped batch workload (B = 16, V = 151,936, bf16, D = 8,
K = 8 (+1 sampled), N = 48, T = 0.7) on synthetic Zipf(1.2) logits.  Inputs for
every depth and the target rows are resident in HBM before the timed region
(515 MB per step, four times the 129 MB L2, so no flush is needed).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference] [--workload NAME]

For N > 1 (torchrun) every rank runs its own replica of the workload on its GPU
(requests are independent: no data-path collective); the timing is the max
over ranks and value counts the tree-steps of all ranks.
"""
from __future__ import annotations

import argparse
import dataclasses
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "tree-steps/sec (expand+prune+verify) at batch B, vocab V; HBM GB/s vs peak"


KERNEL_SOURCES = ("expand.cu", "rheo_device.cuh", "rheo_kernels.h", "stream.cuh")


def kernel_sources_sha() -> str:
    """sha256 over the sources the expand kernel is compiled from (traffic taken
    from an ncu capture is reported only while these are unchanged)."""
    import hashlib

    h = hashlib.sha256()
    for name in KERNEL_SOURCES:
        with open(os.path.join(ROOT, "paper_2609_21827_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def _traffic(key: str):
    """DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) from
    the committed ncu summary, or None if absent or taken on other sources."""
    try:
        with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
            e = json.load(f).get(key)
        if e and e.get("sources_sha256") == kernel_sources_sha():
            return e["bytes_per_launch"]
    except Exception:
        pass
    return None


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, interval_ms: int = 20):
        self.path = tempfile.mktemp(prefix="rheo_clocks_", suffix=".csv")
        self.proc = None
        self.gpu = gpu_index
        self.interval_ms = interval_ms

    def __enter__(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", str(self.interval_ms)],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *a):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.fh.close()

    def summary(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"], "samples": 0}
        with open(self.path) as f:
            lines = f.readlines()
        os.unlink(self.path)
        return self.parse(lines)

    @staticmethod
    def parse(lines):
        """Median SM clock, max clock and active throttle reasons of nvidia-smi CSV lines."""
        rows = []
        for line in lines:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), parts[5:9]))
            except ValueError:
                continue
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for _, _, fl in rows for n, v in zip(names, fl) if v.lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


def _dist():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def reduce_max_time(seconds: float, world: int, device=None) -> float:
    """Max of a per-rank duration over all ranks (no-op for one rank)."""
    if world == 1:
        return seconds
    import torch
    import torch.distributed as dist

    t = torch.tensor([seconds], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


def oracle_cycle(w, draft, reqs):
    """One CPU-oracle cycle on requests `reqs` of the workload inputs.

    Expansion and prune are timed, target rows are built (untimed) from the
    oracle's own pruned tree, then verification is timed.  Returns the seconds
    and the oracle's tree, pruned tree and verification outputs."""
    import numpy as np
    import torch

    import oracle
    from paper_2609_21827_gb300 import synth

    reqs = list(reqs)
    ocfg = oracle.Config(B=len(reqs), V=w.vocab, K=w.K, m=w.m, S=min(w.support, w.vocab), D=w.depth, N=w.budget)
    rows = [r[reqs].float().cpu().numpy() for r in draft.rows]
    T = draft.temperature.cpu().numpy()[reqs]
    seed = draft.seed.cpu().numpy().view(np.uint64)[reqs]
    off = draft.offset.cpu().numpy().view(np.uint64)[reqs]
    t0 = time.perf_counter()
    tree = oracle.Tree(ocfg)
    frontiers = []
    for d in range(1, w.depth + 1):
        oracle.expand(ocfg, d, rows[d - 1], T, seed, off, tree)
        if d < w.depth:
            frontiers.append(tree.frontier.copy())
    pr = oracle.prune(ocfg, tree)
    t_build = time.perf_counter() - t0
    sub = synth.DraftInputs(w, [r[reqs] for r in draft.rows], draft.temperature[reqs], draft.seed[reqs],
                            draft.offset[reqs])
    tgt = synth.target_rows(w, sub, [torch.from_numpy(f) for f in frontiers], torch.from_numpy(pr.gen_id.copy()),
                            request_ids=reqs).float().cpu().numpy()
    t1 = time.perf_counter()
    out = oracle.verify(ocfg, tgt, T, seed, off, tree, pr)
    return t_build + (time.perf_counter() - t1), tree, pr, out


PRUNED_FIELDS = ("gen_id", "token", "parent", "depth", "first_child", "n_child", "sampled_child")
FLIP_GAP = 1e-6


def gpu_outputs(tree, pr, out):
    """Host copies of the integer results of a GPU cycle (for the parity report)."""
    g = {k: getattr(tree, k).cpu().numpy() for k in ("token", "parent", "slot")}
    g.update({"pr_" + k: getattr(pr, k).cpu().numpy() for k in PRUNED_FIELDS})
    g.update(acc_len=out.accepted_len.cpu().numpy(), acc_tok=out.accepted_tokens.cpu().numpy(),
             acc_node=out.accepted_nodes.cpu().numpy(), bonus=out.bonus_token.cpu().numpy())
    return g


def parity_summary(w, g, reqs, ot, op, oo):
    """GPU against oracle on requests `reqs`: every integer result compared
    bit for bit (trees depth by depth, the pruned tree, the accepted path and
    the bonus token).  A request that differs is an explained near-tie flip
    when the oracle's relative margin at the first divergent decision is below
    FLIP_GAP, else unexplained."""
    import numpy as np

    K, D = w.K, w.depth
    exact, flips, bad = 0, [], []
    for j, b in enumerate(reqs):
        why = None
        for d in range(1, D + 1):
            F = 1 if d == 1 else K
            base = 1 if d == 1 else 1 + (K + 1) + (d - 2) * K * (K + 1)
            sl = slice(base, base + F * (K + 1))
            if d >= 2 and not np.array_equal(g["parent"][b, sl], ot.parent[j, sl]):
                why = ("frontier", float(ot.gap_frontier[j, d - 2]))
            elif not np.array_equal(g["token"][b, sl], ot.token[j, sl]):
                for f in range(F):
                    ps = slice(base + f * (K + 1), base + (f + 1) * (K + 1))
                    if not np.array_equal(g["token"][b, ps], ot.token[j, ps]):
                        e = 0 if d == 1 else 1 + (d - 2) * K + f
                        why = ("sample", float(ot.gap_sample[j, e]))
                        break
            elif not np.array_equal(g["slot"][b, sl], ot.slot[j, sl]):
                why = ("pool", 1.0)
            if why:
                break
        if why is None and not np.array_equal(g["pr_gen_id"][b], op.gen_id[j]):
            why = ("prune", float(op.gap_prune[j]))
        if why is None and any(not np.array_equal(g["pr_" + k][b], getattr(op, k)[j]) for k in PRUNED_FIELDS):
            why = ("pruned_fields", 1.0)
        if why is None:
            lvl = None
            for i in range(D):
                if g["acc_node"][b, i] != oo.accepted_nodes[j, i] or g["acc_tok"][b, i] != oo.accepted_tokens[j, i]:
                    lvl = i
                    break
            if lvl is None and (g["acc_len"][b] != oo.accepted_len[j] or g["bonus"][b] != oo.bonus_token[j]):
                lvl = min(int(oo.accepted_len[j]), int(g["acc_len"][b]))
            if lvl is not None:
                why = ("verify", float(oo.gap_level[j, lvl]))
        if why is None:
            exact += 1
        elif why[1] < FLIP_GAP:
            flips.append({"request": int(b), "at": why[0], "gap": why[1]})
        else:
            bad.append({"request": int(b), "at": why[0], "gap": why[1]})
    return {"requests": len(reqs), "exact": exact, "explained_flips": len(flips), "unexplained": len(bad),
            "flips": flips, "mismatches": bad[:8], "flip_gap": FLIP_GAP,
            "compared": "tree tokens, parents and slots at every depth, pruned tree, accepted path, bonus token"}


def cpu_model() -> str:
    """The host CPU's model name (lscpu), else the machine type."""
    import platform
    import subprocess

    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return f"{line.split(':', 1)[1].strip()} ({platform.machine()}, {os.cpu_count()} logical CPUs)"
    except Exception:
        pass
    return f"{platform.machine()} ({os.cpu_count()} logical CPUs)"


def cpu_baseline(w, draft, gpu=None, budget_s=12.0, budget_1t_s=6.0):
    """The oracle as it stands, on the host cores, over a bounded sample: whole
    cycles of the batch (or of its first requests) repeated for about budget_s
    with every core, then cycles of single requests on one thread for about
    budget_1t_s.  With `gpu` (the GPU's results of the same inputs), the last
    all-core cycle's results are also compared with them (parity report)."""
    import oracle

    oracle.build()
    threads0 = oracle.max_threads()
    first, *_ = oracle_cycle(w, draft, [0])
    n = max(1, min(w.batch, int(budget_s / max(first, 1e-3))))
    oracle.threads_used(reset=True)
    secs, cycles, last = 0.0, 0, None
    while cycles == 0 or (secs < budget_s * 0.7 and cycles < 50):
        t, *last = oracle_cycle(w, draft, range(n))
        secs += t
        cycles += 1
    used = oracle.threads_used(reset=True)
    per_step = secs / cycles * w.batch / n
    # one thread: single requests in turn
    oracle.set_threads(1)
    secs1, cyc1 = 0.0, 0
    try:
        while cyc1 == 0 or (secs1 < budget_1t_s and cyc1 < 4 * w.batch):
            t, *_ = oracle_cycle(w, draft, [cyc1 % w.batch])
            secs1 += t
            cyc1 += 1
        used1 = oracle.threads_used(reset=True)
    finally:
        oracle.set_threads(threads0)
    base = {"value": 1.0 / per_step, "unit": "tree-steps/s", "cores": used, "kind": "oracle", "cpu": cpu_model(),
            "sample": f"{cycles} cycles of {n} of {w.batch} requests of {w.name} ({secs:.1f} s), scaled to the "
                      f"full batch; cores = OpenMP threads that ran part of the oracle's loops",
            "one_thread": {"value": 1.0 / (secs1 / cyc1 * w.batch), "unit": "tree-steps/s", "cores": used1,
                           "sample": f"{cyc1} cycles of single requests ({secs1:.1f} s), scaled to the full batch"}}
    par = parity_summary(w, gpu, list(range(n)), *last) if gpu is not None else None
    return base, par


def build_inputs(w, device):
    import torch

    from paper_2609_21827_gb300 import rheo, synth

    draft = synth.make_draft_inputs(w, device=device)
    cfg = rheo.Config(batch=w.batch, vocab=w.vocab, K=w.K, depth=w.depth, budget=w.budget, m=w.m,
                      support=min(w.support, w.vocab), dtype=w.dtype)
    tree, pr, out, ws = rheo.Tree(cfg), rheo.Pruned(cfg), rheo.VerifyOut(cfg, row_lse=False), rheo.Workspace(cfg)
    frontiers = []
    for d in range(1, cfg.depth + 1):
        rheo.expand(cfg, d, draft.rows[d - 1], draft.temperature, draft.seed, draft.offset, tree, ws)
        if d < cfg.depth:
            frontiers.append(tree.frontier.clone())
    rheo.prune(cfg, tree, pr, ws)
    target = synth.target_rows(w, draft, frontiers, pr.gen_id)
    torch.cuda.synchronize()
    return cfg, draft, target, tree, pr, out, ws


def run_reference(args, w):
    """--impl reference: the CPU oracle on this machine's host cores, same workload and metric.
    Each step is a bounded sample (one request of the batch), scaled to B requests."""
    import torch

    world, rank, local = _dist()
    if rank != 0:
        return 0
    import oracle
    from paper_2609_21827_gb300 import synth

    oracle.build()
    device = "cuda" if torch.cuda.is_available() else "cpu"
    draft = synth.make_draft_inputs(w, device=device)
    times = []
    oracle.threads_used(reset=True)
    for i in range(args.warmup + args.steps):
        t, *_ = oracle_cycle(w, draft, [i % w.batch])
        if i >= args.warmup:
            times.append(t * w.batch)
    per_step = sum(times) / len(times)
    cores = oracle.threads_used(reset=True)
    value = 1.0 / per_step
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tree-steps/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": per_step * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": w.name, "batch": w.batch, "vocab": w.vocab, "depth": w.depth, "K": w.K,
                       "support": min(w.support, w.vocab) if w.support else "full",
                       "budget": w.budget, "logits": w.dtype},
            "cpu_baseline": {"value": value, "unit": "tree-steps/s", "cores": cores, "kind": "oracle",
                             "cpu": cpu_model(),
                             "sample": f"1 of {w.batch} requests per step, scaled to the full batch; cores = "
                                       f"OpenMP threads that ran part of the oracle's loops"},
            "e2e": {"value": value, "unit": "tree-steps/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--workload", default="qwen3_batch")
    ap.add_argument("--e2e-steps", type=int, default=50,
                    help="steps of the end-to-end measurement through host buffers (0: leave it out)")
    ap.add_argument("--copy-streams", type=int, default=2,
                    help="copy streams sharing the host-to-device copies of the end-to-end measurement")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--batch", type=int, default=0,
                    help="override the workload's batch (a smaller case of the same kernels, for profiling)")
    ap.add_argument("--no-extras", action="store_true",
                    help="skip the verification variants, the synthetic-model cycles and the full-support step "
                         "(for launch lists of the tree step alone)")
    ap.add_argument("--depth", type=int, default=0,
                    help="override the workload's depth (fewer expansion launches of the same shape, for profiling)")
    ap.add_argument("--support", type=int, default=-1,
                    help="override the workload's top-S support; 0 = full support (App. B, Table "
                         "tab:sparse_support, row Full: the sampled token over the whole vocabulary)")
    args = ap.parse_args(argv)
    args.warmup = max(3, args.warmup)

    from paper_2609_21827_gb300 import build as lib_build
    from paper_2609_21827_gb300 import synth

    w = synth.WORKLOADS[args.workload]
    if args.batch > 0 and args.batch != w.batch:
        w = dataclasses.replace(w, name=f"{w.name}_b{args.batch}", batch=args.batch)
    if args.depth > 0 and args.depth != w.depth:
        w = dataclasses.replace(w, name=f"{w.name}_d{args.depth}", depth=args.depth)
    if args.support >= 0 and args.support != w.support:
        w = dataclasses.replace(w, name=f"{w.name}_s{args.support}" if args.support else f"{w.name}_full",
                                support=args.support)
    if args.impl == "reference":
        return run_reference(args, w)

    import torch

    world, rank, local = _dist()
    if world > 1:
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    device = f"cuda:{local}" if world > 1 else "cuda:0"
    torch.cuda.set_device(device)
    lib_build.build()
    from paper_2609_21827_gb300 import rheo

    cfg, draft, target, tree, pr, out, ws = build_inputs(w, device)
    D = cfg.depth
    esz = 2 if w.dtype == "bf16" else 4
    exp_rows = [w.batch * (1 if d == 1 else w.K) for d in range(1, D + 1)]
    expand_bytes = sum(exp_rows) * w.vocab * esz
    verify_bytes = w.batch * (w.budget + 1) * w.vocab * esz

    full = cfg.support == 0  # full support verifies against the expanded nodes' draft rows

    def verify_call(tgt, rows, T, seed, off, s):
        if full:
            rheo.verify_full(cfg, tgt, rows, T, seed, off, tree, pr, out, ws, s)
        else:
            rheo.verify(cfg, tgt, T, seed, off, tree, pr, out, ws, s)

    stream = torch.cuda.Stream(device=device)
    stream.wait_stream(torch.cuda.current_stream())
    try:  # events that become record nodes of the captured graph
        ev = [torch.cuda.Event(enable_timing=True, external=True) for _ in range(D + 3)]
        graph_events = True
    except TypeError:
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(D + 3)]
        graph_events = False

    def step(s, with_events):
        if with_events:
            ev[0].record(s)
        for d in range(1, D + 1):
            rheo.expand(cfg, d, draft.rows[d - 1], draft.temperature, draft.seed, draft.offset, tree, ws, s)
            if with_events:
                ev[d].record(s)
        rheo.prune(cfg, tree, pr, ws, s)
        if with_events:
            ev[D + 1].record(s)
        verify_call(target, draft.rows, draft.temperature, draft.seed, draft.offset, s)
        if with_events:
            ev[D + 2].record(s)

    # the depth >= 2 expansions back to back, as in the timed step, bracketed
    # by two events only (the launches between them keep their programmatic
    # dependent launch): their average duration is the dominant kernel's
    evb = [torch.cuda.Event(enable_timing=True, external=True) if graph_events else
           torch.cuda.Event(enable_timing=True) for _ in range(2)]

    def step_blk(s):
        rheo.expand(cfg, 1, draft.rows[0], draft.temperature, draft.seed, draft.offset, tree, ws, s)
        evb[0].record(s)
        for d in range(2, D + 1):
            rheo.expand(cfg, d, draft.rows[d - 1], draft.temperature, draft.seed, draft.offset, tree, ws, s)
        evb[1].record(s)
        rheo.prune(cfg, tree, pr, ws, s)
        verify_call(target, draft.rows, draft.temperature, draft.seed, draft.offset, s)

    # the whole step as one CUDA graph of its kernels alone (timed); a second
    # graph with event record nodes between the calls gives per-call durations
    graph = torch.cuda.CUDAGraph()
    graph_ev = torch.cuda.CUDAGraph() if graph_events else None
    with torch.cuda.stream(stream):
        step(stream, False)
        stream.synchronize()
        with torch.cuda.graph(graph, stream=stream):
            step(stream, False)
        if graph_events:
            with torch.cuda.graph(graph_ev, stream=stream):
                step(stream, True)
            graph_blk = torch.cuda.CUDAGraph()
            with torch.cuda.graph(graph_blk, stream=stream):
                step_blk(stream)
    for _ in range(args.warmup):
        graph.replay()
    torch.cuda.synchronize()
    assert rheo.status(cfg, ws, stream) == 0

    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    soak_s = 0.4
    with Clocks(torch.cuda.current_device()) as clk:
        # the same graph replayed for soak_s right before the timed steps, so
        # that the sampler (every 20 ms) sees this load's clocks even when the
        # timed steps last a few milliseconds
        with torch.cuda.stream(stream):
            t_end = time.time() + soak_s
            while time.time() < t_end:
                for _ in range(25):
                    graph.replay()
                stream.synchronize()
        barrier(world)
        torch.cuda.synchronize()
        with torch.cuda.stream(stream):
            start.record(stream)
            for _ in range(args.steps):
                graph.replay()
            stop.record(stream)
        torch.cuda.synchronize()
        barrier(world)
    local_s = start.elapsed_time(stop) / 1e3
    secs = reduce_max_time(local_s, world, device)
    clocks = clk.summary()
    clocks["window"] = f"{soak_s} s of the same step replayed right before the timed steps, and the timed steps"
    gpu_res = gpu_outputs(tree, pr, out) if rank == 0 else None

    # per-kernel durations: replays (or eager steps when captured events are not
    # available) with a synchronise after each, events read every time
    n_k = min(200, args.steps)
    exp_ms, prune_ms, ver_ms = 0.0, 0.0, 0.0
    by_depth = [0.0] * D
    with torch.cuda.stream(stream):
        for _ in range(n_k):
            if graph_events:
                graph_ev.replay()
            else:
                step(stream, True)
            stream.synchronize()
            exp_ms += ev[0].elapsed_time(ev[D])
            for d in range(D):
                by_depth[d] += ev[d].elapsed_time(ev[d + 1])
            prune_ms += ev[D].elapsed_time(ev[D + 1])
            ver_ms += ev[D + 1].elapsed_time(ev[D + 2])
    exp_ms /= n_k
    prune_ms /= n_k
    ver_ms /= n_k
    blk_ms = 0.0
    if D >= 2:
        with torch.cuda.stream(stream):
            for _ in range(n_k):
                if graph_events:
                    graph_blk.replay()
                else:
                    step_blk(stream)
                stream.synchronize()
                blk_ms += evb[0].elapsed_time(evb[1])
        blk_ms /= n_k
    assert rheo.status(cfg, ws, stream) == 0


    variants, synthetic_lm, full_support, attn_us = None, None, None, None
    if not args.no_extras and not full:
        # tree-attention inputs of the target forward (not part of the tree step):
        # 20 launches in one graph, averaged over replays
        attn = rheo.TreeAttn(cfg, device=device)
        g_attn = torch.cuda.CUDAGraph()
        with torch.cuda.stream(stream):
            rheo.tree_attention(cfg, pr, attn, ws, stream)
            stream.synchronize()
            with torch.cuda.graph(g_attn, stream=stream):
                for _ in range(20):
                    rheo.tree_attention(cfg, pr, attn, ws, stream)
            for _ in range(3):
                g_attn.replay()
            a0, a1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a0.record(stream)
            for _ in range(10):
                g_attn.replay()
            a1.record(stream)
            stream.synchronize()
        attn_us = a0.elapsed_time(a1) * 1e3 / 200
        assert rheo.status(cfg, ws, stream) == 0
        # verification variants (App. A, App. D.2) on the same trees and targets:
        # per-call time on this step's tree, and the mean accepted length over the
        # requests of 8 more cycles (Philox offsets 1..8), paired across variants
        variants = {}
        names = {"rheo": rheo.VERIFY_RHEO, "rrsw": rheo.VERIFY_RRSW, "onehot": rheo.VERIFY_ONEHOT}
        vout = rheo.VerifyOut(cfg, row_lse=False, device=device)
        for name, v in names.items():
            with torch.cuda.stream(stream):
                for _ in range(3):
                    rheo.verify_variant(cfg, v, target, draft.temperature, draft.seed, draft.offset, tree, pr, vout, ws,
                                        stream)
                v0, v1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                v0.record(stream)
                for _ in range(50):
                    rheo.verify_variant(cfg, v, target, draft.temperature, draft.seed, draft.offset, tree, pr, vout, ws,
                                        stream)
                v1.record(stream)
                stream.synchronize()
            variants[name] = {"verify_us": v0.elapsed_time(v1) * 1e3 / 50, "accepted": []}
        off0 = draft.offset.clone()
        for off in range(1, 9):
            draft.offset.fill_(off)
            tr2, pr2 = rheo.Tree(cfg, device=device), rheo.Pruned(cfg, device=device)
            fr2 = []
            for d in range(1, D + 1):
                rheo.expand(cfg, d, draft.rows[d - 1], draft.temperature, draft.seed, draft.offset, tr2, ws)
                if d < D:
                    fr2.append(tr2.frontier.clone())
            rheo.prune(cfg, tr2, pr2, ws)
            tg2 = synth.target_rows(w, draft, fr2, pr2.gen_id)
            for name, v in names.items():
                rheo.verify_variant(cfg, v, tg2, draft.temperature, draft.seed, draft.offset, tr2, pr2, vout, ws)
                variants[name]["accepted"] += vout.accepted_len.cpu().tolist()
        draft.offset.copy_(off0)
        assert rheo.status(cfg, ws) == 0
        for name in names:
            acc = variants[name].pop("accepted")
            variants[name]["mean_accepted"] = sum(acc) / len(acc)
            variants[name]["samples"] = len(acc)

        # synthetic analogue of the ablations over m and T (Sec. 5.3, Sec. 5.4):
        # multi-cycle decoding against k-gram draft / target models (V = 64, k = 2),
        # tau = mean tokens emitted per cycle
        from paper_2609_21827_gb300 import cycles as cyc
        lm_gen = torch.Generator().manual_seed(2609)
        d_lm = cyc.KGramLM.random(64, 2, 1.5, lm_gen, device=device)
        t_lm = cyc.KGramLM.random(64, 2, 1.5, lm_gen, device=device, base=d_lm, noise=0.8)
        tau = {}
        lm_ms = 0.0
        for m_ in (0, 1, 2, 3):
            for T_ in (0.5, 1.0):
                c2 = rheo.Config(batch=1024, vocab=64, K=8, depth=6, budget=40, m=m_, support=64, dtype="f32")
                win = torch.randint(0, 64, (1024, 2), generator=lm_gen).to(device)
                sd = torch.arange(1024, dtype=torch.int64, device=device) * 7919 + 31 * m_ + int(10 * T_)
                t0 = time.time()
                res = cyc.run_cycles(c2, d_lm, t_lm, win, torch.full((1024,), T_), sd, cycles=6, L=1)
                torch.cuda.synchronize()
                lm_ms += (time.time() - t0) * 1e3 / 6
                tau[f"m{m_}_T{T_}"] = float(res.accepted.float().mean().item()) + 1.0
        synthetic_lm = {"vocab": 64, "k": 2, "K": 8, "depth": 6, "budget": 40, "sequences": 1024, "cycles": 6,
                        "tau": tau, "host_ms_per_cycle": lm_ms / 8}

        # full support (App. B, Table tab:sparse_support, row Full): the same
        # workload with the sampled token drawn over the whole vocabulary; a graph
        # of its 14 launches timed like the main step, plus per-call times
        cfg_f = rheo.Config(batch=w.batch, vocab=w.vocab, K=w.K, depth=w.depth, budget=w.budget, m=w.m, support=0,
                            dtype=w.dtype)
        tf, pf, wf = rheo.Tree(cfg_f, device), rheo.Pruned(cfg_f, device), rheo.Workspace(cfg_f, device)
        of = rheo.VerifyOut(cfg_f, row_lse=False, device=device)
        fr_f = []
        for d in range(1, D + 1):
            rheo.expand(cfg_f, d, draft.rows[d - 1], draft.temperature, draft.seed, draft.offset, tf, wf)
            if d < D:
                fr_f.append(tf.frontier.clone())
        rheo.prune(cfg_f, tf, pf, wf)
        tgt_f = synth.target_rows(w, draft, fr_f, pf.gen_id)

        def step_f(s_, marks=None):
            for d in range(1, D + 1):
                rheo.expand(cfg_f, d, draft.rows[d - 1], draft.temperature, draft.seed, draft.offset, tf, wf, s_)
            if marks:
                marks[0].record(s_)
            rheo.prune(cfg_f, tf, pf, wf, s_)
            if marks:
                marks[1].record(s_)
            rheo.verify_full(cfg_f, tgt_f, draft.rows, draft.temperature, draft.seed, draft.offset, tf, pf, of, wf, s_)

        g_f = torch.cuda.CUDAGraph()
        with torch.cuda.stream(stream):
            step_f(stream)
            stream.synchronize()
            with torch.cuda.graph(g_f, stream=stream):
                step_f(stream)
            for _ in range(3):
                g_f.replay()
            f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            n_f = max(20, min(200, args.steps))
            f0.record(stream)
            for _ in range(n_f):
                g_f.replay()
            f1.record(stream)
            stream.synchronize()
            ms_f = f0.elapsed_time(f1) / n_f
            mk = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
            mk[0].record(stream)
            step_f(stream, marks=(mk[1], mk[2]))
            mk[3].record(stream)
            stream.synchronize()
        assert rheo.status(cfg_f, wf, stream) == 0
        full_support = {"tree_steps_per_s": 1e3 / ms_f, "ms_per_step": ms_f,
                        "expand_ms": mk[0].elapsed_time(mk[1]), "prune_ms": mk[1].elapsed_time(mk[2]),
                        "verify_ms": mk[2].elapsed_time(mk[3]),
                        "note": "eager per-call times; the step time is the CUDA graph of its 14 launches"}

    # end to end through the public API with host buffers: H2D of every input, D2H of the results
    e2e = None
    if args.e2e_steps > 0 and (rank == 0 or world > 1):
        pin = lambda t: t.cpu().pin_memory()
        h_rows = [pin(r) for r in draft.rows]
        h_tgt = pin(target)
        h_T, h_seed, h_off = pin(draft.temperature), pin(draft.seed), pin(draft.offset)
        d_rows = [torch.empty_like(r) for r in draft.rows]
        d_tgt = torch.empty_like(target)
        d_T, d_seed, d_off = (torch.empty_like(draft.temperature), torch.empty_like(draft.seed),
                              torch.empty_like(draft.offset))
        res = [torch.empty(x.shape, dtype=x.dtype, pin_memory=True)
               for x in (out.accepted_len, out.accepted_tokens, out.bonus_token)]
        h2d = sum(r.numel() * r.element_size() for r in h_rows) + h_tgt.numel() * h_tgt.element_size() + \
            sum(x.numel() * x.element_size() for x in (h_T, h_seed, h_off))
        d2h = sum(x.numel() * x.element_size() for x in res)

        # the inputs are copied while the kernels run, every tensor cut into
        # row blocks spread over `copy_streams` copy streams (so that several
        # copy engines share each tensor); each kernel waits only for the copies
        # it reads, each copy only for the previous step's kernel that read the
        # same buffer
        NC = max(1, args.copy_streams)
        cstreams = [torch.cuda.Stream(device=device) for _ in range(NC)]
        ev_rows = [[torch.cuda.Event() for _ in range(NC)] for _ in range(D)]
        ev_rows_used = [torch.cuda.Event() for _ in range(D)]
        ev_tgt = [torch.cuda.Event() for _ in range(NC)]
        ev_small, ev_step = torch.cuda.Event(), torch.cuda.Event()
        ev_step.record(stream)

        def split_copy(dst, src, after, done):
            # rows [i*n/NC, (i+1)*n/NC) of the flattened [rows, V] tensor on stream i
            d2, s2 = dst.view(-1, dst.shape[-1]), src.view(-1, src.shape[-1])
            nr = d2.shape[0]
            for i, cs in enumerate(cstreams):
                cs.wait_event(after)
                r0, r1 = nr * i // NC, nr * (i + 1) // NC
                with torch.cuda.stream(cs):
                    if r1 > r0:
                        d2[r0:r1].copy_(s2[r0:r1], non_blocking=True)
                    done[i].record(cs)

        def e2e_step(s):
            c0 = cstreams[0]
            c0.wait_event(ev_step)  # the small inputs are read by every kernel of the step
            with torch.cuda.stream(c0):
                d_T.copy_(h_T, non_blocking=True)
                d_seed.copy_(h_seed, non_blocking=True)
                d_off.copy_(h_off, non_blocking=True)
                ev_small.record(c0)
            for d in range(D):
                split_copy(d_rows[d], h_rows[d], ev_rows_used[d], ev_rows[d])
            split_copy(d_tgt, h_tgt, ev_step, ev_tgt)
            s.wait_event(ev_small)
            for d in range(1, D + 1):
                for e in ev_rows[d - 1]:
                    s.wait_event(e)
                rheo.expand(cfg, d, d_rows[d - 1], d_T, d_seed, d_off, tree, ws, s)
                ev_rows_used[d - 1].record(s)
            rheo.prune(cfg, tree, pr, ws, s)
            for e in ev_tgt:
                s.wait_event(e)
            verify_call(d_tgt, d_rows, d_T, d_seed, d_off, s)
            for x, h in zip((out.accepted_len, out.accepted_tokens, out.bonus_token), res):
                h.copy_(x, non_blocking=True)
            ev_step.record(s)

        with torch.cuda.stream(stream):
            for _ in range(3):
                e2e_step(stream)
            stream.synchronize()
            barrier(world)
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(args.e2e_steps):
                e2e_step(stream)
            e1.record(stream)
            stream.synchronize()
            torch.cuda.synchronize()
        e2e_s = reduce_max_time(e0.elapsed_time(e1) / 1e3, world, device)
        e2e = {"value": world * args.e2e_steps / e2e_s, "unit": "tree-steps/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "copy_streams": NC, "h2d_gbs": h2d * args.e2e_steps / e2e_s / 1e9}

    if rank != 0:
        return 0
    peak, peak_kind = _peaks()
    exp_gbs = expand_bytes / (exp_ms / 1e3) / 1e9
    ver_gbs = verify_bytes / (ver_ms / 1e3) / 1e9
    step_gbs = (expand_bytes + verify_bytes) / (secs / args.steps) / 1e9
    # the dominant kernel: expand_kernel at depths >= 2 (B*K frontier rows per
    # launch, most of the step's time); algorithmic bytes = one read of its rows
    if D >= 2:
        dom_name = f"expand_kernel (depth >= 2, {w.batch * w.K} rows per launch)"
        dom_bytes = w.batch * w.K * w.vocab * esz
        dom_ms = blk_ms / (D - 1)
        dom_key = f"{w.name}:expand_d2"
    else:
        dom_name, dom_bytes, dom_ms, dom_key = f"expand_kernel (depth 1, {w.batch} rows)", \
            w.batch * w.vocab * esz, by_depth[0] / n_k, f"{w.name}:expand_d1"
    ach = dom_bytes / (dom_ms / 1e3) / 1e9
    traffic = _traffic(dom_key)
    cpu, parity = (None, None) if args.no_cpu_baseline else cpu_baseline(w, draft, gpu_res)
    line = {
        "metric": METRIC, "value": world * args.steps / secs, "unit": "tree-steps/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": secs / args.steps * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": w.dtype, "data": "synthetic",
        "config": {"workload": w.name, "batch": w.batch, "vocab": w.vocab, "depth": w.depth, "K": w.K,
                   "support": min(w.support, w.vocab) if w.support else "full",
                   "budget": w.budget, "temperature": sorted(set(w.temperatures)), "logits": w.dtype,
                   "bytes_per_step": expand_bytes + verify_bytes, "l2": "inputs 4x larger than L2, no flush",
                   "parallelism": f"replicas{world}", "cuda_graph": True,
                   "kernel_timing": ("per-call times from a separate graph with event nodes between the "
                                     "calls (an event node also removes the programmatic-launch overlap "
                                     "of the calls it separates, so they are upper bounds)")
                   if graph_events else "eager steps"},
        "roofline": {"bound": "hbm", "kernel": dom_name, "achieved": ach, "peak": peak, "unit": "GB/s",
                     "frac": ach / peak, "peak_kind": peak_kind, "traffic": traffic,
                     "bytes_per_launch": dom_bytes, "ms_per_launch": dom_ms,
                     "timing": "CUDA events around the depth 2..D launches replayed back to back as in the step"},
        "request_steps_per_s": world * args.steps / secs * w.batch,
        "kernels": {"expand_ms_per_step": exp_ms, "expand_ms_by_depth": [x / n_k for x in by_depth],
                    "expand_gbs": exp_gbs, "prune_ms": prune_ms,
                    "verify_ms": ver_ms, "verify_gbs": ver_gbs, "step_gbs": step_gbs,
                    "step_frac_of_peak": step_gbs / peak,
                    "tree_attention_us": attn_us,
                    "verify_variants": variants,
                    "synthetic_lm": synthetic_lm,
                    "full_support": full_support,
                    "tree_attention_bytes": w.batch * (w.budget + 1) * ((w.budget + 1) + 4 + 4 * (w.depth + 1) + 12)},
        "clocks": clocks,
        # D expand, 1 prune, verify: prep, stream, table, residual (full support:
        # and the overlap rows)
        "gpu_launches": args.steps * (D + 5 + (1 if full else 0)),
        "e2e": e2e,
        "cpu_baseline": cpu,
        "parity": parity,
    }
    print(json.dumps(line))
    return 0


if __name__ == "__main__":
    sys.exit(main())
