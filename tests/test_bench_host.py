"""Host-side logic of bench.py: max-over-ranks timing with world size 2 (gloo,
CPU) and the clock-log parser."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    w, r, _ = bench._dist()
    bench.barrier(w)
    t = bench.reduce_max_time(0.25 + rank, w)
    q.put((r, w, t))
    dist.destroy_process_group()


def test_max_over_ranks_world2_gloo():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert got == [(0, 2, 1.25), (1, 2, 1.25)]


def test_single_rank_is_identity():
    assert bench.reduce_max_time(0.5, 1) == 0.5


def test_clock_log_parser():
    lines = ["0, 1965, 2070, 900.1, 0x0, Not Active, Not Active, Not Active, Not Active\n",
             "0, 1980, 2070, 1100.5, 0x4, Not Active, Not Active, Not Active, Active\n",
             "0, 1995, 2070, 1200.0, 0x0, Not Active, Not Active, Not Active, Not Active\n",
             "garbage\n"]
    s = bench.Clocks.parse(lines)
    assert s["sm_mhz"] == 1980 and s["sm_max_mhz"] == 2070 and s["samples"] == 3
    assert s["reasons"] == ["sw_power_cap"]
    assert bench.Clocks.parse([])["samples"] == 0


def test_peaks_are_read():
    peak, kind = bench._peaks()
    assert peak > 1000 and kind in ("measured", "fallback")


def test_parity_summary_classifies_differences():
    """The bench's parity report: identical results are exact; a changed bonus
    token or a changed tree node with a wide oracle margin is unexplained."""
    import copy
    import dataclasses

    import numpy as np

    from paper_2609_21827_gb300 import synth

    w = dataclasses.replace(synth.WORKLOADS["tiny"], name="tiny_b3", batch=3)
    draft = synth.make_draft_inputs(w, device="cpu")
    _, ot, op, oo = bench.oracle_cycle(w, draft, range(3))
    g = {"token": ot.token.copy(), "parent": ot.parent.copy(), "slot": ot.slot.copy(),
         "acc_len": oo.accepted_len.copy(), "acc_tok": oo.accepted_tokens.copy(),
         "acc_node": oo.accepted_nodes.copy(), "bonus": oo.bonus_token.copy()}
    g.update({"pr_" + k: getattr(op, k).copy() for k in bench.PRUNED_FIELDS})
    rep = bench.parity_summary(w, g, [0, 1, 2], ot, op, oo)
    assert (rep["exact"], rep["explained_flips"], rep["unexplained"]) == (3, 0, 0)
    bad = copy.deepcopy(g)
    bad["bonus"][1] = (bad["bonus"][1] + 1) % w.vocab
    bad["token"][2, 1 + w.m] = -7  # the sampled child of the root
    rep = bench.parity_summary(w, bad, [0, 1, 2], ot, op, oo)
    gaps = {1: float(oo.gap_level[1, int(oo.accepted_len[1])]), 2: float(ot.gap_sample[2, 0])}
    want_bad = sum(1 for b in (1, 2) if gaps[b] >= bench.FLIP_GAP)
    assert rep["exact"] == 1 and rep["unexplained"] == want_bad and rep["explained_flips"] == 2 - want_bad
    assert np.all(g["bonus"] == oo.bonus_token)


def test_oracle_reports_threads_it_ran():
    import oracle

    oracle.build()
    n = oracle.max_threads()
    oracle.set_threads(1)
    try:
        assert oracle.max_threads() == 1
    finally:
        oracle.set_threads(n)
    assert oracle.max_threads() == n


def test_reference_arm_full_support_line(capsys):
    """--impl reference with --support 0 times the oracle's full-support cycle
    (App. B, row Full) and names it in the config, on the host alone."""
    import json

    assert bench.main(["--impl", "reference", "--workload", "tiny", "--support", "0", "--steps", "1",
                       "--warmup", "0"]) == 0
    line = json.loads(capsys.readouterr().out.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["value"] > 0
    assert line["config"]["workload"] == "tiny_full" and line["config"]["support"] == "full"
    assert line["cpu_baseline"]["kind"] == "oracle"
