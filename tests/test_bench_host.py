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
