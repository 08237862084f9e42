"""The multi-rank path of the bench on CPU (gloo, world size 2): each rank
processes its own batch (same shapes, distinct seeds, no exchange of data), and
the reported step time is the maximum over ranks, computed by an all-reduce."""
import os
import socket

import numpy as np
import pytest

import synth

torch = pytest.importorskip("torch")
dist = pytest.importorskip("torch.distributed")


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def worker(rank, world, port, out):
    import bench

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w = bench.rank_shard(bench.PREFILL, rank)
        box = synth.host_tensor(w, "q", (0, 0, 0, 0), (1, 4, w.Hq, w.d))
        d = bench.rank_shard(bench.DECODE, rank)
        needles = synth.needle_chunk_ids(d)
        ms = 10.0 + 5.0 * rank  # rank 1 is the slower one
        worst = bench.reduce_max(ms, world, torch.device("cpu"))
        out.put((rank, w.number, box.tobytes(), tuple(int(x) for x in needles[:4]), worst))
    finally:
        dist.destroy_process_group()


def test_two_ranks_process_distinct_batches_and_report_the_slowest():
    ctx = torch.multiprocessing.get_context("spawn")
    out = ctx.Queue()
    port = free_port()
    procs = [ctx.Process(target=worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    got = {}
    for _ in procs:
        rank, number, box, needles, worst = out.get(timeout=120)
        got[rank] = (number, box, needles, worst)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert got[0][0] != got[1][0]           # distinct seeds
    assert got[0][1] != got[1][1]           # hence distinct inputs
    assert got[0][2] != got[1][2]           # and distinct decode needles
    assert got[0][3] == got[1][3] == 15.0  # every rank sees the slowest rank's time


def test_rank_zero_keeps_the_workload():
    import bench

    assert bench.rank_shard(bench.PREFILL, 0) is bench.PREFILL
    w1 = bench.rank_shard(bench.PREFILL, 1)
    assert (w1.B, w1.L, w1.Hq, w1.Hkv, w1.d, w1.topk) == (bench.PREFILL.B, bench.PREFILL.L, bench.PREFILL.Hq,
                                                         bench.PREFILL.Hkv, bench.PREFILL.d, bench.PREFILL.topk)
    a = synth.host_tensor(bench.PREFILL, "K", (0, 0, 0, 0), (1, 2, 1, 8))
    b = synth.host_tensor(w1, "K", (0, 0, 0, 0), (1, 2, 1, 8))
    assert not np.array_equal(a, b)
