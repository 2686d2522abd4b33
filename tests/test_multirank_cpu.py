"""The N > 1 path of bench.py on CPU: two ranks over gloo on 127.0.0.1.

Under torchrun every rank evicts its own request (weak scaling, no collective on the
data path); the only cross-rank work is the barrier and the max over ranks of the
timed region, and the whole-job throughput counts every rank's request. The reference
arm runs on rank 0 alone; the other ranks exit without work.
"""
import os
import socket
import sys

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.abspath(os.path.join(os.path.dirname(__file__), ".."))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port),
                       "RANK": str(rank), "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w, r, local = bench._dist()
        # each rank times a different region; the job time is the slowest rank's
        mine = 0.010 + 0.005 * rank
        job = bench._max_over_ranks(mine, w, torch.device("cpu"))
        dist.barrier()
        # the reference arm: rank 0 only; other ranks return at once without work
        ref = None
        if r != 0:
            class A:
                steps, warmup = 1, 0
            ref = bench.run_reference(A())
        out.put((r, w, local, job, bench._job_tok_s(w, 32768, job), ref))
    finally:
        dist.destroy_process_group()


def test_two_ranks_gloo():
    world = 2
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(out.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [x[0] for x in res] == [0, 1]
    for r, w, local, job, tok_s, ref in res:
        assert w == world and local == r
        assert job == pytest.approx(0.015)                 # max over ranks, on every rank
        assert tok_s == pytest.approx(2 * 32768 / 0.015)   # whole-job: both ranks' requests
    assert res[1][5] is None                               # rank 1 of the reference arm: no work


def test_single_rank_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench._max_over_ranks(0.25, 1, None) == 0.25
    assert bench._job_tok_s(1, 32768, 0.5) == 65536.0
