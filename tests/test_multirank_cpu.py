"""The N > 1 path of bench.py on CPU: ranks over gloo on 127.0.0.1.

Under torchrun a one-request workload gives every rank its own request (weak
scaling); a batch of requests is split across the ranks by prefix tokens (strong
scaling). Neither has a collective on the data path: the only cross-rank work is the
barrier and the max over ranks of the timed region, and the whole-job throughput
counts every rank's tokens. The reference arm runs on rank 0 alone; the other ranks
exit without work.
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


def _fake_outputs(spec, req_ids, seq):
    """Per-unit outputs in the layouts of include/kv_evict.h for the requests
    req_ids (lengths seq), filled with values that identify (request, layer, head,
    slot) -- what a rank's plan over those requests returns."""
    N_L, Hkv, B = spec["num_layers"], spec["num_kv_heads"], spec["budget"]
    idx, mu = [], []
    for rid, L in zip(req_ids, seq):
        for layer in range(N_L):
            for h in range(Hkv):
                idx.append([((rid * 100 + layer) * 10 + h) * 1000 + b for b in range(B)])
                mu.append([((rid * 100 + layer) * 10 + h) + i / (L + 1.0) for i in range(L)])
    return idx, [x for row in mu for x in row]


def _split_rank_main(rank, world, port, out):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port),
                       "RANK": str(rank), "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
    sys.path.insert(0, ROOT)
    import bench
    from paper_2609_30738_gb300.workloads import WORKLOADS, scaled
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        full = scaled(WORKLOADS["mistral-32layer-ragged16"], num_layers=2, num_kv_heads=2, budget=3,
                      seq_lens=[37, 90, 41, 66, 52, 75, 48, 33, 81])
        reqs, scaling = bench._rank_requests(full, world, rank)
        seq = [full["seq_lens"][r] for r in reqs]
        idx, mu = _fake_outputs(full, reqs, seq)
        parts = [None] * world
        dist.all_gather_object(parts, (reqs, idx, mu))
        out.put((rank, scaling, parts))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 4])
def test_batch_split_across_ranks_gloo(world):
    """The ragged batch under torchrun: every request on exactly one rank, prefix
    tokens balanced, and the ranks' outputs (per-request blocks of units and of
    mu / sigma) reassemble into the single-GPU layout of the whole batch."""
    sys.path.insert(0, ROOT)
    from paper_2609_30738_gb300.workloads import WORKLOADS, request_layout, scaled
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_split_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted((q.get(timeout=120) for _ in range(world)), key=lambda x: x[0])
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    full = scaled(WORKLOADS["mistral-32layer-ragged16"], num_layers=2, num_kv_heads=2, budget=3,
                  seq_lens=[37, 90, 41, 66, 52, 75, 48, 33, 81])
    seq = full["seq_lens"]
    parts = res[0][2]
    assert all(r[1] == "strong" for r in res)
    owned = sorted(r for reqs, _, _ in parts for r in reqs)
    assert owned == list(range(len(seq)))                      # a disjoint cover
    loads = [sum(seq[r] for r in reqs) for reqs, _, _ in parts]
    assert max(loads) - min(loads) <= max(seq)                 # greedy balance bound
    # reassemble into the whole batch's layout and compare with a single-GPU run
    want_idx, want_mu = _fake_outputs(full, list(range(len(seq))), seq)
    lay_full = request_layout(seq, full["num_layers"], full["num_kv_heads"])
    got_idx = [None] * len(want_idx)
    got_mu = [None] * len(want_mu)
    for reqs, idx, mu in parts:
        lay = request_layout([seq[r] for r in reqs], full["num_layers"], full["num_kv_heads"])
        for j, r in enumerate(reqs):
            u0, n_u, e0, n_e = lay[j]
            U0, _, E0, _ = lay_full[r]
            got_idx[U0:U0 + n_u] = idx[u0:u0 + n_u]
            got_mu[E0:E0 + n_e] = mu[e0:e0 + n_e]
    assert got_idx == want_idx and got_mu == want_mu


def test_batch_subset_inputs_equal_whole_batch_slices():
    """A rank's subset of the batch is generated with the requests' own seeds: its
    tensors equal the corresponding slices of the whole batch."""
    sys.path.insert(0, ROOT)
    from paper_2609_30738_gb300 import synth
    from paper_2609_30738_gb300.workloads import WORKLOADS, scaled
    full = scaled(WORKLOADS["mistral-32layer-ragged16"], num_layers=1, num_kv_heads=2, num_q_heads=8,
                  seq_lens=[40, 70, 55])
    whole = synth.make_batch(full, seed=2609)
    sub = synth.make_batch(dict(full, seq_lens=[70, 40]), seed=2609, request_ids=[1, 0])
    assert torch.equal(sub["k"][:, :, :70], whole["k"][:, :, 40:110])
    assert torch.equal(sub["k"][:, :, 70:], whole["k"][:, :, :40])
    assert torch.equal(sub["q_win"][:, 0], whole["q_win"][:, 1])
    assert torch.equal(sub["v"][:, :, 70:], whole["v"][:, :, :40])
