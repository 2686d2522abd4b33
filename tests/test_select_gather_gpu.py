"""kv_evict_select_gather (steps 3 and 4 in one launch) against kv_evict_select
followed by kv_evict_gather: the same indices, order, margins and compact cache, bit
for bit, on ragged, short, layered, per-query-head and every-candidate plans, with
values in device or pinned host memory. GPU only. (The oracle checks of every other
GPU test run through the fused call as well: run_step uses it.)"""

import pytest

torch = pytest.importorskip("torch")

from paper_2609_30738_gb300 import synth
from paper_2609_30738_gb300.workloads import WORKLOADS, lambda_arrays, scaled

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_30738_gb300 import kv_evict as K
    K.library()
    return K


def _both(spec, seed, layer_budgets=None, per_query_head=False, host_v=False):
    from paper_2609_30738_gb300 import kv_evict as K
    batch = synth.make_batch(spec, seed=seed)
    plan = K.Plan(spec, batch["seq_lens"], layer_budgets=layer_budgets, per_query_head=per_query_head)
    lam = lambda_arrays(spec, K.profile)
    q, k, v = (batch[x].to(DEV) for x in ("q_win", "k", "v"))
    sep, fus = K.Buffers(plan), K.Buffers(plan)
    K.run_step(plan, sep, q, k, v, lam[0], lam[1], fused=False)
    assert plan.status(sep.ws) == K.KVE_OK
    for t in (fus.indices, fus.order, fus.k_out, fus.v_out):
        t.fill_(7)
    fus.margins.fill_(7.0)
    plan.score(q, k, fus.mu, fus.sigma, fus.ws)   # (bit-identical to sep's; it also readies fus.ws)
    vv = batch["v"].contiguous().pin_memory() if host_v else v
    plan.select_gather(fus.mu, fus.sigma, k, vv, lam[0], lam[1], fus.indices, fus.k_out, fus.v_out,
                       fus.ws, fus.order, fus.margins)
    assert plan.status(fus.ws) == K.KVE_OK
    for name in ("indices", "order", "margins", "k_out", "v_out"):
        a, b = getattr(sep, name), getattr(fus, name)
        assert torch.equal(a.view(torch.int32) if a.dtype == torch.float32 else a,
                           b.view(torch.int32) if b.dtype == torch.float32 else b), name
    return plan, batch


@pytest.mark.parametrize("case", ["ragged", "window8", "short", "tiny_budget", "cf2"])
def test_fused_equals_select_then_gather(case):
    base = WORKLOADS["mistral-1layer-L2048"]
    spec = {
        "ragged": scaled(base, num_layers=2, budget=16, seq_lens=[300, 777, 1500, 40, 513]),
        "window8": scaled(base, window=8, budget=32, seq_lens=[1000, 129]),
        "short": scaled(base, seq_lens=[33, 40, 100], budget=64),        # Lc below B: every token kept
        "tiny_budget": scaled(base, seq_lens=[129, 2048], budget=8, pool_kernel=1),
        "cf2": scaled(base, seq_lens=[4097], budget=64, candidate_factor=2),
    }[case]
    _both(spec, seed=len(case))


def test_fused_with_layer_budgets_and_per_query_head():
    from paper_2609_30738_gb300 import kv_evict as K
    spec = scaled(WORKLOADS["mistral-1layer-L2048"], num_layers=4, budget=40, seq_lens=[1500, 300, 2100])
    _both(spec, seed=13, layer_budgets=K.budget_pyramid(24, 4, 0.4))
    spec = scaled(WORKLOADS["mistral-1layer-L2048"], num_layers=2, budget=16, seq_lens=[700, 1300])
    _both(spec, seed=14, per_query_head=True)


def test_fused_every_candidate_plan():
    """candidate_factor 0 beyond 512 prefix tokens: the every-candidate selector, then
    the gather, behind the same call."""
    spec = scaled(WORKLOADS["mistral-1layer-L2048"], seq_lens=[1500], budget=32, candidate_factor=0)
    _both(spec, seed=15)


def test_fused_reads_pinned_host_values_and_refuses_pageable():
    from paper_2609_30738_gb300 import kv_evict as K
    spec = scaled(WORKLOADS["mistral-1layer-L2048"], num_layers=2, budget=16, seq_lens=[300, 1500, 513])
    plan, batch = _both(spec, seed=16, host_v=True)
    bufs = K.Buffers(plan)
    lam = lambda_arrays(spec, K.profile)
    q, k = batch["q_win"].to(DEV), batch["k"].to(DEV)
    plan.score(q, k, bufs.mu, bufs.sigma, bufs.ws)
    pv = batch["v"].contiguous()
    assert not pv.is_pinned()
    with pytest.raises(ValueError):
        plan.select_gather(bufs.mu, bufs.sigma, k, pv, lam[0], lam[1], bufs.indices, bufs.k_out,
                           bufs.v_out, bufs.ws)
    import numpy as np
    l1 = np.ascontiguousarray(lam[0], dtype=np.float32)
    l2 = np.ascontiguousarray(lam[1], dtype=np.float32)
    bufs.v_out.fill_(1)
    st = K.library().kv_evict_select_gather(plan._h, bufs.mu.data_ptr(), bufs.sigma.data_ptr(), k.data_ptr(),
                                            pv.data_ptr(), l1.ctypes.data, l2.ctypes.data,
                                            bufs.indices.data_ptr(), None, None, bufs.k_out.data_ptr(),
                                            bufs.v_out.data_ptr(), bufs.ws.data_ptr(), None)
    assert st == K.KVE_EINVAL
    torch.cuda.synchronize()
    assert bool((bufs.v_out == 1).all())   # refused before any launch: nothing written
