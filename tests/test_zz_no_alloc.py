"""kv_evict_select_noalloc: selection for callers that cannot allocate device memory.

Serving engines that reserve almost all of HBM for their own KV-cache pool, and
plugin hosts that hand a kernel only its inputs and outputs, cannot give the
selector a workspace. This entry point keeps the selector's scratch in a fixed
array inside the library instead, and its device-side error word beside it. These
tests check, through the C ABI, that two calls in a row return what the workspace
entry point returns for the same inputs, that the library's error word reads clean
after them, and that requests too large for the fixed array are refused before any
launch. The file is named so that pytest collects it last.
"""

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from paper_2609_30738_gb300 import synth
from paper_2609_30738_gb300.workloads import WORKLOADS, scaled
from tests import parity as PT

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def K():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_30738_gb300 import kv_evict
    kv_evict.library()
    return kv_evict


def _select_both(K, plan, bufs, k, lam1, lam2):
    """Workspace entry point, then the no-allocation one, on the same mu/sigma."""
    n, B = bufs.indices.shape
    plan.select(bufs.mu, bufs.sigma, k, lam1, lam2, bufs.indices, bufs.ws, bufs.order, bufs.margins)
    assert plan.status(bufs.ws) == K.KVE_OK
    ref = (bufs.indices.clone(), bufs.order.clone(), bufs.margins.clone())
    idx = torch.full((n, B), -7, dtype=torch.int32, device=k.device)
    order = torch.full((n, B), -7, dtype=torch.int32, device=k.device)
    margins = torch.full((n, B), float("nan"), dtype=torch.float32, device=k.device)
    plan.select_noalloc(bufs.mu, bufs.sigma, k, lam1, lam2, idx, order, margins)
    # the no-allocation call's own error word (kept in the library, not in bufs.ws)
    assert plan.status(None) == K.KVE_OK
    return ref, (idx, order, margins)


def _same(ref, got):
    assert torch.equal(ref[0], got[0]), "indices differ"
    assert torch.equal(ref[1], got[1]), "admission order differs"
    m_ref, m_got = ref[2].cpu().numpy(), got[2].cpu().numpy()
    assert np.array_equal(np.isfinite(m_ref), np.isfinite(m_got))
    fin = np.isfinite(m_ref)
    assert np.all(np.abs(m_ref[fin] - m_got[fin]) <= PT.TIE_TOL)


def test_noalloc_matches_workspace_select_twice(K):
    spec = scaled(WORKLOADS["mistral-1layer-L2048"], num_layers=2, seq_lens=[3000, 1777], budget=32)
    batch = synth.make_batch(spec, seed=31)
    plan = K.Plan(spec, batch["seq_lens"])
    bufs = K.Buffers(plan)
    q, k = batch["q_win"].cuda(), batch["k"].cuda()
    plan.score(q, k, bufs.mu, bufs.sigma, bufs.ws)
    assert plan.status(bufs.ws) == K.KVE_OK
    # first call
    l1, l2 = np.full(2, 0.5, np.float32), np.full(2, -0.5, np.float32)
    ref, got = _select_both(K, plan, bufs, k, l1, l2)
    _same(ref, got)
    # second call in a row, other coefficients: the array still holds the first
    # call's scores and must be rewritten, not trusted
    l1, l2 = np.array([0.0, 0.3], np.float32), np.array([-0.15, 0.6], np.float32)
    ref, got = _select_both(K, plan, bufs, k, l1, l2)
    _same(ref, got)


def test_noalloc_refuses_requests_beyond_its_array(K):
    lib = K.library()
    lam = np.zeros(32, np.float32)
    # 32 layers x 8 KV heads x 20000 tokens = 5.12 M scores > 4194304 (16 MiB)
    spec = scaled(WORKLOADS["mistral-32layer-L8192"], seq_lens=[20000])
    plan = K.Plan(spec, spec["seq_lens"])
    st = lib.kv_evict_select_noalloc(plan._h, 16, 16, 16, lam.ctypes.data, lam.ctypes.data, 16,
                                     None, None, None)
    assert st == K.KVE_EINVAL
    # a per-query-head plan counts Hq units per layer: 32 x 32 x 4100 > 4194304
    perq = K.Plan(scaled(spec, seq_lens=[4100]), [4100], per_query_head=True)
    st = lib.kv_evict_select_noalloc(perq._h, 16, 16, 16, lam.ctypes.data, lam.ctypes.data, 16,
                                     None, None, None)
    assert st == K.KVE_EINVAL
    assert perq.status(None) == K.KVE_OK
