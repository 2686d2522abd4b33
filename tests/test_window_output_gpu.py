"""kv_evict_score_attn: the score pass that also returns the window rows' own attention
output O[r] = sum_i A[r, i] v_i (Section 3.2 scores tokens with the prefill's existing
attention; these rows are that attention's output). GPU only, through the C ABI.

Tolerance of O, from the arithmetic: every probability enters the value product as
bf16 (8 significant bits: relative rounding error <= 2^-8), the product accumulates in
fp32, and O is rounded to bf16 once (<= 2^-8 |O|); so
|O - O_ref| <= 2^-8 sum_i A_ri |v_ij| + 2^-8 |O_ref| (the probabilities' own fp32 error,
~1e-5 relative, is far below), checked here at twice that plus 1e-6 absolute. mu and
sigma must equal kv_evict_score's bit for bit (within 1e-5 relative at full size, see
that test), and the selection made from them likewise.
"""

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import kv_evict_oracle as O
from paper_2609_30738_gb300 import synth
from paper_2609_30738_gb300.workloads import WORKLOADS, lambda_arrays, scaled
from tests import parity as PT

pytestmark = pytest.mark.gpu

DEV = "cuda"
O_REL = 2.0 ** -7


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_30738_gb300 import kv_evict as K
    K.library()
    return K


def _run_both(spec, batch, per_query_head=False, kt=None, vt=None, k_strides=None, v_strides=None):
    """kv_evict_score on one plan, kv_evict_score_attn on another (same inputs)."""
    from paper_2609_30738_gb300 import kv_evict as K
    q, k, v = (batch[x].to(DEV) for x in ("q_win", "k", "v"))
    plan = K.Plan(spec, batch["seq_lens"], per_query_head=per_query_head)
    bufs = K.Buffers(plan)
    plan.score(q, k, bufs.mu, bufs.sigma, bufs.ws)
    assert plan.status(bufs.ws) == K.KVE_OK
    plan2 = K.Plan(spec, batch["seq_lens"], per_query_head=per_query_head, k_strides=k_strides,
                   v_strides=v_strides)
    bufs2 = K.Buffers(plan2)
    attn_ws = torch.empty(plan2.score_attn_workspace(), dtype=torch.uint8, device=DEV)
    o_win = torch.full_like(q, 7.0)
    plan2.score_attn(q, kt if kt is not None else k, vt if vt is not None else v, bufs2.mu, bufs2.sigma,
                     o_win, bufs2.ws, attn_ws)
    assert plan2.status(bufs2.ws) == K.KVE_OK
    return (plan, bufs), (plan2, bufs2), (q, k, v), o_win


def _check_outputs(spec, batch, o_win, per_query_head=False, units=None):
    """O of the listed units (r, layer, head) against the oracle; returns the worst
    |O - O_ref| / bound."""
    seq = batch["seq_lens"]
    W, Hq, Hkv = spec["window"], spec["num_q_heads"], spec["num_kv_heads"]
    G = Hq // Hkv
    ug = 1 if per_query_head else G                      # query heads per unit
    uheads = Hq if per_query_head else Hkv
    if units is None:
        units = [(r, l, h) for r in range(len(seq)) for l in range(spec["num_layers"]) for h in range(uheads)]
    ow = o_win.float().cpu().numpy()
    worst = 0.0
    for (r, layer, h) in units:
        L, off = seq[r], sum(seq[:r])
        kvh = h // G if per_query_head else h
        qb = PT.to_bits(batch["q_win"][layer, r, h * ug:(h + 1) * ug]).reshape(ug * W, -1)
        kb = PT.to_bits(batch["k"][layer, kvh, off:off + L])
        vb = PT.to_bits(batch["v"][layer, kvh, off:off + L])
        vf = O.bf16_bits_to_f64(vb)
        A = O.window_attention(O.bf16_bits_to_f64(qb), O.bf16_bits_to_f64(kb), L, W, ug)
        o_ref = O.window_output(A, vf)
        o_gpu = ow[layer, r, h * ug:(h + 1) * ug].reshape(ug * W, -1)
        bound = O_REL * (A @ np.abs(vf)) + O_REL * np.abs(o_ref) + 1e-6
        err = np.abs(o_gpu - o_ref)
        bad = np.argwhere(~(err <= bound))
        assert len(bad) == 0, (f"unit (r={r}, l={layer}, h={h}) O mismatch at {bad[:3].tolist()}: "
                               f"gpu {o_gpu[tuple(bad[0])]}, ref {o_ref[tuple(bad[0])]}")
        worst = max(worst, float((err / bound).max()))
    return worst


@pytest.mark.parametrize("case", ["L2048", "ragged"])
def test_window_output_every_unit(case):
    """Every unit's window output against the oracle; mu, sigma and the selection made
    from them equal the plain score pass bit for bit."""
    from paper_2609_30738_gb300 import kv_evict as K
    if case == "L2048":
        spec = WORKLOADS["mistral-1layer-L2048"]
    else:
        spec = scaled(WORKLOADS["mistral-1layer-L2048"], num_layers=2, budget=16, seq_lens=[300, 777, 1500, 513])
    batch = synth.make_batch(spec, seed=71)
    (plan, bufs), (plan2, bufs2), (q, k, v), o_win = _run_both(spec, batch)
    assert torch.equal(bufs.mu, bufs2.mu) and torch.equal(bufs.sigma, bufs2.sigma)
    lam = lambda_arrays(spec, K.profile)
    for pl, bf in ((plan, bufs), (plan2, bufs2)):
        pl.select(bf.mu, bf.sigma, k, lam[0], lam[1], bf.indices, bf.ws, bf.order, bf.margins)
    assert plan2.status(bufs2.ws) == K.KVE_OK
    assert torch.equal(bufs.indices, bufs2.indices) and torch.equal(bufs.margins, bufs2.margins)
    worst = _check_outputs(spec, batch, o_win)
    print(f"window output, worst |O - O_ref| / bound = {worst:.3f}")


def test_window_output_short_rows_and_per_query_head():
    """n < 128 window rows: W = 8 (n = 32, the rows past n hold no probabilities), and
    per-query-head units (n = W = 32)."""
    spec = scaled(WORKLOADS["mistral-1layer-L2048"], window=8, budget=16, seq_lens=[1000, 129])
    batch = synth.make_batch(spec, seed=72)
    (_, bufs), (_, bufs2), _, o_win = _run_both(spec, batch)
    assert torch.equal(bufs.mu, bufs2.mu) and torch.equal(bufs.sigma, bufs2.sigma)
    _check_outputs(spec, batch, o_win)
    spec = scaled(WORKLOADS["mistral-1layer-L2048"], budget=16, seq_lens=[900, 300])
    batch = synth.make_batch(spec, seed=73)
    (_, bufs), (_, bufs2), _, o_win = _run_both(spec, batch, per_query_head=True)
    assert torch.equal(bufs.mu, bufs2.mu) and torch.equal(bufs.sigma, bufs2.sigma)
    _check_outputs(spec, batch, o_win, per_query_head=True)


def test_window_output_strided_values():
    """v read in place from a token-major cache (plan strides): the same output as the
    dense layout, bit for bit."""
    spec = scaled(WORKLOADS["mistral-1layer-L2048"], num_layers=2, budget=16, seq_lens=[700, 1300])
    batch = synth.make_batch(spec, seed=74)
    (_, _), (_, _), (q, k, v), o_dense = _run_both(spec, batch)
    vt = v.permute(0, 2, 1, 3).contiguous()              # [N_L][SL][Hkv][d]
    v_str = (vt.stride(0), vt.stride(2), vt.stride(1))
    (_, _), (_, _), _, o_strided = _run_both(spec, batch, vt=vt, v_strides=v_str)
    assert torch.equal(o_dense, o_strided)


def test_window_output_full_size_sampled_units():
    """The L = 32768 workload (256 units, 38 work items each): sampled units' window
    output against the oracle. Here the window-output pass folds a unit's 38 row
    partials in batches of 16 (its smaller merge buffer) where the plain pass folds them
    in one batch of 40, so the normalisers, and with them mu and sigma, may differ from
    the plain pass in the last bits: they are compared within 1e-5 relative."""
    spec = WORKLOADS["mistral-32layer-L32768-B64"]
    batch = synth.make_batch(spec, seed=2609, device=DEV)
    (_, bufs), (_, bufs2), _, o_win = _run_both(spec, batch)
    for a, b in ((bufs.mu, bufs2.mu), (bufs.sigma, bufs2.sigma)):
        rel = ((a.double() - b.double()).abs() / a.double().abs().clamp_min(1e-30)).max().item()
        assert rel <= 1e-5, rel
    units = [(0, 0, 0), (0, 13, 5), (0, 31, 7)]
    worst = _check_outputs(spec, batch, o_win, units=units)
    print(f"full size window output, worst |O - O_ref| / bound = {worst:.3f}")
