"""kv_evict_score_attn: the score pass that also returns the window rows' own attention
output O[r] = sum_i A[r, i] v_i (Section 3.2 scores tokens with the prefill's existing
attention; these rows are that attention's output). GPU only, through the C ABI.

Tolerance of O, from the arithmetic: every probability enters the value product as
bf16 (8 significant bits: relative rounding error <= 2^-8), the product accumulates in
fp32, and O is rounded to bf16 once (<= 2^-8 |O|); so
|O - O_ref| <= 2^-8 sum_i A_ri |v_ij| + 2^-8 |O_ref| (the probabilities' own fp32 error,
~1e-5 relative, is far below), checked here at twice that plus 1e-6 absolute. mu and
sigma meet the oracle tolerances of every parity test, and stay within 1e-5 relative of
kv_evict_score's (the two calls may fold a unit's row partials in different batches, so
the normalisers can round differently in the last bits).
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


def _close(a, b, rtol=1e-5):
    """Elementwise |a - b| <= rtol |b| + 1e-30 (float tensors on the device)."""
    a, b = a.double(), b.double()
    return bool(((a - b).abs() <= rtol * b.abs() + 1e-30).all())


def _check_outputs(spec, batch, o_win, per_query_head=False, units=None, bufs=None):
    """O of the listed units (r, layer, head) against the oracle, and (bufs given) mu and
    sigma of the same call; returns the worst |O - O_ref| / bound."""
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
        if bufs is not None:
            mu_ref = O.mean_attention(A)
            sg_ref = O.dispersion(A, mu_ref)
            o0 = spec["num_layers"] * uheads * off + (layer * uheads + h) * L
            PT.check_mu_sigma(bufs.mu[o0:o0 + L].cpu().numpy(), bufs.sigma[o0:o0 + L].cpu().numpy(),
                              mu_ref, sg_ref, f"unit (r={r}, l={layer}, h={h})")
        bound = O_REL * (A @ np.abs(vf)) + O_REL * np.abs(o_ref) + 1e-6
        err = np.abs(o_gpu - o_ref)
        bad = np.argwhere(~(err <= bound))
        assert len(bad) == 0, (f"unit (r={r}, l={layer}, h={h}) O mismatch at {bad[:3].tolist()}: "
                               f"gpu {o_gpu[tuple(bad[0])]}, ref {o_ref[tuple(bad[0])]}")
        worst = max(worst, float((err / bound).max()))
    return worst


@pytest.mark.parametrize("case", ["L2048", "ragged"])
def test_window_output_every_unit(case):
    """Every unit's window output, mu and sigma against the oracle; mu and sigma within
    1e-5 relative of the plain score pass."""
    if case == "L2048":
        spec = WORKLOADS["mistral-1layer-L2048"]
    else:
        spec = scaled(WORKLOADS["mistral-1layer-L2048"], num_layers=2, budget=16, seq_lens=[300, 777, 1500, 513])
    batch = synth.make_batch(spec, seed=71)
    (plan, bufs), (plan2, bufs2), (q, k, v), o_win = _run_both(spec, batch)
    assert _close(bufs2.mu, bufs.mu) and _close(bufs2.sigma, bufs.sigma)
    worst = _check_outputs(spec, batch, o_win, bufs=bufs2)
    print(f"window output, worst |O - O_ref| / bound = {worst:.3f}")


def test_window_output_logit_jump():
    """Keys whose logits exceed everything earlier in their work item by far (planted:
    k = c q_r for one window row r, logit about 200 in natural units, i.e. 2^288 times
    the rest): the rows' maxima and normalisers jump in the middle of an item. O, mu and
    sigma against the oracle on every unit."""
    spec = scaled(WORKLOADS["mistral-1layer-L2048"], budget=16, seq_lens=[2048, 1536])
    batch = synth.make_batch(spec, seed=75)
    q, k = batch["q_win"], batch["k"]
    W, G, d = spec["window"], spec["num_q_heads"] // spec["num_kv_heads"], spec["head_dim"]
    off = 0
    for r, L in enumerate(spec["seq_lens"]):
        for h in range(spec["num_kv_heads"]):
            for j, pos in enumerate((128 * 5 + 7, 128 * 11 + 3)):
                if pos >= L - W:
                    continue
                qr = q[0, r, h * G + (j % G), (3 * j + h) % W].double()
                c = 200.0 * d ** 0.5 / float((qr * qr).sum())
                k[0, h, off + pos] = (c * qr).to(k.dtype)
        off += L
    (_, bufs), (_, bufs2), _, o_win = _run_both(spec, batch)
    worst = _check_outputs(spec, batch, o_win, bufs=bufs2)
    assert _close(bufs2.mu, bufs.mu, 1e-4) and _close(bufs2.sigma, bufs.sigma, 1e-4)
    print(f"logit jump, worst |O - O_ref| / bound = {worst:.3f}")


def test_window_output_short_rows_and_per_query_head():
    """n < 128 window rows: W = 8 (n = 32, the rows past n hold no probabilities), and
    per-query-head units (n = W = 32)."""
    spec = scaled(WORKLOADS["mistral-1layer-L2048"], window=8, budget=16, seq_lens=[1000, 129])
    batch = synth.make_batch(spec, seed=72)
    (_, bufs), (_, bufs2), _, o_win = _run_both(spec, batch)
    assert _close(bufs2.mu, bufs.mu) and _close(bufs2.sigma, bufs.sigma)
    _check_outputs(spec, batch, o_win, bufs=bufs2)
    spec = scaled(WORKLOADS["mistral-1layer-L2048"], budget=16, seq_lens=[900, 300])
    batch = synth.make_batch(spec, seed=73)
    (_, bufs), (_, bufs2), _, o_win = _run_both(spec, batch, per_query_head=True)
    assert _close(bufs2.mu, bufs.mu) and _close(bufs2.sigma, bufs.sigma)
    _check_outputs(spec, batch, o_win, per_query_head=True, bufs=bufs2)


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
    output, mu and sigma against the oracle; mu and sigma within 1e-5 relative of the
    plain score pass everywhere."""
    spec = WORKLOADS["mistral-32layer-L32768-B64"]
    batch = synth.make_batch(spec, seed=2609, device=DEV)
    (_, bufs), (_, bufs2), _, o_win = _run_both(spec, batch)
    assert _close(bufs2.mu, bufs.mu) and _close(bufs2.sigma, bufs.sigma)
    units = [(0, 0, 0), (0, 13, 5), (0, 31, 7)]
    worst = _check_outputs(spec, batch, o_win, units=units, bufs=bufs2)
    print(f"full size window output, worst |O - O_ref| / bound = {worst:.3f}")
