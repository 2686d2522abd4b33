"""kv_evict_score_lse (the column pass given every window row's softmax normaliser)
against the fp64 oracle, element by element, on every unit of small cases (ragged
requests, W = 8, per-query-head plans), and against the two-pass kv_evict_score at full
size. GPU only."""

import math

import numpy as np
import pytest

torch = pytest.importorskip("torch")

from oracle import kv_evict_oracle as O
from paper_2609_30738_gb300 import synth
from paper_2609_30738_gb300.workloads import WORKLOADS, scaled

from tests import parity as PT

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no GPU")
    from paper_2609_30738_gb300 import kv_evict as K
    K.library()
    return K


def _oracle_lse_and_stats(spec, batch, per_query_head=False):
    """lse in q_win's row order [N_L][n_req][Hq][W] (fp64) and the oracle's mu / sigma per
    unit, keyed by (r, layer, head)."""
    N_L, Hq, Hkv, W = spec["num_layers"], spec["num_q_heads"], spec["num_kv_heads"], spec["window"]
    G = Hq // Hkv
    seq = batch["seq_lens"]
    lse = np.zeros((N_L, len(seq), Hq, W))
    stats = {}
    for r, L in enumerate(seq):
        off = sum(seq[:r])
        for layer in range(N_L):
            for h in range(Hkv):
                kb = O.bf16_bits_to_f64(PT.to_bits(batch["k"][layer, h, off:off + L]))
                qb = O.bf16_bits_to_f64(PT.to_bits(batch["q_win"][layer, r, h * G:(h + 1) * G])).reshape(G * W, -1)
                lse[layer, r, h * G:(h + 1) * G] = O.window_lse(qb, kb, L, W, G).reshape(G, W)
                if per_query_head:
                    for g in range(G):
                        qg = qb[g * W:(g + 1) * W]
                        stats[(r, layer, h * G + g)] = O.score_unit(qg, kb, L, W, 1)
                else:
                    stats[(r, layer, h)] = O.score_unit(qb, kb, L, W, G)
    return lse, stats


@pytest.mark.parametrize("case", ["single_layer", "ragged_w8", "per_query_head"])
def test_score_lse_every_unit(case):
    from paper_2609_30738_gb300 import kv_evict as K
    base = WORKLOADS["mistral-1layer-L2048"]
    spec, pqh = {
        "single_layer": (base, False),
        "ragged_w8": (scaled(base, num_layers=2, window=8, budget=16, seq_lens=[300, 777, 1500, 40]), False),
        "per_query_head": (scaled(base, num_layers=2, budget=16, seq_lens=[700, 1300]), True),
    }[case]
    batch = synth.make_batch(spec, seed=31 + len(case))
    plan = K.Plan(spec, batch["seq_lens"], per_query_head=pqh)
    bufs = K.Buffers(plan)
    q, k = batch["q_win"].to(DEV), batch["k"].to(DEV)
    lse, stats = _oracle_lse_and_stats(spec, batch, per_query_head=pqh)
    lse_dev = torch.from_numpy(lse.astype(np.float32)).to(DEV)
    plan.score_lse(q, k, lse_dev, bufs.mu, bufs.sigma, bufs.ws)
    assert plan.status(bufs.ws) == K.KVE_OK
    mu_l, sg_l = bufs.mu.clone(), bufs.sigma.clone()
    plan.score(q, k, bufs.mu, bufs.sigma, bufs.ws)
    assert plan.status(bufs.ws) == K.KVE_OK
    # the one-pass and two-pass paths differ only by the rounding of the normaliser (the
    # two-pass kernel's fp32 sums of up to L terms: a few 1e-5 of Z at worst)
    assert torch.allclose(mu_l, bufs.mu, rtol=1e-4, atol=0) and torch.allclose(sg_l, bufs.sigma, rtol=1e-4, atol=1e-30)
    mu_all, sg_all = mu_l.cpu().numpy(), sg_l.cpu().numpy()
    seq, N_L = batch["seq_lens"], spec["num_layers"]
    heads = spec["num_q_heads"] if pqh else spec["num_kv_heads"]
    worst = 0.0
    for (r, layer, h), (mu_ref, sg_ref) in stats.items():
        L = seq[r]
        o = N_L * heads * sum(seq[:r]) + (layer * heads + h) * L
        worst = max(worst, PT.check_mu_sigma(mu_all[o:o + L], sg_all[o:o + L], mu_ref, sg_ref,
                                             f"unit(r={r},l={layer},h={h})"))
    print(f"{case}: max mu rel err {worst:.2e}")


def test_score_lse_full_size_against_two_pass():
    """The headline workload with lse from a float32 GPU computation of the window rows'
    logits (TF32 off): mu and sigma within 1e-4 of the two-pass kernel's everywhere,
    and one sampled unit against the oracle."""
    from paper_2609_30738_gb300 import kv_evict as K
    spec = WORKLOADS["mistral-32layer-L32768-B64"]
    batch = synth.make_batch(spec, seed=2609, device=DEV, with_values=False)
    N_L, Hq, Hkv, W, d = (spec[x] for x in ("num_layers", "num_q_heads", "num_kv_heads", "window", "head_dim"))
    G, L = Hq // Hkv, batch["seq_lens"][0]
    q, k = batch["q_win"], batch["k"]
    prev = torch.backends.cuda.matmul.allow_tf32
    torch.backends.cuda.matmul.allow_tf32 = False
    try:
        lse = torch.empty((N_L, 1, Hq, W), dtype=torch.float32, device=DEV)
        pos = torch.arange(L - W, L, device=DEV)
        vis = torch.arange(L, device=DEV)[None, :] <= pos[:, None]           # [W, L]
        for layer in range(N_L):
            for h in range(Hkv):
                qq = q[layer, 0, h * G:(h + 1) * G].float()                  # [G, W, d]
                lg = torch.einsum("gwd,ld->gwl", qq, k[layer, h].float()) / math.sqrt(d)
                lse[layer, 0, h * G:(h + 1) * G] = torch.logsumexp(lg.masked_fill(~vis, -math.inf), dim=-1)
    finally:
        torch.backends.cuda.matmul.allow_tf32 = prev
    plan = K.Plan(spec, batch["seq_lens"])
    bufs = K.Buffers(plan, with_trace=False)
    plan.score_lse(q, k, lse, bufs.mu, bufs.sigma, bufs.ws)
    assert plan.status(bufs.ws) == K.KVE_OK
    mu_l, sg_l = bufs.mu.clone(), bufs.sigma.clone()
    plan.score(q, k, bufs.mu, bufs.sigma, bufs.ws)
    assert plan.status(bufs.ws) == K.KVE_OK
    assert torch.allclose(mu_l, bufs.mu, rtol=1e-4, atol=0)
    assert torch.allclose(sg_l, bufs.sigma, rtol=1e-4, atol=1e-30)
    layer, h = 17, 3
    kb = O.bf16_bits_to_f64(PT.to_bits(k[layer, h]))
    qb = O.bf16_bits_to_f64(PT.to_bits(q[layer, 0, h * G:(h + 1) * G])).reshape(G * W, -1)
    mu_ref, sg_ref = O.score_unit(qb, kb, L, W, G)
    o = (layer * Hkv + h) * L
    PT.check_mu_sigma(mu_l[o:o + L].cpu().numpy(), sg_l[o:o + L].cpu().numpy(), mu_ref, sg_ref, "lse unit")
