"""Seeded synthetic inputs shaped like Mistral-7B end-of-prefill K/V caches.

This module only draws inputs: it holds none of the eviction method's arithmetic
and imports neither the CUDA library nor the oracle, so both sides of a parity
test can consume the very same tensors.

Recipe, per (request r, layer l) with its own torch.Generator seeded from
(seed, r, l), vectorised over the KV heads:
  * 64 cluster centres per head, Gaussian directions of unit norm.
  * Key i = centre z_i (z_i uniform) + Gaussian noise of per-component std
    noise/sqrt(d) (noise norm ~ `noise`).
  * A fraction `dup_frac` of the tokens i >= 1 are near-duplicates: they copy the
    nearest preceding original token plus noise of per-component std
    dup_noise/sqrt(d).
  * Window queries (G*W rows per KV head): a centre each (a fraction
    `salient_frac` of the rows share one salient centre) plus the same noise,
    scaled per head so that the logits q.k/sqrt(d) over the non-sink keys have a
    standard deviation of `logit_std`.
  * Token 0 is an attention sink: its key points along the mean window-query
    direction, with the norm that gives it about half of a typical row's mass.
  * Values: the same key recipe from the same generator (no sink).
Keys are treated as already rotated (post-RoPE); no RoPE is applied.
Everything is produced in float32 and rounded once to bf16.
"""

from __future__ import annotations

import hashlib
import math

import torch


def _seed(*parts) -> int:
    h = hashlib.sha256(("/".join(str(p) for p in parts)).encode()).digest()
    return int.from_bytes(h[:8], "little") & ((1 << 63) - 1)


def _normal(gen, shape, device):
    return torch.randn(shape, generator=gen, device=device, dtype=torch.float32)


def _clustered(gen, H, L, d, centres, noise, dup_frac, dup_noise, device):
    """[H, L, d] tokens around `centres` [H, 64, d] with near-duplicate runs."""
    nc = centres.shape[1]
    z = torch.randint(0, nc, (H, L), generator=gen, device=device)
    x = torch.gather(centres, 1, z[..., None].expand(H, L, d)).clone()
    x += _normal(gen, (H, L, d), device) * (noise / math.sqrt(d))
    dup = torch.rand((H, L), generator=gen, device=device) < dup_frac
    dup[:, 0] = False
    pos = torch.arange(L, device=device).expand(H, L)
    base = torch.where(dup, torch.zeros_like(pos), pos).cummax(dim=1).values
    copy = torch.gather(x, 1, base[..., None].expand(H, L, d))
    jitter = _normal(gen, (H, L, d), device) * (dup_noise / math.sqrt(d))
    return torch.where(dup[..., None], copy + jitter, x)


def unit_tensors(seed, r, layer, L, Hkv, G, W, d=128, salient_frac=0.0, noise=0.1,
                 dup_frac=0.3, dup_noise=0.01, logit_std=3.0, device="cpu"):
    """Keys [Hkv, L, d], values [Hkv, L, d] and window queries [Hkv, G*W, d] (fp32)."""
    gen = torch.Generator(device=device)
    gen.manual_seed(_seed(seed, r, layer))
    n = G * W
    centres = _normal(gen, (Hkv, 64, d), device)
    centres /= centres.norm(dim=-1, keepdim=True)
    k = _clustered(gen, Hkv, L, d, centres, noise, dup_frac, dup_noise, device)
    zq = torch.randint(0, 64, (Hkv, n), generator=gen, device=device)
    salient = torch.rand((Hkv, n), generator=gen, device=device) < salient_frac
    zq = torch.where(salient, torch.zeros_like(zq), zq)
    q = torch.gather(centres, 1, zq[..., None].expand(Hkv, n, d)).clone()
    q += _normal(gen, (Hkv, n, d), device) * (noise / math.sqrt(d))
    # scale queries so the non-sink logits have the requested spread
    logits = torch.einsum("hnd,hld->hnl", q, k[:, 1:]) / math.sqrt(d)
    scale = logit_std / logits.std(dim=(1, 2), keepdim=True).clamp_min(1e-6)
    q *= scale
    logits *= scale
    # attention sink at token 0: along the mean query direction, sized so that its
    # logit matches the median row log-sum-exp of the other keys (about half the mass)
    u = q.mean(dim=1)
    u /= u.norm(dim=-1, keepdim=True).clamp_min(1e-6)
    lse = torch.logsumexp(logits, dim=2)                      # [Hkv, n]
    proj = torch.einsum("hnd,hd->hn", q, u) / math.sqrt(d)     # logit per unit sink norm
    ratio = torch.where(proj > 1e-3, lse / proj.clamp_min(1e-3), torch.zeros_like(lse))
    beta = ratio.median(dim=1).values.clamp(0.0, 1e4)
    k[:, 0] = u * beta[:, None]
    v = _clustered(gen, Hkv, L, d, _normal(gen, (Hkv, 64, d), device), noise, dup_frac,
                   dup_noise, device)
    return k, v, q


def make_batch(spec: dict, seed: int = 2609, device="cpu", with_values: bool = True,
               request_ids=None):
    """Inputs of a whole call in the library's layouts (see include/kv_evict.h):
    q_win [N_L][n_req][Hq][W][d], k/v [N_L][Hkv][SL][d], all bf16 (torch tensors).
    request_ids[j] (default j) is the request number that seeds the j-th request, so
    that a subset of a batch's requests gets the same tensors as in the whole batch."""
    N_L, Hq, Hkv, d, W = (spec["num_layers"], spec["num_q_heads"], spec["num_kv_heads"],
                          spec["head_dim"], spec["window"])
    lens = [int(x) for x in spec["seq_lens"]]
    G = Hq // Hkv
    SL = sum(lens)
    q_win = torch.empty((N_L, len(lens), Hq, W, d), dtype=torch.bfloat16, device=device)
    k = torch.empty((N_L, Hkv, SL, d), dtype=torch.bfloat16, device=device)
    v = torch.empty((N_L, Hkv, SL, d), dtype=torch.bfloat16, device=device) if with_values else None
    ids = list(range(len(lens))) if request_ids is None else [int(x) for x in request_ids]
    assert len(ids) == len(lens)
    off = 0
    for r, L in enumerate(lens):
        for layer in range(N_L):
            kk, vv, qq = unit_tensors(seed, ids[r], layer, L, Hkv, G, W, d,
                                      salient_frac=spec.get("salient_frac", 0.0), device=device)
            k[layer, :, off:off + L] = kk.to(torch.bfloat16)
            if with_values:
                v[layer, :, off:off + L] = vv.to(torch.bfloat16)
            q_win[layer, r] = qq.reshape(Hkv, G, W, d).reshape(Hq, W, d).to(torch.bfloat16)
        off += L
    return dict(q_win=q_win, k=k, v=v, seq_lens=lens)
