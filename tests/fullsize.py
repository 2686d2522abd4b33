"""Every unit of a full-size call against the fp64 oracle, on the host cores.

TEST INFRASTRUCTURE (GPU tests only). The CUDA path's outputs are copied to the
host one (request, layer) slice at a time -- the Hkv units that share its window
queries -- and checked in spawned worker processes, one BLAS thread each, so that
a 32-layer, 16-request call (4096 units) is checked unit by unit in about a
minute. At most two slices per worker are in flight, so host memory stays
bounded whatever the call's size. Each worker runs the oracle's Eq. 1 / Eq. 3
statistics and replays the GPU's admission order through the oracle's selection
(tests/parity.py: tolerances, near-tie swaps) and returns error statistics:

  mu_rel        max |mu - mu_ref| / mu_ref
  sigma_rel     max |sigma - sigma_ref| / sigma_ref over sigma_ref >= 1e-20
  sigma_tiny    keys with 0 < sigma_ref < 1e-20 (A below about 2^-103: the kernel's
                fp32 squares underflow there, and the 1e-30 absolute floor holds)
  sigma_floor   checks whose |sigma - sigma_ref| exceeds 1e-3 sigma_ref + 1e-30,
                i.e. that would need a mu-proportional floor (none is applied here)
  sigma_ratio   max |sigma - sigma_ref| / (1e-3 sigma_ref + 1e-4 mu_ref + 1e-30)
  swaps         accepted near-tie swaps (unit, step, gpu pick, oracle pick, gap, kind)
  failures      messages of every check that failed
"""

from __future__ import annotations

import multiprocessing as mp
import os

import numpy as np


def _slice_check(task):
    """One (request, layer) slice: every KV head's unit (runs in a worker)."""
    from oracle import kv_evict_oracle as O
    from tests import parity as PT
    (r, layer, L, W, G, B, lam1, lam2, pool_kernel, cand_factor, eps,
     q_bits, k_bits, mu, sigma, order, indices, margins) = task
    out = dict(units=0, mu_rel=0.0, sigma_rel=0.0, sigma_tiny=0, sigma_floor=0, sigma_ratio=0.0,
               swaps=[], failures=[])
    for h in range(k_bits.shape[0]):
        tag = f"unit(r={r},l={layer},h={h})"
        qf = O.bf16_bits_to_f64(q_bits[h])
        kf = O.bf16_bits_to_f64(k_bits[h])
        mu_ref, sg_ref = O.score_unit(qf, kf, L, W, G)
        m, s = mu[h].astype(np.float64), sigma[h].astype(np.float64)
        dmu = np.abs(m - mu_ref)
        dsg = np.abs(s - sg_ref)
        out["mu_rel"] = max(out["mu_rel"], float((dmu / np.maximum(mu_ref, 1e-300)).max()))
        pos = sg_ref >= 1e-20
        if pos.any():
            out["sigma_rel"] = max(out["sigma_rel"], float((dsg[pos] / sg_ref[pos]).max()))
        out["sigma_tiny"] += int(np.count_nonzero((sg_ref > 0) & (sg_ref < 1e-20)))
        out["sigma_floor"] += int(np.count_nonzero(dsg > PT.SIGMA_RTOL * sg_ref + PT.ABS_FLOOR))
        tol = PT.SIGMA_RTOL * sg_ref + PT.SIGMA_MU_FLOOR * mu_ref + PT.ABS_FLOOR
        out["sigma_ratio"] = max(out["sigma_ratio"], float((dsg / tol).max()))
        try:
            PT.check_mu_sigma(m, s, mu_ref, sg_ref, tag)
            sw = PT.check_selection(order[h], indices[h], mu_ref, sg_ref, kf, L, W, B, lam1, lam2,
                                    pool_kernel, cand_factor, eps, margins_gpu=margins[h], what=tag)
            out["swaps"] += [(tag,) + tuple(x) for x in sw]
        except AssertionError as e:
            out["failures"].append(str(e)[:400])
        out["units"] += 1
    return out


def _bits(t):
    import torch
    return t.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def _slices(spec, batch, plan, bufs, lambdas):
    """Host copies of the inputs and outputs of every (request, layer) slice."""
    seq = [int(x) for x in batch["seq_lens"]]
    N_L, Hkv, Hq = spec["num_layers"], spec["num_kv_heads"], spec["num_q_heads"]
    W, G, B = spec["window"], Hq // Hkv, spec["budget"]
    off = 0
    for r, L in enumerate(seq):
        base = N_L * Hkv * off
        for layer in range(N_L):
            q = _bits(batch["q_win"][layer, r]).reshape(Hkv, G * W, -1)
            k = _bits(batch["k"][layer, :, off:off + L])
            o = base + layer * Hkv * L
            mu = bufs.mu[o:o + Hkv * L].view(Hkv, L).cpu().numpy()
            sg = bufs.sigma[o:o + Hkv * L].view(Hkv, L).cpu().numpy()
            u0 = (r * N_L + layer) * Hkv
            yield (r, layer, L, W, G, int(plan.layer_budgets[layer]), float(lambdas[0][layer]),
                   float(lambdas[1][layer]), spec["pool_kernel"], spec["candidate_factor"],
                   spec["norm_eps"], q, k, mu, sg, bufs.order[u0:u0 + Hkv].cpu().numpy(),
                   bufs.indices[u0:u0 + Hkv].cpu().numpy(), bufs.margins[u0:u0 + Hkv].cpu().numpy())
        off += L


def check_every_unit(spec, batch, plan, bufs, lambdas, workers=None):
    """Oracle check of every unit of a call (default per-KV-head plan). Returns the
    merged statistics (see the module docstring)."""
    workers = workers or max(1, os.cpu_count() or 1)
    for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[var] = "1"
    total = dict(units=0, mu_rel=0.0, sigma_rel=0.0, sigma_tiny=0, sigma_floor=0, sigma_ratio=0.0,
                 swaps=[], failures=[])

    def merge(res):
        total["units"] += res["units"]
        total["sigma_floor"] += res["sigma_floor"]
        total["sigma_tiny"] += res["sigma_tiny"]
        for key in ("mu_rel", "sigma_rel", "sigma_ratio"):
            total[key] = max(total[key], res[key])
        total["swaps"] += res["swaps"]
        total["failures"] += res["failures"]

    with mp.get_context("spawn").Pool(workers) as pool:
        pending = []
        for task in _slices(spec, batch, plan, bufs, lambdas):
            pending.append(pool.apply_async(_slice_check, (task,)))
            while len(pending) >= 2 * workers:
                merge(pending.pop(0).get())
        for p in pending:
            merge(p.get())
    return total


def check_every_gather(spec, batch, plan, bufs):
    """The compact cache of every unit against plain torch indexing on the device:
    kept rows (ascending) then the W window rows, zero rows after them; bit-exact."""
    import torch
    seq = [int(x) for x in batch["seq_lens"]]
    N_L, Hkv, W, B = spec["num_layers"], spec["num_kv_heads"], spec["window"], spec["budget"]
    d = spec["head_dim"]
    off = 0
    for r, L in enumerate(seq):
        for layer in range(N_L):
            u0 = (r * N_L + layer) * Hkv
            idx = bufs.indices[u0:u0 + Hkv].long()
            m = int((idx[0] >= 0).sum())
            assert bool(((idx >= 0).sum(1) == m).all())
            rows = torch.cat([idx[:, :m], torch.arange(L - W, L, device=idx.device).expand(Hkv, W)], 1)
            for src, out in ((batch["k"], bufs.k_out), (batch["v"], bufs.v_out)):
                ref = torch.gather(src[layer, :, off:off + L], 1, rows[..., None].expand(-1, -1, d))
                got = out[u0:u0 + Hkv]
                assert torch.equal(got[:, :m + W].view(torch.int16), ref.view(torch.int16)), (r, layer)
                assert bool((got[:, m + W:].view(torch.int16) == 0).all()), (r, layer)
        off += L
