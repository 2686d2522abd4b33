"""Comparison of the CUDA path with the fp64 oracle (test helpers).

Tolerances (the kernels compute A, mu and sigma in fp32 from bf16 inputs):
  mu:    |d| <= 1e-3 |mu_ref| + 1e-30                      (1e-3 relative)
  sigma: |d| <= 1e-3 |sigma_ref| + 1e-30                   (1e-3 relative)
         Columns whose window rows give nearly equal A (sigma << mu, e.g. zero
         queries) carry an error set by the fp32 error of each A, which scales with
         mu, not sigma; the test that builds such columns passes a floor
         sigma_mu_floor * mu_ref (1e-4). No other workload needs it.
  The 1e-30 absolute floor covers keys with A below about 2^-103 (mu ~ 1e-31),
  whose squares underflow in the kernel's fp32 column sums.
  selection: the GPU's admissions are replayed through the oracle; at every step the
  GPU's pick must be the oracle's argmax, or within TIE_TOL = 1e-4 (in s~ units) of
  it; a pick outside the oracle's top-C pool must lie within TIE_TOL of the cut.
  gather: bit-exact.
"""

from __future__ import annotations

import numpy as np

from oracle import kv_evict_oracle as O

MU_RTOL = 1e-3
SIGMA_RTOL = 1e-3
SIGMA_MU_FLOOR = 1e-4      # only where a test builds near-constant columns
ABS_FLOOR = 1e-30
TIE_TOL = 1e-4


def to_bits(t) -> np.ndarray:
    """bf16 torch tensor -> uint16 numpy bit patterns."""
    import torch
    return t.detach().view(torch.int16).cpu().numpy().view(np.uint16)


def check_mu_sigma(mu_gpu, sigma_gpu, mu_ref, sigma_ref, what="", sigma_mu_floor=0.0):
    mu_gpu = np.asarray(mu_gpu, dtype=np.float64)
    sigma_gpu = np.asarray(sigma_gpu, dtype=np.float64)
    dmu = np.abs(mu_gpu - mu_ref)
    tol_mu = MU_RTOL * np.abs(mu_ref) + ABS_FLOOR
    bad = np.flatnonzero(~(dmu <= tol_mu))
    assert len(bad) == 0, (f"{what} mu mismatch at {bad[:5]}: gpu {mu_gpu[bad[:5]]} "
                           f"ref {mu_ref[bad[:5]]}")
    ds = np.abs(sigma_gpu - sigma_ref)
    tol_s = SIGMA_RTOL * np.abs(sigma_ref) + sigma_mu_floor * np.abs(mu_ref) + ABS_FLOOR
    bad = np.flatnonzero(~(ds <= tol_s))
    assert len(bad) == 0, (f"{what} sigma mismatch at {bad[:5]}: gpu {sigma_gpu[bad[:5]]} "
                           f"ref {sigma_ref[bad[:5]]} mu {mu_ref[bad[:5]]}")
    rel = dmu / np.maximum(np.abs(mu_ref), 1e-300)
    return float(rel.max())


def check_selection(order_gpu, indices_gpu, mu_ref, sigma_ref, keys_f64, L, W, B, lambda1, lambda2,
                    pool_kernel=7, candidate_factor=4, norm_eps=1e-12, margins_gpu=None, what=""):
    """Replay the GPU's admission order through the oracle. Returns the list of
    accepted near-tie swaps (step, gpu pick, oracle pick, gap, kind): kind "argmax"
    when the GPU admitted a pool member whose value is within TIE_TOL below the
    oracle's argmax (gap = v_best - v_pick >= 0), "cut" when the GPU's pool held a
    position the oracle's top-C pool left out, its s~ within TIE_TOL of the cut
    (gap = the oracle's cut value minus its s~)."""
    Lc = L - W
    C = Lc if candidate_factor == 0 else min(candidate_factor * B, Lc)
    nsel = min(B, C)
    order_gpu = [int(x) for x in order_gpu[:nsel]]
    idx = np.asarray(indices_gpu)
    assert np.all(idx[nsel:] == -1), f"{what} padding"
    assert np.array_equal(np.sort(order_gpu), idx[:nsel]), f"{what} indices != sorted order"
    assert len(set(order_gpu)) == nsel and min(order_gpu) >= 0 and max(order_gpu) < Lc, what
    ref = O.select_unit(mu_ref, sigma_ref, keys_f64, L, W, B, lambda1, lambda2, pool_kernel,
                        candidate_factor, norm_eps, follow=order_gpu)
    pool = set(int(x) for x in ref["pool"])
    st = ref["s_tilde"]
    ranked = O.rank_desc(st)
    cut_value = st[ranked[C - 1]]
    swaps = []
    for t, step in enumerate(ref["steps"]):
        if step["pick"] != step["best"]:
            gap = step["v_best"] - step["v_pick"]
            assert gap <= TIE_TOL, (f"{what} step {t}: gpu admitted {step['pick']} but the oracle's "
                                    f"argmax {step['best']} is better by {gap:.3e}")
        if step["pick"] not in pool:
            assert st[step["pick"]] >= cut_value - TIE_TOL, (
                f"{what} step {t}: pick {step['pick']} outside the top-C pool")
            swaps.append((t, step["pick"], step["best"], float(cut_value - st[step["pick"]]), "cut"))
        elif step["pick"] != step["best"]:
            swaps.append((t, step["pick"], step["best"], step["v_best"] - step["v_pick"], "argmax"))
    if margins_gpu is not None and not swaps:
        m_ref = np.array([s["margin"] for s in ref["steps"]])
        m_gpu = np.asarray(margins_gpu[:nsel], dtype=np.float64)
        finite = np.isfinite(m_ref)
        assert np.all(np.isfinite(m_gpu) == finite), f"{what} margin finiteness"
        assert np.all(np.abs(m_gpu[finite] - m_ref[finite]) <= TIE_TOL), f"{what} margins"
    return swaps


def check_gather(k_out_bits, v_out_bits, k_bits, v_bits, indices, L, W, B):
    ko, vo = O.gather_unit(k_bits, v_bits, indices[indices >= 0], L, W, B)
    assert np.array_equal(k_out_bits, ko)
    assert np.array_equal(v_out_bits, vo)
