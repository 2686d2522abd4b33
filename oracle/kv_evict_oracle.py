"""Plain fp64 CPU oracle of the diversified KV-eviction step.

TEST INFRASTRUCTURE. This module is the correctness reference for the CUDA
library. Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import it; the library never calls it, and it shares no code with
the library (no kernels, headers, helpers or constants).

It restates "Beyond Mean Attention: Diversity-Aware, Layer-Wise Scoring for KV
Cache Eviction", Section 3, one unit (request, layer, KV head) at a time, in
float64 from the bf16-decoded inputs, in the paper's order:

  window_attention   Section 3.1, context of Eq. 1: softmax attention A[q, i] of
                     the window queries over the causal prefix.
  window_lse         the same rows' natural-log softmax normalisers (what a prefill's
                     attention computes for its own output; input of the one-pass score).
  mean_attention     Eq. 1: mu_i = (1/|W|) sum_q A[q, i].
  dispersion         Eq. 3: sample standard deviation, divisor |W| - 1.
  max_pool           Section 3.1: the baselines' max-pooling of the scores.
  base_score         Eq. 2 without the redundancy term: s_i = mu_i + lambda1 sigma_i.
  candidate_pool     Section 3.2: candidates restricted to the top 4B by s.
  normalise          Eq. 5: s~_i = s_i / max_j s_j, denominator clamped positive.
  corr               Eq. 4: max(0, max_{j in S} cos(k_i, k_j)), corr(i, {}) = 0.
  greedy_mmr         Eq. 5: S <- S + argmax_{i not in S}(s~_i + lambda2 corr(i, S)),
                     first admission argmax s~, until |S| = B.
  gather             Section 1: the layer keeps B entries (plus the window).
  window_output      Section 3.2 ("uses existing attention"): the window rows' own
                     attention output O[r] = sum_i A[r, i] v_i, from the same A as Eq. 1.
  depth_profile      Eq. 6: a(l) = c0 + c1 t + c2 t^2, t = l/(N_L - 1),
                     lambda = sinh(a); Global / Segments / Curve.

Readings where the paper is silent:
  * GQA: the window rows of a KV head are all n = G*W rows of the G query heads
    that share it; mu and sigma are taken over those n rows (sigma divisor n - 1,
    sigma = 0 when n = 1).
  * Window tokens count in every softmax denominator, are not candidates, and are
    always kept; the candidates are positions 0 .. L - W - 1.
  * Pooling: max-pool of mu and of sigma separately, odd kernel k, stride 1, the
    window clipped to the candidate range.
  * Ties (top-C cut and every argmax): larger value first, then lower position.
  * A zero-norm key has cos = 0 with every key.

Parity pins: every function here is checked in tests/test_oracle_pins.py against
closed forms, invariants, special cases that reduce to library routines, and
brute force on tiny inputs. The end-to-end effect on LongBench accuracy is
parity unpinned (no datasets or model weights are available).
"""

from __future__ import annotations

import math

import numpy as np

# ----------------------------------------------------------------------------
# Input decoding


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """Decode bf16 bit patterns (uint16) exactly into float64."""
    b = np.ascontiguousarray(bits).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


# ----------------------------------------------------------------------------
# Section 3.1: window attention, Eq. 1 and Eq. 3


def window_positions(L: int, W: int, G: int) -> np.ndarray:
    """Token position of every window row r = g*W + w (query of head g at L-W+w)."""
    return np.tile(np.arange(L - W, L, dtype=np.int64), G)


def window_attention(q: np.ndarray, k: np.ndarray, L: int, W: int, G: int) -> np.ndarray:
    """A[r, i] for the n = G*W window rows over the L prefix keys.

    Logits are q_r . k_i / sqrt(d); the row at position p attends to keys 0..p
    (prefill is causal), window keys included; A is the softmax of each row over
    its unmasked keys and is 0 where masked.
    """
    n, d = q.shape
    assert k.shape == (L, d) and n == G * W
    logits = (q @ k.T) / math.sqrt(d)
    pos = window_positions(L, W, G)
    visible = np.arange(L)[None, :] <= pos[:, None]
    logits = np.where(visible, logits, -np.inf)
    row_max = logits.max(axis=1, keepdims=True)
    e = np.where(visible, np.exp(logits - row_max), 0.0)
    return e / e.sum(axis=1, keepdims=True)


def window_lse(q: np.ndarray, k: np.ndarray, L: int, W: int, G: int) -> np.ndarray:
    """The natural-log softmax normaliser of every window row: ln sum_i exp(q_r . k_i /
    sqrt(d)) over the keys the row sees (the same causal mask as window_attention), so
    that A[r, i] = exp(q_r . k_i / sqrt(d) - lse_r) on those keys."""
    n, d = q.shape
    assert k.shape == (L, d) and n == G * W
    logits = (q @ k.T) / math.sqrt(d)
    pos = window_positions(L, W, G)
    visible = np.arange(L)[None, :] <= pos[:, None]
    logits = np.where(visible, logits, -np.inf)
    row_max = logits.max(axis=1)
    return row_max + np.log(np.where(visible, np.exp(logits - row_max[:, None]), 0.0).sum(axis=1))


def mean_attention(A: np.ndarray) -> np.ndarray:
    """Eq. 1: mu_i = (1/n) sum_r A[r, i]."""
    return A.sum(axis=0) / A.shape[0]


def dispersion(A: np.ndarray, mu: np.ndarray) -> np.ndarray:
    """Eq. 3: sigma_i = sqrt( sum_r (A[r, i] - mu_i)^2 / (n - 1) ), two-pass."""
    n = A.shape[0]
    if n < 2:
        return np.zeros(A.shape[1])
    dev = A - mu[None, :]
    return np.sqrt((dev * dev).sum(axis=0) / (n - 1))


# ----------------------------------------------------------------------------
# Section 3.1 pooling, Eq. 2, Section 3.2 candidate restriction, Eq. 5


def max_pool(x: np.ndarray, kernel: int) -> np.ndarray:
    """y_i = max of x_j over |j - i| <= (kernel-1)/2, j inside [0, len(x))."""
    assert kernel >= 1 and kernel % 2 == 1
    h = kernel // 2
    padded = np.concatenate([np.full(h, -np.inf), x, np.full(h, -np.inf)])
    # window i of the padded array covers x[i-h .. i+h]; the -inf padding stands for
    # positions outside [0, len(x)), which the clipped window leaves out
    return np.lib.stride_tricks.sliding_window_view(padded, kernel).max(axis=1)


def base_score(mu_hat: np.ndarray, sigma_hat: np.ndarray, lambda1: float) -> np.ndarray:
    """Eq. 2 without corr: s_i = mu_i + lambda1 * sigma_i."""
    return mu_hat + lambda1 * sigma_hat


def pooled_base_score(mu: np.ndarray, sigma: np.ndarray, Lc: int, kernel: int,
                      lambda1: float) -> np.ndarray:
    """Section 3.1 pooling, then Eq. 2 without corr, over the candidates [0, Lc):
    mu and sigma are max-pooled separately, then s_i = mu^_i + lambda1 sigma^_i."""
    return base_score(max_pool(mu[:Lc], kernel), max_pool(sigma[:Lc], kernel), lambda1)


def rank_desc(values: np.ndarray) -> np.ndarray:
    """Positions sorted by value descending, ties to the lower position."""
    return np.lexsort((np.arange(len(values)), -values))


def candidate_pool(s: np.ndarray, C: int) -> np.ndarray:
    """Section 3.2: the C candidate positions with the largest base score."""
    return rank_desc(s)[:C]


def normalise(s: np.ndarray, pool: np.ndarray, eps: float) -> np.ndarray:
    """Eq. 5: s~ = s / max(max_{j in pool} s_j, eps)."""
    return s / max(float(s[pool].max()), eps)


# ----------------------------------------------------------------------------
# Eq. 4 and Eq. 5: redundancy and greedy admission


def cosine(a: np.ndarray, b: np.ndarray) -> float:
    """cos(a, b); 0 when either vector is zero."""
    na = math.sqrt(float(a @ a))
    nb = math.sqrt(float(b @ b))
    if na == 0.0 or nb == 0.0:
        return 0.0
    return float(a @ b) / (na * nb)


def corr(i: int, S, keys: np.ndarray) -> float:
    """Eq. 4: max(0, max_{j in S} cos(k_i, k_j)); 0 for the empty set."""
    best = 0.0
    for j in S:
        best = max(best, cosine(keys[i], keys[j]))
    return best


def cosine_table(keys: np.ndarray, rows, cols) -> np.ndarray:
    """cos(k_i, k_j) for i in rows, j in cols (one matmul); 0 where a key is zero."""
    a = keys[np.asarray(rows, dtype=np.int64)]
    b = keys[np.asarray(cols, dtype=np.int64)]
    na = np.sqrt((a * a).sum(axis=1))
    nb = np.sqrt((b * b).sum(axis=1))
    inv_a = np.where(na > 0, 1.0 / np.where(na > 0, na, 1.0), 0.0)
    inv_b = np.where(nb > 0, 1.0 / np.where(nb > 0, nb, 1.0), 0.0)
    return (a @ b.T) * inv_a[:, None] * inv_b[None, :]


def greedy_mmr(s_tilde: np.ndarray, keys: np.ndarray, cand: np.ndarray, lambda2: float,
               B: int, follow=None):
    """Eq. 5 over the candidate positions `cand`.

    Admits min(B, len(cand)) positions. corr is kept incrementally: after each
    admission j, corr_i <- max(corr_i, cos(k_i, k_j)), which equals Eq. 4 for the
    grown set (the max over S of a set grows by one term; corr starts at 0, which
    is both corr(i, {}) and the clamp of Eq. 4).

    Returns a list of steps; step t is a dict with
      pick    -- the admitted position,
      best    -- the oracle's own argmax (larger value, then lower position),
      v_best  -- its greedy value, v_pick -- the admitted position's value,
      margin  -- v_best minus the best value among the other remaining candidates
                 (inf when no other remains).
    With `follow` (a sequence of positions) the oracle admits follow[t] instead of
    its own argmax at every step (forced replay); a position outside `cand` joins
    the candidates when it is admitted, with its corr recomputed from Eq. 4.
    """
    cand = np.asarray(cand, dtype=np.int64)
    cos = cosine_table(keys, cand, cand)
    corr_v = np.zeros(len(cand))
    taken = np.zeros(len(cand), dtype=bool)
    selected: list[int] = []
    steps = []
    n_adm = min(B, len(cand)) if follow is None else len(follow)
    for t in range(n_adm):
        vals = s_tilde[cand] + lambda2 * corr_v
        rem = np.flatnonzero(~taken)
        order = rem[np.lexsort((cand[rem], -vals[rem]))]
        best = int(order[0])
        margin = vals[order[0]] - vals[order[1]] if len(order) > 1 else math.inf
        if follow is None:
            p = best
        else:
            hit = np.flatnonzero(cand == int(follow[t]))
            if len(hit) == 0:  # forced pick outside this oracle's candidates
                pick = int(follow[t])
                cand = np.append(cand, pick)
                corr_v = np.append(corr_v, corr(pick, selected, keys))
                taken = np.append(taken, False)
                cos = cosine_table(keys, cand, cand)
                vals = np.append(vals, s_tilde[pick] + lambda2 * corr_v[-1])
                p = len(cand) - 1
            else:
                p = int(hit[0])
        steps.append(dict(pick=int(cand[p]), best=int(cand[best]), v_best=float(vals[best]),
                          v_pick=float(vals[p]), margin=float(margin)))
        selected.append(int(cand[p]))
        taken[p] = True
        corr_v = np.maximum(corr_v, cos[:, p])
    return steps


# ----------------------------------------------------------------------------
# One unit end to end


def select_unit(mu: np.ndarray, sigma: np.ndarray, keys: np.ndarray, L: int, W: int, B: int,
                lambda1: float, lambda2: float, pool_kernel: int = 7,
                candidate_factor: int = 4, norm_eps: float = 1e-12, follow=None):
    """Pooling, Eq. 2, Section 3.2, Eq. 5 for one unit.

    Returns dict(indices=sorted admitted positions, steps=greedy trace,
    pool=candidate positions, s_tilde=normalised base scores over [0, Lc),
    cut_margin=s~ of the last pool member minus the first one left out).
    """
    Lc = L - W
    s = pooled_base_score(mu, sigma, Lc, pool_kernel, lambda1)
    C = Lc if candidate_factor == 0 else min(candidate_factor * B, Lc)
    ranked = rank_desc(s)
    pool = ranked[:C]
    s_tilde = normalise(s, pool, norm_eps)
    cut_margin = (s_tilde[ranked[C - 1]] - s_tilde[ranked[C]]) if C < Lc else math.inf
    steps = greedy_mmr(s_tilde, keys, pool, lambda2, B, follow=follow)
    idx = np.sort(np.array([st["pick"] for st in steps], dtype=np.int64))
    return dict(indices=idx, steps=steps, pool=pool, s_tilde=s_tilde, cut_margin=cut_margin)


def window_output(A: np.ndarray, v: np.ndarray) -> np.ndarray:
    """The attention output of the window rows: O[r] = sum_i A[r, i] v_i over the
    prefix (A from window_attention: causal softmax rows, 0 where masked). Section 3.2
    scores tokens with the prefill's existing attention; these rows are that
    attention's output for the last W positions of every query head."""
    return A @ v


def score_unit(q: np.ndarray, k: np.ndarray, L: int, W: int, G: int):
    """Steps 1-2 for one unit: (mu, sigma) over all L tokens (Eq. 1, Eq. 3)."""
    A = window_attention(q, k, L, W, G)
    mu = mean_attention(A)
    return mu, dispersion(A, mu)


def gather_unit(k_bits: np.ndarray, v_bits: np.ndarray, indices: np.ndarray, L: int, W: int,
                B: int):
    """Compact cache of one unit as bit patterns: kept rows ascending, then the W
    window rows, then zero rows up to B + W."""
    d = k_bits.shape[1]
    rows = list(indices) + list(range(L - W, L))
    ko = np.zeros((B + W, d), dtype=k_bits.dtype)
    vo = np.zeros((B + W, d), dtype=v_bits.dtype)
    ko[: len(rows)] = k_bits[rows]
    vo[: len(rows)] = v_bits[rows]
    return ko, vo


# ----------------------------------------------------------------------------
# Eq. 6: depth profiles


def depth_profile(kind: str, c, num_layers: int, seg_bounds=None) -> np.ndarray:
    """lambda^(l) = sinh(a(l)) for l = 0..N_L-1.

    global:   a(l) = c[0]
    segments: a(l) = c[0], c[1], c[2] on the shallow, middle and deep parts,
              split at seg_bounds = (b0, b1), by default thirds
              (b0 = ceil(N_L/3), b1 = ceil(2 N_L/3))
    curve:    a(l) = c0 + c1 t + c2 t^2 with t = l / (N_L - 1)
    """
    ells = np.arange(num_layers)
    if kind == "global":
        a = np.full(num_layers, float(c[0]))
    elif kind == "segments":
        if seg_bounds is None:
            seg_bounds = (-(-num_layers // 3), -(-2 * num_layers // 3))
        b0, b1 = seg_bounds
        a = np.where(ells < b0, float(c[0]), np.where(ells < b1, float(c[1]), float(c[2])))
    elif kind == "curve":
        t = ells / (num_layers - 1) if num_layers > 1 else np.zeros(num_layers)
        a = float(c[0]) + float(c[1]) * t + float(c[2]) * t * t
    else:
        raise ValueError(kind)
    return np.sinh(a)


# ----------------------------------------------------------------------------
# Layout helpers for the batched tensors (documented in include/kv_evict.h)


def unit_slices(q_bits, k_bits, seq_lens, r, layer, h, n_kv_heads, W):
    """Window rows [n, d] and keys [L, d] (bf16 bits) of unit (r, layer, h) from the
    batched q_win [N_L][n_req][Hq][W][d] and k [N_L][Hkv][SL][d] arrays."""
    Hq = q_bits.shape[2]
    G = Hq // n_kv_heads
    d = q_bits.shape[-1]
    off = int(sum(seq_lens[:r]))
    L = int(seq_lens[r])
    q = q_bits[layer, r, h * G:(h + 1) * G].reshape(G * W, d)
    k = k_bits[layer, h, off:off + L]
    return q, k


def evict_unit(q_bits, k_bits, L, W, G, B, lambda1, lambda2, pool_kernel=7,
               candidate_factor=4, norm_eps=1e-12):
    """The whole step for one unit from bf16 bit patterns: mu, sigma and the
    selection (see select_unit)."""
    q = bf16_bits_to_f64(q_bits)
    k = bf16_bits_to_f64(k_bits)
    mu, sigma = score_unit(q, k, L, W, G)
    sel = select_unit(mu, sigma, k, L, W, B, lambda1, lambda2, pool_kernel,
                      candidate_factor, norm_eps)
    return mu, sigma, sel
