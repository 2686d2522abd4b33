"""Named workloads (Mistral-7B attention shapes) and their layer-wise coefficients.

Every workload uses 32 query heads, 8 KV heads (GQA group 4) and head_dim 128, a
window of W = 32 queries and max-pooling kernel 7. The coefficient profiles are
inputs of a call; "segments" values are latent a-values mapped by lambda = sinh(a)
(Eq. 6), "quadratic" is the literal lambda2(l) = -0.6 + 1.2((l-15.5)/15.5)^2 - 0.6.
"""

from __future__ import annotations

import numpy as np

MISTRAL = dict(num_q_heads=32, num_kv_heads=8, head_dim=128, window=32, pool_kernel=7,
               candidate_factor=4, norm_eps=1e-12)


def _ragged_lens(seed: int, n: int, lo: int, hi: int):
    rng = np.random.default_rng(seed)
    return [int(x) for x in rng.integers(lo, hi + 1, size=n)]


WORKLOADS = {
    # one layer at L=2048: the small parity case
    "mistral-1layer-L2048": dict(MISTRAL, num_layers=1, seq_lens=[2048], budget=64,
                                 lambdas=("global", 0.5, -0.5)),
    # full 32-layer model shape at L=8192
    "mistral-32layer-L8192": dict(MISTRAL, num_layers=32, seq_lens=[8192], budget=64,
                                  lambdas=("global", 0.5, -0.5)),
    # long-context budget sweep at L=32768 with a salient query cluster
    "mistral-32layer-L32768-B32": dict(MISTRAL, num_layers=32, seq_lens=[32768], budget=32,
                                       salient_frac=0.2, lambdas=("global", 0.5, -0.5)),
    "mistral-32layer-L32768-B64": dict(MISTRAL, num_layers=32, seq_lens=[32768], budget=64,
                                       salient_frac=0.2, lambdas=("global", 0.5, -0.5)),
    "mistral-32layer-L32768-B128": dict(MISTRAL, num_layers=32, seq_lens=[32768], budget=128,
                                        salient_frac=0.2, lambdas=("global", 0.5, -0.5)),
    # three-segment profile with the mid-layer sign flip of lambda2, L=16384, B=128
    "mistral-32layer-L16384-segments": dict(MISTRAL, num_layers=32, seq_lens=[16384],
                                            budget=128,
                                            lambdas=("segments", (0.3, 0.3, 0.3),
                                                     (-0.8, 0.6, -0.8))),
    # 16 ragged requests, L_r ~ U[4096, 32768], quadratic lambda2 over depth
    "mistral-32layer-ragged16": dict(MISTRAL, num_layers=32,
                                     seq_lens=_ragged_lens(2609, 16, 4096, 32768), budget=64,
                                     lambdas=("quadratic", 0.2)),
}


def scaled(spec: dict, **over) -> dict:
    """A copy of `spec` with fields replaced (e.g. fewer layers for a quick case)."""
    out = dict(spec)
    out.update(over)
    return out


def lambda_arrays(spec: dict, profile_fn):
    """(lambda1[N_L], lambda2[N_L]) as float64 arrays.

    profile_fn(kind, c, num_layers) -> array implements Eq. 6 (the caller chooses
    whose implementation: the oracle's or the library's)."""
    N_L = spec["num_layers"]
    kind = spec["lambdas"][0]
    if kind == "global":
        _, l1, l2 = spec["lambdas"]
        return np.full(N_L, float(l1)), np.full(N_L, float(l2))
    if kind == "segments":
        _, a1, a2 = spec["lambdas"]
        return (np.asarray(profile_fn("segments", a1, N_L), dtype=np.float64),
                np.asarray(profile_fn("segments", a2, N_L), dtype=np.float64))
    if kind == "quadratic":
        _, l1 = spec["lambdas"]
        ell = np.arange(N_L, dtype=np.float64)
        mid = (N_L - 1) / 2.0
        return (np.full(N_L, float(l1)),
                -0.6 + 1.2 * ((ell - mid) / mid) ** 2 - 0.6)
    raise ValueError(kind)


def partition_requests(seq_lens, world: int):
    """Split the requests of one batch across `world` ranks, balanced by prefix tokens
    (the score kernel's work is proportional to them): longest first, each to the
    rank with the fewest tokens so far (ties to the lower rank). Returns one sorted
    list of request indices per rank; every request goes to exactly one rank. A
    rank may get none when there are fewer requests than ranks."""
    loads = [0] * world
    parts = [[] for _ in range(world)]
    for r in sorted(range(len(seq_lens)), key=lambda i: (-int(seq_lens[i]), i)):
        j = min(range(world), key=lambda w: (loads[w], w))
        parts[j].append(r)
        loads[j] += int(seq_lens[r])
    return [sorted(p) for p in parts]


def request_layout(seq_lens, num_layers: int, unit_heads: int):
    """Per request r, (first unit, units, first mu/sigma element, elements) in the
    layouts of include/kv_evict.h: units are request-major (N_L * unit_heads per
    request) and mu / sigma are packed per request (N_L * unit_heads * L_r)."""
    out = []
    unit = elem = 0
    for L in seq_lens:
        n_u = num_layers * unit_heads
        out.append((unit, n_u, elem, n_u * int(L)))
        unit += n_u
        elem += n_u * int(L)
    return out
