"""Host-side checks that need no GPU: the library loads and exports every entry
point of include/kv_evict.h, plan validation and the Eq. 6 profile helper."""

import ctypes
import os
import re

import numpy as np
import pytest

from oracle import kv_evict_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
LIB = os.path.join(ROOT, "paper_2609_30738_gb300", "libkvevict.so")


def _need_lib():
    if not os.path.exists(LIB):
        pytest.skip("library not built")


def _spec(**over):
    s = dict(num_layers=2, num_q_heads=32, num_kv_heads=8, head_dim=128, window=32, budget=64,
             pool_kernel=7, candidate_factor=4, norm_eps=1e-12)
    s.update(over)
    return s


def test_header_symbols_are_exported():
    _need_lib()
    header = open(os.path.join(ROOT, "include", "kv_evict.h")).read()
    names = set(re.findall(r"\b(kv_evict_\w+)\s*\(", header))
    assert len(names) >= 9
    lib = ctypes.CDLL(LIB)
    for n in sorted(names):
        assert hasattr(lib, n), n
    from paper_2609_30738_gb300 import kv_evict as K
    assert names == set(K.EXPORTS)


def test_plan_sizes_and_validation():
    _need_lib()
    from paper_2609_30738_gb300 import kv_evict as K
    p = K.Plan(_spec(), [2048, 777])
    assert p.n_units == 2 * 2 * 8
    assert p.score_elems == 2 * 8 * (2048 + 777)
    assert p.workspace_bytes > 0 and p.workspace_bytes % 256 == 0
    bad = [
        (_spec(head_dim=64), [100]),          # d != 128
        (_spec(window=33), [100]),            # G*W > 128
        (_spec(num_q_heads=30), [100]),       # Hq not a multiple of Hkv
        (_spec(pool_kernel=4), [100]),        # even pooling kernel
        (_spec(budget=0), [100]),
        (_spec(budget=200), [5000]),          # 4B > 512 candidates
        (_spec(), [32]),                      # L <= W
        (_spec(norm_eps=0.0), [100]),
        (_spec(num_layers=0), [100]),
        (_spec(), [100] * 65),                # too many requests
    ]
    for spec, lens in bad:
        with pytest.raises(K.KvEvictError) as e:
            K.Plan(spec, lens)
        assert e.value.status == K.KVE_EINVAL


def test_null_arguments_rejected_without_gpu():
    _need_lib()
    from paper_2609_30738_gb300 import kv_evict as K
    lib = K.library()
    p = K.Plan(_spec(), [300])
    assert lib.kv_evict_score(p._h, None, None, None, None, None, None) == K.KVE_EINVAL
    assert lib.kv_evict_gather(None, None, None, None, None, None, None) == K.KVE_EINVAL
    assert lib.kv_evict_plan_set_debug(p._h, 0, 0) == K.KVE_EINVAL
    assert lib.kv_evict_strerror(K.KVE_ETIMEOUT) == b"device-side wait timed out"
    # mu / sigma must be 16-byte aligned (the selector reads them 16 bytes at a time);
    # the check fails before any launch, so fake device addresses suffice
    lam = np.zeros(2, np.float32)
    good, odd = ctypes.c_void_p(1 << 20), ctypes.c_void_p((1 << 20) + 4)
    for mu, sg in [(odd, good), (good, odd)]:
        assert lib.kv_evict_select(p._h, mu, sg, good, lam.ctypes.data, lam.ctypes.data, good, None, None,
                                   good, None) == K.KVE_EINVAL
        assert lib.kv_evict_select_noalloc(p._h, mu, sg, good, lam.ctypes.data, lam.ctypes.data, good, None,
                                           None, None) == K.KVE_EINVAL


@pytest.mark.parametrize("kind,c", [("global", [0.3]), ("segments", [-0.8, 0.6, -0.8]),
                                    ("curve", [0.1, -0.7, 1.3])])
@pytest.mark.parametrize("N", [1, 5, 32])
def test_profile_matches_oracle(kind, c, N):
    _need_lib()
    from paper_2609_30738_gb300 import kv_evict as K
    lib_vals = K.profile(kind, c, N)
    ref = O.depth_profile(kind, c, N)
    np.testing.assert_allclose(lib_vals, ref, rtol=2e-7, atol=1e-7)


@pytest.mark.parametrize("B,N,r", [(64, 32, 0.5), (64, 32, 1.0), (64, 32, 0.1), (32, 5, 0.3),
                                   (1, 4, 1.0), (7, 3, 0.2), (128, 1, 0.5), (16, 2, 0.25)])
def test_budget_pyramid_properties(B, N, r):
    """Depth-decreasing budgets with the uniform total: non-increasing, sum N*B,
    first >= B >= last >= 1, last near r*B, uniform for r = 1."""
    _need_lib()
    from paper_2609_30738_gb300 import kv_evict as K
    b = K.budget_pyramid(B, N, r).astype(np.int64)
    assert b.sum() == N * B
    assert np.all(np.diff(b) <= 0) and b.min() >= 1
    assert b[0] >= B >= b[-1]
    if N > 1:
        assert abs(b[-1] - max(1, int(np.floor(r * B)))) <= 1
        # linear in depth: second differences of at most one unit (rounding)
        assert np.all(np.abs(np.diff(b, 2)) <= 2)
    if r == 1.0:
        assert np.all(b == B)


def test_budget_pyramid_and_layered_plan_validation():
    _need_lib()
    from paper_2609_30738_gb300 import kv_evict as K
    for args in [(0, 4, 0.5), (64, 0, 0.5), (64, 4, 0.0), (64, 4, 1.5)]:
        with pytest.raises(K.KvEvictError) as e:
            K.budget_pyramid(*args)
        assert e.value.status == K.KVE_EINVAL
    spec = _spec(num_layers=4, budget=24)
    p = K.Plan(spec, [2048], layer_budgets=[24, 18, 14, 8])
    assert p.layer_budgets == [24, 18, 14, 8]
    assert p.workspace_bytes == K.Plan(spec, [2048]).workspace_bytes
    for lb in ([24, 25, 14, 8], [24, 18, 0, 8]):          # above the stride, below one
        with pytest.raises(K.KvEvictError) as e:
            K.Plan(spec, [2048], layer_budgets=lb)
        assert e.value.status == K.KVE_EINVAL


def test_select_profiles_validation_without_gpu():
    """Multi-profile selection: scratch size per profile, and the host checks that
    return before any launch (so fake, aligned device addresses suffice)."""
    _need_lib()
    from paper_2609_30738_gb300 import kv_evict as K
    lib = K.library()
    p = K.Plan(_spec(num_layers=3), [2048, 777])
    words = 3 * 8 * (2048 + 777)
    padded = (words + 63) // 64 * 64
    for n in (1, 2, 14):
        assert p.select_profiles_workspace(n) == 256 + n * padded * 4   # error-word header
    with pytest.raises(K.KvEvictError) as e:
        p.select_profiles_workspace(0)
    assert e.value.status == K.KVE_EINVAL
    fake = ctypes.c_void_p(1 << 20)   # aligned, never dereferenced: validation fails first
    ok = np.zeros((2, 3), np.float32)
    for l1, l2, n in [(ok, ok, 0),
                      (np.array([[0.5, np.nan, 0.5], [0.5, 0.5, 0.5]], np.float32), ok, 2),
                      (ok, np.array([[0.0, 0.0, 0.0], [0.0, np.inf, 0.0]], np.float32), 2)]:
        st = lib.kv_evict_select_profiles(p._h, n, fake, fake, fake, l1.ctypes.data, l2.ctypes.data,
                                          fake, None, None, fake, None)
        assert st == K.KVE_EINVAL
    assert lib.kv_evict_select_profiles(p._h, 1, None, fake, fake, ok.ctypes.data, ok.ctypes.data,
                                        fake, None, None, fake, None) == K.KVE_EINVAL


def test_plan_ex_flags_without_gpu():
    """kv_evict_plan_ex: flag 0 is the layered plan, KVE_PLAN_PER_QUERY_HEAD makes one
    unit per query head, other bits are rejected."""
    _need_lib()
    from paper_2609_30738_gb300 import kv_evict as K
    spec = _spec(num_layers=3)
    base = K.Plan(spec, [2048, 777])
    perq = K.Plan(spec, [2048, 777], per_query_head=True)
    assert perq.n_units == 2 * 3 * 32 and base.n_units == 2 * 3 * 8
    assert perq.score_elems == 3 * 32 * (2048 + 777)
    assert perq.workspace_bytes > base.workspace_bytes
    lib = K.library()
    cfg = K.make_config(spec)
    lens = (ctypes.c_int64 * 1)(500)
    h, ws = ctypes.c_void_p(), ctypes.c_size_t()
    for bad in (2, 4, -1):
        assert lib.kv_evict_plan_ex(ctypes.byref(cfg), lens, 1, None, bad, ctypes.byref(h),
                                    ctypes.byref(ws)) == K.KVE_EINVAL
    assert lib.kv_evict_plan_ex(ctypes.byref(cfg), lens, 1, None, 0, ctypes.byref(h),
                                ctypes.byref(ws)) == K.KVE_OK
    lib.kv_evict_plan_destroy(h)


def test_every_candidate_plan_limits_without_gpu():
    """candidate_factor = 0: pools up to 512 candidates use the pooled selector; longer
    prefixes the every-candidate selector (Lc <= 32768, B <= 1024, with its own scratch
    in the workspace); multi-profile selection is refused for such plans."""
    _need_lib()
    from paper_2609_30738_gb300 import kv_evict as K
    small = K.Plan(_spec(candidate_factor=0), [500])
    big = K.Plan(_spec(candidate_factor=0), [5000])
    pooled = K.Plan(_spec(candidate_factor=4), [5000])
    assert big.workspace_bytes > pooled.workspace_bytes
    assert small.workspace_bytes > 0
    for spec, lens in [(_spec(candidate_factor=0), [32768 + 32 + 1]),
                       (_spec(candidate_factor=0, budget=1025), [5000])]:
        with pytest.raises(K.KvEvictError) as e:
            K.Plan(spec, lens)
        assert e.value.status == K.KVE_EINVAL
    K.Plan(_spec(candidate_factor=0), [32768 + 32])   # Lc = 32768: the largest
    with pytest.raises(K.KvEvictError) as e:
        big.select_profiles_workspace(2)
    assert e.value.status == K.KVE_EINVAL


def test_gather_refuses_pageable_host_memory_without_gpu():
    """kv_evict_gather reads k and v in place only from host memory the CUDA runtime
    pinned: the binding refuses a pageable CPU tensor, and the C ABI returns
    KVE_EINVAL for a pointer the runtime cannot classify (here: no GPU), both before
    any launch."""
    _need_lib()
    torch = pytest.importorskip("torch")
    from paper_2609_30738_gb300 import kv_evict as K
    p = K.Plan(_spec(num_layers=1), [300])
    k = torch.zeros((1, 8, 300, 128), dtype=torch.bfloat16)   # pageable
    idx = torch.zeros((8, 64), dtype=torch.int32)
    out = torch.zeros((8, 96, 128), dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        p.gather(k, k, idx, out, out)
    if torch.cuda.is_available():
        return   # the GPU suite checks the C ABI's refusal of pageable memory
    buf = np.zeros(1 << 16, dtype=np.uint8)
    ptr = buf.ctypes.data + (-buf.ctypes.data) % 16            # 16-byte aligned
    assert K.library().kv_evict_gather(p._h, ptr, ptr, ptr, ptr, ptr, None) == K.KVE_EINVAL


def test_noalloc_size_limit_counts_units_per_layer_without_gpu():
    """kv_evict_select_noalloc refuses, before any CUDA call, a plan whose scratch
    (one word per prefix token of every unit) exceeds its fixed 4194304-word array;
    a per-query-head plan has Hq units per layer, not Hkv, so it reaches the limit
    G times sooner."""
    _need_lib()
    from paper_2609_30738_gb300 import kv_evict as K
    lib = K.library()
    lam = np.zeros(32, np.float32)
    fake = ctypes.c_void_p(1 << 20)
    spec = _spec(num_layers=32)
    # 32 layers x 32 query heads x 4100 tokens = 4198400 words: over the limit
    perq = K.Plan(spec, [4100], per_query_head=True)
    assert perq.score_elems > 4194304
    assert lib.kv_evict_select_noalloc(perq._h, fake, fake, fake, lam.ctypes.data, lam.ctypes.data,
                                       fake, None, None, None) == K.KVE_EINVAL
    # the same prefix grouped per KV head needs 1049600 words: within the limit
    assert K.Plan(spec, [4100]).score_elems <= 4194304
    # 32 layers x 8 KV heads x 16385 tokens: over the limit
    big = K.Plan(spec, [16385])
    assert lib.kv_evict_select_noalloc(big._h, fake, fake, fake, lam.ctypes.data, lam.ctypes.data,
                                       fake, None, None, None) == K.KVE_EINVAL


def test_fused_and_given_normaliser_calls_validate_without_gpu():
    """kv_evict_select_gather and kv_evict_score_lse refuse null and misaligned
    arguments, and the binding refuses a pageable value tensor, before any launch."""
    _need_lib()
    torch = pytest.importorskip("torch")
    from paper_2609_30738_gb300 import kv_evict as K
    lib = K.library()
    p = K.Plan(_spec(num_layers=1), [300])
    assert lib.kv_evict_score_lse(p._h, None, None, None, None, None, None, None) == K.KVE_EINVAL
    good, odd = ctypes.c_void_p(1 << 20), ctypes.c_void_p((1 << 20) + 2)
    # lse must be 4-byte aligned; the check comes before any CUDA call
    assert lib.kv_evict_score_lse(p._h, good, good, odd, good, good, good, None) == K.KVE_EINVAL
    lam = np.zeros(1, np.float32)
    assert lib.kv_evict_select_gather(None, good, good, good, good, lam.ctypes.data, lam.ctypes.data, good,
                                      None, None, good, good, good, None) == K.KVE_EINVAL
    assert lib.kv_evict_select_gather(p._h, good, good, good, None, lam.ctypes.data, lam.ctypes.data, good,
                                      None, None, good, good, good, None) == K.KVE_EINVAL
    # misaligned mu, then a misaligned output row block
    assert lib.kv_evict_select_gather(p._h, odd, good, good, good, lam.ctypes.data, lam.ctypes.data, good,
                                      None, None, good, good, good, None) == K.KVE_EINVAL
    assert lib.kv_evict_select_gather(p._h, good, good, good, good, lam.ctypes.data, lam.ctypes.data, good,
                                      None, None, odd, good, good, None) == K.KVE_EINVAL
    k = torch.zeros((1, 8, 300, 128), dtype=torch.bfloat16)   # pageable
    mu = torch.zeros(8 * 300, dtype=torch.float32)
    idx = torch.zeros((8, 64), dtype=torch.int32)
    out = torch.zeros((8, 96, 128), dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        p.select_gather(mu, mu, k, k, lam, lam, idx, out, out, mu)


def test_kv_strides_validation_without_gpu():
    """kv_evict_plan_set_kv_strides: strides in elements (layer, KV head, token), each a
    multiple of 8 and below 2^37, the token stride at least d; NULL restores the dense
    layout; a refused call leaves the plan as it was."""
    _need_lib()
    from paper_2609_30738_gb300 import kv_evict as K
    SL, Hkv, d = 2048 + 777, 8, 128
    p = K.Plan(_spec(), [2048, 777])
    p.set_kv_strides((SL * Hkv * d, d, Hkv * d), (Hkv * SL * 2 * d, SL * 2 * d, 2 * d))
    p.set_kv_strides(None, None)
    p.set_kv_strides((Hkv * SL * d, SL * d, d))
    for bad in [(SL * Hkv * d, d, 64),            # token stride below d
                (SL * Hkv * d + 4, d, Hkv * d),    # not a multiple of 8 elements
                (-8, d, Hkv * d),
                (1 << 37, d, Hkv * d)]:
        with pytest.raises(K.KvEvictError) as e:
            p.set_kv_strides(bad, None)
        assert e.value.status == K.KVE_EINVAL
        with pytest.raises(K.KvEvictError) as e:
            p.set_kv_strides(None, bad)
        assert e.value.status == K.KVE_EINVAL
    assert K.library().kv_evict_plan_set_kv_strides(None, None, None) == K.KVE_EINVAL
