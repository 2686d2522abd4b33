"""Pins of the fp64 oracle to facts fixed outside it: closed forms, invariants,
special cases that reduce to library routines, hand-worked examples and brute
force on tiny inputs. CPU only."""

import itertools
import math
import os

import numpy as np
import pytest
import scipy.ndimage
import scipy.special

from oracle import kv_evict_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rand_unit(rng, L, W, G, d=16, scale=2.0):
    q = rng.standard_normal((G * W, d)) * scale
    k = rng.standard_normal((L, d))
    return q, k


# --------------------------------------------------------------------------
# Window attention and Eq. 1 / Eq. 3


def test_two_key_softmax_closed_form():
    """Golden: one row, two keys, logits a/sqrt(d) and 0 -> logistic closed form."""
    for line in open(os.path.join(GOLDEN, "two_key_softmax.txt")):
        if not line.startswith("a "):
            continue
        parts = line.split()
        a, A0, A1 = float(parts[1]), float(parts[3]), float(parts[4])
        q = np.array([[a, 0.0, 0.0, 0.0]])
        k = np.array([[1.0, 0.0, 0.0, 0.0], [0.0, 0.0, 0.0, 0.0]])
        A = O.window_attention(q, k, L=2, W=1, G=1)
        np.testing.assert_allclose(A[0], [A0, A1], rtol=1e-12)
        mu, sigma = O.score_unit(q, k, 2, 1, 1)
        np.testing.assert_allclose(mu, [A0, A1], rtol=1e-12)
        assert np.all(sigma == 0.0)


def test_rows_are_distributions_and_mu_sums_to_one():
    rng = np.random.default_rng(1)
    for L, W, G in [(40, 8, 4), (17, 16, 1), (64, 1, 3)]:
        q, k = _rand_unit(rng, L, W, G)
        A = O.window_attention(q, k, L, W, G)
        assert np.all(A >= 0) and np.all(A <= 1)
        np.testing.assert_allclose(A.sum(axis=1), 1.0, rtol=1e-12)
        mu = O.mean_attention(A)
        assert abs(mu.sum() - 1.0) < 1e-12


def test_causal_mask_counts():
    """Row at window offset w sees exactly L - W + w + 1 keys."""
    rng = np.random.default_rng(2)
    L, W, G = 30, 6, 2
    q, k = _rand_unit(rng, L, W, G)
    A = O.window_attention(q, k, L, W, G)
    for g in range(G):
        for w in range(W):
            row = A[g * W + w]
            assert np.count_nonzero(row) == L - W + w + 1
            assert np.all(row[L - W + w + 1:] == 0)


def test_softmax_matches_scipy_on_visible_prefix():
    rng = np.random.default_rng(3)
    L, W, G, d = 25, 5, 2, 8
    q, k = _rand_unit(rng, L, W, G, d)
    A = O.window_attention(q, k, L, W, G)
    for r in range(G * W):
        p = L - W + (r % W)
        ref = scipy.special.softmax(np.array([np.dot(q[r], k[i]) for i in range(p + 1)]) / math.sqrt(d))
        np.testing.assert_allclose(A[r, :p + 1], ref, rtol=1e-12, atol=1e-300)


def test_uniform_keys_closed_form():
    """All keys equal -> A[r, i] = 1/(p_r + 1) for i <= p_r: pins mask, mean and divisor."""
    rng = np.random.default_rng(4)
    L, W, G, d = 20, 4, 3, 8
    k = np.tile(rng.standard_normal(d), (L, 1))
    q = rng.standard_normal((G * W, d))
    mu, sigma = O.score_unit(q, k, L, W, G)
    n = G * W
    A = np.zeros((n, L))
    for g in range(G):
        for w in range(W):
            p = L - W + w
            A[g * W + w, :p + 1] = 1.0 / (p + 1)
    np.testing.assert_allclose(mu, A.mean(axis=0), rtol=1e-12)
    np.testing.assert_allclose(sigma, A.std(axis=0, ddof=1), rtol=1e-10, atol=1e-15)
    # the first column is seen by every row: mu_0 = (1/W) sum_w 1/(L-W+w+1)
    assert abs(mu[0] - np.mean([1.0 / (L - W + w + 1) for w in range(W)])) < 1e-15


def test_window_lse_closed_form_and_library():
    """The window rows' normaliser: equal keys give c_r + ln(p_r + 1) (closed form); random
    rows equal scipy's logsumexp over each row's visible prefix; exp(l - lse) over the
    visible keys sums to 1 and equals window_attention's row."""
    rng = np.random.default_rng(41)
    L, W, G, d = 20, 4, 3, 8
    kv = rng.standard_normal(d)
    k = np.tile(kv, (L, 1))
    q = rng.standard_normal((G * W, d)) * 3.0
    lse = O.window_lse(q, k, L, W, G)
    for r in range(G * W):
        p = L - W + (r % W)
        c = float(np.dot(q[r], kv)) / math.sqrt(d)
        assert abs(lse[r] - (c + math.log(p + 1))) < 1e-12
    L, W, G, d = 33, 6, 2, 16
    q, k = _rand_unit(rng, L, W, G, d, scale=4.0)
    lse = O.window_lse(q, k, L, W, G)
    A = O.window_attention(q, k, L, W, G)
    for r in range(G * W):
        p = L - W + (r % W)
        logits = np.array([np.dot(q[r], k[i]) for i in range(p + 1)]) / math.sqrt(d)
        assert abs(lse[r] - scipy.special.logsumexp(logits)) < 1e-12
        np.testing.assert_allclose(np.exp(logits - lse[r]), A[r, :p + 1], rtol=1e-12, atol=1e-300)
        assert abs(np.exp(logits - lse[r]).sum() - 1.0) < 1e-12


def test_identical_rows_give_zero_sigma():
    """W = 1 and G identical query heads: every row is the same distribution."""
    rng = np.random.default_rng(5)
    L, d = 33, 16
    q1 = rng.standard_normal(d) * 2
    q = np.tile(q1, (4, 1))
    k = rng.standard_normal((L, d))
    mu, sigma = O.score_unit(q, k, L, 1, 4)
    ref = scipy.special.softmax(k @ q1 / math.sqrt(d))
    np.testing.assert_allclose(mu, ref, rtol=1e-12)
    assert np.all(np.abs(sigma) < 1e-15)


def test_two_rows_sigma_closed_form():
    """n = 2 -> sigma_i = |A1 - A2| / sqrt(2) (sample std of two numbers)."""
    rng = np.random.default_rng(6)
    L, d = 21, 8
    q = rng.standard_normal((2, d)) * 2
    k = rng.standard_normal((L, d))
    mu, sigma = O.score_unit(q, k, L, 1, 2)
    A1 = scipy.special.softmax(k @ q[0] / math.sqrt(d))
    A2 = scipy.special.softmax(k @ q[1] / math.sqrt(d))
    np.testing.assert_allclose(sigma, np.abs(A1 - A2) / math.sqrt(2), rtol=1e-10, atol=1e-16)
    np.testing.assert_allclose(mu, (A1 + A2) / 2, rtol=1e-12)


def test_dispersion_is_sample_std():
    rng = np.random.default_rng(7)
    A = rng.random((12, 40))
    mu = O.mean_attention(A)
    np.testing.assert_allclose(mu, A.mean(axis=0), rtol=1e-13)
    np.testing.assert_allclose(O.dispersion(A, mu), A.std(axis=0, ddof=1), rtol=1e-12)
    assert np.all(O.dispersion(A[:1], A[0]) == 0)


def test_planted_divisor_bug_is_caught(monkeypatch):
    """A wrong Eq. 3 divisor (n instead of n - 1) must fail the closed-form pin."""
    def bad(A, mu):
        return np.sqrt(((A - mu) ** 2).sum(axis=0) / A.shape[0])
    monkeypatch.setattr(O, "dispersion", bad)
    with pytest.raises(AssertionError):
        test_two_rows_sigma_closed_form()


def test_planted_scale_bug_is_caught(monkeypatch):
    """Dropping the 1/sqrt(d) logit scale must fail the two-key closed form."""
    orig = O.window_attention

    def bad(q, k, L, W, G):
        return orig(q * math.sqrt(q.shape[1]), k, L, W, G)
    monkeypatch.setattr(O, "window_attention", bad)
    with pytest.raises(AssertionError):
        test_two_key_softmax_closed_form()


# --------------------------------------------------------------------------
# Pooling, Eq. 2, candidate pool, Eq. 5


@pytest.mark.parametrize("k", [1, 3, 5, 7])
def test_max_pool_matches_scipy(k):
    rng = np.random.default_rng(8)
    for m in [1, 2, 5, 50]:
        x = rng.random(m)
        ref = scipy.ndimage.maximum_filter1d(x, size=k, mode="nearest")
        np.testing.assert_array_equal(O.max_pool(x, k), ref)
    x = rng.random(9)
    np.testing.assert_array_equal(O.max_pool(x, 1), x)


def test_rank_ties_go_to_lower_position():
    s = np.array([0.5, 0.9, 0.5, 0.9, 0.1, 0.5])
    ref = sorted(range(len(s)), key=lambda i: (-s[i], i))
    np.testing.assert_array_equal(O.rank_desc(s), ref)
    np.testing.assert_array_equal(O.candidate_pool(s, 3), [1, 3, 0])


def test_normalise_range_and_clamp():
    s = np.array([0.2, 0.8, 0.4])
    st = O.normalise(s, np.arange(3), 1e-12)
    assert st.max() == 1.0 and st.min() >= 0.0
    neg = np.array([-0.2, -0.5])
    np.testing.assert_allclose(O.normalise(neg, np.arange(2), 1e-3), neg / 1e-3)


# --------------------------------------------------------------------------
# Eq. 4 and Eq. 5


def test_cosine_and_corr_special_cases():
    a = np.array([1.0, 2.0, -1.0])
    assert abs(O.cosine(a, a) - 1) < 1e-15 and abs(O.cosine(a, -a) + 1) < 1e-15
    assert O.cosine(a, np.zeros(3)) == 0.0
    keys = np.array([[1.0, 0.0], [-1.0, 0.0], [0.0, 1.0]])
    assert O.corr(0, [], keys) == 0.0
    assert O.corr(1, [0], keys) == 0.0          # cos = -1 clamps to 0
    assert abs(O.corr(2, [0, 1], keys)) < 1e-15


def _golden_mmr():
    lines = [l for l in open(os.path.join(GOLDEN, "mmr_worked_example.txt")) if not l.startswith("#")]
    keys = np.array([[float(x) for x in row.split()] for row in lines[0][5:].split(";")])
    s_tilde = np.array([float(x) for x in lines[1].split()[1:]])
    cases = []
    for l in lines[2:]:
        p = l.split()
        lam2, B = float(p[1]), int(p[2])
        i = p.index("order")
        j = p.index("margins")
        cases.append((lam2, B, [int(x) for x in p[i + 1:j]], [float(x) for x in p[j + 1:]]))
    return keys, s_tilde, cases


def test_mmr_worked_example():
    keys, s_tilde, cases = _golden_mmr()
    for lam2, B, order, margins in cases:
        steps = O.greedy_mmr(s_tilde, keys, np.arange(4), lam2, B)
        assert [st["pick"] for st in steps] == order
        np.testing.assert_allclose([st["margin"] for st in steps], margins, atol=6e-8)


def _brute_force_greedy(s_tilde, keys, cand, lam2, B):
    """Every ordered B-tuple; keep those in which each element is the argmax
    (value, then lower position) given its predecessors, corr recomputed from scratch."""
    def cos(i, j):
        a, b = keys[i], keys[j]
        na, nb = math.sqrt(sum(x * x for x in a)), math.sqrt(sum(x * x for x in b))
        return 0.0 if na == 0 or nb == 0 else sum(x * y for x, y in zip(a, b)) / (na * nb)

    good = []
    for tup in itertools.permutations(cand, B):
        ok = True
        for t in range(B):
            prefix = tup[:t]

            def val(i):
                c = max([0.0] + [cos(i, j) for j in prefix])
                return s_tilde[i] + lam2 * c
            rest = [i for i in cand if i not in prefix]
            best = sorted(rest, key=lambda i: (-val(i), i))[0]
            if best != tup[t]:
                ok = False
                break
        if ok:
            good.append(list(tup))
    return good


@pytest.mark.parametrize("seed", range(6))
def test_greedy_matches_brute_force(seed):
    rng = np.random.default_rng(100 + seed)
    C, B, d = 6, 3, 4
    keys = rng.standard_normal((C, d))
    keys[1] = keys[0] + 0.05 * rng.standard_normal(d)     # a near-duplicate pair
    s_tilde = rng.random(C)
    s_tilde /= s_tilde.max()
    for lam2 in [-0.8, -0.15, 0.0, 0.6]:
        sols = _brute_force_greedy(s_tilde, keys, list(range(C)), lam2, B)
        assert len(sols) == 1
        steps = O.greedy_mmr(s_tilde, keys, np.arange(C), lam2, B)
        assert [st["pick"] for st in steps] == sols[0]


def test_greedy_lambda2_zero_is_a_sort():
    rng = np.random.default_rng(9)
    s_tilde = np.round(rng.random(40), 2)   # rounding creates exact ties
    keys = rng.standard_normal((40, 8))
    steps = O.greedy_mmr(s_tilde, keys, np.arange(40), 0.0, 12)
    ref = sorted(range(40), key=lambda i: (-s_tilde[i], i))[:12]
    assert [st["pick"] for st in steps] == ref


def test_incremental_corr_equals_recomputed():
    rng = np.random.default_rng(10)
    keys = rng.standard_normal((30, 8))
    s_tilde = rng.random(30)
    steps = O.greedy_mmr(s_tilde, keys, np.arange(30), -0.5, 10)
    picks = [st["pick"] for st in steps]
    for t, st in enumerate(steps):
        expect = s_tilde[st["pick"]] - 0.5 * O.corr(st["pick"], picks[:t], keys)
        assert abs(st["v_pick"] - expect) < 1e-12
    assert steps[0]["pick"] == int(np.argmax(s_tilde))


# --------------------------------------------------------------------------
# Whole-unit selection (Section 3.2 special cases)


def _unit(seed, L=160, W=8, G=4, d=16):
    rng = np.random.default_rng(seed)
    q, k = _rand_unit(rng, L, W, G, d, scale=3.0)
    mu, sigma = O.score_unit(q, k, L, W, G)
    return mu, sigma, k


def test_lambda_zero_recovers_mean_attention_ranking():
    """lambda1 = lambda2 = 0: top-B by pooled mean attention (SnapKV/PyramidKV)."""
    L, W, B = 160, 8, 12
    mu, sigma, k = _unit(11, L, W)
    for pk in [1, 5, 7]:
        sel = O.select_unit(mu, sigma, k, L, W, B, 0.0, 0.0, pool_kernel=pk)
        pooled = scipy.ndimage.maximum_filter1d(mu[:L - W], size=pk, mode="nearest")
        ref = np.sort(sorted(range(L - W), key=lambda i: (-pooled[i], i))[:B])
        np.testing.assert_array_equal(sel["indices"], ref)


def test_candidate_restriction():
    L, W, B = 160, 8, 10
    mu, sigma, k = _unit(12, L, W)
    full = O.select_unit(mu, sigma, k, L, W, B, 0.5, -0.5, candidate_factor=0)
    big = O.select_unit(mu, sigma, k, L, W, B, 0.5, -0.5, candidate_factor=100)
    np.testing.assert_array_equal(full["indices"], big["indices"])
    four = O.select_unit(mu, sigma, k, L, W, B, 0.5, -0.5, candidate_factor=4)
    assert len(four["pool"]) == 4 * B
    assert set(four["indices"]) <= set(four["pool"])
    # lambda2 = 0: the restriction does not change the answer
    a = O.select_unit(mu, sigma, k, L, W, B, 0.5, 0.0, candidate_factor=4)
    b = O.select_unit(mu, sigma, k, L, W, B, 0.5, 0.0, candidate_factor=0)
    np.testing.assert_array_equal(a["indices"], b["indices"])


def test_normalised_scores_in_unit_interval_for_nonnegative_lambda1():
    L, W, B = 160, 8, 10
    mu, sigma, k = _unit(13, L, W)
    sel = O.select_unit(mu, sigma, k, L, W, B, 0.7, -0.3)
    st = sel["s_tilde"]
    assert st.min() >= 0 and abs(st.max() - 1.0) < 1e-15


def test_budget_at_least_candidates_keeps_everything():
    L, W = 40, 8
    mu, sigma, k = _unit(14, L, W)
    sel = O.select_unit(mu, sigma, k, L, W, 64, 0.5, -0.5)
    np.testing.assert_array_equal(sel["indices"], np.arange(L - W))


# --------------------------------------------------------------------------
# Base score with lambda1 != 0: mu and sigma pooled separately (Section 3.1, Eq. 2)


def _golden_pooled():
    lines = [l.split() for l in open(os.path.join(GOLDEN, "pooled_base_score.txt"))
             if l.strip() and not l.startswith("#")]
    head = {p[0]: p[1:] for p in lines if p[0] != "case"}
    kernel = int(head["kernel"][0])
    mu = np.array([float(x) for x in head["mu"]])
    sigma = np.array([float(x) for x in head["sigma"]])
    cases = []
    for p in lines:
        if p[0] == "case":
            i, j = p.index("s"), p.index("top2")
            cases.append((float(p[1]), [float(x) for x in p[i + 1:j]], [int(x) for x in p[j + 1:]]))
    return kernel, mu, sigma, cases


def test_pooled_base_score_worked_example():
    """Hand-worked s = mu^ + lambda1 sigma^ (separate pooling) for lambda1 in
    {0.5, -0.3, 2}, and the top 2 by the whole-unit selection at lambda2 = 0."""
    kernel, mu, sigma, cases = _golden_pooled()
    Lc = len(mu)
    W = 1
    keys = np.eye(Lc + W, 4)            # irrelevant at lambda2 = 0
    mu_all = np.append(mu, 0.0)         # the window token (not a candidate)
    sg_all = np.append(sigma, 0.0)
    for lam1, s_ref, top2 in cases:
        s = O.pooled_base_score(mu_all, sg_all, Lc, kernel, lam1)
        np.testing.assert_allclose(s, s_ref, rtol=0, atol=1e-15)
        sel = O.select_unit(mu_all, sg_all, keys, Lc + W, W, 2, lam1, 0.0, pool_kernel=kernel)
        assert [st["pick"] for st in sel["steps"]] == top2
        np.testing.assert_allclose(sel["s_tilde"], np.array(s_ref) / max(s_ref), rtol=1e-15)


def _pooled_reference(mu, sigma, Lc, k, lam1, B, eps=1e-12):
    """Built outside the oracle: scipy's max filter on mu and on sigma separately,
    then a plain sort (value descending, then position ascending)."""
    mh = scipy.ndimage.maximum_filter1d(mu[:Lc], size=k, mode="nearest")
    sh = scipy.ndimage.maximum_filter1d(sigma[:Lc], size=k, mode="nearest")
    s = mh + lam1 * sh
    order = sorted(range(Lc), key=lambda i: (-s[i], i))
    return s / max(max(s), eps), order[:B]


@pytest.mark.parametrize("lam1", [0.5, -0.3, 2.0])
@pytest.mark.parametrize("k", [3, 7])
def test_pooled_base_score_lambda1_matches_scipy(lam1, k):
    """lambda2 = 0 makes the greedy a sort, so the whole-unit selection is the top-B
    of the pooled base score; with lambda1 != 0, how sigma is pooled and weighted
    decides the set. s~ and the admissions match the reference built above."""
    L, W, B = 160, 8, 12
    for seed in (21, 22):
        mu, sigma, k_ = _unit(seed, L, W)
        sel = O.select_unit(mu, sigma, k_, L, W, B, lam1, 0.0, pool_kernel=k)
        st_ref, top = _pooled_reference(mu, sigma, L - W, k, lam1, B)
        np.testing.assert_allclose(sel["s_tilde"], st_ref, rtol=1e-13, atol=1e-300)
        assert [s["pick"] for s in sel["steps"]] == top


def _joint_pooling(mu, sigma, Lc, kernel, lambda1):
    return O.max_pool(mu[:Lc] + lambda1 * sigma[:Lc], kernel)


@pytest.mark.parametrize("bad", [
    ("pool", _joint_pooling),                                   # s = maxpool(mu + l1 sigma)
    ("base", lambda m, s, l1: m + l1 * s * s),                  # s = mu + l1 sigma^2
    ("base", lambda m, s, l1: m + 0.5 * l1 * s),                # s = mu + l1 sigma / 2
])
def test_planted_base_score_bugs_are_caught(monkeypatch, bad):
    """Each plausible mistake in the pooled base score fails a pin above."""
    where, fn = bad
    monkeypatch.setattr(O, "pooled_base_score" if where == "pool" else "base_score", fn)
    failed = 0
    try:
        test_pooled_base_score_worked_example()
    except AssertionError:
        failed += 1
    for lam1 in (0.5, -0.3, 2.0):
        try:
            test_pooled_base_score_lambda1_matches_scipy(lam1, 7)
        except AssertionError:
            failed += 1
    assert failed >= 2


# --------------------------------------------------------------------------
# Forced replay (the branch parity checking runs through on every near-tie swap)


def _brute_value(i, prior, s_tilde, keys, lam2):
    """s~_i + lambda2 * corr(i, prior) with corr from Eq. 4 by plain loops."""
    c = 0.0
    for j in prior:
        a, b = keys[i], keys[j]
        na = math.sqrt(sum(x * x for x in a))
        nb = math.sqrt(sum(x * x for x in b))
        cs = 0.0 if na == 0 or nb == 0 else sum(x * y for x, y in zip(a, b)) / (na * nb)
        c = max(c, cs)
    return s_tilde[i] + lam2 * c


def _forced_case():
    """A unit where the forced sequence takes a position outside the top-4B pool,
    with that key a near-duplicate of a pool member, so its corr and the corr it
    adds to others are both far from 0."""
    L, W, B = 200, 8, 6
    rng = np.random.default_rng(31)
    mu, sigma, keys = _unit(31, L, W)
    sel = O.select_unit(mu, sigma, keys, L, W, B, 0.5, -0.6)
    pool = [int(x) for x in sel["pool"]]
    ranked = O.rank_desc(sel["s_tilde"])
    outside = int(ranked[len(pool) + 3])                   # not in the pool
    keys = keys.copy()
    mate = pool[5]
    keys[outside] = keys[mate] + 0.05 * rng.standard_normal(keys.shape[1])
    first = [int(s["pick"]) for s in O.select_unit(mu, sigma, keys, L, W, B, 0.5, -0.6)["steps"]]
    follow = first[:2] + [outside] + first[2:5]
    return mu, sigma, keys, L, W, B, pool, outside, mate, follow


def test_forced_replay_out_of_pool_pick():
    """follow = the oracle's own picks with one position from outside the pool forced
    in at step 2: every step's v_pick, v_best, best and margin equal brute force over
    the grown admitted set (the forced key counts in later corr, Eq. 4)."""
    mu, sigma, keys, L, W, B, pool, outside, mate, follow = _forced_case()
    lam2 = -0.6
    ref = O.select_unit(mu, sigma, keys, L, W, B, 0.5, lam2, follow=follow)
    st = ref["s_tilde"]
    assert outside not in pool
    assert [s["pick"] for s in ref["steps"]] == follow
    taken = []
    for t, step in enumerate(ref["steps"]):
        assert abs(step["v_pick"] - _brute_value(step["pick"], taken, st, keys, lam2)) < 1e-12
        rest = [i for i in pool if i not in taken]
        vals = sorted(((-_brute_value(i, taken, st, keys, lam2), i) for i in rest))
        assert step["best"] == vals[0][1]
        assert abs(step["v_best"] + vals[0][0]) < 1e-12
        assert abs(step["margin"] - (vals[1][0] - vals[0][0])) < 1e-12
        taken.append(step["pick"])
    # the forced key is a near-duplicate of `mate`: after step 2 mate's corr is ~1
    t_after = 3
    if mate not in follow[:t_after]:
        v_mate = _brute_value(mate, follow[:t_after], st, keys, lam2)
        assert v_mate < st[mate] + lam2 * 0.9


def test_planted_forced_replay_bug_is_caught(monkeypatch):
    """Admitting an out-of-pool position with corr = 0 instead of Eq. 4 fails the pin."""
    monkeypatch.setattr(O, "corr", lambda i, S, keys: 0.0)
    with pytest.raises(AssertionError):
        test_forced_replay_out_of_pool_pick()


def test_gather_rows_and_zero_tail():
    rng = np.random.default_rng(15)
    L, W, B, d = 20, 4, 8, 6
    kb = rng.integers(0, 2 ** 16, (L, d), dtype=np.uint16)
    vb = rng.integers(0, 2 ** 16, (L, d), dtype=np.uint16)
    idx = np.array([1, 5, 7])
    ko, vo = O.gather_unit(kb, vb, idx, L, W, B)
    np.testing.assert_array_equal(ko[:3], kb[idx])
    np.testing.assert_array_equal(ko[3:3 + W], kb[L - W:])
    assert np.all(ko[3 + W:] == 0) and np.all(vo[3 + W:] == 0)
    np.testing.assert_array_equal(vo[:3], vb[idx])


def test_bf16_decode():
    bits = np.array([0x3F80, 0xBF80, 0x4049, 0x0000, 0x8000, 0x7F7F], dtype=np.uint16)
    vals = O.bf16_bits_to_f64(bits)
    assert vals[0] == 1.0 and vals[1] == -1.0 and vals[3] == 0.0
    assert abs(vals[2] - 3.140625) < 1e-15
    assert vals[5] == float(np.float32(3.3895314e38))


# --------------------------------------------------------------------------
# The window rows' attention output (Section 3.2: the existing attention)


def test_window_output_uniform_keys_closed_form():
    """All keys equal: every visible key gets 1/(p+1), so O[r] is the mean of the
    values at positions 0 .. p_r (prefix means by cumulative sums)."""
    rng = np.random.default_rng(41)
    L, W, G, d = 24, 5, 3, 8
    k = np.tile(rng.standard_normal(d), (L, 1))
    q = rng.standard_normal((G * W, d))
    v = rng.standard_normal((L, d))
    O_ = O.window_output(O.window_attention(q, k, L, W, G), v)
    prefix_mean = np.cumsum(v, axis=0) / np.arange(1, L + 1)[:, None]
    for g in range(G):
        for w in range(W):
            np.testing.assert_allclose(O_[g * W + w], prefix_mean[L - W + w], rtol=1e-12, atol=1e-14)


def test_window_output_single_visible_key():
    """A window row at position 0 sees only key 0: its output is v_0 exactly."""
    rng = np.random.default_rng(42)
    L = W = 6
    q = rng.standard_normal((W, 4)) * 3
    k = rng.standard_normal((L, 4))
    v = rng.standard_normal((L, 4))
    O_ = O.window_output(O.window_attention(q, k, L, W, 1), v)
    np.testing.assert_array_equal(O_[0], v[0])


def test_window_output_matches_scipy_softmax():
    rng = np.random.default_rng(43)
    L, W, G, d = 30, 4, 2, 8
    q, k = _rand_unit(rng, L, W, G, d)
    v = rng.standard_normal((L, d))
    O_ = O.window_output(O.window_attention(q, k, L, W, G), v)
    for r in range(G * W):
        p = L - W + (r % W)
        a = scipy.special.softmax(np.array([q[r] @ k[i] for i in range(p + 1)]) / math.sqrt(d))
        np.testing.assert_allclose(O_[r], a @ v[:p + 1], rtol=1e-12, atol=1e-14)


def test_planted_window_output_bugs_are_caught(monkeypatch):
    """Values paired with the wrong keys (positions reversed), or attention without the
    causal mask, fail the pins."""
    orig = O.window_attention
    monkeypatch.setattr(O, "window_output", lambda A, v: A[:, ::-1] @ v)
    with pytest.raises(AssertionError):
        test_window_output_matches_scipy_softmax()
    monkeypatch.setattr(O, "window_output", lambda A, v: A @ v)

    def unmasked(q, k, L, W, G):
        lg = (q @ k.T) / math.sqrt(q.shape[1])
        e = np.exp(lg - lg.max(axis=1, keepdims=True))
        return e / e.sum(axis=1, keepdims=True)
    monkeypatch.setattr(O, "window_attention", unmasked)
    with pytest.raises(AssertionError):
        test_window_output_single_visible_key()
    monkeypatch.setattr(O, "window_attention", orig)


# --------------------------------------------------------------------------
# Eq. 6


def test_profiles_against_paper_statements():
    for line in open(os.path.join(GOLDEN, "sinh_profile.txt")):
        p = line.split()
        if not p or p[0].startswith("#"):
            continue
        if p[0] == "sinh":
            lam = O.depth_profile("global", [float(p[1])], 4)
            np.testing.assert_allclose(lam, float(p[2]), rtol=1e-15, atol=1e-300)
        if p[0] == "asinh":
            lam = O.depth_profile("global", [float(p[2])], 3)
            np.testing.assert_allclose(lam, float(p[1]), rtol=1e-14)


def test_profile_families_contain_global():
    g = O.depth_profile("global", [0.4], 32)
    np.testing.assert_allclose(O.depth_profile("segments", [0.4, 0.4, 0.4], 32), g, rtol=0)
    np.testing.assert_allclose(O.depth_profile("curve", [0.4, 0.0, 0.0], 32), g, rtol=0)
    seg = O.depth_profile("segments", [-0.8, 0.6, -0.8], 32)
    assert np.all(seg[:11] == math.sinh(-0.8)) and np.all(seg[11:22] == math.sinh(0.6))
    assert np.all(seg[22:] == math.sinh(-0.8))
    cur = O.depth_profile("curve", [0.1, 0.2, 0.3], 5)
    np.testing.assert_allclose(cur[[0, 4]], [math.sinh(0.1), math.sinh(0.6)], rtol=1e-15)
    np.testing.assert_allclose(cur[2], math.sinh(0.1 + 0.1 + 0.075), rtol=1e-15)
