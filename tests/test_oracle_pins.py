"""Pins of the fp64 oracle to things other than itself (CPU only).

Each test ties one oracle function to a hand-worked value from tests/golden/, a
closed form, an invariant the paper states, brute force on tiny inputs, or a
special case that reduces to a library routine (scipy, numpy, torch).  They are
chosen so that a dropped term, a wrong sign or index, a missing mask or a
transposed operand in the oracle fails at least one of them.
"""
import itertools
import json
import math
import os

import numpy as np
import pytest
import scipy.ndimage
import scipy.special
import torch

import oracle

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def gold(name):
    with open(os.path.join(GOLD, name)) as f:
        return json.load(f)


# ---------------------------------------------------------------- Eq. 1 --------
def test_eq1_golden_cases():
    g = gold("eq1_retention.json")
    for c in g["cases"]:
        r = oracle.retention_ratio(c["history"], c["base"], c["delta"])
        assert abs(r - c["ratio"]) < 1e-7, c
        assert oracle.keep_count(r, c["L"], c["w"]) == c["m"], c


def test_eq1_bounds_and_monotone():
    """lambda_i stays in [lambda - delta, lambda + delta] (Sec. 3.2) and falls as v_i rises."""
    rng = np.random.default_rng(1)
    for _ in range(300):
        n = int(rng.integers(2, 20))
        h = rng.random(n).astype(np.float32)
        r = oracle.retention_ratio(h, 0.25, 0.1)
        assert 0.15 - 1e-12 <= r <= 0.35 + 1e-12
        h2 = h.copy()
        h2[-1] = np.float32(min(1.0, h2[-1] + 0.1))
        assert oracle.retention_ratio(h2, 0.25, 0.1) <= r + 1e-12
    # the extremes are reached only by the extreme rewards
    assert abs(oracle.retention_ratio([0.0, 1.0], 0.25, 0.1) - (0.25 - 0.1 * 0.5)) < 1e-12
    assert abs(oracle.retention_ratio([1.0, 0.0], 0.25, 0.1) - (0.25 + 0.1 * 0.5)) < 1e-12


def test_eq1_depends_on_current_reward_not_position():
    """The adjustment uses the last entry as v_i: reversing a history flips its sign."""
    h = [0.1, 0.4, 0.9]
    a = oracle.retention_ratio(h, 0.25, 0.1) - 0.25
    b = oracle.retention_ratio(h[::-1], 0.25, 0.1) - 0.25
    assert a < 0 < b


# ---------------------------------------------------------------- Eq. 2 --------
def test_eq2_hand_example_and_selection():
    g = gold("eq2_score.json")
    q = np.array(g["q"], np.float32)
    k = np.array(g["k"], np.float32)
    raw, _ = oracle.score_unit(q, k, g["w"], g["scale"], 1)
    np.testing.assert_allclose(raw, g["raw"], atol=g["raw_tol"])
    L = k.shape[0]
    for s in g["selections"]:
        _, pooled = oracle.score_unit(q, k, g["w"], g["scale"], s["pool"])
        kept = oracle.select_unit(pooled.astype(np.float32), L, g["w"], s["m"])
        assert kept.tolist() == s["kept"], s


def _harmonic(n):
    return sum(1.0 / i for i in range(1, n + 1))


@pytest.mark.parametrize("G,w,L", [(1, 1, 9), (3, 5, 20), (7, 32, 300)])
def test_eq2_zero_query_closed_form(G, w, L):
    """q = 0 gives a uniform softmax over the visible keys, so window query t spreads
    1/(L-w+t+1) over keys 0..L-w+t.  A candidate j < L-w therefore scores
    H(L) - H(L-w); window key L-w+s scores H(L) - H(L-w+s).  Fails without the
    causal mask, with an off-by-one window position, or with a sum over heads."""
    d = 4
    q = np.zeros((G, w, d), np.float32)
    k = np.random.default_rng(0).standard_normal((L, d)).astype(np.float32)
    raw, _ = oracle.score_unit(q, k, w, 0.5, 1)
    HL = _harmonic(L)
    for j in range(L - w):
        assert abs(raw[j] - (HL - _harmonic(L - w))) < 1e-12
    for s in range(w):
        assert abs(raw[L - w + s] - (HL - _harmonic(L - w + s))) < 1e-12


def test_eq2_single_query_is_a_softmax_row():
    """G = 1, w = 1: the score is one softmax row of scale * K q (scipy)."""
    rng = np.random.default_rng(2)
    for L, d, scale in [(7, 3, 1.0), (50, 16, 0.25), (200, 64, 0.125)]:
        q = rng.standard_normal((1, 1, d)).astype(np.float32)
        k = rng.standard_normal((L, d)).astype(np.float32)
        raw, _ = oracle.score_unit(q, k, 1, scale, 1)
        ref = scipy.special.softmax(scale * (k.astype(np.float64) @ q[0, 0].astype(np.float64)))
        np.testing.assert_allclose(raw, ref, rtol=1e-12, atol=1e-15)


def test_eq2_mass_is_window_size():
    """Every softmax row sums to 1, so the unpooled scores over all L keys sum to w
    (a sum over heads instead of the mean would give G*w)."""
    rng = np.random.default_rng(3)
    for G, w, L, d in [(2, 4, 30, 8), (4, 16, 128, 16), (6, 3, 11, 5)]:
        q = rng.standard_normal((G, w, d)).astype(np.float32)
        k = rng.standard_normal((L, d)).astype(np.float32)
        raw, _ = oracle.score_unit(q, k, w, 1.0 / math.sqrt(d), 1)
        assert abs(raw.sum() - w) < 1e-9


def test_eq2_gqa_mean_of_heads():
    """The GQA score is the mean of the per-head scores (checked head by head)."""
    rng = np.random.default_rng(4)
    G, w, L, d = 3, 4, 25, 8
    q = rng.standard_normal((G, w, d)).astype(np.float32)
    k = rng.standard_normal((L, d)).astype(np.float32)
    raw, _ = oracle.score_unit(q, k, w, 0.3, 1)
    per = [oracle.score_unit(q[g:g + 1], k, w, 0.3, 1)[0] for g in range(G)]
    np.testing.assert_allclose(raw, np.mean(per, axis=0), rtol=1e-12)


def test_eq2_head_grouping_in_batched_scores():
    """KV head h serves query heads h*G .. h*G+G-1: changing query heads 2,3 of a
    4/2-head layer changes KV head 1's scores and leaves KV head 0's alone."""
    rng = np.random.default_rng(5)
    Ly, B, Hq, Hkv, w, L, d = 1, 2, 4, 2, 3, 20, 8
    q = rng.standard_normal((Ly, B, Hq, w, d)).astype(np.float32)
    K = rng.standard_normal((Ly, B, Hkv, L, d)).astype(np.float32)
    lens = np.full((Ly, B, Hkv), L, np.int32)
    a = oracle.score_cache(q, K, lens, w, 1, 0.3)
    q2 = q.copy()
    q2[:, :, 2:4] = rng.standard_normal(q2[:, :, 2:4].shape)
    b = oracle.score_cache(q2, K, lens, w, 1, 0.3)
    nc = L - w
    np.testing.assert_array_equal(a[:, :, 0, :nc], b[:, :, 0, :nc])
    assert np.abs(a[:, :, 1, :nc] - b[:, :, 1, :nc]).max() > 1e-3
    # and each unit equals the single-unit definition on its own slice
    for bb in range(B):
        for h in range(Hkv):
            _, pooled = oracle.score_unit(q[0, bb, h * 2:h * 2 + 2], K[0, bb, h], w, 0.3, 1)
            np.testing.assert_array_equal(a[0, bb, h, :nc], pooled)


def test_eq2_scale_enters_the_logits():
    rng = np.random.default_rng(6)
    q = rng.standard_normal((2, 3, 8)).astype(np.float32)
    k = rng.standard_normal((17, 8)).astype(np.float32)
    a, _ = oracle.score_unit(q, k, 3, 0.5, 1)
    b, _ = oracle.score_unit((q * 0.5).astype(np.float32), k, 3, 1.0, 1)  # 0.5 is exact in float32
    np.testing.assert_allclose(a, b, rtol=1e-12)
    c, _ = oracle.score_unit(q, k, 3, 1.0, 1)
    assert np.abs(a - c).max() > 1e-3


@pytest.mark.parametrize("pool", [1, 3, 7, 9])
def test_maxpool_matches_scipy(pool):
    """Max-pool with the window clipped to [0, L-w) equals scipy's maximum filter
    with edge replication (a max over a clipped window)."""
    rng = np.random.default_rng(7)
    q = rng.standard_normal((2, 4, 8)).astype(np.float32)
    k = rng.standard_normal((40, 8)).astype(np.float32)
    raw, pooled = oracle.score_unit(q, k, 4, 0.3, pool)
    ref = scipy.ndimage.maximum_filter1d(raw[:36], size=pool, mode="nearest")
    np.testing.assert_array_equal(pooled, ref)


# ---------------------------------------------------------------- top-m ---------
def _rank_select(s, L, w, m):
    """Brute force by rank: candidate j is kept iff fewer than m-w candidates beat it
    (a higher score, or an equal score at a lower index)."""
    nc = L - w
    kept = []
    for j in range(nc):
        beat = sum(1 for i in range(nc) if s[i] > s[j] or (s[i] == s[j] and i < j))
        if beat < m - w:
            kept.append(j)
    return kept + list(range(nc, L))


def test_select_matches_rank_brute_force_with_ties():
    rng = np.random.default_rng(8)
    for trial in range(200):
        L = int(rng.integers(1, 14))
        w = int(rng.integers(1, L + 1))
        s = (rng.integers(0, 4, L - w) / 4.0).astype(np.float32)  # many exact ties
        for m in range(w, L + 1):
            got = oracle.select_unit(s, L, w, m).tolist()
            assert got == _rank_select(s, L, w, m), (L, w, m, s)


def test_select_exhaustive_subsets():
    """On tiny inputs, the kept candidates are the (m-w)-subset with the largest score
    sum, and among equal sums the lexicographically smallest index set."""
    rng = np.random.default_rng(9)
    for trial in range(60):
        L = int(rng.integers(2, 10))
        w = int(rng.integers(1, L))
        s = (rng.integers(0, 3, L - w) / 2.0).astype(np.float32)
        nc = L - w
        for m in range(w, L + 1):
            best = max(itertools.combinations(range(nc), m - w),
                       key=lambda c: (sum(float(s[i]) for i in c), [-i for i in c]))
            got = oracle.select_unit(s, L, w, m).tolist()
            assert got == sorted(best) + list(range(nc, L))


def test_select_invariants_and_identity():
    rng = np.random.default_rng(10)
    L, w = 300, 16
    s = rng.random(L - w).astype(np.float32)
    for m in [w, 17, 75, 299, 300]:
        idx = oracle.select_unit(s, L, w, m)
        assert idx.size == m
        assert np.all(np.diff(idx) > 0) and idx[0] >= 0 and idx[-1] < L
        assert set(range(L - w, L)) <= set(idx.tolist())
    assert oracle.select_unit(s, L, w, L).tolist() == list(range(L))


def test_gather_matches_numpy_indexing():
    rng = np.random.default_rng(11)
    rows = rng.standard_normal((50, 6)).astype(np.float32)
    idx = np.sort(rng.choice(50, 20, replace=False)).astype(np.int32)
    np.testing.assert_array_equal(oracle.gather_unit(rows, idx), rows[idx])


# ---------------------------------------------------------------- decode ----------
def test_decode_matches_torch_sdpa():
    rng = np.random.default_rng(12)
    for length, d in [(1, 8), (5, 16), (300, 64), (1000, 128)]:
        q = rng.standard_normal(d).astype(np.float32)
        k = rng.standard_normal((length, d)).astype(np.float32)
        v = rng.standard_normal((length, d)).astype(np.float32)
        scale = 1.0 / math.sqrt(d)
        out, lse = oracle.decode_unit(q, k, v, length, scale)
        tq = torch.from_numpy(q).double().view(1, 1, 1, d)
        tk = torch.from_numpy(k).double().view(1, 1, length, d)
        tv = torch.from_numpy(v).double().view(1, 1, length, d)
        ref = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, scale=scale).view(d).numpy()
        np.testing.assert_allclose(out, ref, rtol=1e-10, atol=1e-12)
        ref_lse = torch.logsumexp(scale * (tk[0, 0] @ tq[0, 0, 0]), 0).item()
        assert abs(lse - ref_lse) < 1e-10


def test_decode_special_cases():
    rng = np.random.default_rng(13)
    d = 16
    q = rng.standard_normal(d).astype(np.float32)
    v = rng.standard_normal((9, d)).astype(np.float32)
    k = rng.standard_normal((9, d)).astype(np.float32)
    out, _ = oracle.decode_unit(q, k, v, 1, 0.25)
    np.testing.assert_allclose(out, v[0], rtol=0, atol=1e-12)  # one key: o = v_0
    kk = np.repeat(k[:1], 9, axis=0)
    out, lse = oracle.decode_unit(q, kk, v, 9, 0.25)
    np.testing.assert_allclose(out, v.astype(np.float64).mean(0), atol=1e-12)  # equal keys: mean of V
    assert abs(lse - (0.25 * float(k[0].astype(np.float64) @ q.astype(np.float64)) + math.log(9))) < 1e-12


def test_decode_lse_is_the_eq2_row_normaliser():
    """The identity the one-pass scoring rests on, between two separate oracle functions:
    the decode of window query t over the keys 0..L-w+t (its cache when it was decoded)
    returns lse_t, and exp(logit - lse_t) summed over the window and averaged over the G
    heads is Eq. 2's raw score.  A causal off-by-one or a wrong window position on either
    side breaks it."""
    rng = np.random.default_rng(12)
    G, w, L, d, scale = 3, 5, 23, 8, 0.37
    q = rng.standard_normal((G, w, d)).astype(np.float32)
    k = rng.standard_normal((L, d)).astype(np.float32)
    v = rng.standard_normal((L, d)).astype(np.float32)
    raw_ref, _ = oracle.score_unit(q, k, w, scale, 1)
    raw = np.zeros(L)
    for g in range(G):
        for t in range(w):
            n = L - w + t + 1
            _, lse = oracle.decode_unit(q[g, t], k[:n], v[:n], n, scale)
            logits = scale * (k[:n].astype(np.float64) @ q[g, t].astype(np.float64))
            raw[:n] += np.exp(logits - lse)
    np.testing.assert_allclose(raw / G, raw_ref, rtol=1e-12, atol=1e-15)


def test_decode_batch_head_grouping():
    rng = np.random.default_rng(14)
    Ly, B, Hq, Hkv, Lc, d = 2, 2, 6, 2, 12, 8
    q = rng.standard_normal((Ly, B, Hq, d)).astype(np.float32)
    K = rng.standard_normal((Ly, B, Hkv, Lc, d)).astype(np.float32)
    V = rng.standard_normal((Ly, B, Hkv, Lc, d)).astype(np.float32)
    lens = rng.integers(1, Lc + 1, (Ly, B, Hkv)).astype(np.int32)
    out, lse = oracle.decode_batch(q, K, V, lens, 0.3)
    for l, b, hq in itertools.product(range(Ly), range(B), range(Hq)):
        h = hq // 3
        o, s = oracle.decode_unit(q[l, b, hq], K[l, b, h], V[l, b, h], int(lens[l, b, h]), 0.3)
        np.testing.assert_array_equal(out[l, b, hq], o)
        assert lse[l, b, hq] == s


# ---------------------------------------------------------------- Eq. 3 / 4 --------
def test_eq3_bands_golden():
    g = gold("eq34_penalty.json")
    for c in g["bands"]:
        assert oracle.penalty_band(c["v"], g["tau_l"], g["tau_h"]) == c["band"], c
        z, beta_i, _ = oracle.reflect_penalty(np.zeros((1, 4), np.float32), [1], [c["v"]],
                                              g["tau_l"], g["tau_h"], g["beta"])
        assert beta_i[0] == c["beta_i"]
        assert z[0, 1] == -c["beta_i"] and z[0, 0] == 0.0


def test_eq4_logit_example_and_set_semantics():
    g = gold("eq34_penalty.json")
    ex = g["logit_example"]
    z, _, _ = oracle.reflect_penalty(np.array([[0.0, ex["z"]]], np.float32), [1], [ex["v"]],
                                     g["tau_l"], g["tau_h"], g["beta"])
    assert z[0, 1] == np.float32(ex["z_penalised"])
    dup = g["duplicate_example"]
    z, _, _ = oracle.reflect_penalty(np.array([dup["z"]], np.float32), dup["ids"], [dup["v"]],
                                     g["tau_l"], g["tau_h"], g["beta"])
    np.testing.assert_array_equal(z[0], np.array(dup["z_penalised"], np.float32))


def test_eq4_untouched_ids_are_bit_identical():
    rng = np.random.default_rng(15)
    B, V = 4, 500
    z0 = (rng.standard_normal((B, V)) * 2).astype(np.float32)
    ids = rng.choice(V, 12, replace=False).astype(np.int32)
    rewards = np.array([0.1, 0.5, 0.8, 0.95], np.float32)
    z, beta_i, bad = oracle.reflect_penalty(z0, ids, rewards)
    assert bad == 0
    mask = np.zeros(V, bool)
    mask[ids] = True
    np.testing.assert_array_equal(z[:, ~mask].view(np.uint32), z0[:, ~mask].view(np.uint32))
    np.testing.assert_array_equal(beta_i, np.array([0, 2, 4, 4], np.float32))
    for b in range(B):
        np.testing.assert_array_equal(z[b, mask], z0[b, mask] - beta_i[b])  # float32 subtract


def test_eq4_out_of_range_ids_are_ignored():
    z, _, bad = oracle.reflect_penalty(np.zeros((1, 5), np.float32), [-1, 2, 5], [1.0])
    assert bad == 2 and z[0].tolist() == [0, 0, -4, 0, 0]


def test_probe_trigger_golden():
    for c in gold("eq34_penalty.json")["probe_trigger"]:
        assert oracle.probe_trigger(c["v_prev"], c["v_cur"], 0.8) == c["fire"], c


# ---------------------------------------------------------------- Eq. 5 / 6 --------
def test_eq5_golden():
    g = gold("eq56_ppl.json")
    t = g["two_token"]
    ppl, stop = oracle.answer_ppl(np.array([t["logits"]], np.float32), np.array([t["tokens"]], np.int32),
                                  tau_p=g["tau_p"])
    assert abs(ppl[0] - t["ppl"]) < 1e-6 and stop[0] == t["stop"]
    u = g["uniform"]
    ppl, stop = oracle.answer_ppl(np.zeros((1, u["n"], u["V"]), np.float32),
                                  np.array([[1, 7, 1000]], np.int32), tau_p=g["tau_p"])
    assert abs(ppl[0] - u["ppl"]) < 1e-9 and not stop[0]
    c = g["confident"]
    z = np.zeros((1, 2, c["V"]), np.float32)
    z[0, 0, 3] = c["boost"]
    z[0, 1, 9] = c["boost"]
    ppl, stop = oracle.answer_ppl(z, np.array([[3, 9]], np.int32), tau_p=g["tau_p"])
    assert abs(ppl[0] - 1.0) < 1e-12 and stop[0]


def test_eq5_matches_torch_cross_entropy_and_ragged_lengths():
    rng = np.random.default_rng(16)
    B, n, V = 3, 6, 300
    z = (rng.standard_normal((B, n, V)) * 2).astype(np.float32)
    tok = rng.integers(0, V, (B, n)).astype(np.int32)
    nv = np.array([6, 1, 4], np.int32)
    ppl, _ = oracle.answer_ppl(z, tok, nv)
    for b in range(B):
        ce = torch.nn.functional.cross_entropy(torch.from_numpy(z[b, :nv[b]]).double(),
                                               torch.from_numpy(tok[b, :nv[b]]).long())
        assert abs(ppl[b] - math.exp(ce.item())) < 1e-9 * ppl[b]


def test_eq6_stop_boundary_is_inclusive():
    # a single token with p = 1/1.1 has PPL exactly 1.1 in exact arithmetic; use a clear margin instead
    V = 2
    for p_target, expect in [(0.95, True), (0.85, False)]:
        zt = math.log(p_target / (1 - p_target))
        z = np.array([[[zt, 0.0]]], np.float32)
        ppl, stop = oracle.answer_ppl(z, np.array([[0]], np.int32), tau_p=1.1)
        assert stop[0] == expect, (p_target, ppl)
    ppl, stop = oracle.answer_ppl(np.zeros((1, 2, 3), np.float32), np.zeros((1, 2), np.int32),
                                  np.array([0], np.int32))
    assert math.isnan(ppl[0]) and not stop[0]  # empty answer: no perplexity, no stop


# ---------------------------------------------------------------- sampling after Eq. 4 --------
def _sample(z, u, ids=(), rewards=None, **kw):
    z = np.atleast_2d(np.asarray(z, np.float32))
    B = z.shape[0]
    rewards = np.zeros(B, np.float32) if rewards is None else rewards
    return oracle.penalty_sample(z, np.asarray(ids, np.int32), rewards, np.asarray(u, np.float32), **kw)


def test_sample_golden_cdf_boundaries():
    g = gold("sample_inversion.json")
    t = g["two_token"]
    for u, tok in t["cases"]:
        assert _sample([t["logits"]], [u])[1][0] == tok, (u, tok)
    un = g["uniform"]
    for u, tok in un["cases"]:
        assert _sample(np.zeros((1, un["V"])), [u])[1][0] == tok, (u, tok)
    oh = g["one_hot"]
    z = np.zeros((1, oh["V"]), np.float32)
    z[0, oh["hot"]] = oh["boost"]
    for u in oh["uniforms"]:
        assert _sample(z, [u])[1][0] == oh["hot"]
    m = g["masked"]
    zm = [float(x) for x in m["logits"]]
    for u, tok in m["cases"]:
        assert _sample([zm], [u])[1][0] == tok, (u, tok)


def test_sample_draws_after_the_penalty():
    g = gold("sample_inversion.json")["penalty"]
    for c in g["cases"]:
        _, tok, _, _, _ = _sample([g["z"]], [c["u"]], g["ids"], np.array([c["v"]], np.float32),
                                  tau_l=g["tau_l"], tau_h=g["tau_h"], beta=g["beta"])
        assert tok[0] == c["token"], c


def test_sample_matches_searchsorted_on_the_cumulative_softmax():
    rng = np.random.default_rng(21)
    B, V = 64, 300
    z = (rng.standard_normal((B, V)) * 2).astype(np.float32)
    ids = rng.choice(V, 10, replace=False).astype(np.int32)
    rw = rng.uniform(0, 1, B).astype(np.float32)
    u = rng.uniform(0, 1, B).astype(np.float32)
    zp, tok, lo, hi, bad = _sample(z, u, ids, rw)
    assert bad == 0
    for b in range(B):
        p = scipy.special.softmax(zp[b].astype(np.float64))
        cdf = np.cumsum(p)
        ref = int(np.searchsorted(cdf, float(u[b]), side="right"))
        if abs(cdf[ref] - u[b]) > 1e-12 and (ref == 0 or abs(cdf[ref - 1] - u[b]) > 1e-12):
            assert tok[b] == ref, (b, tok[b], ref)
        assert abs(lo[b] - (cdf[tok[b] - 1] if tok[b] else 0.0)) < 1e-12 and abs(hi[b] - cdf[tok[b]]) < 1e-12


def test_sample_stratified_counts_follow_the_probabilities():
    """With stratified draws u_k = (k + 1/2)/N, inversion gives token j exactly the number of
    grid points inside its CDF interval, i.e. N p_j to within one, for every j."""
    rng = np.random.default_rng(22)
    V, N = 50, 4000
    z = (rng.standard_normal(V) * 2).astype(np.float32)
    u = ((np.arange(N) + 0.5) / N).astype(np.float32)
    _, tok, _, _, _ = _sample(np.repeat(z[None], N, 0), u)
    counts = np.bincount(tok, minlength=V)
    p = scipy.special.softmax(z.astype(np.float64))
    assert np.abs(counts - N * p).max() <= 1.0 + 1e-6, np.abs(counts - N * p).max()
    assert counts.sum() == N
