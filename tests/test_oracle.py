"""Pins of the CPU oracle against what the paper and the mathematics fix.

Nothing here compares the oracle with itself: every expected value is a closed
form, a brute-force loop written independently of the oracle's numpy code, a
textbook table (tests/golden/) or an invariant of the method (Eq. 3, Eq. 8,
Eq. 9, Eq. 10 and the refresh schedule).
"""
import copy
import math
import os

import numpy as np
import pytest

import oracle as O
import synth


# --------------------------------------------------------------------------
# Attention (Eq. 3)
# --------------------------------------------------------------------------

def brute_attention(q, k, v, heads):
    """Triple loop over queries, keys and head dims with math.exp; no max shift."""
    n_q, D = len(q), len(q[0])
    dh = D // heads
    out = [[0.0] * D for _ in range(n_q)]
    for h in range(heads):
        for i in range(n_q):
            scores = []
            for j in range(len(k)):
                acc = 0.0
                for d in range(h * dh, (h + 1) * dh):
                    acc += float(q[i][d]) * float(k[j][d])
                scores.append(math.exp(acc / math.sqrt(dh)))
            z = math.fsum(scores)
            for d in range(h * dh, (h + 1) * dh):
                out[i][d] = math.fsum(scores[j] * float(v[j][d]) for j in range(len(k))) / z
    return np.array(out)


@pytest.mark.parametrize("n_q,T,D,heads", [(1, 1, 2, 1), (3, 5, 4, 1), (4, 6, 8, 2), (2, 7, 6, 3)])
def test_attention_matches_brute_force(n_q, T, D, heads):
    rng = np.random.default_rng(n_q * 100 + T)
    q, k, v = rng.normal(size=(n_q, D)), rng.normal(size=(T, D)), rng.normal(size=(T, D))
    np.testing.assert_allclose(O.attention(q, k, v, heads), brute_attention(q, k, v, heads), rtol=1e-12, atol=1e-13)


def test_attention_worked_example():
    # One head of width 2: q = e1, keys e1 and e2. Scores 1/sqrt(2) and 0, so the
    # weight on the first key is 1 / (1 + exp(-1/sqrt(2))).
    q = np.array([[1.0, 0.0]])
    k = np.array([[1.0, 0.0], [0.0, 1.0]])
    v = np.array([[1.0, 2.0], [3.0, 4.0]])
    w1 = 1.0 / (1.0 + math.exp(-1.0 / math.sqrt(2.0)))
    expect = w1 * v[0] + (1 - w1) * v[1]
    np.testing.assert_allclose(O.attention(q, k, v, 1)[0], expect, rtol=1e-14)
    assert abs(expect[0] - 1.66048) < 1e-4  # 0.66976 * 1 + 0.33024 * 3


def test_attention_equal_keys_average_values():
    rng = np.random.default_rng(7)
    q = rng.normal(size=(3, 8))
    k = np.tile(rng.normal(size=(1, 8)), (5, 1))
    v = rng.normal(size=(5, 8))
    np.testing.assert_allclose(O.attention(q, k, v, 2), np.tile(v.mean(0), (3, 1)), rtol=1e-13)


def test_attention_heads_are_independent_slices():
    rng = np.random.default_rng(8)
    q, k, v = rng.normal(size=(3, 8)), rng.normal(size=(6, 8)), rng.normal(size=(6, 8))
    base = O.attention(q, k, v, 2)
    k2 = k.copy()
    k2[:, 4:] = rng.normal(size=(6, 4))       # perturb head 1's keys only
    out = O.attention(q, k2, v, 2)
    np.testing.assert_array_equal(out[:, :4], base[:, :4])
    assert np.abs(out[:, 4:] - base[:, 4:]).max() > 1e-3


# --------------------------------------------------------------------------
# LayerNorm, GELU, linear
# --------------------------------------------------------------------------

def test_layer_norm_closed_form():
    x = np.array([[1.0, 2.0, 3.0, 4.0]])
    # mean 2.5, biased variance 1.25
    expect = (x - 2.5) / math.sqrt(1.25 + 1e-6)
    np.testing.assert_allclose(O.layer_norm(x, np.ones(4), np.zeros(4), 1e-6), expect, rtol=1e-14)
    g, b = np.array([2.0, -1.0, 0.5, 3.0]), np.array([0.1, 0.2, 0.3, 0.4])
    np.testing.assert_allclose(O.layer_norm(x, g, b, 1e-6), expect * g + b, rtol=1e-14)


def test_gelu_textbook_values(golden_dir):
    rows = [l.split() for l in open(os.path.join(golden_dir, "normal_cdf.txt")) if l.strip() and l[0] != "#"]
    xs = np.array([float(r[0]) for r in rows])
    phi = np.array([float(r[1]) for r in rows])
    np.testing.assert_allclose(O.gelu(xs), xs * phi, rtol=1e-14, atol=1e-16)


def test_linear_orientation():
    x = np.array([[1.0, 2.0]])
    w = np.array([[1.0, 0.0], [0.0, 1.0], [1.0, 1.0]])   # [out=3, in=2]
    np.testing.assert_array_equal(O.linear(x, w, np.array([10.0, 20.0, 30.0])), [[11.0, 22.0, 33.0]])


# --------------------------------------------------------------------------
# The block: closed forms and invariants
# --------------------------------------------------------------------------

def _rand_block(rng, D, H4, scale=0.3):
    return {
        "ln1_g": 1 + 0.1 * rng.normal(size=D), "ln1_b": 0.1 * rng.normal(size=D),
        "w_qkv": scale * rng.normal(size=(3 * D, D)), "b_qkv": 0.1 * rng.normal(size=3 * D),
        "w_o": scale * rng.normal(size=(D, D)), "b_o": 0.1 * rng.normal(size=D),
        "ln2_g": 1 + 0.1 * rng.normal(size=D), "ln2_b": 0.1 * rng.normal(size=D),
        "w1": scale * rng.normal(size=(H4, D)), "b1": 0.1 * rng.normal(size=H4),
        "w2": scale * rng.normal(size=(D, H4)), "b2": 0.1 * rng.normal(size=D),
    }


def test_block_closed_form_with_zero_projections():
    # W_qkv = 0: every key equals b_k, so attention weights are uniform and every
    # token's attention output is b_v. W_o is a (non-symmetric) permutation P and
    # W1 = 0, so the block output is x + b_v P^T + b_o + GELU(b1) W2^T + b2.
    rng = np.random.default_rng(1)
    D, H4, T = 6, 12, 5
    bw = _rand_block(rng, D, H4)
    bw["w_qkv"] = np.zeros((3 * D, D))
    perm = np.array([2, 0, 5, 1, 3, 4])
    bw["w_o"] = np.eye(D)[perm]
    bw["w1"] = np.zeros((H4, D))
    x = rng.normal(size=(T, D))
    out, k, v = O.block_full(bw, x, heads=2, eps=1e-6)
    b_v = bw["b_qkv"][2 * D:]
    gel = np.array([u * 0.5 * (1 + math.erf(u / math.sqrt(2))) for u in bw["b1"]])
    expect = x + b_v[perm] + bw["b_o"] + bw["w2"] @ gel + bw["b2"]
    np.testing.assert_allclose(out, expect, rtol=1e-13, atol=1e-13)
    np.testing.assert_allclose(k, np.tile(bw["b_qkv"][D:2 * D], (T, 1)), rtol=1e-15)
    np.testing.assert_allclose(v, np.tile(b_v, (T, 1)), rtol=1e-15)


def test_block_is_permutation_equivariant():
    # Bidirectional attention without a mask (Eq. 3): permuting the tokens of a
    # sequence permutes the block's outputs and nothing else.
    rng = np.random.default_rng(2)
    D, T = 8, 7
    bw = _rand_block(rng, D, 4 * D)
    x = rng.normal(size=(T, D))
    p = rng.permutation(T)
    out, k, v = O.block_full(bw, x, heads=2, eps=1e-6)
    out_p, k_p, v_p = O.block_full(bw, x[p], heads=2, eps=1e-6)
    np.testing.assert_allclose(out_p, out[p], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(k_p, k[p], rtol=1e-13)


def test_block_cached_over_all_tokens_is_the_full_block():
    rng = np.random.default_rng(3)
    D, T = 8, 6
    bw = _rand_block(rng, D, 4 * D)
    x = rng.normal(size=(T, D))
    out, k, v = O.block_full(bw, x, heads=2, eps=1e-6)
    kc, vc = rng.normal(size=(T, D)), rng.normal(size=(T, D))   # stale cache contents
    out_c = O.block_cached(bw, x, np.arange(T), kc, vc, heads=2, eps=1e-6)
    np.testing.assert_allclose(out_c, out, rtol=1e-13, atol=1e-13)
    np.testing.assert_array_equal(kc, k)
    np.testing.assert_array_equal(vc, v)


def test_block_cached_uses_cached_keys_for_unselected_tokens():
    # Eq. 9: a computed token attends to the cached K/V of I_cache tokens. With the
    # cache filled from the same inputs, the subset result equals the full block's
    # rows; with a perturbed cache row it does not.
    rng = np.random.default_rng(4)
    D, T = 8, 6
    bw = _rand_block(rng, D, 4 * D)
    x = rng.normal(size=(T, D))
    out, k, v = O.block_full(bw, x, heads=2, eps=1e-6)
    idx = np.array([1, 4])
    kc, vc = k.copy(), v.copy()
    np.testing.assert_allclose(O.block_cached(bw, x[idx], idx, kc, vc, 2, 1e-6), out[idx], rtol=1e-13, atol=1e-13)
    vc2 = v.copy()
    vc2[0] += 1.0
    assert np.abs(O.block_cached(bw, x[idx], idx, k.copy(), vc2, 2, 1e-6) - out[idx]).max() > 1e-3


# --------------------------------------------------------------------------
# Selection (Eq. 8)
# --------------------------------------------------------------------------

def test_cosine_similarity_special_cases():
    rng = np.random.default_rng(5)
    v = rng.normal(size=16)
    w = rng.normal(size=16)
    w -= (w @ v) / (v @ v) * v      # orthogonal to v
    assert abs(O.cosine_similarity(v, v) - 1) < 1e-15
    assert abs(O.cosine_similarity(v, -v) + 1) < 1e-15
    assert abs(O.cosine_similarity(v, 3.5 * v) - 1) < 1e-15
    assert abs(O.cosine_similarity(v, w)) < 1e-15
    assert O.cosine_similarity(np.zeros(16), v) == 0.0
    assert O.cosine_similarity(np.zeros(16), np.zeros(16)) == 0.0


def test_cosine_similarity_matches_fsum_loop():
    rng = np.random.default_rng(6)
    a, b = rng.normal(size=(5, 33)), rng.normal(size=(5, 33))
    got = O.cosine_similarity(a, b)
    for i in range(5):
        dot = math.fsum(float(x) * float(y) for x, y in zip(a[i], b[i]))
        na = math.fsum(float(x) * float(x) for x in a[i])
        nb = math.fsum(float(y) * float(y) for y in b[i])
        assert abs(got[i] - dot / math.sqrt(na * nb)) < 1e-15


@pytest.mark.parametrize("T,n", [(1, 0), (1, 1), (10, 0), (10, 3), (10, 10), (80, 20), (320, 50)])
def test_select_matches_brute_force_sort(T, n):
    rng = np.random.default_rng(T * 7 + n)
    S = rng.normal(size=T)
    if T > 4:                                  # inject exact ties
        S[rng.integers(0, T, size=T // 3)] = S[0]
    expect = sorted(t for _, t in sorted((float(S[t]), t) for t in range(T))[:n])
    assert list(O.select_compute(S, n)) == expect


def test_select_picks_least_similar_and_nan_first():
    S = np.array([0.99, 0.2, 0.999, np.nan, 0.5, 0.2])
    # NaN counts as -inf; the tie at 0.2 goes to the lower index.
    assert list(O.select_compute(S, 1)) == [3]
    assert list(O.select_compute(S, 3)) == [1, 3, 5]
    assert list(O.select_compute(S, 4)) == [1, 3, 4, 5]


def _rule_precedes(a, b, S, rule, prio, keys):
    """Token a is taken before token b under a selection rule of Table 3,
    written as explicit comparisons (priority, then the rule, then index)."""
    pa, pb = (prio[a], prio[b]) if prio is not None else (0, 0)
    if pa != pb:
        return pa > pb
    if rule == O.SELECT_RANDOM:
        ka, kb = int(keys[a]), int(keys[b])
    else:
        sa = -math.inf if math.isnan(S[a]) else S[a]
        sb = -math.inf if math.isnan(S[b]) else S[b]
        ka, kb = (sa, sb) if rule == O.SELECT_LEAST_SIMILAR else (-sa, -sb)
    if ka != kb:
        return ka < kb
    return a < b


@pytest.mark.parametrize("rule", [O.SELECT_LEAST_SIMILAR, O.SELECT_MOST_SIMILAR, O.SELECT_RANDOM])
@pytest.mark.parametrize("with_prio", [False, True])
@pytest.mark.parametrize("T,n", [(1, 0), (1, 1), (9, 4), (16, 7), (16, 16)])
def test_select_by_rule_is_a_prefix_of_the_order(rule, with_prio, T, n):
    """Every selected token precedes every unselected one under the stated
    order, the set has n members, ascending; ties in S, -0/+0 and NaN included."""
    rng = np.random.default_rng(T * 31 + n + rule * 7 + with_prio)
    S = np.round(rng.standard_normal(T), 1)  # rounding makes ties
    if T > 3:
        S[1] = np.nan
        S[2], S[3] = 0.0, -0.0
    prio = rng.integers(0, 2, T) if with_prio else None
    keys = rng.integers(0, 6, T).astype(np.uint32)  # repeated keys: ties
    got = list(O.select_by_rule(S, n, rule, prio, keys))
    assert len(got) == n and got == sorted(got)
    rest = [t for t in range(T) if t not in got]
    for a in got:
        for b in rest:
            assert _rule_precedes(a, b, S, rule, prio, keys), (a, b)


def test_select_by_rule_worked_cases():
    """Hand-worked six-token row (Table 3 strategies; priority 1 marks tokens
    that must be recomputed, as the observation-based strategy does for
    tokens decoded at steps t-1 and t)."""
    S = np.array([0.9, 0.1, np.nan, 0.5, 0.1, -0.2])
    prio = np.array([0, 0, 0, 1, 0, 1])
    keys = np.array([5, 3, 9, 1, 0, 2], np.uint32)
    # strategy V: least similar first; NaN counts as -inf
    assert list(O.select_by_rule(S, 3)) == [1, 2, 5]
    # strategy IV: most similar first; the NaN token comes last
    assert list(O.select_by_rule(S, 3, O.SELECT_MOST_SIMILAR)) == [0, 1, 3]
    # strategy III: ascending random keys
    assert list(O.select_by_rule(S, 3, O.SELECT_RANDOM, keys=keys)) == [3, 4, 5]
    # priority first (tokens 3 and 5), then each rule fills the remaining slot
    assert list(O.select_by_rule(S, 3, O.SELECT_LEAST_SIMILAR, prio)) == [2, 3, 5]
    assert list(O.select_by_rule(S, 3, O.SELECT_MOST_SIMILAR, prio)) == [0, 3, 5]
    assert list(O.select_by_rule(S, 3, O.SELECT_RANDOM, prio, keys)) == [3, 4, 5]
    # more priority tokens than the budget: the rule orders them
    assert list(O.select_by_rule(S, 1, O.SELECT_LEAST_SIMILAR, prio)) == [5]
    assert list(O.select_by_rule(S, 1, O.SELECT_MOST_SIMILAR, prio)) == [3]
    # without priority, the default rule is select_compute
    for n in range(7):
        assert list(O.select_by_rule(S, n)) == list(O.select_compute(S, n))


def test_selection_recomputes_the_changed_tokens():
    # Strategy V (Table 3): the tokens whose representation moved most since the
    # last step are recomputed.
    rng = np.random.default_rng(9)
    ref = rng.normal(size=(12, 16))
    cur = ref + 1e-3 * rng.normal(size=(12, 16))
    cur[[2, 7, 9]] = rng.normal(size=(3, 16))
    assert list(O.select_compute(O.cosine_similarity(cur, ref), 3)) == [2, 7, 9]


# --------------------------------------------------------------------------
# Embedding (Eq. 6)
# --------------------------------------------------------------------------

def test_embed_token_kinds():
    cfg = synth.config("tiny")
    W = synth.make_weights(cfg)
    lat = synth.make_latent_table(cfg)
    mask = np.ones((1, cfg["n_img"]), np.uint8)
    mask[0, [0, 5]] = 0
    lat = np.where(mask[:, :, None] == 0, lat, 0).astype(np.float32)
    labels = np.array([17], np.int32)
    X = O.embed(cfg, W, lat, mask, labels, "both")
    nb = cfg["n_buffer"]
    assert X.shape == (2, cfg["T"], cfg["width"])
    pos = W["pos_emb"].astype(np.float64)
    np.testing.assert_allclose(X[0, 3], pos[3] + W["class_emb"][17], rtol=1e-15)
    np.testing.assert_allclose(X[1, 3], pos[3], rtol=1e-15)                 # fake cond token = 0
    np.testing.assert_allclose(X[0, nb + 1], pos[nb + 1] + W["mask_emb"], rtol=1e-15)
    e5 = np.array([sum(float(W["embed_w"][d, i]) * float(lat[0, 5, i]) for i in range(16)) for d in range(cfg["width"])])
    np.testing.assert_allclose(X[0, nb + 5], pos[nb + 5] + e5 + W["embed_b"], rtol=1e-12, atol=1e-15)
    np.testing.assert_array_equal(X[0, nb:], X[1, nb:])                     # pair shares image tokens


# --------------------------------------------------------------------------
# Steps: invariants of the token cache and the condition cache
# --------------------------------------------------------------------------

@pytest.fixture(scope="module")
def tiny():
    cfg = synth.config("tiny")
    W = synth.make_weights(cfg)
    order, table = synth.make_order(cfg), synth.make_latent_table(cfg)
    (lat0, m0), (lat1, m1) = synth.tiny_state(cfg, order, table)
    labels = synth.make_labels(cfg)
    cache = O.Cache(cfg, cfg["batch"])
    O.full_step(cfg, W, cache, lat0, m0, labels, 3.0)
    return cfg, W, cache, (lat1, m1, labels)


def test_full_ratio_cached_step_equals_full_step(tiny):
    cfg, W, cache, (lat, m, labels) = tiny
    c_full, c_cached = copy.deepcopy(cache), copy.deepcopy(cache)
    z_f, g_f = O.full_step(cfg, W, c_full, lat, m, labels, 3.0)
    z_c, g_c, I, _ = O.cached_step(cfg, W, c_cached, lat, m, labels, cfg["T"], False, 3.0)
    assert (I == np.arange(cfg["T"])).all()
    np.testing.assert_allclose(z_c, z_f, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(g_c, g_f, rtol=1e-12, atol=1e-12)
    for l in c_full.K:
        np.testing.assert_allclose(c_cached.K[l], c_full.K[l], rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(c_cached.V[l], c_full.V[l], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(c_cached.delta, c_full.delta, rtol=1e-12, atol=1e-12)


def test_cached_step_leaves_unselected_cache_rows_untouched(tiny):
    cfg, W, cache, (lat, m, labels) = tiny
    c = copy.deepcopy(cache)
    n = synth.n_compute(cfg)
    z, g, I, S = O.cached_step(cfg, W, c, lat, m, labels, n, False, 3.0)
    assert I.shape == (2, n)
    # the image tokens decoded since the cache was filled changed most (their
    # input went from the mask embedding to a latent) and must be recomputed
    order, table = synth.make_order(cfg), synth.make_latent_table(cfg)
    (_, m_before), _ = synth.tiny_state(cfg, order, table)
    newly = cfg["n_buffer"] + np.where(m_before[0] != m[0])[0]
    assert len(newly) == 8
    for r in range(2):
        assert set(newly) <= set(I[r])
        keep = np.setdiff1d(np.arange(cfg["T"]), I[r])
        for l in c.K:
            np.testing.assert_array_equal(c.K[l][r][keep], cache.K[l][r][keep])
            np.testing.assert_array_equal(c.V[l][r][keep], cache.V[l][r][keep])
            assert (np.abs(c.K[l][r][I[r]] - cache.K[l][r][I[r]]).max(axis=1) > 0).all()
        np.testing.assert_array_equal(c.x_last[r][keep], cache.x_last[r][keep])


def test_cond_reuse_with_same_step_residual_is_exact(tiny):
    # Condition cache (Eq. 10): when the residual comes from the same inputs, the
    # rebuilt unconditional output equals the computed one.
    cfg, W, cache, (lat, m, labels) = tiny
    c = copy.deepcopy(cache)
    z_f, g_f = O.full_step(cfg, W, c, lat, m, labels, 3.0)
    z_r, g_r, _, _ = O.cached_step(cfg, W, c, lat, m, labels, cfg["T"], True, 3.0)
    np.testing.assert_allclose(z_r, z_f, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(g_r, g_f, rtol=1e-11, atol=1e-12)


def test_guidance_closed_form():
    c, u = np.array([1.0, -2.0]), np.array([0.5, 1.0])
    np.testing.assert_array_equal(O.guidance(c, u, 1.0), c)     # gamma = 1 -> conditional
    np.testing.assert_array_equal(O.guidance(c, u, 0.0), u)     # gamma = 0 -> unconditional
    np.testing.assert_allclose(O.guidance(c, u, 3.0), [2.0, -8.0])
    d = O.cond_cache_store(c, u)
    np.testing.assert_array_equal(O.cond_cache_reuse(c, d), u)


def test_cfg_interval_one_never_reuses():
    # A condition-cache interval of 1 means every step runs both pathways, i.e.
    # standard classifier-free guidance.
    assert not any(O.plan(k, 4, 9, 1)[1] for k in range(64))
    assert not any(O.plan(k, 4, 9, 9, cond_cache=False)[1] for k in range(64))


def test_schedule_paper_settings(golden_dir):
    for line in open(os.path.join(golden_dir, "schedule.txt")):
        if not line.strip() or line[0] == "#":
            continue
        head, full = line.split(":")
        steps, k0, tau = map(int, head.split())
        expect = [int(t) for t in full.split()]
        got = [k for k in range(steps) if O.plan(k, k0, tau, tau)[0]]
        assert got == expect
        # with tau_cfg = tau every cached step reuses the condition cache
        assert all(O.plan(k, k0, tau, tau)[1] for k in range(steps) if k not in expect)


def test_schedule_cfg_every_other_step():
    kinds = [O.plan(k, 4, 9, 2) for k in range(4, 14)]
    assert kinds[0] == (True, False)
    assert [r for f, r in kinds[1:9]] == [True, False, True, False, True, False, True, False]
    assert kinds[9] == (True, False)


def test_mask_schedule_structure():
    for steps, n in [(64, 256), (32, 256), (64, 1024), (64, 64)]:
        m = synth.mask_counts(steps, n)
        dec = [n - m[0]] + [m[k - 1] - m[k] for k in range(1, steps)]
        assert m[-1] == 0 and min(dec) >= 1 and sum(dec) == n
