"""Closed-form pins of the oracle's decoding steps: which representation Eq. 8
compares, at which block, what the final features are made of, and how the
caches carry over across full, cached and condition-reuse steps.

The model here has every block reduced to a constant shift. With W_o = 0,
W1 = 0, W2 = 0 and b2 = 0, block l maps x to x + b_o[l] whatever its attention
and MLP compute, while its Q/K/V projection (LN1 then W_qkv) still runs on
the real input. So:

* the output of block l is X + b_o[0] + ... + b_o[l] (X the embedded tokens);
* the value matrix of block l is LN1_l(X + b_o[0] + ... + b_o[l-1]) W_v^T + b_v;
* the last block's output, and from it the final features, follow in closed
  form for any step sequence.

Every expected value below is computed by scalar loops with math.fsum. It is
not computed by the oracle's numpy code. A slip in the oracle fails one of
these tests: the wrong block for the selection reference, K or the block
output in place of V, the reference not overwritten, the buffer tokens
sliced instead of the image tokens, or the unconditional rows' state not
kept over a reuse step.
"""
import copy
import math

import numpy as np
import pytest

import oracle as O

GAMMA = 3.0
EPS = 1e-6


def shift_model(seed, depth=3, s=2, D=8, heads=2, nb=3, n_img=5, td=2, n_classes=4, criterion="value"):
    """Config and weights of a `depth`-block model whose blocks are constant shifts."""
    rng = np.random.default_rng(seed)
    T = nb + n_img
    cfg = dict(depth=depth, width=D, heads=heads, mlp_ratio=4, n_buffer=nb, n_img=n_img, T=T, token_dim=td,
               n_classes=n_classes, sel_layers=s, ln_eps=EPS, criterion=criterion)
    blocks = []
    for _ in range(depth):
        blocks.append({
            "ln1_g": 1 + 0.3 * rng.normal(size=D), "ln1_b": 0.3 * rng.normal(size=D),
            "w_qkv": rng.normal(size=(3 * D, D)), "b_qkv": rng.normal(size=3 * D),
            "w_o": np.zeros((D, D)), "b_o": rng.normal(size=D),
            "ln2_g": 1 + 0.3 * rng.normal(size=D), "ln2_b": 0.3 * rng.normal(size=D),
            "w1": np.zeros((4 * D, D)), "b1": rng.normal(size=4 * D),
            "w2": np.zeros((D, 4 * D)), "b2": np.zeros(D),
        })
    W = {"pos_emb": rng.normal(size=(T, D)), "class_emb": rng.normal(size=(n_classes, D)),
         "mask_emb": rng.normal(size=D), "embed_w": rng.normal(size=(D, td)), "embed_b": rng.normal(size=D),
         "lnf_g": 1 + 0.3 * rng.normal(size=D), "lnf_b": 0.3 * rng.normal(size=D), "blocks": blocks}
    return cfg, W


def inputs(seed, B, n_img, td, n_decoded):
    """Latents and masks of B pairs with the first n_decoded positions of a
    fixed per-pair order decoded."""
    rng = np.random.default_rng(seed)
    table = rng.normal(size=(B, n_img, td))
    order = [rng.permutation(n_img) for _ in range(B)]

    def state(k):
        mask = np.ones((B, n_img), np.uint8)
        for b in range(B):
            mask[b, order[b][:k]] = 0
        return np.where(mask[:, :, None] == 0, table, 0.0), mask
    return [state(k) for k in n_decoded]


# ---- scalar closed forms ----------------------------------------------------

def ln_loop(x, g, b):
    D = len(x)
    mu = math.fsum(x) / D
    var = math.fsum((v - mu) ** 2 for v in x) / D
    r = 1.0 / math.sqrt(var + EPS)
    return [(x[i] - mu) * r * g[i] + b[i] for i in range(D)]


def embedded(cfg, W, lat, mask, labels, b, uncond):
    """Row `b` of the embedded tokens (Eq. 6) as lists, by scalar loops."""
    nb, D, td = cfg["n_buffer"], cfg["width"], cfg["token_dim"]
    rows = []
    for t in range(cfg["T"]):
        base = [float(W["pos_emb"][t][d]) for d in range(D)]
        if t < nb:
            add = [0.0] * D if uncond else [float(W["class_emb"][labels[b]][d]) for d in range(D)]
        else:
            i = t - nb
            if mask[b][i]:
                add = [float(W["mask_emb"][d]) for d in range(D)]
            else:
                add = [math.fsum(float(W["embed_w"][d][j]) * float(lat[b][i][j]) for j in range(td))
                       + float(W["embed_b"][d]) for d in range(D)]
        rows.append([base[d] + add[d] for d in range(D)])
    return rows


def shifted(cfg, W, x, upto):
    """x + b_o[0] + ... + b_o[upto - 1], token by token."""
    D = cfg["width"]
    return [[x[t][d] + math.fsum(float(W["blocks"][j]["b_o"][d]) for j in range(upto)) for d in range(D)]
            for t in range(len(x))]


def value_matrix(cfg, W, x, l):
    """V of block l: LN1_l(block input) W_v^T + b_v, W_v the third D x D slice of W_qkv."""
    D = cfg["width"]
    bw = W["blocks"][l]
    xin = shifted(cfg, W, x, l)
    out = []
    for t in range(len(x)):
        n = ln_loop(xin[t], bw["ln1_g"], bw["ln1_b"])
        out.append([math.fsum(float(bw["w_qkv"][2 * D + e][d]) * n[d] for d in range(D))
                    + float(bw["b_qkv"][2 * D + e]) for e in range(D)])
    return out


def representation(cfg, W, x):
    """What Eq. 8 compares: V of block s-1 (value criterion) or block s-1's output."""
    s = cfg["sel_layers"]
    if cfg["criterion"] == "value":
        return value_matrix(cfg, W, x, s - 1)
    return shifted(cfg, W, x, s)


def cos_loop(a, b):
    dot = math.fsum(u * v for u, v in zip(a, b))
    na = math.fsum(u * u for u in a)
    nb = math.fsum(v * v for v in b)
    return dot / math.sqrt(max(na * nb, 1e-16))


def final_features(cfg, W, x_last):
    """Final LayerNorm of the image tokens of the last block's output."""
    return [ln_loop(x_last[t], W["lnf_g"], W["lnf_b"]) for t in range(cfg["n_buffer"], cfg["T"])]


class Model:
    """Closed-form state of every row: the representation each row last ran
    with, and its last-block output (the token cache of the model output)."""

    def __init__(self, cfg, W, B):
        self.cfg, self.W, self.B = cfg, W, B
        self.ref = [None] * (2 * B)
        self.x_last = [None] * (2 * B)
        self.delta = None

    def rows_x(self, lat, mask, labels, reuse):
        n_rows = self.B if reuse else 2 * self.B
        return [embedded(self.cfg, self.W, lat, mask, labels, r % self.B, r >= self.B) for r in range(n_rows)]

    def z(self):
        return np.array([final_features(self.cfg, self.W, self.x_last[r]) for r in range(2 * self.B)])

    def full(self, lat, mask, labels):
        L = self.cfg["depth"]
        for r, x in enumerate(self.rows_x(lat, mask, labels, False)):
            self.ref[r] = representation(self.cfg, self.W, x)
            self.x_last[r] = shifted(self.cfg, self.W, x, L)
        z = self.z()
        self.delta = z[:self.B] - z[self.B:]
        return z

    def cached(self, lat, mask, labels, n, reuse):
        """Returns (S per row, I per row, z of both pathways)."""
        L = self.cfg["depth"]
        S_all, I_all = [], []
        for r, x in enumerate(self.rows_x(lat, mask, labels, reuse)):
            cur = representation(self.cfg, self.W, x)
            S = [cos_loop(cur[t], self.ref[r][t]) for t in range(len(x))]
            self.ref[r] = cur
            I = sorted(t for _, t in sorted((S[t], t) for t in range(len(x)))[:n])
            new = shifted(self.cfg, self.W, x, L)
            self.x_last[r] = [new[t] if t in I else self.x_last[r][t] for t in range(len(x))]
            S_all.append(S)
            I_all.append(I)
        z = self.z()
        if reuse:
            z[self.B:] = z[:self.B] - self.delta
        else:
            self.delta = z[:self.B] - z[self.B:]
        return np.array(S_all), np.array(I_all), z


# ---- tests -------------------------------------------------------------------

@pytest.mark.parametrize("criterion", ["value", "feature"])
def test_full_step_final_features_are_the_image_tokens(criterion):
    """z of a full step is the final LayerNorm of the last block's output at
    the n_img image positions (not the n_buffer class positions), cond rows
    first; the guided output is u + gamma (c - u)."""
    cfg, W = shift_model(1, criterion=criterion)
    B = 2
    labels = np.array([1, 3])
    (lat, mask), = inputs(2, B, cfg["n_img"], cfg["token_dim"], [2])
    m = Model(cfg, W, B)
    z_ref = m.full(lat, mask, labels)
    cache = O.Cache(cfg, B)
    z, g = O.full_step(cfg, W, cache, lat, mask, labels, GAMMA)
    assert z.shape == (2 * B, cfg["n_img"], cfg["width"])
    np.testing.assert_allclose(z, z_ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(g, z_ref[B:] + GAMMA * (z_ref[:B] - z_ref[B:]), rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(cache.ref, np.array(m.ref), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("criterion", ["value", "feature"])
def test_step_sequence_matches_closed_form(criterion):
    """full -> cached (both) -> cached (reuse) -> cached (both) -> cached (both).

    At every cached step S is Eq. 8's cosine between this step's
    representation (V of block s-1, or block s-1's output) and the one the row
    last ran with. After a reuse step the unconditional rows compare against
    the step before it, and their cached outputs are the ones from before
    too. I_cache tokens keep their last-block output."""
    cfg, W = shift_model(3, criterion=criterion)
    B, n = 2, 3
    labels = np.array([0, 2])
    states = inputs(4, B, cfg["n_img"], cfg["token_dim"], [1, 2, 3, 4, 5])
    m = Model(cfg, W, B)
    cache = O.Cache(cfg, B)
    lat, mask = states[0]
    m.full(lat, mask, labels)
    O.full_step(cfg, W, cache, lat, mask, labels, GAMMA)
    for (lat, mask), reuse in zip(states[1:], [False, True, False, False]):
        S_ref, I_ref, z_ref = m.cached(lat, mask, labels, n, reuse)
        z, g, I, S = O.cached_step(cfg, W, cache, lat, mask, labels, n, reuse, GAMMA)
        np.testing.assert_allclose(S, S_ref, rtol=0, atol=1e-13)
        assert I.tolist() == I_ref.tolist()
        np.testing.assert_allclose(z, z_ref, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(g, z_ref[B:] + GAMMA * (z_ref[:B] - z_ref[B:]), rtol=1e-12, atol=1e-12)


def test_value_and_feature_criteria_compare_different_things():
    """The two criteria give different similarities on the same inputs, so
    the branch taken is visible; each matches its own closed form."""
    got = {}
    for criterion in ("value", "feature"):
        cfg, W = shift_model(5, criterion=criterion)
        (lat0, m0), (lat1, m1) = inputs(6, 1, cfg["n_img"], cfg["token_dim"], [1, 3])
        cache = O.Cache(cfg, 1)
        O.full_step(cfg, W, cache, lat0, m0, np.array([1]), GAMMA)
        _, _, _, S = O.cached_step(cfg, W, cache, lat1, m1, np.array([1]), 2, False, GAMMA)
        m = Model(cfg, W, 1)
        m.full(lat0, m0, np.array([1]))
        S_ref, _, _ = m.cached(lat1, m1, np.array([1]), 2, False)
        np.testing.assert_allclose(S, S_ref, rtol=0, atol=1e-13)
        got[criterion] = S
    assert np.abs(got["value"] - got["feature"]).max() > 1e-3


def test_selection_layer_is_block_s_minus_1():
    """Full mixing weights everywhere except block s-1, whose W_v is zero and
    b_v nonzero: every value-matrix row there equals b_v, in every step, so
    S = 1 for every token and the tie rule recomputes tokens 0..N-1. Taking V
    from any other block, or K, would give varying similarities."""
    rng = np.random.default_rng(7)
    D, depth, s, nb, n_img = 8, 4, 2, 3, 6
    cfg, W = shift_model(8, depth=depth, s=s, D=D, nb=nb, n_img=n_img)
    for bw in W["blocks"]:                 # full blocks: attention and MLP mix the tokens
        bw["w_o"] = 0.5 * rng.normal(size=(D, D))
        bw["w1"] = 0.5 * rng.normal(size=(4 * D, D))
        bw["w2"] = 0.5 * rng.normal(size=(D, 4 * D))
        bw["b2"] = rng.normal(size=D)
    W["blocks"][s - 1]["w_qkv"][2 * D:] = 0.0
    (lat0, m0), (lat1, m1) = inputs(9, 2, n_img, cfg["token_dim"], [1, 4])
    labels = np.array([0, 1])
    cache = O.Cache(cfg, 2)
    O.full_step(cfg, W, cache, lat0, m0, labels, GAMMA)
    n = 4
    _, _, I, S = O.cached_step(cfg, W, cache, lat1, m1, labels, n, False, GAMMA)
    assert (S == 1.0).all()
    assert (I == np.arange(n)).all()
    # the same model with block s-1's W_v restored: the similarities vary
    W2 = copy.deepcopy(W)
    W2["blocks"][s - 1]["w_qkv"][2 * D:] = rng.normal(size=(D, D))
    cache = O.Cache(cfg, 2)
    O.full_step(cfg, W2, cache, lat0, m0, labels, GAMMA)
    _, _, _, S2 = O.cached_step(cfg, W2, cache, lat1, m1, labels, n, False, GAMMA)
    assert S2.min() < 0.999


def test_feature_criterion_recomputes_exactly_the_changed_tokens():
    """Blocks 0..s-1 that act token by token (W_qkv = 0 makes every score the
    same constant and every value row b_v, so the attention output is one
    vector for all tokens): tokens whose input did not change keep the same
    block s-1 output, so S = 1 for them and S < 1 for the tokens decoded in
    between. With N = (newly decoded) + 2 the selection is those tokens plus
    the two lowest-index unchanged ones (ties go to the lower index). Block s
    mixes tokens, so reading its output instead would move every similarity."""
    rng = np.random.default_rng(10)
    D, depth, s = 8, 3, 2
    cfg, W = shift_model(11, depth=depth, s=s, D=D, nb=3, n_img=6, criterion="feature")
    for l, bw in enumerate(W["blocks"]):
        bw["w1"] = 0.5 * rng.normal(size=(4 * D, D))
        bw["w2"] = 0.5 * rng.normal(size=(D, 4 * D))
        if l < s:
            bw["w_qkv"][:] = 0.0             # the same attention output for every token
        bw["w_o"] = 0.5 * rng.normal(size=(D, D))
    (lat0, m0), (lat1, m1) = inputs(12, 1, cfg["n_img"], cfg["token_dim"], [1, 3])
    newly = sorted(cfg["n_buffer"] + i for i in np.where(m0[0] != m1[0])[0])
    assert len(newly) == 2
    cache = O.Cache(cfg, 1)
    O.full_step(cfg, W, cache, lat0, m0, np.array([2]), GAMMA)
    n = len(newly) + 2
    _, _, I, S = O.cached_step(cfg, W, cache, lat1, m1, np.array([2]), n, False, GAMMA)
    for r in range(2):
        unchanged = [t for t in range(cfg["T"]) if t not in newly]
        assert all(S[r][t] == 1.0 for t in unchanged)
        assert all(S[r][t] < 1.0 for t in newly)
        assert I[r].tolist() == sorted(newly + unchanged[:2])
