"""Plain fp64 CPU oracle of LazyMAR's cached MAR decoding step.

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's CPU
baseline / reference leg import this module. The product path (the CUDA
library and its binding) never does, and this module imports nothing from it.
Its inputs come from the seeded generators in `synth/` or from the tests.

Each function restates one passage of the paper (cited in its docstring) in
direct numpy form: fp64 throughout, matrix products as the only library
primitive, no blocking, fusion or reordering beyond what the passage states.
Where the paper is silent, ambiguous or garbled the docstring says "reading"
and states the choice; the same list is kept in the design notes.

Layout. A batch of B cond/uncond pairs runs as rows: rows 0..B-1 are the
conditional pathway of pairs 0..B-1, rows B..2B-1 the unconditional pathway of
the same pairs (a condition-cache reuse step runs rows 0..B-1 only). Each row
is a sequence of T = n_buffer + n_img tokens of width D: n_buffer conditional
(class) tokens first, then the image tokens (Eq. 6; 64 cls tokens, Sec. 4.1).
Weight matrices use the [out, in] layout, y = x W^T + b.

Parity status: every function below is pinned by tests/test_oracle.py against
closed forms, brute force or invariants the paper fixes. The overall quality of
the cached approximation against full recomputation is not something the paper
prints values for (its FID/IS need trained weights): that comparison is a
measurement, not a pin.
"""
import numpy as np
from scipy.special import erf

F64 = np.float64

# ----------------------------------------------------------------------------
# Transformer pieces (Eq. 3 and the MAR block the paper builds on)
# ----------------------------------------------------------------------------


def layer_norm(x, g, b, eps):
    """LayerNorm over the width: (x - mean) / sqrt(var + eps) * g + b.

    Reading: the paper's blocks are MAR's pre-LN transformer blocks (Sec. 4.1
    uses MAR's default settings); biased variance, eps = 1e-6.
    """
    x = np.asarray(x, F64)
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * np.asarray(g, F64) + np.asarray(b, F64)


def gelu(x):
    """GELU with the exact normal CDF: x * Phi(x), Phi(x) = (1 + erf(x / sqrt 2)) / 2."""
    x = np.asarray(x, F64)
    return 0.5 * x * (1.0 + erf(x / np.sqrt(2.0)))


def linear(x, w, b):
    """y = x W^T + b with W in [out, in] layout."""
    return np.asarray(x, F64) @ np.asarray(w, F64).T + np.asarray(b, F64)


def attention(q, k, v, heads):
    """Bidirectional multi-head attention of Eq. 3 for one sequence.

    Every query attends to every key (no mask): O = softmax(Q K^T / sqrt(d)) V
    per head, with d the head width and the heads taking consecutive slices of
    the width. q is [n_q, D]; k and v are [T, D]. The row maximum is subtracted
    before exponentiating (softmax is invariant to that shift).
    """
    q = np.asarray(q, F64)
    k = np.asarray(k, F64)
    v = np.asarray(v, F64)
    n_q, D = q.shape
    dh = D // heads
    out = np.empty((n_q, D), F64)
    for h in range(heads):
        sl = slice(h * dh, (h + 1) * dh)
        s = q[:, sl] @ k[:, sl].T / np.sqrt(F64(dh))
        s = s - s.max(axis=1, keepdims=True)
        p = np.exp(s)
        p = p / p.sum(axis=1, keepdims=True)
        out[:, sl] = p @ v[:, sl]
    return out


def embed(cfg, W, latents, mask, labels, pathways):
    """Input tokens of Eq. 6 for every row: X joined with C conditional tokens.

    Conditional pathway: the C = n_buffer buffer positions hold the class
    embedding c(y); unconditional pathway: the fake conditional tokens are zero
    (Eq. 6). Image positions hold Linear(token_dim -> D)(latent) once decoded and
    a learned mask embedding while masked (reading: MAR's encoder input with
    masked positions kept in the sequence). A learned position embedding is
    added at all T positions.

    latents [B, n_img, token_dim], mask [B, n_img] (1 = masked), labels [B].
    pathways: "both" -> 2B rows, "cond" -> B rows.
    """
    B = latents.shape[0]
    nb, D = cfg["n_buffer"], cfg["width"]
    img = linear(latents.reshape(-1, latents.shape[-1]), W["embed_w"], W["embed_b"]).reshape(B, -1, D)
    img = np.where(np.asarray(mask)[:, :, None] != 0, np.asarray(W["mask_emb"], F64)[None, None, :], img)
    cond_buf = np.asarray(W["class_emb"], F64)[np.asarray(labels)][:, None, :].repeat(nb, axis=1)
    rows = [np.concatenate([cond_buf, img], axis=1)]
    if pathways == "both":
        rows.append(np.concatenate([np.zeros_like(cond_buf), img], axis=1))
    X = np.concatenate(rows, axis=0)
    return X + np.asarray(W["pos_emb"], F64)[None]


def block_qkv(bw, x, eps):
    """Pre-LN attention input: Q, K, V = LN1(x) W_qkv^T + b_qkv, split along the width."""
    D = x.shape[-1]
    qkv = linear(layer_norm(x, bw["ln1_g"], bw["ln1_b"], eps), bw["w_qkv"], bw["b_qkv"])
    return qkv[:, :D], qkv[:, D:2 * D], qkv[:, 2 * D:]


def block_rest(bw, x, o, eps):
    """Rest of the block: y = x + O W_o^T + b_o; out = y + MLP(LN2(y)), MLP = W2 GELU(W1 . + b1) + b2."""
    y = x + linear(o, bw["w_o"], bw["b_o"])
    h = gelu(linear(layer_norm(y, bw["ln2_g"], bw["ln2_b"], eps), bw["w1"], bw["b1"]))
    return y + linear(h, bw["w2"], bw["b2"])


def block_full(bw, x, heads, eps):
    """One bidirectional block over all tokens of a sequence (Eq. 3). Returns (out, K, V)."""
    q, k, v = block_qkv(bw, x, eps)
    return block_rest(bw, x, attention(q, k, v, heads), eps), k, v


def block_cached(bw, x_sel, idx, k_cache, v_cache, heads, eps):
    """One block under the token cache, Eq. 9, for one sequence.

    Only the tokens in I_compute (= idx, x_sel holds their input features) are
    computed. Their fresh K and V overwrite the cached rows idx; their queries
    then attend over all T keys: fresh ones for I_compute, cached ones for
    I_cache (applying the cache to self-attention and to the MLP, Sec. 3.2.1).
    Rows of k_cache / v_cache outside idx are left untouched. Returns the block
    output for the rows in idx; the caches are updated in place.
    """
    q, k, v = block_qkv(bw, x_sel, eps)
    k_cache[idx] = k
    v_cache[idx] = v
    return block_rest(bw, x_sel, attention(q, k_cache, v_cache, heads), eps)


# ----------------------------------------------------------------------------
# Token selection (Eq. 8)
# ----------------------------------------------------------------------------


def cosine_similarity(cur, ref, eps=1e-8):
    """S(x_i) of Eq. 8: cosine between a token's current and cached representation.

    Over the last axis: <cur, ref> / sqrt(max(|cur|^2 |ref|^2, eps^2)), in fp64.
    Reading: the eps guard of common cosine implementations; a zero vector
    gives S = 0.
    """
    cur = np.asarray(cur, F64)
    ref = np.asarray(ref, F64)
    dot = np.sum(cur * ref, axis=-1)
    n1 = np.sum(cur * cur, axis=-1)
    n2 = np.sum(ref * ref, axis=-1)
    return dot / np.sqrt(np.maximum(n1 * n2, F64(eps) * F64(eps)))


def select_compute(S, n):
    """I_compute of Eq. 8 for one row: which N tokens are recomputed.

    Reading: Eq. 8 prints argmax, but the text skips the tokens most similar to
    their cached values and strategy V of Table 3 caches the maximum-similarity
    tokens, so I_compute is the N tokens with the SMALLEST S. Ties go to the
    lower token index; a NaN similarity counts as -inf (always recomputed).
    Returned ascending.
    """
    S = np.asarray(S, F64)
    S = np.where(np.isnan(S), -np.inf, S)
    order = np.lexsort((np.arange(S.shape[0]), S))
    return np.sort(order[:n]).astype(np.int64)


# Token-selection rules (Table 3): which tokens fill the recompute budget N.
SELECT_LEAST_SIMILAR = 0  # strategy V (LazyMAR): cache the most similar, recompute the least
SELECT_MOST_SIMILAR = 1   # strategy IV: cache the least similar, recompute the most
SELECT_RANDOM = 2         # strategy III: caller-drawn random priority keys


def select_by_rule(S, n, rule=SELECT_LEAST_SIMILAR, priority=None, keys=None):
    """I_compute for one row under the selection strategies of Sec. 4.4 (Table 3)
    and the observation-based strategy of Sec. 3.2.1.

    Tokens are taken in the order: priority descending (when given), then the
    rule, then token index ascending; the first n are recomputed, returned
    ascending. Rules: SELECT_LEAST_SIMILAR, S ascending (strategy V, the
    default, equal to select_compute); SELECT_MOST_SIMILAR, S descending
    (strategy IV); SELECT_RANDOM, ascending `keys` (strategy III: the random
    draw is an input). A NaN S counts as -inf under both similarity rules.
    Reading: the priority classes express the strategies that choose by token
    type. Observation-based: 1 for tokens decoded at step t-1 or decoded at
    step t, which are always recomputed. Strategy I (cache the unpredicted
    tokens): 1 for decoded tokens. Strategy II (cache the predicted tokens): 1
    for masked tokens. The paper gives no order inside a class; the rule
    decides.
    """
    S = np.asarray(S, F64)
    T = S.shape[0]
    if rule == SELECT_RANDOM:
        key = np.asarray(keys, np.int64)
    else:
        Sm = np.where(np.isnan(S), -np.inf, S)
        key = Sm if rule == SELECT_LEAST_SIMILAR else -Sm
    prio = np.zeros(T, np.int64) if priority is None else np.asarray(priority, np.int64)
    order = np.lexsort((np.arange(T), key, -prio))
    return np.sort(order[:n]).astype(np.int64)


# ----------------------------------------------------------------------------
# Classifier-free guidance and the condition cache (Eq. 7, Eq. 10)
# ----------------------------------------------------------------------------


def guidance(z_cond, z_uncond, gamma):
    """Guided output from the two pathways.

    Reading: Eq. 7 as printed (F_cond + gamma F_uncond) is not a guidance mix;
    the standard classifier-free guidance u + gamma (c - u) is used.
    """
    z_cond = np.asarray(z_cond, F64)
    z_uncond = np.asarray(z_uncond, F64)
    return z_uncond + F64(gamma) * (z_cond - z_uncond)


def cond_cache_store(z_cond, z_uncond):
    """Condition cache of Eq. 10, stored as cond - uncond (the paper stores
    uncond - cond and adds it; storing the negation and subtracting gives the
    same reconstruction)."""
    return np.asarray(z_cond, F64) - np.asarray(z_uncond, F64)


def cond_cache_reuse(z_cond, delta):
    """Unconditional output rebuilt from the condition cache (Sec. 3.2.2): u = c - delta."""
    return np.asarray(z_cond, F64) - np.asarray(delta, F64)


# ----------------------------------------------------------------------------
# Periodic cache-reuse-refreshment schedule
# ----------------------------------------------------------------------------


def plan(k, k0, tau, tau_cfg, cond_cache=True):
    """Kind of decoding step k (0-based) under periodic cache-reuse-refreshment.

    Reading of Sec. 1 ("every K steps ... full computation"), Fig. 3 and Sec. 4.1
    (64 steps: caching from the 5th step, tau = 9): steps k < k0 are full; after
    that a full step comes whenever (k - k0) is a multiple of tau, and the
    others are cached steps. The condition cache is refreshed whenever both
    pathways run; a cached step reuses it when (k - k0) is not a multiple of
    tau_cfg (tau_cfg = 0 or cond_cache False: never).
    Returns (full, cond_reuse).
    """
    if k < k0 or (k - k0) % tau == 0:
        return True, False
    reuse = bool(cond_cache) and tau_cfg > 0 and (k - k0) % tau_cfg != 0
    return False, reuse


# ----------------------------------------------------------------------------
# Decoding steps
# ----------------------------------------------------------------------------


class Cache:
    """Token cache, selection reference and condition cache for 2B rows.

    K[l], V[l] : keys/values of blocks l >= s (I_cache rows are read from here)
    ref        : block s-1 value matrix (or output features) of the last step
                 each row ran: the C^{l=3} of Eq. 8
    x_last     : output features of the last block (the token cache of the
                 model output, from which I_cache rows of the output come)
    delta      : condition cache, cond - uncond of the final features
    """

    def __init__(self, cfg, batch):
        rows, T, D = 2 * batch, cfg["T"], cfg["width"]
        s, L = cfg["sel_layers"], cfg["depth"]
        self.batch = batch
        self.K = {l: np.zeros((rows, T, D), F64) for l in range(s, L)}
        self.V = {l: np.zeros((rows, T, D), F64) for l in range(s, L)}
        self.ref = np.zeros((rows, T, D), F64)
        self.x_last = np.zeros((rows, T, D), F64)
        self.delta = np.zeros((batch, cfg["n_img"], D), F64)


def _final(cfg, W, x_last):
    """Output features of the image tokens: final LayerNorm of the last block's output."""
    return layer_norm(x_last[:, cfg["n_buffer"]:], W["lnf_g"], W["lnf_b"], cfg["ln_eps"])


def full_step(cfg, W, cache, latents, mask, labels, gamma):
    """A refresh step: every token, both pathways, all caches refreshed (Fig. 3).

    Returns z [2B, n_img, D] (final features of both pathways) and the guided
    output [B, n_img, D]. Fills the token cache C_token^l := F^l(X) (Sec.
    3.2.1), the selection reference and the condition cache (Eq. 10).
    """
    s, H, eps = cfg["sel_layers"], cfg["heads"], cfg["ln_eps"]
    B = latents.shape[0]
    X = embed(cfg, W, latents, mask, labels, "both")
    for r in range(2 * B):
        x = X[r]
        for l, bw in enumerate(W["blocks"]):
            x_new, k, v = block_full(bw, x, H, eps)
            if l == s - 1:
                cache.ref[r] = v if cfg.get("criterion", "value") == "value" else x_new
            if l >= s:
                cache.K[l][r] = k
                cache.V[l][r] = v
            x = x_new
        cache.x_last[r] = x
    z = _final(cfg, W, cache.x_last[:2 * B])
    cache.delta = cond_cache_store(z[:B], z[B:])
    return z, guidance(z[:B], z[B:], gamma)


def cached_step(cfg, W, cache, latents, mask, labels, n, cond_reuse, gamma, idx=None, rule=SELECT_LEAST_SIMILAR,
                priority=None, keys=None):
    """A cached step: token cache (Eq. 8, Eq. 9) and optionally the condition cache.

    Blocks 0..s-1 run over all tokens (the paper's "first three layers"). At
    block s-1 every token's value matrix (criterion "value", Sec. 4.4) or
    output feature is compared with the selection reference by Eq. 8's cosine;
    the N least similar tokens form I_compute and the reference is overwritten
    with the current values. Blocks s..L-1 run only I_compute (Eq. 9); their
    results are written back into the token cache. The final features of I_cache
    tokens come from the cache.

    cond_reuse: only the conditional rows run; the unconditional output is
    rebuilt as c - delta (Sec. 3.2.2). Otherwise both pathways run and the
    condition cache is refreshed.
    idx: optional [rows, N] caller-chosen I_compute (used instead of Eq. 8).
    rule, priority [rows, T], keys [rows, T]: the selection strategy of
    select_by_rule (default: strategy V, the N least similar tokens).

    Returns z [2B, n_img, D], guided [B, n_img, D], I_compute [rows, N] and the
    similarities S [rows, T].
    """
    s, L, H, eps = cfg["sel_layers"], cfg["depth"], cfg["heads"], cfg["ln_eps"]
    B = latents.shape[0]
    X = embed(cfg, W, latents, mask, labels, "cond" if cond_reuse else "both")
    rows = X.shape[0]
    I_all = np.zeros((rows, n), np.int64)
    S_all = np.zeros((rows, cfg["T"]), F64)
    for r in range(rows):
        x = X[r]
        cur = None
        for l in range(s):
            x_new, _, v = block_full(W["blocks"][l], x, H, eps)
            if l == s - 1:
                cur = v if cfg.get("criterion", "value") == "value" else x_new
            x = x_new
        S = cosine_similarity(cur, cache.ref[r])
        cache.ref[r] = cur
        if idx is not None:
            I = np.asarray(idx[r], np.int64)
        else:
            I = select_by_rule(S, n, rule, None if priority is None else priority[r], None if keys is None else keys[r])
        xs = x[I]
        for l in range(s, L):
            xs = block_cached(W["blocks"][l], xs, I, cache.K[l][r], cache.V[l][r], H, eps)
        cache.x_last[r][I] = xs
        I_all[r] = I
        S_all[r] = S
    z = _final(cfg, W, cache.x_last[:rows])
    if cond_reuse:
        z = np.concatenate([z, cond_cache_reuse(z[:B], cache.delta)], axis=0)
    else:
        cache.delta = cond_cache_store(z[:B], z[B:])
    return z, guidance(z[:B], z[B:], gamma), I_all, S_all
