"""Seeded synthetic MAR-shaped workloads.

The paper evaluates on ImageNet 256x256 class-conditional generation with
trained MAR-B/L/H weights (Sec. 4.1). Neither the dataset nor the weights are
available, so every input here is synthetic with the paper's shapes: 64 buffer
(class) tokens prepended to 256 KL-16 image tokens of latent dimension 16, 1000
classes, 64-step decoding. Weights are N(0, 0.02); LayerNorm gains are
1 + N(0, 0.1) and shifts N(0, 0.02) so that a swapped gain/shift is visible.

Generators (numpy PCG64, fixed seeds):
  weights            seed 0 (+ config-independent stream order, see make_weights)
  class labels       seed 1, uniform over [0, n_classes)
  decode order       seed 2, one permutation of the image positions per
                     cond/uncond pair
  token latents      seed 3, one N(0, 1) latent per (pair, image position),
                     revealed once that position is decoded

bf16 configurations store weights as bf16: `round_bf16` maps fp32 values to
the nearest bf16 value (ties to even) and keeps them in fp32 containers, so
both sides read identical numbers.
"""
import math

import numpy as np

# Model/workload shapes. `batch` counts cond/uncond pairs (B); the forward runs
# rows = 2B (both pathways) or B (condition-cache reuse step).
CONFIGS = {
    # 2 blocks, width 256, 4 heads, 16 buffer + 64 image tokens, one pair, fp32.
    "tiny": dict(depth=2, width=256, heads=4, mlp_ratio=4, n_buffer=16, n_img=64,
                 token_dim=16, n_classes=1000, batch=1, sel_layers=1, dtype="fp32",
                 steps=64, k0=4, tau=9, tau_cfg=9, ratio=0.25),
    # 12 encoder + 12 decoder blocks, width 768, 12 heads, B = 32.
    "mar_b": dict(depth=24, width=768, heads=12, mlp_ratio=4, n_buffer=64, n_img=256,
                  token_dim=16, n_classes=1000, batch=32, sel_layers=3, dtype="bf16",
                  steps=64, k0=4, tau=9, tau_cfg=2, ratio=50 / 320),
    # 16 + 16 blocks, width 1024, 16 heads, B = 64.
    "mar_l": dict(depth=32, width=1024, heads=16, mlp_ratio=4, n_buffer=64, n_img=256,
                  token_dim=16, n_classes=1000, batch=64, sel_layers=3, dtype="bf16",
                  steps=64, k0=4, tau=9, tau_cfg=9, ratio=50 / 320),
    # 20 + 20 blocks, width 1280, 16 heads (head dim 80), B = 128.
    "mar_h": dict(depth=40, width=1280, heads=16, mlp_ratio=4, n_buffer=64, n_img=256,
                  token_dim=16, n_classes=1000, batch=128, sel_layers=3, dtype="bf16",
                  steps=64, k0=4, tau=9, tau_cfg=9, ratio=50 / 320),
    # MAR-L shapes at 32x32 latents: 64 + 1024 tokens, B = 16, 25 % recompute.
    "hires": dict(depth=32, width=1024, heads=16, mlp_ratio=4, n_buffer=64, n_img=1024,
                  token_dim=16, n_classes=1000, batch=16, sel_layers=3, dtype="bf16",
                  steps=64, k0=4, tau=9, tau_cfg=0, ratio=0.25),
}


def config(name, **overrides):
    """Return a copy of a named configuration with derived fields filled in."""
    c = dict(CONFIGS[name])
    c.update(overrides)
    c["name"] = name
    c["T"] = c["n_buffer"] + c["n_img"]
    c["head_dim"] = c["width"] // c["heads"]
    c["ln_eps"] = 1e-6
    c.setdefault("criterion", "value")
    return c


def n_compute(cfg, ratio=None):
    """Tokens recomputed per row: round-half-up(ratio * T)."""
    r = cfg["ratio"] if ratio is None else ratio
    return int(math.floor(r * cfg["T"] + 0.5))


def round_bf16(x):
    """Nearest bf16 value (ties to even) of each fp32 element, as fp32."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    u = (u + (((u >> 16) & 1) + 0x7FFF)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32)


def _normal(rng, shape, std):
    return (rng.standard_normal(shape, dtype=np.float32) * np.float32(std)).astype(np.float32)


def make_weights(cfg, seed=0):
    """Random-init weights of the MAR-shaped transformer (nn.Linear layout [out, in]).

    Returns a dict of fp32 arrays; for bf16 configurations every value is
    already bf16-representable.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    D, T, H4 = cfg["width"], cfg["T"], cfg["width"] * cfg["mlp_ratio"]
    w = {
        "pos_emb": _normal(rng, (T, D), 0.02),
        "class_emb": _normal(rng, (cfg["n_classes"], D), 0.02),
        "mask_emb": _normal(rng, (D,), 0.02),
        "embed_w": _normal(rng, (D, cfg["token_dim"]), 0.02),
        "embed_b": _normal(rng, (D,), 0.02),
        "lnf_g": (1.0 + _normal(rng, (D,), 0.1)).astype(np.float32),
        "lnf_b": _normal(rng, (D,), 0.02),
        "blocks": [],
    }
    for _ in range(cfg["depth"]):
        w["blocks"].append({
            "ln1_g": (1.0 + _normal(rng, (D,), 0.1)).astype(np.float32),
            "ln1_b": _normal(rng, (D,), 0.02),
            "w_qkv": _normal(rng, (3 * D, D), 0.02),
            "b_qkv": _normal(rng, (3 * D,), 0.02),
            "w_o": _normal(rng, (D, D), 0.02),
            "b_o": _normal(rng, (D,), 0.02),
            "ln2_g": (1.0 + _normal(rng, (D,), 0.1)).astype(np.float32),
            "ln2_b": _normal(rng, (D,), 0.02),
            "w1": _normal(rng, (H4, D), 0.02),
            "b1": _normal(rng, (H4,), 0.02),
            "w2": _normal(rng, (D, H4), 0.02),
            "b2": _normal(rng, (D,), 0.02),
        })
    if cfg["dtype"] == "bf16":
        for k in list(w):
            if k != "blocks":
                w[k] = round_bf16(w[k])
        for b in w["blocks"]:
            for k in b:
                b[k] = round_bf16(b[k])
    return w


def make_labels(cfg, seed=1):
    rng = np.random.Generator(np.random.PCG64(seed))
    return rng.integers(0, cfg["n_classes"], size=cfg["batch"], dtype=np.int64).astype(np.int32)


def make_order(cfg, seed=2):
    """Decode order: one permutation of image positions per pair, [B, n_img]."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return np.stack([rng.permutation(cfg["n_img"]) for _ in range(cfg["batch"])]).astype(np.int32)


def make_latent_table(cfg, seed=3):
    """Latent revealed for each (pair, image position) once decoded, [B, n_img, token_dim]."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return rng.standard_normal((cfg["batch"], cfg["n_img"], cfg["token_dim"]), dtype=np.float32)


def mask_counts(steps, n_img):
    """Masked image tokens left after each decoding step (cosine schedule, as in MAR/MaskGIT).

    m[k] = floor(n_img * cos(pi/2 * (k+1)/steps)), clamped so that every step
    decodes at least one token and the last step decodes the rest (m[-1] = 0).
    This is workload structure for the synthetic driver, not part of LazyMAR.
    """
    m, prev = [], n_img
    for k in range(steps):
        if k == steps - 1:
            cur = 0
        else:
            cur = int(math.floor(n_img * math.cos(math.pi / 2 * (k + 1) / steps)))
            cur = max(1, min(cur, prev - 1))
        m.append(cur)
        prev = cur
    return m


def step_state(cfg, order, table, n_decoded):
    """Inputs of one forward: latents [B, n_img, token_dim] fp32, mask [B, n_img] u8 (1 = masked).

    The first `n_decoded` positions of each pair's order are decoded and carry
    their latent; the rest are masked (their latent entries are zero).
    """
    B, n = order.shape
    mask = np.ones((B, n), dtype=np.uint8)
    for b in range(B):
        mask[b, order[b, :n_decoded]] = 0
    lat = np.where(mask[:, :, None] == 0, table, 0.0).astype(np.float32)
    return lat, mask


def tiny_state(cfg, order, table, before=24, after=32):
    """The tiny workload: a forward with 24 decoded tokens, then one with 8 more."""
    return step_state(cfg, order, table, before), step_state(cfg, order, table, after)


def tensor(shape, seed, std=1.0, dtype="fp32", mean=0.0):
    """Seeded N(mean, std^2) fp32 tensor; bf16-representable when dtype == 'bf16'."""
    rng = np.random.Generator(np.random.PCG64(seed))
    x = (rng.standard_normal(shape, dtype=np.float32) * np.float32(std) + np.float32(mean)).astype(np.float32)
    return round_bf16(x) if dtype == "bf16" else x


def similarity_inputs(rows, T, D, seed, dtype="fp32", changed=0.1):
    """Current / cached representations for the selection test.

    Most tokens move a little between steps, a `changed` fraction moves a lot
    (the tokens decoded at the last step); token 1 duplicates token 0 (an exact
    tie), token 2 is the zero vector when T > 2.
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    ref = rng.standard_normal((rows, T, D), dtype=np.float32)
    cur = ref + np.float32(0.05) * rng.standard_normal((rows, T, D), dtype=np.float32)
    big = rng.random((rows, T)) < changed
    cur[big] = rng.standard_normal((int(big.sum()), D), dtype=np.float32)
    if T > 1:
        cur[:, 1], ref[:, 1] = cur[:, 0], ref[:, 0]
    if T > 2:
        cur[:, 2] = 0.0
    if dtype == "bf16":
        cur, ref = round_bf16(cur), round_bf16(ref)
    return cur.astype(np.float32), ref.astype(np.float32)


def distinct_rows(n, total, seed):
    """n distinct row indices out of `total`, in random order (a scatter map)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return rng.permutation(total)[:n].astype(np.int32)


# ----------------------------------------------------------------------------
# Diffusion head (the per-token denoiser that draws each decoded token's latent)
# ----------------------------------------------------------------------------
# Width and depth follow the MAR head sizes that go with the transformer
# configurations; n_steps sampling steps over n_train training steps.
HEAD_CONFIGS = {
    "tiny": dict(width=128, depth=2, freq_dim=256, n_train=1000, n_steps=10),
    "mar_b": dict(width=1024, depth=6, freq_dim=256, n_train=1000, n_steps=100),
    "mar_l": dict(width=1280, depth=8, freq_dim=256, n_train=1000, n_steps=100),
    "mar_h": dict(width=1536, depth=12, freq_dim=256, n_train=1000, n_steps=100),
}


def head_config(name, **overrides):
    c = dict(HEAD_CONFIGS[name])
    c.update(overrides)
    c["name"] = name
    return c


def make_head_weights(hc, cond_dim, token_dim, seed=4, bf16=True):
    """Random-init head weights ([out, in] layout), N(0, 0.02) throughout."""
    rng = np.random.Generator(np.random.PCG64(seed))
    w, f = hc["width"], hc["freq_dim"]
    W = {
        "t_w1": _normal(rng, (w, f), 0.02), "t_b1": _normal(rng, (w,), 0.02),
        "t_w2": _normal(rng, (w, w), 0.02), "t_b2": _normal(rng, (w,), 0.02),
        "c_w": _normal(rng, (w, cond_dim), 0.02), "c_b": _normal(rng, (w,), 0.02),
        "in_w": _normal(rng, (w, token_dim), 0.02), "in_b": _normal(rng, (w,), 0.02),
        "blocks": [],
    }
    for _ in range(hc["depth"]):
        W["blocks"].append({
            "ada_w": _normal(rng, (3 * w, w), 0.02), "ada_b": _normal(rng, (3 * w,), 0.02),
            "w1": _normal(rng, (w, w), 0.02), "b1": _normal(rng, (w,), 0.02),
            "w2": _normal(rng, (w, w), 0.02), "b2": _normal(rng, (w,), 0.02),
        })
    W["f_ada_w"] = _normal(rng, (2 * w, w), 0.02)
    W["f_ada_b"] = _normal(rng, (2 * w,), 0.02)
    W["out_w"] = _normal(rng, (2 * token_dim, w), 0.02)
    W["out_b"] = _normal(rng, (2 * token_dim,), 0.02)
    if bf16:
        for k in list(W):
            if k != "blocks":
                W[k] = round_bf16(W[k])
        for b in W["blocks"]:
            for k in b:
                b[k] = round_bf16(b[k])
    return W


def make_head_noise(n_steps, M, token_dim, seed=5):
    """noise[0] = starting latents, noise[i] = noise added after denoising step i."""
    rng = np.random.Generator(np.random.PCG64(seed))
    return rng.standard_normal((n_steps, M, token_dim), dtype=np.float32)
