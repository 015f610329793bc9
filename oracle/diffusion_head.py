"""Plain fp64 CPU oracle of the per-token diffusion head and its sampler.

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's CPU
baseline leg import this module; the product path (the CUDA library and its
binding) never does, and this module imports nothing from it.

The paper's transformer produces one feature vector z per image token; the
token's continuous latent is then drawn by a small denoising network run for
100 diffusion steps, following "the standard setting" of the diffusion papers
it cites (Sec. 4.1, implementation details; 16-dim KL-16 latents). The paper
gives no further detail, so every piece below is a reading, listed here and in
the design notes:

- Denoiser: the MAR head, a residual MLP of `depth` blocks of width `width`
  whose LayerNorms (no gain or shift of their own) are modulated by the
  condition y = t_emb(t) + W_c z + b_c (adaptive LayerNorm: shift, scale and a
  residual gate per block, from a linear map of SiLU(y)); a final modulated
  LayerNorm and a linear map to 2 * token_dim outputs, the noise prediction
  eps and the variance interpolation v.
- Timestep embedding: 256 sinusoids [cos(t f_i), sin(t f_i)],
  f_i = 10000^(-i/128), then Linear, SiLU, Linear.
- Noise schedule: the cosine schedule, alpha_bar(t) = f(t) / f(0) with
  f(t) = cos^2(((t / T) + s) / (1 + s) * pi / 2), s = 0.008, over T = 1000
  training steps, beta_t = min(1 - alpha_bar(t+1)/alpha_bar(t), 0.999).
- 100 sampling steps: the training steps round(i (T - 1) / (n - 1)),
  i = 0..n-1, with the betas recomputed so that the cumulative products at the
  kept steps are unchanged; the network is called with the kept training-step
  index.
- Sampler: ancestral sampling. From x and the predicted noise eps,
  x0 = x / sqrt(alpha_bar) - sqrt(1 / alpha_bar - 1) eps, the mean is the
  Gaussian posterior mean of x_{t-1} given (x_t, x0), the log variance is
  interpolated between log beta_t and the (clipped) log posterior variance
  by frac = (v + 1) / 2, and noise times a temperature is added on every step
  but the last.
- Guidance: the network runs on (x, z_cond) and (x, z_uncond) with the same x;
  eps = eps_u + gamma (eps_c - eps_u); v comes from the conditional run.

Random numbers are inputs: noise[0] is x at the first (noisiest) step and
noise[i] (i >= 1) the noise added after the i-th denoising step.

Parity status: pinned by tests/test_head_oracle.py against closed forms (a
denoiser that knows x0 returns x0; the sampling mean equals the Gaussian
posterior mean derived from the two Gaussians; the variance interpolation hits
its end points), invariants (the respaced cumulative products equal the kept
ones; gates of zero make every block the identity; guidance of 1 or equal
conditions reduce to a single run) and brute force.
"""
import math

import numpy as np

F64 = np.float64


def silu(x):
    """x * sigmoid(x)."""
    x = np.asarray(x, F64)
    return x / (1.0 + np.exp(-x))


def linear(x, w, b):
    """y = x W^T + b with W in [out, in] layout."""
    return np.asarray(x, F64) @ np.asarray(w, F64).T + np.asarray(b, F64)


def layer_norm_plain(x, eps=1e-6):
    """LayerNorm without gain or shift: (x - mean) / sqrt(var + eps), biased variance."""
    x = np.asarray(x, F64)
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps)


def modulate(x, shift, scale):
    """Adaptive LayerNorm modulation x (1 + scale) + shift."""
    return x * (1.0 + scale) + shift


# ----------------------------------------------------------------------------
# Noise schedule
# ----------------------------------------------------------------------------


def cosine_alpha_bar(t, n_train, s=0.008):
    """alpha_bar at training step t (of n_train): f(t) / f(0)."""
    f = lambda u: math.cos((u / n_train + s) / (1.0 + s) * math.pi / 2.0) ** 2
    return f(t) / f(0)


def train_betas(n_train, max_beta=0.999):
    """beta_i = min(1 - alpha_bar(i + 1) / alpha_bar(i), max_beta), i = 0..n_train-1."""
    return np.array([min(1.0 - cosine_alpha_bar(i + 1, n_train) / cosine_alpha_bar(i, n_train), max_beta)
                     for i in range(n_train)], F64)


def kept_steps(n_train, n_steps):
    """Training steps used for sampling: round(i (n_train - 1) / (n_steps - 1))."""
    if n_steps == 1:
        return np.array([0])
    stride = (n_train - 1) / (n_steps - 1)
    return np.array([int(round(i * stride)) for i in range(n_steps)])


class Schedule:
    """Sampling schedule over the kept steps j = 0..n_steps-1 (j = 0 last)."""

    def __init__(self, n_train=1000, n_steps=100):
        ab_train = np.cumprod(1.0 - train_betas(n_train))
        self.t = kept_steps(n_train, n_steps)
        ab = ab_train[self.t]
        prev = np.concatenate([[1.0], ab[:-1]])
        self.beta = 1.0 - ab / prev                      # respaced betas
        self.alpha_bar = ab
        self.alpha_bar_prev = prev
        self.post_var = self.beta * (1.0 - prev) / (1.0 - ab)
        # the posterior variance is 0 at j = 0: its log is clipped to j = 1's
        pv = self.post_var.copy()
        if len(pv) > 1:
            pv[0] = pv[1]
        # with a single kept step the posterior variance is 0 (log -inf); that
        # step is the last one and adds no noise, so the value is never used
        with np.errstate(divide="ignore"):
            self.post_log_var = np.log(pv)
        self.coef_x0 = self.beta * np.sqrt(prev) / (1.0 - ab)
        self.coef_xt = (1.0 - prev) * np.sqrt(1.0 - self.beta) / (1.0 - ab)

    def __len__(self):
        return len(self.t)


# ----------------------------------------------------------------------------
# Denoiser
# ----------------------------------------------------------------------------


def timestep_embedding(t, dim=256, max_period=10000.0):
    """[cos(t f_0..f_{h-1}), sin(t f_0..f_{h-1})], f_i = max_period^(-i/h), h = dim / 2."""
    t = np.asarray(t, F64).reshape(-1)
    half = dim // 2
    f = np.exp(-math.log(max_period) * np.arange(half, dtype=F64) / half)
    a = t[:, None] * f[None, :]
    return np.concatenate([np.cos(a), np.sin(a)], axis=1)


def time_embed(W, t):
    """Linear, SiLU, Linear of the sinusoidal embedding of training step t."""
    e = timestep_embedding(t, W["t_w1"].shape[1])
    return linear(silu(linear(e, W["t_w1"], W["t_b1"])), W["t_w2"], W["t_b2"])


def denoiser(W, x, t, z, eps=1e-6):
    """Network output [R, 2 token_dim] for latents x [R, token_dim] at training
    step t (scalar) under conditions z [R, cond_dim]."""
    y = time_embed(W, [t]) + linear(z, W["c_w"], W["c_b"])          # [R, w]
    sy = silu(y)
    h = linear(x, W["in_w"], W["in_b"])
    for blk in W["blocks"]:
        shift, scale, gate = np.split(linear(sy, blk["ada_w"], blk["ada_b"]), 3, axis=1)
        a = modulate(layer_norm_plain(h, eps), shift, scale)
        a = linear(silu(linear(a, blk["w1"], blk["b1"])), blk["w2"], blk["b2"])
        h = h + gate * a
    shift, scale = np.split(linear(sy, W["f_ada_w"], W["f_ada_b"]), 2, axis=1)
    return linear(modulate(layer_norm_plain(h, eps), shift, scale), W["out_w"], W["out_b"])


def guided_output(W, x, t, z_cond, z_uncond, gamma):
    """eps = eps_u + gamma (eps_c - eps_u) and v of the conditional run."""
    td = x.shape[1]
    oc = denoiser(W, x, t, z_cond)
    ou = denoiser(W, x, t, z_uncond)
    eps = ou[:, :td] + gamma * (oc[:, :td] - ou[:, :td])
    return eps, oc[:, td:]


# ----------------------------------------------------------------------------
# Sampler
# ----------------------------------------------------------------------------


def sample_step(sched, j, x, eps, v, noise, temperature):
    """x_{t-1} from x_t at kept step j (Gaussian posterior of x_{t-1} given x_t
    and the predicted x0; learned-range variance; no noise at j = 0)."""
    ab = sched.alpha_bar[j]
    x0 = x / math.sqrt(ab) - math.sqrt(1.0 / ab - 1.0) * eps
    mean = sched.coef_x0[j] * x0 + sched.coef_xt[j] * x
    if j == 0:
        return mean
    frac = (v + 1.0) / 2.0
    log_var = frac * math.log(sched.beta[j]) + (1.0 - frac) * sched.post_log_var[j]
    return mean + np.exp(0.5 * log_var) * temperature * noise


def sample(W, sched, z_cond, z_uncond, noise, gamma, temperature=1.0):
    """Latents [M, token_dim] of M tokens: noise [n_steps, M, token_dim]."""
    noise = np.asarray(noise, F64)
    x = noise[0].copy()
    n = len(sched)
    for i in range(n):
        j = n - 1 - i
        eps, v = guided_output(W, x, float(sched.t[j]), z_cond, z_uncond, gamma)
        x = sample_step(sched, j, x, eps, v, noise[i + 1] if j > 0 else None, temperature)
    return x
