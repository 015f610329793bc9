"""Pins of the diffusion-head oracle (oracle/diffusion_head.py) against closed
forms, invariants and hand-worked values; no GPU."""
import math

import numpy as np
import pytest

from oracle import diffusion_head as H
from synth import inputs as S

TD = 16


def tiny_weights(depth=2, width=128, cond=64, seed=7):
    return S.make_head_weights(dict(width=width, depth=depth, freq_dim=256), cond, TD, seed=seed, bf16=False)


# ----------------------------------------------------------------------------
# schedule
# ----------------------------------------------------------------------------

def test_train_betas_telescope_to_the_cosine_alpha_bar():
    """prod_{i < t} (1 - beta_i) = alpha_bar(t) / alpha_bar(0) wherever no beta is
    clipped: the index convention of the betas (beta_i links steps i and i+1)."""
    n = 1000
    b = H.train_betas(n)
    ab = np.cumprod(1.0 - b)
    f = lambda u: math.cos((u / n + 0.008) / 1.008 * math.pi / 2) ** 2
    for t in (1, 10, 500, 900, 990):
        assert ab[t - 1] == pytest.approx(f(t) / f(0), rel=1e-12)
    assert b[-1] == 0.999                       # alpha_bar(1000) = 0: clipped
    assert np.all(b[:-1] < 0.999) and np.all(np.diff(b) > 0)


def test_kept_steps_hand_worked():
    assert H.kept_steps(1000, 10).tolist() == [0, 111, 222, 333, 444, 555, 666, 777, 888, 999]
    k = H.kept_steps(1000, 100)
    # stride 999 / 99 = 10.0909...: 5 * stride = 50.45 -> 50, 6 * stride = 60.55 -> 61
    assert k[:8].tolist() == [0, 10, 20, 30, 40, 50, 61, 71]
    assert len(k) == 100 and k[-1] == 999 and np.all(np.diff(k) > 0)


def test_respaced_products_equal_the_kept_alpha_bars():
    s = H.Schedule(1000, 100)
    ab_train = np.cumprod(1.0 - H.train_betas(1000))
    np.testing.assert_allclose(np.cumprod(1.0 - s.beta), ab_train[s.t], rtol=1e-10)
    assert np.all((s.beta > 0) & (s.beta < 1))


def test_posterior_mean_and_variance_from_the_two_gaussians():
    """q(x_{t-1} | x_t, x0) from N(x_{t-1}; sqrt(ab_prev) x0, 1 - ab_prev) times
    N(x_t; sqrt(1 - beta) x_{t-1}, beta): precision-weighted mean and variance."""
    s = H.Schedule(1000, 100)
    rng = np.random.default_rng(0)
    for j in (1, 2, 37, 98, 99):
        x0, xt = rng.standard_normal(5), rng.standard_normal(5)
        a, b, abp = 1.0 - s.beta[j], s.beta[j], s.alpha_bar_prev[j]
        prec = 1.0 / (1.0 - abp) + a / b
        mean = (math.sqrt(abp) * x0 / (1.0 - abp) + math.sqrt(a) * xt / b) / prec
        np.testing.assert_allclose(s.coef_x0[j] * x0 + s.coef_xt[j] * xt, mean, rtol=1e-10, atol=1e-12)
        assert s.post_var[j] == pytest.approx(1.0 / prec, rel=1e-10)
    assert s.post_log_var[0] == pytest.approx(math.log(s.post_var[1]))   # clipped at the last step


def test_a_denoiser_that_knows_x0_returns_x0():
    """With eps = (x_t - sqrt(ab) x0) / sqrt(1 - ab) and no noise every step's mean
    keeps x0, and the last step returns it."""
    s = H.Schedule(1000, 100)
    rng = np.random.default_rng(1)
    x0 = rng.standard_normal((3, TD))
    x = rng.standard_normal((3, TD))
    for j in range(len(s) - 1, -1, -1):
        ab = s.alpha_bar[j]
        eps = (x - math.sqrt(ab) * x0) / math.sqrt(1.0 - ab)
        x = H.sample_step(s, j, x, eps, np.zeros_like(x), np.zeros_like(x), 1.0)
    np.testing.assert_allclose(x, x0, rtol=1e-7, atol=1e-9)


def test_variance_interpolation_end_points():
    """v = 1 gives variance beta, v = -1 the clipped posterior variance."""
    s = H.Schedule(1000, 100)
    x = np.zeros((1, TD))
    eps = np.zeros((1, TD))
    n = np.ones((1, TD))
    for j in (1, 50, 99):
        for v, var in ((1.0, s.beta[j]), (-1.0, math.exp(s.post_log_var[j]))):
            vv = np.full((1, TD), v)
            up = H.sample_step(s, j, x, eps, vv, n, 1.0)
            dn = H.sample_step(s, j, x, eps, vv, -n, 1.0)
            np.testing.assert_allclose((up - dn) / 2, math.sqrt(var), rtol=1e-12)
            half = H.sample_step(s, j, x, eps, vv, n, 0.5)
            np.testing.assert_allclose((half - dn) / 2, 0.75 * math.sqrt(var), rtol=1e-12)


def test_sampler_loop_with_a_constant_denoiser():
    """All weights zero but the output bias: eps and v are constants and the loop
    is the recurrence x <- (x - beta / sqrt(1 - ab) eps) / sqrt(1 - beta)
    + sqrt(beta) temperature noise (v = 1), from noise[0], steps j = n-1..0."""
    W = tiny_weights()
    Z = {k: np.zeros_like(v) for k, v in W.items() if k != "blocks"}
    Z["blocks"] = [{k: np.zeros_like(v) for k, v in b.items()} for b in W["blocks"]]
    eps_c = np.linspace(-1, 1, TD)
    Z["out_b"] = np.concatenate([eps_c, np.ones(TD)])
    s = H.Schedule(1000, 10)
    rng = np.random.default_rng(2)
    noise = rng.standard_normal((10, 4, TD))
    z = rng.standard_normal((2, 4, 64))
    got = H.sample(Z, s, z[0], z[1], noise, gamma=3.0, temperature=0.7)
    x = noise[0].copy()
    for i, j in enumerate(range(9, -1, -1)):
        b, ab = s.beta[j], s.alpha_bar[j]
        x = (x - b / math.sqrt(1.0 - ab) * eps_c) / math.sqrt(1.0 - b)
        if j > 0:
            x = x + math.sqrt(b) * 0.7 * noise[i + 1]
    np.testing.assert_allclose(got, x, rtol=1e-9, atol=1e-12)


# ----------------------------------------------------------------------------
# denoiser
# ----------------------------------------------------------------------------

def test_silu_identities():
    x = np.linspace(-30, 30, 121)
    np.testing.assert_allclose(H.silu(x) - H.silu(-x), x, rtol=1e-12, atol=1e-12)
    assert H.silu(0.0) == 0.0 and H.silu(1.0) == pytest.approx(1.0 / (1.0 + math.exp(-1.0)))


def test_timestep_embedding_values():
    e = H.timestep_embedding([0.0, 1.0, 999.0], 256)
    assert np.all(e[0, :128] == 1.0) and np.all(e[0, 128:] == 0.0)
    assert e[1, 0] == pytest.approx(math.cos(1.0)) and e[1, 128] == pytest.approx(math.sin(1.0))
    f_last = 10000.0 ** (-127 / 128)
    assert e[2, 127] == pytest.approx(math.cos(999.0 * f_last)) and e[2, 255] == pytest.approx(math.sin(999.0 * f_last))
    # cos a cos b + sin a sin b = cos(a - b) for every frequency pair
    np.testing.assert_allclose(e[1, :128] * e[2, :128] + e[1, 128:] * e[2, 128:],
                               np.cos((1.0 - 999.0) * 10000.0 ** (-np.arange(128) / 128)), atol=1e-12)


def test_plain_layer_norm_and_modulation():
    x = np.random.default_rng(3).standard_normal((5, 96)) * 3 + 2
    y = H.layer_norm_plain(x, 0.0)
    np.testing.assert_allclose(y.mean(-1), 0, atol=1e-12)
    np.testing.assert_allclose((y ** 2).mean(-1), 1, rtol=1e-12)
    np.testing.assert_allclose(H.modulate(y, 0.0, 0.0), y)
    np.testing.assert_allclose(H.modulate(y, 1.5, -1.0), 1.5)


def test_zero_gates_make_every_block_the_identity():
    """Gate rows of zero: the blocks' MLPs drop out, so their weights do not matter
    and the output equals that of a network without blocks; a non-zero gate
    changes it."""
    W = tiny_weights()
    w = W["in_w"].shape[0]
    for b in W["blocks"]:
        b["ada_w"][2 * w:] = 0
        b["ada_b"][2 * w:] = 0
    rng = np.random.default_rng(4)
    x, z = rng.standard_normal((3, TD)), rng.standard_normal((3, 64))
    ref = H.denoiser(W, x, 250.0, z)
    W2 = dict(W, blocks=[dict(b, w1=b["w1"] * 3 + 0.1, b2=b["b2"] - 1) for b in W["blocks"]])
    np.testing.assert_allclose(H.denoiser(W2, x, 250.0, z), ref, rtol=1e-12)
    np.testing.assert_allclose(H.denoiser(dict(W, blocks=[]), x, 250.0, z), ref, rtol=1e-12)
    W3 = dict(W, blocks=[dict(b, ada_b=b["ada_b"] + 0.5) for b in W["blocks"]])
    assert np.abs(H.denoiser(W3, x, 250.0, z) - ref).max() > 1e-3


def test_block_residual_and_gate_order():
    """One block with shift = scale = 0 and gate = 1 (ada weights zero, gate bias
    one) adds MLP(LN(h)) to h: checked against a network whose input projection
    already holds h + MLP(LN(h)) and has no blocks."""
    W = tiny_weights(depth=1)
    w = W["in_w"].shape[0]
    b = W["blocks"][0]
    b["ada_w"][:] = 0
    b["ada_b"][:] = 0
    b["ada_b"][2 * w:] = 1.0
    rng = np.random.default_rng(5)
    x = rng.standard_normal((2, TD))
    z = rng.standard_normal((2, 64))
    h = H.linear(x, W["in_w"], W["in_b"])
    mlp = H.linear(H.silu(H.linear(H.layer_norm_plain(h), b["w1"], b["b1"])), b["w2"], b["b2"])
    # a network without blocks whose input projection lands on h + mlp: append
    # the residual as extra input columns of an identity map
    Wn = dict(W, blocks=[], in_w=np.concatenate([W["in_w"], np.eye(w)], axis=1))
    xn = np.concatenate([x, mlp], axis=1)
    np.testing.assert_allclose(H.denoiser(W, x, 10.0, z), H.denoiser(Wn, xn, 10.0, z), rtol=1e-10, atol=1e-12)


def test_guidance_reductions():
    W = tiny_weights()
    rng = np.random.default_rng(6)
    x = rng.standard_normal((3, TD))
    zc, zu = rng.standard_normal((2, 3, 64))
    oc = H.denoiser(W, x, 500.0, zc)
    e1, v1 = H.guided_output(W, x, 500.0, zc, zu, 1.0)
    np.testing.assert_allclose(e1, oc[:, :TD], rtol=1e-12)
    np.testing.assert_allclose(v1, oc[:, TD:], rtol=1e-12)
    e3, _ = H.guided_output(W, x, 500.0, zc, zc, 3.0)
    np.testing.assert_allclose(e3, oc[:, :TD], rtol=1e-12)
    eu = H.denoiser(W, x, 500.0, zu)[:, :TD]
    e0, _ = H.guided_output(W, x, 500.0, zc, zu, 0.0)
    np.testing.assert_allclose(e0, eu, rtol=1e-12)


def test_condition_and_timestep_enter_through_y():
    """The denoiser depends on t and z only through y = t_emb(t) + W_c z + b_c:
    moving the conditioning bias into the time embedding's last bias changes
    nothing."""
    W = tiny_weights()
    rng = np.random.default_rng(8)
    x, z = rng.standard_normal((2, TD)), rng.standard_normal((2, 64))
    ref = H.denoiser(W, x, 321.0, z)
    W2 = dict(W, t_b2=W["t_b2"].astype(np.float64) + W["c_b"], c_b=np.zeros_like(W["c_b"]))
    np.testing.assert_allclose(H.denoiser(W2, x, 321.0, z), ref, rtol=1e-10)
    assert np.abs(H.denoiser(W, x, 322.0, z) - ref).max() > 1e-6


def test_final_layer_shift_then_scale():
    """Final modulation with zero ada weights, shift s0 and scale -1: LN(h) drops
    out and the output is W_out s0 + b_out for every input."""
    W = tiny_weights()
    w = W["in_w"].shape[0]
    s0 = np.linspace(-0.5, 0.5, w)
    W["f_ada_w"] = np.zeros_like(W["f_ada_w"])
    W["f_ada_b"] = np.concatenate([s0, -np.ones(w)])
    rng = np.random.default_rng(9)
    x, z = rng.standard_normal((3, TD)), rng.standard_normal((3, 64))
    want = np.asarray(W["out_w"], np.float64) @ s0 + W["out_b"]
    np.testing.assert_allclose(H.denoiser(W, x, 77.0, z), np.tile(want, (3, 1)), rtol=1e-10, atol=1e-12)


def test_time_embedding_mlp_applies_silu_between_its_linears():
    """With identity linears the time embedding is SiLU of the sinusoids: at t = 0,
    SiLU(1) on the cosine half and SiLU(0) = 0 on the sine half."""
    W = tiny_weights(width=256)
    W["t_w1"], W["t_b1"] = np.eye(256), np.zeros(256)
    W["t_w2"], W["t_b2"] = np.eye(256), np.zeros(256)
    e = H.time_embed(W, [0.0])[0]
    np.testing.assert_allclose(e[:128], 1.0 / (1.0 + math.exp(-1.0)), rtol=1e-12)
    np.testing.assert_allclose(e[128:], 0.0, atol=1e-15)
