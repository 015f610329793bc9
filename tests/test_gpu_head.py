"""GPU parity of the diffusion head (per-token denoiser and its guided sampler)
against the fp64 oracle (oracle/diffusion_head.py), through the C ABI."""
import numpy as np
import pytest

from oracle import diffusion_head as HO
from paper_2503_12450_gb300 import lazymar as lm
import synth
from synth import inputs as S
from _gpu import COS_MIN, TOL, dev, dev_int, empty, host, max_rel, min_cos, torch_cuda

pytestmark = pytest.mark.gpu
TD = 16


def z_rows(z, B, n_img, pos):
    """Oracle view of the rows the head gathers: cond rows of pair b at pos[b],
    then the uncond rows."""
    n_new = pos.shape[1]
    zc = np.concatenate([z[b, pos[b]] for b in range(B)])
    zu = np.concatenate([z[B + b, pos[b]] for b in range(B)])
    return zc.reshape(B * n_new, -1), zu.reshape(B * n_new, -1)


def setup(name, cond_dim, B, n_img, n_new, seed, z_dtype="bf16", steps=None):
    torch_cuda()
    hc = S.head_config(name, **({} if steps is None else {"n_steps": steps}))
    W = S.make_head_weights(hc, cond_dim, TD, seed=seed)
    rng = np.random.default_rng(seed)
    z = rng.standard_normal((2 * B, n_img, cond_dim)).astype(np.float32)
    if z_dtype == "bf16":
        z = S.round_bf16(z)
    pos = np.stack([rng.choice(n_img, n_new, replace=False) for _ in range(B)]).astype(np.int32)
    h = lm.lazymar_head_create(hc, cond_dim, TD, W, max_tokens=B * n_new, z_dtype=z_dtype)
    return hc, W, z, pos, h


@pytest.mark.parametrize("name,cond_dim,B,n_img,n_new,z_dtype", [
    ("mar_b", 768, 3, 256, 50, "bf16"),     # 300 rows: three row tiles, ragged
    ("mar_b", 768, 1, 256, 1, "bf16"),      # a single token
    ("tiny", 256, 2, 64, 5, "fp32"),        # fp32 features, width 128
    ("mar_h", 1280, 2, 256, 7, "bf16"),     # width 1536, 12 blocks
])
def test_network_output_matches_oracle(name, cond_dim, B, n_img, n_new, z_dtype):
    hc, W, z, pos, h = setup(name, cond_dim, B, n_img, n_new, seed=11, z_dtype=z_dtype)
    M = B * n_new
    x = np.random.default_rng(12).standard_normal((M, TD)).astype(np.float32)
    zc, zu = z_rows(z, B, n_img, pos)
    sched = HO.Schedule(hc["n_train"], hc["n_steps"])
    for j in (hc["n_steps"] - 1, hc["n_steps"] // 2, 0):
        out = empty((2 * M, 2 * TD))
        lm.lazymar_head_eval(h, dev(z, z_dtype), B, n_img, pos, n_new, x, j, out)
        lm.lazymar_head_sync(h)
        t = float(sched.t[j])
        want = np.concatenate([HO.denoiser(W, x, t, zc), HO.denoiser(W, x, t, zu)])
        got = host(out)
        assert max_rel(got, want) < TOL["bf16"], (j, max_rel(got, want))
        assert min_cos(got, want) >= COS_MIN
    h.close()


@pytest.mark.parametrize("name,cond_dim,B,n_new,gamma,temp", [
    ("mar_b", 768, 2, 4, 3.0, 1.0),
    ("tiny", 256, 3, 3, 1.5, 0.5),
])
def test_sampler_matches_oracle(name, cond_dim, B, n_new, gamma, temp):
    n_img = 256
    hc, W, z, pos, h = setup(name, cond_dim, B, n_img, n_new, seed=21)
    M = B * n_new
    noise = S.make_head_noise(hc["n_steps"], M, TD, seed=22)
    zc, zu = z_rows(z, B, n_img, pos)
    want = HO.sample(W, HO.Schedule(hc["n_train"], hc["n_steps"]), zc, zu, noise, gamma, temp)
    x = empty((M, TD))
    lm.lazymar_head_sample(h, dev(z, "bf16"), B, n_img, pos, n_new, noise, gamma, temp, x)
    lm.lazymar_head_sync(h)
    got = host(x)
    assert max_rel(got, want) < TOL["bf16"], max_rel(got, want)
    assert min_cos(got, want) >= COS_MIN
    h.close()


def test_sampler_graph_replay_and_host_buffers():
    """Eager first call, captured second, replayed third: identical bits, on
    device or host buffers; a changed gamma is honoured by the replay."""
    torch = torch_cuda()
    hc, W, z, pos, h = setup("tiny", 256, 2, 64, 4, seed=31)
    M = 8
    noise = S.make_head_noise(hc["n_steps"], M, TD, seed=32)
    zd = dev(z, "bf16")
    outs = []
    for k in range(3):
        x = empty((M, TD))
        lm.lazymar_head_sample(h, zd, 2, 64, dev_int(pos), 4, dev(noise), 3.0, 1.0, x)
        lm.lazymar_head_sync(h)
        outs.append(host(x))
    xh = torch.empty((M, TD), dtype=torch.float32).pin_memory()
    lm.lazymar_head_sample(h, zd, 2, 64, pos, 4, noise, 3.0, 1.0, xh)
    lm.lazymar_head_sync(h)
    outs.append(xh.numpy().astype(np.float64))
    for o in outs[1:]:
        assert np.array_equal(o, outs[0])
    x = empty((M, TD))
    lm.lazymar_head_sample(h, zd, 2, 64, pos, 4, noise, 1.0, 1.0, x)
    lm.lazymar_head_sync(h)
    zc, zu = z_rows(z, 2, 64, pos)
    want = HO.sample(W, HO.Schedule(hc["n_train"], hc["n_steps"]), zc, zu, noise, 1.0, 1.0)
    assert max_rel(host(x), want) < TOL["bf16"]
    n, f = lm.lazymar_head_counters(h)
    assert n > 5 * hc["n_steps"] and f > 0
    h.close()


def test_out_of_range_position_is_reported():
    torch_cuda()
    hc, W, z, pos, h = setup("tiny", 256, 1, 64, 2, seed=41)
    bad = pos.copy()
    bad[0, 1] = 64
    x = empty((2, TD))
    lm.lazymar_head_sample(h, dev(z, "bf16"), 1, 64, bad, 2, S.make_head_noise(hc["n_steps"], 2, TD), 3.0, 1.0, x)
    with pytest.raises(lm.LazymarError) as e:
        lm.lazymar_head_sync(h)
    assert e.value.status == 7
    # the handle stays usable
    lm.lazymar_head_sample(h, dev(z, "bf16"), 1, 64, pos, 2, S.make_head_noise(hc["n_steps"], 2, TD), 3.0, 1.0, x)
    lm.lazymar_head_sync(h)
    h.close()


def test_argument_checks():
    torch_cuda()
    hc, W, z, pos, h = setup("tiny", 256, 1, 64, 2, seed=51)
    x = empty((2, TD))
    noise = S.make_head_noise(hc["n_steps"], 2, TD)
    with pytest.raises(lm.LazymarError):      # more tokens than max_tokens
        lm.lazymar_head_sample(h, dev(z, "bf16"), 1, 64, np.zeros((1, 3), np.int32), 3, noise, 3.0, 1.0, x)
    with pytest.raises(lm.LazymarError):      # z on the host
        lm.lazymar_head_sample(h, z, 1, 64, pos, 2, noise, 3.0, 1.0, x)
    with pytest.raises(lm.LazymarError):      # step outside 0..n_steps-1
        lm.lazymar_head_eval(h, dev(z, "bf16"), 1, 64, pos, 2, np.zeros((2, TD), np.float32), hc["n_steps"],
                             empty((4, 2 * TD)))
    h.close()


@pytest.mark.parametrize("td,steps,B,n_new", [(4, 1, 2, 3), (64, 3, 1, 5), (16, 2, 3, 1)])
def test_sampler_edge_shapes(td, steps, B, n_new):
    """One kept step (no noise added at all), a few steps, latent widths 4 and 64."""
    torch_cuda()
    hc = S.head_config("tiny", n_steps=steps)
    cond_dim, n_img = 128, 16
    W = S.make_head_weights(hc, cond_dim, td, seed=61)
    rng = np.random.default_rng(62)
    z = S.round_bf16(rng.standard_normal((2 * B, n_img, cond_dim)).astype(np.float32))
    pos = np.stack([rng.choice(n_img, n_new, replace=False) for _ in range(B)]).astype(np.int32)
    h = lm.lazymar_head_create(hc, cond_dim, td, W, max_tokens=B * n_new)
    M = B * n_new
    noise = S.make_head_noise(steps, M, td, seed=63)
    x = empty((M, td))
    lm.lazymar_head_sample(h, dev(z, "bf16"), B, n_img, pos, n_new, noise, 2.0, 0.8, x)
    lm.lazymar_head_sync(h)
    zc, zu = z_rows(z, B, n_img, pos)
    want = HO.sample(W, HO.Schedule(hc["n_train"], steps), zc, zu, noise, 2.0, 0.8)
    got = host(x)
    assert max_rel(got, want) < TOL["bf16"], max_rel(got, want)
    assert min_cos(got, want) >= COS_MIN
    h.close()


def sampler_case(name, cond_dim, B, n_new, steps, max_tokens, seed):
    torch_cuda()
    n_img = 256
    hc = S.head_config(name, n_steps=steps)
    W = S.make_head_weights(hc, cond_dim, TD, seed=seed)
    rng = np.random.default_rng(seed + 1)
    z = S.round_bf16(rng.standard_normal((2 * B, n_img, cond_dim)).astype(np.float32))
    pos = np.stack([rng.choice(n_img, n_new, replace=False) for _ in range(B)]).astype(np.int32)
    h = lm.lazymar_head_create(hc, cond_dim, TD, W, max_tokens=max_tokens)
    noise = S.make_head_noise(steps, B * n_new, TD, seed=seed + 2)
    return hc, W, z, pos, noise, h


@pytest.mark.parametrize("name,cond_dim,B,n_new,steps,max_tokens", [
    ("mar_b", 768, 3, 50, 6, 150),     # 300 rows: three 128-row tiles, the last ragged
    ("mar_l", 1024, 2, 5, 4, 10),      # width 1280, 8 blocks
    ("mar_h", 1280, 2, 7, 3, 14),      # width 1536, 12 blocks
    ("mar_b", 768, 2, 4, 100, 128),    # 100 kept steps whose modulations take two GEMMs (95 + 5 steps)
])
def test_sampler_widths_tiles_and_modulation_chunks(name, cond_dim, B, n_new, steps, max_tokens):
    """The guided sampler at the MAR-B, MAR-L and MAR-H head widths, over
    several ragged row tiles, and with the modulations of the kept steps
    computed in two chunks, against the oracle."""
    hc, W, z, pos, noise, h = sampler_case(name, cond_dim, B, n_new, steps, max_tokens, seed=71)
    M = B * n_new
    x = empty((M, TD))
    lm.lazymar_head_sample(h, dev(z, "bf16"), B, 256, pos, n_new, noise, 3.0, 1.0, x)
    lm.lazymar_head_sync(h)
    zc, zu = z_rows(z, B, 256, pos)
    want = HO.sample(W, HO.Schedule(hc["n_train"], steps), zc, zu, noise, 3.0, 1.0)
    got = host(x)
    assert max_rel(got, want) < TOL["bf16"], max_rel(got, want)
    assert min_cos(got, want) >= COS_MIN
    h.close()


def test_sampler_graph_replay_is_bitwise_stable_at_mar_b_width():
    """Eager, captured and replayed runs at width 1024 (tcgen05 block GEMMs)
    give the same bits; a changed temperature is honoured by the replay."""
    hc, W, z, pos, noise, h = sampler_case("mar_b", 768, 2, 6, 5, 12, seed=81)
    zd = dev(z, "bf16")
    outs = []
    for _ in range(3):
        x = empty((12, TD))
        lm.lazymar_head_sample(h, zd, 2, 256, dev_int(pos), 6, dev(noise), 3.0, 1.0, x)
        lm.lazymar_head_sync(h)
        outs.append(host(x))
    for o in outs[1:]:
        assert np.array_equal(o, outs[0])
    x = empty((12, TD))
    lm.lazymar_head_sample(h, zd, 2, 256, dev_int(pos), 6, dev(noise), 3.0, 0.5, x)
    lm.lazymar_head_sync(h)
    zc, zu = z_rows(z, 2, 256, pos)
    want = HO.sample(W, HO.Schedule(hc["n_train"], 5), zc, zu, noise, 3.0, 0.5)
    assert max_rel(host(x), want) < TOL["bf16"]
    h.close()
