"""FP8 (E4M3) arithmetic for the oracle, and the approximation error of FP8
GEMMs in the token-cached blocks.

TEST INFRASTRUCTURE, like the rest of oracle/: only tests/ and bench.py's CPU
legs use it; the CUDA library never does.

The paper ran FP16 (Sec. 4.1) and says nothing about 8-bit arithmetic. The
GPU path can run the Q/K/V projection of the blocks under the token cache
(Eq. 9) on 8-bit tensor cores: the LayerNorm output and the weights are
rounded to E4M3 (the OCP 8-bit floating-point format: 1 sign bit, 4 exponent
bits with bias 7, 3 mantissa bits; subnormals; no infinities; largest finite
value 448), each weight row with its own scale. This module states that
rounding from the format's definition and runs the oracle's cached step with
it, so that the error of any choice of FP8 GEMMs can be measured against the
fp64 oracle (the paper's method at full precision).

    python -m oracle.fp8 mar_b                # error of each FP8 choice
"""
import sys

import numpy as np

from . import lazymar_oracle as OM

E4M3_MAX = 448.0        # largest finite value: 1.110b x 2^8
E4M3_MIN_EXP = -6       # smallest normal exponent (1 - bias)
E4M3_MANT_BITS = 3


def e4m3_round(x):
    """Nearest E4M3 value of each element (ties to even), saturating at +-448.

    The spacing of E4M3 values in the binade [2^e, 2^(e+1)) is 2^(e-3); below
    the smallest normal 2^-6 the subnormals keep the spacing 2^-9. A tie
    between two neighbours goes to the one with an even mantissa.
    """
    x = np.asarray(x, np.float64)
    a = np.abs(x)
    e = np.floor(np.log2(np.where(a > 0, a, 1.0)))
    e = np.maximum(e, E4M3_MIN_EXP)
    step = np.exp2(e - E4M3_MANT_BITS)
    q = np.round(a / step) * step          # numpy rounds half to even
    q = np.minimum(q, E4M3_MAX)
    return np.where(a > 0, np.copysign(q, x), x * 0.0)


def e4m3_decode(byte):
    """Value of an E4M3 byte: sign s, exponent field E (4 bits), mantissa m
    (3 bits): (-1)^s 2^(E-7) (1 + m/8) for E > 0, (-1)^s 2^-6 (m/8) for E = 0;
    0x7F / 0xFF are NaN."""
    b = np.asarray(byte, np.int64) & 0xFF
    s = np.where(b & 0x80, -1.0, 1.0)
    E = (b >> 3) & 0xF
    m = (b & 0x7).astype(np.float64)
    v = np.where(E > 0, np.exp2(E - 7.0) * (1.0 + m / 8.0), np.exp2(-6.0) * (m / 8.0))
    v = np.where((b & 0x7F) == 0x7F, np.nan, v)
    return s * v


def quantize_rows(w):
    """Per-row (output-channel) scaling of a weight matrix [out, in]: scale_n =
    max_k |W[n, k]| / 448, W[n, :] ~ scale_n * e4m3(W[n, :] / scale_n). Returns
    (e4m3 values of W / scale as float64, scale). A zero row has scale 1."""
    w = np.asarray(w, np.float64)
    amax = np.abs(w).max(axis=1)
    scale = np.where(amax > 0, amax / E4M3_MAX, 1.0)
    return e4m3_round(w / scale[:, None]), scale


def linear_e4m3(x, w, b):
    """y = e4m3(x) (scale_n e4m3(W / scale_n))^T + b: an 8-bit GEMM with unit
    activation scale and per-output-channel weight scales, accumulated exactly
    (the GPU accumulates in fp32)."""
    wq, scale = quantize_rows(w)
    return (e4m3_round(x) @ wq.T) * scale[None, :] + np.asarray(b, np.float64)


def cached_step_fp8(cfg, W, cache, latents, mask, labels, n, cond_reuse, gamma, idx=None, gemms=("qkv",)):
    """OM.cached_step with the named GEMMs of the token-cached blocks (a subset
    of qkv, out, fc1, fc2) computed by linear_e4m3. The full blocks 0..s-1
    (which decide the selection) are unchanged."""
    gemms = set(gemms)

    def lin(which, x, w, b):
        return linear_e4m3(x, w, b) if which in gemms else OM.linear(x, w, b)

    def block_cached(bw, x_sel, I, k_cache, v_cache, heads, eps):
        D = x_sel.shape[-1]
        qkv = lin("qkv", OM.layer_norm(x_sel, bw["ln1_g"], bw["ln1_b"], eps), bw["w_qkv"], bw["b_qkv"])
        k_cache[I] = qkv[:, D:2 * D]
        v_cache[I] = qkv[:, 2 * D:]
        o = OM.attention(qkv[:, :D], k_cache, v_cache, heads)
        y = x_sel + lin("out", o, bw["w_o"], bw["b_o"])
        h = OM.gelu(lin("fc1", OM.layer_norm(y, bw["ln2_g"], bw["ln2_b"], eps), bw["w1"], bw["b1"]))
        return y + lin("fc2", h, bw["w2"], bw["b2"])

    saved = OM.block_cached
    OM.block_cached = block_cached
    try:
        return OM.cached_step(cfg, W, cache, latents, mask, labels, n, cond_reuse, gamma, idx=idx)
    finally:
        OM.block_cached = saved


def _report(name, pair=0):
    import copy

    import synth
    cfg = synth.config(name)
    W = synth.make_weights(cfg)
    order, table = synth.make_order(cfg), synth.make_latent_table(cfg)
    labels = synth.make_labels(cfg)[pair:pair + 1]
    sl = slice(pair, pair + 1)
    (l0, m0), (l1, m1) = synth.step_state(cfg, order, table, 100), synth.step_state(cfg, order, table, 104)
    N = synth.n_compute(cfg)
    c = OM.Cache(cfg, 1)
    OM.full_step(cfg, W, c, l0[sl], m0[sl], labels, 3.0)
    base = copy.deepcopy(c)
    z_ref, _, I, _ = OM.cached_step(cfg, W, c, l1[sl], m1[sl], labels, N, False, 3.0)
    for gemms in (("qkv",), ("out",), ("fc1",), ("fc2",), ("fc1", "fc2"), ("qkv", "out", "fc1", "fc2")):
        z, _, _, _ = cached_step_fp8(cfg, W, copy.deepcopy(base), l1[sl], m1[sl], labels, N, False, 3.0, idx=I,
                                     gemms=gemms)
        a, b = z.reshape(-1, z.shape[-1]), z_ref.reshape(-1, z_ref.shape[-1])
        cos = float(((a * b).sum(-1) / np.sqrt((a * a).sum(-1) * (b * b).sum(-1))).min())
        err = float(np.abs(z - z_ref).max() / np.abs(z_ref).max())
        print("%s, E4M3 %-22s max rel err %.4f  min cosine %.5f" % (name, "+".join(gemms) + ":", err, cos), flush=True)


if __name__ == "__main__":
    for n in sys.argv[1:] or ["mar_b"]:
        _report(n)
