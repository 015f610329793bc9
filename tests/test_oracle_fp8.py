"""Pins of the oracle's E4M3 arithmetic against the 8-bit format's definition
(1 sign bit, 4 exponent bits with bias 7, 3 mantissa bits, subnormals, no
infinities, 0x7F / 0xFF NaN, largest finite value 448)."""
import copy
import math

import numpy as np
import pytest

import oracle as O
from oracle import fp8
import synth


def test_e4m3_decode_table_values():
    # values fixed by the format: exponent bias 7, subnormals below 2^-6
    cases = {0x00: 0.0, 0x01: 2.0 ** -9, 0x07: 7 * 2.0 ** -9, 0x08: 2.0 ** -6, 0x38: 1.0, 0x3C: 1.5,
             0x40: 2.0, 0x7E: 448.0, 0x77: 240.0, 0x80: -0.0, 0xB8: -1.0, 0xFE: -448.0}
    for b, v in cases.items():
        assert fp8.e4m3_decode(b) == v, hex(b)
    assert math.isnan(fp8.e4m3_decode(0x7F)) and math.isnan(fp8.e4m3_decode(0xFF))


def test_e4m3_round_fixed_points_and_brute_force():
    codes = np.arange(256)
    vals = fp8.e4m3_decode(codes)
    finite = np.isfinite(vals)
    # every finite E4M3 value rounds to itself
    np.testing.assert_array_equal(fp8.e4m3_round(vals[finite]), vals[finite])
    # any other value goes to the nearest E4M3 value; a tie to the code with
    # an even mantissa; beyond 448 to +-448
    table = np.unique(vals[finite])
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(4000) * 10.0 ** rng.uniform(-4, 3, 4000),
                        (table[:-1] + table[1:]) / 2])                     # every midpoint: a tie
    got = fp8.e4m3_round(x)
    for xi, gi in zip(x, got):
        if abs(xi) > 448:
            assert gi == math.copysign(448.0, xi)
            continue
        d = np.abs(table - xi)
        near = table[d == d.min()]
        if len(near) == 1:
            assert gi == near[0], xi
        else:                                     # tie: the neighbour whose code has mantissa bit 0 clear
            even = [v for v in near if int(codes[finite][vals[finite] == v][0]) & 1 == 0]
            assert gi == even[0], xi


def test_e4m3_round_worked_ties():
    assert fp8.e4m3_round(1 + 1 / 16) == 1.0            # between 1.0 (m=0) and 1.125 (m=1)
    assert fp8.e4m3_round(1 + 3 / 16) == 1.25           # between 1.125 (m=1) and 1.25 (m=2)
    assert fp8.e4m3_round(2.0 ** -10) == 0.0            # half the smallest subnormal
    assert fp8.e4m3_round(3 * 2.0 ** -10) == 2.0 ** -8  # between 2^-9 (m=1) and 2^-8 (m=2)
    assert fp8.e4m3_round(500.0) == 448.0 and fp8.e4m3_round(-1e9) == -448.0


def test_quantize_rows_scales_each_row_to_448():
    rng = np.random.default_rng(1)
    w = rng.standard_normal((5, 7)) * np.array([1e-3, 1.0, 30.0, 0.02, 5.0])[:, None]
    w[3] = 0.0
    q, s = fp8.quantize_rows(w)
    np.testing.assert_array_equal(np.abs(q).max(axis=1)[[0, 1, 2, 4]], 448.0)
    assert s[3] == 1.0 and (q[3] == 0).all()
    np.testing.assert_allclose(s[[0, 1, 2, 4]], np.abs(w[[0, 1, 2, 4]]).max(axis=1) / 448.0, rtol=1e-15)
    # every element within half an E4M3 spacing of its scaled value: relative
    # 2^-4 in the normal range, absolute 2^-10 among the subnormals
    u = np.abs(w / s[:, None])
    err = np.abs(q - w / s[:, None])
    normal = u >= 2.0 ** -6
    assert (err[normal] <= 2.0 ** -4 * u[normal] + 1e-12).all()
    assert (err[~normal] <= 2.0 ** -10 + 1e-15).all()


def test_linear_e4m3_is_exact_on_representable_operands():
    rng = np.random.default_rng(2)
    codes = rng.integers(0, 256, size=(6, 16))
    codes[(codes & 0x7F) == 0x7F] = 0x38
    x = fp8.e4m3_decode(codes)
    w = fp8.e4m3_decode(np.where(((c := rng.integers(0, 256, size=(4, 16))) & 0x7F) == 0x7F, 0x38, c))
    w[:, 0] = 448.0                                  # every row's scale is exactly 1
    b = rng.standard_normal(4)
    expect = np.array([[math.fsum(x[i, k] * w[j, k] for k in range(16)) + b[j] for j in range(4)] for i in range(6)])
    np.testing.assert_allclose(fp8.linear_e4m3(x, w, b), expect, rtol=1e-15, atol=1e-15)


def test_fp8_cached_step_without_fp8_gemms_is_the_oracle():
    cfg = synth.config("tiny")
    W = synth.make_weights(cfg)
    order, table = synth.make_order(cfg), synth.make_latent_table(cfg)
    (l0, m0), (l1, m1) = synth.tiny_state(cfg, order, table)
    labels = synth.make_labels(cfg)
    c = O.Cache(cfg, 1)
    O.full_step(cfg, W, c, l0, m0, labels, 3.0)
    base = copy.deepcopy(c)
    c2 = copy.deepcopy(c)
    N = synth.n_compute(cfg)
    z, g, I, S = O.cached_step(cfg, W, c, l1, m1, labels, N, False, 3.0)
    z2, g2, I2, S2 = fp8.cached_step_fp8(cfg, W, c2, l1, m1, labels, N, False, 3.0, gemms=())
    np.testing.assert_array_equal(z, z2)
    np.testing.assert_array_equal(I, I2)
    # with the Q/K/V projection in E4M3 the selection (decided in the full
    # blocks) is the same and the features move, but little
    z3, _, I3, _ = fp8.cached_step_fp8(cfg, W, base, l1, m1, labels, N, False, 3.0, gemms=("qkv",))
    assert I3.tolist() == I.tolist()
    assert 0 < np.abs(z3 - z).max() / np.abs(z).max() < 2e-2
