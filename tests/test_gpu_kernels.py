"""Kernel-level parity: each CUDA kernel, called through the C ABI, against
the CPU oracle on the same seeded inputs."""
import numpy as np
import pytest

import oracle as O
from oracle import diffusion_head as HO
from oracle import fp8
import synth
from paper_2503_12450_gb300 import lazymar as lm
from _gpu import DT, TOL, dev, dev_int, empty, host, max_rel, sync, torch_cuda

pytestmark = pytest.mark.gpu


# --------------------------------------------------------------------------
# Selection (Eq. 8): indices bit-exact
# --------------------------------------------------------------------------

@pytest.mark.parametrize("rows,T,D,N,dtype", [
    (2, 80, 256, 20, "fp32"),      # tiny
    (64, 320, 768, 50, "bf16"),    # MAR-B
    (16, 320, 1024, 32, "bf16"),   # MAR-L, 10 %
    (8, 320, 1280, 50, "bf16"),    # MAR-H
    (32, 1088, 1024, 272, "bf16"),  # high resolution, 25 %
    (3, 320, 768, 0, "bf16"),
    (3, 320, 768, 320, "bf16"),
    (1, 1, 8, 1, "fp32"),
    (5, 100, 16, 37, "bf16"),
    (4, 513, 64, 129, "fp32"),     # T spans two scan chunks
])
def test_select_tokens_bit_exact(rows, T, D, N, dtype):
    torch = torch_cuda()
    cur, ref = synth.similarity_inputs(rows, T, D, seed=rows * 1000 + T, dtype=dtype)
    g_cur, g_ref = dev(cur, dtype), dev(ref, dtype)
    idx = torch.full((rows, max(N, 1)), -1, dtype=torch.int32, device="cuda")
    lm.lazymar_select_tokens(DT[dtype], g_cur, g_ref, rows, T, D, N, idx)
    sync()
    got = idx.cpu().numpy()[:, :N]
    for r in range(rows):
        expect = O.select_compute(O.cosine_similarity(cur[r], ref[r]), N)
        assert got[r].tolist() == expect.tolist(), "row %d" % r
    # the reference now holds the current values, bit for bit
    assert torch.equal(g_ref, g_cur)


@pytest.mark.parametrize("rule", [lm.LAZYMAR_SELECT_LEAST_SIMILAR, lm.LAZYMAR_SELECT_MOST_SIMILAR,
                                  lm.LAZYMAR_SELECT_RANDOM])
@pytest.mark.parametrize("with_prio", [False, True])
@pytest.mark.parametrize("rows,T,D,N,dtype", [
    (64, 320, 768, 50, "bf16"),    # MAR-B
    (2, 80, 256, 20, "fp32"),      # tiny
    (5, 100, 16, 37, "bf16"),
    (3, 320, 768, 320, "bf16"),    # N = T
    (4, 513, 64, 129, "fp32"),
])
def test_select_rules_bit_exact(rule, with_prio, rows, T, D, N, dtype):
    """Selection strategies of Table 3 (V, IV, III) with and without priority
    classes (observation-based / type strategies) against the oracle on the
    same buffers: indices bit-exact, reference updated."""
    torch = torch_cuda()
    cur, ref = synth.similarity_inputs(rows, T, D, seed=rows * 1000 + T + rule, dtype=dtype)
    rng = np.random.default_rng(rows + T + 7 * rule + with_prio)
    prio = rng.integers(0, 3, size=(rows, T)).astype(np.uint8) if with_prio else None
    keys = rng.integers(0, 1 << 32, size=(rows, T), dtype=np.uint64).astype(np.uint32)
    keys[:, 1::7] = keys[:, 0:1]  # repeated keys: the index decides
    g_cur, g_ref = dev(cur, dtype), dev(ref, dtype)
    g_prio = torch.from_numpy(prio).cuda() if with_prio else None
    g_keys = torch.from_numpy(keys.view(np.int32)).cuda()
    idx = torch.full((rows, max(N, 1)), -1, dtype=torch.int32, device="cuda")
    lm.lazymar_select_tokens_ex(DT[dtype], g_cur, g_ref, rows, T, D, N, rule, g_prio, g_keys, idx)
    sync()
    got = idx.cpu().numpy()[:, :N]
    for r in range(rows):
        expect = O.select_by_rule(O.cosine_similarity(cur[r], ref[r]), N, rule,
                                  None if prio is None else prio[r], keys[r])
        assert got[r].tolist() == expect.tolist(), "row %d" % r
    assert torch.equal(g_ref, g_cur)


def _selection_edge_inputs(T, D, seed):
    """bf16 rows that exercise both similarity paths of the kernel.

    row 0: every element scaled by 2^u, u uniform in [-60, 60] (exponent span
           far beyond the exact integer sums: the fp64 path);
    row 1: per token either a narrow ([-4, 4]) or a wide ([-30, 30]) span;
    row 2: subnormal and near-subnormal values, zero tokens, cur = -ref;
    row 3: Inf / NaN elements in a few tokens (S is NaN, ranked as -inf).
    """
    rng = np.random.Generator(np.random.PCG64(seed))
    ref = rng.standard_normal((4, T, D)).astype(np.float32)
    cur = ref * (1 + 0.05 * rng.standard_normal((4, T, D))).astype(np.float32)
    big = rng.random((4, T)) < 0.2
    cur[big] = rng.standard_normal((int(big.sum()), D)).astype(np.float32)
    u = rng.integers(-60, 61, size=(T, D))
    cur[0] *= np.exp2(u).astype(np.float32)
    ref[0] *= np.exp2(u).astype(np.float32)
    span = np.where(rng.random(T) < 0.5, 4, 30)[:, None]
    u = rng.integers(-span, span + 1, size=(T, D))
    cur[1] *= np.exp2(u).astype(np.float32)
    ref[1] *= np.exp2(u).astype(np.float32)
    scale = np.where(rng.random((T, 1)) < 0.5, 2.0 ** -130, 2.0 ** -120).astype(np.float32)
    cur[2] *= scale
    ref[2] *= scale
    cur[2, :5] = 0.0
    ref[2, 3:8] = 0.0
    cur[2, 10:20] = -ref[2, 10:20]
    for t, v in [(0, np.inf), (7, -np.inf), (11, np.nan)]:
        cur[3, t, t % D] = v
    ref[3, 20, 5] = np.inf
    ref[3, 21, 6] = np.nan
    return synth.round_bf16(cur), synth.round_bf16(ref)


@pytest.mark.parametrize("D", [768, 1280, 64])
def test_select_tokens_exponent_range_and_specials(D):
    """Selections agree with the oracle on data whose exponent spans, subnormals
    and Inf/NaN elements steer tokens through both the exact integer sums and
    the fp64 fallback. (Where the spans exceed what fp64 sums exactly, both
    sides round; the random data has no near-ties for that to reorder.)"""
    torch = torch_cuda()
    T, N = 200, 60
    cur, ref = _selection_edge_inputs(T, D, seed=D)
    g_cur, g_ref = dev(cur, "bf16"), dev(ref, "bf16")
    idx = torch.full((4, N), -1, dtype=torch.int32, device="cuda")
    lm.lazymar_select_tokens(DT["bf16"], g_cur, g_ref, 4, T, D, N, idx)
    sync()
    got = idx.cpu().numpy()
    with np.errstate(invalid="ignore", over="ignore"):
        for r in range(4):
            expect = O.select_compute(O.cosine_similarity(cur[r], ref[r]), N)
            assert got[r].tolist() == expect.tolist(), "row %d" % r
    # bit patterns: the copied NaNs compare unequal as values
    assert torch.equal(g_ref.view(torch.int16), g_cur.view(torch.int16))


def test_select_tokens_fp32_near_ties():
    """fp32 similarities are fp64 sums rounded at every addition, in the
    kernel's order on the GPU and in numpy's on the CPU, so mathematically
    equal similarities may come out a few ulps apart on either side. Tokens
    t and t + 32 carry the same vectors with their elements permuted (equal
    exact sums, different rounding) and the budget N cuts through those
    pairs. The GPU's selection must be valid against the oracle's S up to
    8 ulps; every token outside that band is selected exactly as the oracle
    selects it."""
    torch = torch_cuda()
    rows, T, D, N = 4, 64, 256, 40
    rng = np.random.default_rng(31)
    ref = rng.standard_normal((rows, T, D)).astype(np.float32)
    cur = (ref + 0.3 * rng.standard_normal((rows, T, D))).astype(np.float32)
    perm = rng.permutation(D)
    cur[:, 32:], ref[:, 32:] = cur[:, :32][:, :, perm], ref[:, :32][:, :, perm]
    g_cur, g_ref = dev(cur), dev(ref)
    idx = torch.full((rows, N), -1, dtype=torch.int32, device="cuda")
    lm.lazymar_select_tokens(DT["fp32"], g_cur, g_ref, rows, T, D, N, idx)
    sync()
    got = idx.cpu().numpy()
    for r in range(rows):
        S = O.cosine_similarity(cur[r], ref[r])
        margin = 8 * np.spacing(np.abs(S).max())
        sel = set(got[r].tolist())
        assert len(sel) == N and got[r].tolist() == sorted(sel)
        for a in sel:
            for b in set(range(T)) - sel:
                assert S[a] <= S[b] + margin, (r, a, b)
        thr = np.sort(S)[N - 1]
        clear = np.abs(S - thr) > margin
        expect = set(O.select_compute(S, N).tolist())
        assert {t for t in range(T) if clear[t] and t in sel} == {t for t in range(T) if clear[t] and t in expect}


# --------------------------------------------------------------------------
# Condition cache / guidance (Eq. 7 reading, Eq. 10)
# --------------------------------------------------------------------------

@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
@pytest.mark.parametrize("mode", [lm.LAZYMAR_CFG_GUIDE, lm.LAZYMAR_CFG_REFRESH, lm.LAZYMAR_CFG_REUSE])
@pytest.mark.parametrize("n", [8 * 1000 + 3, 32 * 256 * 768])
def test_cfg_combine(dtype, mode, n):
    gamma = 3.0
    c = synth.tensor((n,), 11, dtype=dtype)
    u = synth.tensor((n,), 12, dtype=dtype)
    d = synth.tensor((n,), 13, std=0.1, dtype=dtype)
    gc, gu, gd = dev(c, dtype), dev(u, dtype), dev(d, dtype)
    g, uo = empty((n,), dtype), empty((n,), dtype)
    lm.lazymar_cfg_combine(DT[dtype], mode, gc, gu, gd, gamma, n, uo, g)
    sync()
    tol = 8e-3 if dtype == "bf16" else 1e-6
    if mode == lm.LAZYMAR_CFG_REUSE:
        u_ref = O.cond_cache_reuse(c, d)
        assert max_rel(host(uo), u_ref) < tol
    else:
        u_ref = u
    if mode == lm.LAZYMAR_CFG_REFRESH:
        assert max_rel(host(gd), O.cond_cache_store(c, u)) < tol
    assert max_rel(host(g), O.guidance(c, u_ref, gamma)) < tol


# --------------------------------------------------------------------------
# GEMMs (tcgen05 for bf16, CUDA cores for fp32) with every epilogue
# --------------------------------------------------------------------------

GEMM_SHAPES = [
    (1, 384, 128), (40, 768, 256), (200, 2304, 768), (3200, 2304, 768), (3200, 768, 768),
    (3200, 3072, 768), (3200, 768, 3072), (777, 1280, 1280), (384, 3840, 1280),
    (100, 256, 192), (33, 384, 320),  # K not a multiple of 128: 64-deep stages at every width
]


def _linear_case(dtype, epi, M, N, K, flags, seed, scatter=True):
    torch = torch_cuda()
    a = synth.tensor((M, K), seed, dtype=dtype)
    w = synth.tensor((N, K), seed + 1, std=0.05, dtype=dtype)
    b = synth.tensor((N,), seed + 2, std=0.1, dtype=dtype)
    ga, gw, gb = dev(a, dtype), dev(w, dtype), dev(b, dtype)
    ref = O.linear(a, w, b)
    out_dtype_tol = 1e-2 if dtype == "bf16" else 1e-4
    if epi in (lm.LAZYMAR_EPI_BIAS, lm.LAZYMAR_EPI_GELU, lm.LAZYMAR_EPI_SILU):
        out = empty((M, N), dtype)
        lm.lazymar_linear(DT[dtype], epi, ga, gw, gb, M, N, K, out, N, flags=flags)
        sync()
        expect = {lm.LAZYMAR_EPI_BIAS: ref, lm.LAZYMAR_EPI_GELU: O.gelu(ref), lm.LAZYMAR_EPI_SILU: HO.silu(ref)}[epi]
        assert max_rel(host(out), expect) < out_dtype_tol
    elif epi == lm.LAZYMAR_EPI_RESIDUAL:
        r0 = synth.tensor((M, N), seed + 3)
        out = dev(r0, "fp32")
        lm.lazymar_linear(DT[dtype], epi, ga, gw, gb, M, N, K, out, N, flags=flags)
        sync()
        assert max_rel(host(out), r0 + ref) < 1e-4
    elif not scatter:
        D = N // 3
        q, gk, gv = empty((M, D), dtype), empty((M, D), dtype), empty((M, D), dtype)
        lm.lazymar_linear(DT[dtype], epi, ga, gw, gb, M, N, K, q, D, gk, gv, None, flags=flags)
        sync()
        assert max_rel(host(q), ref[:, :D]) < out_dtype_tol
        assert max_rel(host(gk), ref[:, D:2 * D]) < out_dtype_tol
        assert max_rel(host(gv), ref[:, 2 * D:]) < out_dtype_tol
    else:
        D = N // 3
        R = M + 17
        row_map = synth.distinct_rows(M, R, seed + 4)
        k0 = synth.tensor((R, D), seed + 5, dtype=dtype)
        v0 = synth.tensor((R, D), seed + 6, dtype=dtype)
        q, gk, gv = empty((M, D), dtype), dev(k0, dtype), dev(v0, dtype)
        lm.lazymar_linear(DT[dtype], epi, ga, gw, gb, M, N, K, q, D, gk, gv, dev_int(row_map), flags=flags)
        sync()
        assert max_rel(host(q), ref[:, :D]) < out_dtype_tol
        k, v = host(gk), host(gv)
        assert max_rel(k[row_map], ref[:, D:2 * D]) < out_dtype_tol
        assert max_rel(v[row_map], ref[:, 2 * D:]) < out_dtype_tol
        keep = np.setdiff1d(np.arange(R), row_map)
        assert np.array_equal(k[keep], k0[keep]) and np.array_equal(v[keep], v0[keep])


@pytest.mark.parametrize("M,N,K", GEMM_SHAPES)
@pytest.mark.parametrize("epi", [lm.LAZYMAR_EPI_BIAS, lm.LAZYMAR_EPI_GELU, lm.LAZYMAR_EPI_RESIDUAL,
                                 lm.LAZYMAR_EPI_QKV, lm.LAZYMAR_EPI_SILU])
def test_linear_bf16_tcgen05(M, N, K, epi):
    if epi == lm.LAZYMAR_EPI_QKV and (N % 3 or (N // 3) % 32):
        pytest.skip("not a QKV shape")
    for flags in [1, 4] + ([2] if N % 256 == 0 else []) + ([3] if N % 192 == 0 else []):
        _linear_case("bf16", epi, M, N, K, flags, seed=M + N + K + epi)


@pytest.mark.parametrize("M,N,K,epi", [
    (20480, 768, 768, lm.LAZYMAR_EPI_RESIDUAL),    # out-projection: three waves of 256-wide tiles, then 8 row tiles 64 wide
    (20480, 768, 3072, lm.LAZYMAR_EPI_RESIDUAL),   # residual over long K (fc2): one launch
    (20480, 2304, 768, lm.LAZYMAR_EPI_QKV),        # other epilogues: one launch
])
def test_linear_last_wave_split(M, N, K, epi):
    """With the automatic tile width (flags 0) the fp32-residual GEMM over
    short K whose last round of tiles would run mostly empty is launched as
    two: the row tiles of the whole waves, then the remaining rows (their A
    rows and residual rows offset) with narrower tiles."""
    _linear_case("bf16", epi, M, N, K, 0, seed=M + N + K + epi)
    if epi == lm.LAZYMAR_EPI_QKV:
        _linear_case("bf16", epi, M, N, K, 0, seed=M + N + K, scatter=False)


@pytest.mark.parametrize("M,N,K", [(1, 12, 8), (40, 768, 256), (160, 1024, 256), (77, 256, 1024)])
@pytest.mark.parametrize("epi", [lm.LAZYMAR_EPI_BIAS, lm.LAZYMAR_EPI_GELU, lm.LAZYMAR_EPI_RESIDUAL,
                                 lm.LAZYMAR_EPI_QKV, lm.LAZYMAR_EPI_SILU])
def test_linear_fp32(M, N, K, epi):
    if epi == lm.LAZYMAR_EPI_QKV and (N % 3 or (N // 3) % 4):
        pytest.skip("not a QKV shape")
    _linear_case("fp32", epi, M, N, K, 0, seed=M + N + K + epi)


# --------------------------------------------------------------------------
# E4M3 Q/K/V projection (qkv_e4m3): weight quantization, LayerNorm to E4M3,
# the kind::f8f6f4 GEMM
# --------------------------------------------------------------------------

def _e4m3_codes(shape, seed):
    """Random E4M3 bytes over the whole finite range (no NaN codes)."""
    c = np.random.default_rng(seed).integers(0, 256, size=shape).astype(np.uint8)
    c[(c & 0x7F) == 0x7F] = 0x38
    return c


@pytest.mark.parametrize("rows,cols", [(2304, 768), (3840, 1280), (5, 8), (130, 1024)])
def test_quantize_e4m3_bit_exact(rows, cols):
    """Per-row scales and E4M3 codes of a bf16 weight matrix. The rounding
    decision is taken in fp32 on both sides (the kernel's precision): scale =
    fp32(max|w|) / 448, code = E4M3(fp32(w) / scale); the oracle's rounding is
    the format's definition. Rows of zeros, a row with an exact tie and
    mixed magnitudes included."""
    torch = torch_cuda()
    w = synth.tensor((rows, cols), rows + cols, std=0.02, dtype="bf16")
    w[0] = 0.0
    if rows > 2:
        w[1] = synth.round_bf16(np.linspace(-3, 3, cols).astype(np.float32))
        w[2] = synth.round_bf16(w[2] * np.float32(1e4))
    gw = dev(w, "bf16")
    q = torch.zeros((rows, cols), dtype=torch.uint8, device="cuda")
    sc = torch.zeros(rows, dtype=torch.float32, device="cuda")
    lm.lazymar_quantize_e4m3(gw, rows, cols, q, sc)
    sync()
    amax = np.abs(w).max(axis=1).astype(np.float32)
    s32 = np.where(amax > 0, amax / np.float32(448.0), np.float32(1.0)).astype(np.float32)
    np.testing.assert_array_equal(sc.cpu().numpy(), s32)
    expect = fp8.e4m3_round((w.astype(np.float32) / s32[:, None]).astype(np.float32))
    got = fp8.e4m3_decode(q.cpu().numpy())
    np.testing.assert_array_equal(np.abs(got), np.abs(expect))
    nz = expect != 0
    assert (np.sign(got[nz]) == np.sign(expect[nz])).all()


def test_layernorm_e4m3_output():
    """LayerNorm rows to E4M3 (unit scale): every code is the E4M3 rounding of
    the oracle's LayerNorm, or its neighbour where the fp32 value lies within
    rounding distance of the midpoint between two codes."""
    torch = torch_cuda()
    M, D = 300, 768
    x = synth.tensor((M, D), 41, std=3.0, mean=0.5)
    g = synth.tensor((D,), 42, std=0.5, mean=1.0, dtype="bf16")
    b = synth.tensor((D,), 43, std=0.2, dtype="bf16")
    y = torch.zeros((M, D), dtype=torch.uint8, device="cuda")
    lm.lazymar_layernorm(lm.LAZYMAR_E4M3, dev(x), None, dev(g, "bf16"), dev(b, "bf16"), y, M, D, 1e-6)
    sync()
    ref = O.layer_norm(x, g, b, 1e-6)
    got = fp8.e4m3_decode(y.cpu().numpy())
    exact = fp8.e4m3_round(ref)
    bad = got != exact
    assert bad.mean() < 1e-3
    # where they differ, the oracle's value sits at a rounding midpoint of the two codes
    lo, hi = np.minimum(got[bad], exact[bad]), np.maximum(got[bad], exact[bad])
    mid = (lo + hi) / 2
    assert (np.abs(ref[bad] - mid) <= 1e-5 * np.maximum(np.abs(mid), 1.0)).all()
    assert (hi - lo <= np.maximum(np.abs(hi), np.abs(lo)) * 2.0 ** -3 + 2.0 ** -9).all()


@pytest.mark.parametrize("M,N,K", [(3200, 2304, 768), (1600, 2304, 768), (12800, 3840, 1280), (777, 3072, 1024),
                                   (1, 384, 128), (130, 256, 256)])
@pytest.mark.parametrize("epi", [lm.LAZYMAR_EPI_BIAS, lm.LAZYMAR_EPI_QKV])
def test_linear_e4m3(M, N, K, epi):
    """The kind::f8f6f4 GEMM on E4M3 operands with per-column weight scales
    against the oracle's product of the decoded operands (exact in fp64; the
    GPU accumulates in fp32 and writes bf16), every tile width."""
    if epi == lm.LAZYMAR_EPI_QKV and (N % 3 or (N // 3) % 32):
        pytest.skip("not a QKV shape")
    torch = torch_cuda()
    seed = M + N + K + epi
    ac, wc = _e4m3_codes((M, K), seed), _e4m3_codes((N, K), seed + 1)   # subnormals to +-448
    scale = (np.random.default_rng(seed + 2).uniform(0.5, 2.0, N) * 1e-3).astype(np.float32)
    bias = synth.tensor((N,), seed + 3, std=0.1, dtype="bf16")
    ref = fp8.e4m3_decode(ac) @ (fp8.e4m3_decode(wc) * scale[:, None].astype(np.float64)).T + bias
    ga = torch.from_numpy(ac).cuda()
    gw = torch.from_numpy(wc).cuda()
    gs = torch.from_numpy(scale).cuda()
    gb = dev(bias, "bf16")
    for flags in [1] + ([2] if N % 256 == 0 else []) + ([3] if N % 192 == 0 else []):
        if epi == lm.LAZYMAR_EPI_BIAS:
            out = empty((M, N), "bf16")
            lm.lazymar_linear_e4m3(epi, ga, gw, gs, gb, M, N, K, out, N, flags=flags)
            sync()
            assert max_rel(host(out), ref) < 1e-2, flags
        else:
            D = N // 3
            R = M + 17
            row_map = synth.distinct_rows(M, R, seed + 4)
            k0 = synth.tensor((R, D), seed + 5, dtype="bf16")
            v0 = synth.tensor((R, D), seed + 6, dtype="bf16")
            q, gk, gv = empty((M, D), "bf16"), dev(k0, "bf16"), dev(v0, "bf16")
            lm.lazymar_linear_e4m3(epi, ga, gw, gs, gb, M, N, K, q, D, gk, gv, dev_int(row_map), flags=flags)
            sync()
            assert max_rel(host(q), ref[:, :D]) < 1e-2
            k, v = host(gk), host(gv)
            assert max_rel(k[row_map], ref[:, D:2 * D]) < 1e-2 and max_rel(v[row_map], ref[:, 2 * D:]) < 1e-2
            keep = np.setdiff1d(np.arange(R), row_map)
            assert np.array_equal(k[keep], k0[keep]) and np.array_equal(v[keep], v0[keep])


# --------------------------------------------------------------------------
# Attention (Eq. 3 with a query subset)
# --------------------------------------------------------------------------

@pytest.mark.parametrize("rows,n_q,T,heads,dh,dtype,q_std", [
    (2, 50, 320, 12, 64, "bf16", 1.0),    # MAR-B cached layer
    (2, 320, 320, 4, 64, "bf16", 1.0),    # full layer
    (1, 272, 1088, 2, 64, "bf16", 1.0),   # high resolution cached layer
    (3, 50, 320, 4, 80, "bf16", 1.0),     # MAR-H head width, cached layer
    (2, 320, 320, 16, 80, "bf16", 1.0),   # MAR-H full layer (three query tiles)
    (2, 65, 130, 2, 80, "bf16", 1.0),     # ragged queries and keys
    (1, 129, 200, 3, 80, "bf16", 1.0),    # one query past a tile, a ragged key chunk
    (3, 256, 300, 5, 64, "bf16", 1.0),    # whole query tiles only (no shorter last tile)
    (1, 1, 1, 1, 80, "bf16", 1.0),
    (1, 1, 1, 1, 64, "bf16", 1.0),
    # scores of std ~6 (log2 units): the running maximum is raised mid-row
    # and O in tensor memory rescaled
    (2, 50, 320, 4, 64, "bf16", 4.0),
    (2, 50, 320, 4, 80, "bf16", 4.0),
    (2, 20, 80, 4, 64, "fp32", 1.0),      # tiny
    (1, 3, 5, 2, 32, "fp32", 1.0),
])
def test_attention(rows, n_q, T, heads, dh, dtype, q_std):
    D = heads * dh
    q = synth.tensor((rows, n_q, D), 21, std=q_std, dtype=dtype)
    k = synth.tensor((rows, T, D), 22, dtype=dtype)
    v = synth.tensor((rows, T, D), 23, dtype=dtype)
    o = empty((rows, n_q, D), dtype)
    lm.lazymar_attention(DT[dtype], dev(q, dtype), dev(k, dtype), dev(v, dtype), o, rows, n_q, T, heads, dh)
    sync()
    ref = np.stack([O.attention(q[r], k[r], v[r], heads) for r in range(rows)])
    assert max_rel(host(o), ref) < (1e-2 if dtype == "bf16" else 1e-5)


# --------------------------------------------------------------------------
# LayerNorm (gathering rows)
# --------------------------------------------------------------------------

@pytest.mark.parametrize("M,D,gather,dtype", [(100, 768, False, "bf16"), (50, 1280, True, "bf16"),
                                              (80, 256, True, "fp32"), (3, 1024, False, "fp32")])
def test_layernorm(M, D, gather, dtype):
    R = M + 30
    x = synth.tensor((R, D), 31, std=2.0, mean=0.5)
    g = synth.tensor((D,), 32, std=0.1, mean=1.0, dtype=dtype)
    b = synth.tensor((D,), 33, std=0.1, dtype=dtype)
    rm = synth.distinct_rows(M, R, 34) if gather else None
    y = empty((M, D), dtype)
    lm.lazymar_layernorm(DT[dtype], dev(x), None if rm is None else dev_int(rm), dev(g, dtype), dev(b, dtype), y,
                         M, D, 1e-6)
    sync()
    src = x[rm] if gather else x[:M]
    assert max_rel(host(y), O.layer_norm(src, g, b, 1e-6)) < (1e-2 if dtype == "bf16" else 1e-5)


def test_gelu_epilogue_matches_erf_gelu():
    """The MLP epilogue's GELU (the normal tail as 2^P(|x|), P a fitted degree-5
    polynomial, within 2.8e-7 max(1, |x|) in fp32) against the oracle's fp64
    erf GELU. An fp32 GEMM with W = I makes the pre-activation exactly the
    input, on a dense grid over [-8, 8]."""
    M, K = 512, 64
    x = np.linspace(-8.0, 8.0, M * K, dtype=np.float32).reshape(M, K)
    out = empty((M, K), "fp32")
    lm.lazymar_linear(DT["fp32"], lm.LAZYMAR_EPI_GELU, dev(x), dev(np.eye(K, dtype=np.float32)), None, M, K, K,
                      out, K)
    sync()
    err = np.abs(host(out) - O.gelu(x.astype(np.float64)))
    assert (err <= 1e-6 * np.maximum(1.0, np.abs(x))).all(), float(err.max())


# --------------------------------------------------------------------------
# Failure detection: a bounded device wait that runs out
# --------------------------------------------------------------------------

def test_bounded_wait_expires_and_device_stays_usable():
    """The self-test kernel waits 50 ms on an mbarrier nothing completes: the
    wait gives up, the host reads LAZYMAR_ERR_TIMEOUT (then the word is clear),
    and kernels launched afterwards still run correctly."""
    import time
    lm.lazymar_device_check()
    t0 = time.perf_counter()
    lm.lazymar_selftest_wait(50000)
    with pytest.raises(lm.LazymarError) as e:
        lm.lazymar_device_check()
    assert e.value.status == 5                       # LAZYMAR_ERR_TIMEOUT
    assert time.perf_counter() - t0 < 10
    lm.lazymar_device_check()                        # reported once, then clear
    _linear_case("bf16", lm.LAZYMAR_EPI_BIAS, 200, 256, 128, 1, seed=5)
    lm.lazymar_device_check()

