"""The C-ABI library without a GPU: it builds, loads, exports every entry point
include/lazymar.h declares, and its host-only logic (schedule, argument
checks, status strings) behaves as documented. No compute call is made."""
import ctypes
import os
import re

import pytest

import oracle as O
from paper_2503_12450_gb300 import build
from paper_2503_12450_gb300 import lazymar as lm

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    build.build()
    return lm.lib()


def declared_functions():
    text = open(os.path.join(ROOT, "include", "lazymar.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(lazymar_[a-z_]+)\s*\(", text)))


def test_exports_every_declared_symbol(lib):
    names = declared_functions()
    assert len(names) >= 15
    raw = ctypes.CDLL(lm.LIB_PATH)
    missing = [n for n in names if not hasattr(raw, n)]
    assert not missing, missing
    # and the binding exposes the same names
    assert not [n for n in names if not hasattr(lm, n)
                and n not in ("lazymar_destroy", "lazymar_last_error", "lazymar_head_destroy")]


@pytest.mark.parametrize("k0,tau,tau_cfg,cond", [(4, 9, 9, True), (4, 9, 2, True), (3, 5, 5, True),
                                                  (4, 9, 0, True), (4, 9, 9, False), (0, 1, 1, True)])
def test_plan_step_matches_oracle_schedule(lib, k0, tau, tau_cfg, cond):
    for k in range(64):
        assert lm.lazymar_plan_step(k, k0, tau, tau_cfg, cond) == O.plan(k, k0, tau, tau_cfg, cond)


def test_plan_step_rejects_bad_arguments(lib):
    assert lib.lazymar_plan_step(-1, 4, 9, 9, 1) == -1
    assert lib.lazymar_plan_step(3, 4, 0, 9, 1) == -1
    assert lib.lazymar_plan_step(3, 4, 9, -1, 1) == -1


def test_status_strings(lib):
    for s in range(8):
        assert lm.lazymar_status_string(s) not in ("", "unknown status")
    assert lm.lazymar_status_string(99) == "unknown status"


def _cfg(**kw):
    c = dict(depth=2, width=256, heads=4, mlp_ratio=4, n_buffer=16, n_img=64, token_dim=16, n_classes=1000,
             max_batch=1, sel_layers=1, dtype="fp32", criterion="value", ln_eps=1e-6)
    c.update(kw)
    return c


@pytest.mark.parametrize("bad,status", [(dict(sel_layers=0), 1), (dict(sel_layers=3), 1), (dict(width=200), 6),
                                        (dict(width=384, heads=3), 6), (dict(heads=2, dtype="bf16"), 6),
                                        (dict(token_dim=65), 6), (dict(max_batch=0), 1), (dict(dtype=7), 1),
                                        (dict(select_rule=3), 1), (dict(qkv_e4m3=2), 1),
                                        (dict(qkv_e4m3=1), 6)])
def test_create_rejects_bad_configs_before_touching_the_device(lib, bad, status):
    with pytest.raises(lm.LazymarError) as e:
        _create_raw(lib, _cfg(**bad))
    assert e.value.status == status


def _create_raw(lib, cfg):
    c = lm.lazymar_config()
    for n, _ in lm.lazymar_config._fields_:
        if n not in ("dtype", "criterion", "ln_eps", "select_rule", "qkv_e4m3"):
            setattr(c, n, cfg[n])
    c.qkv_e4m3 = cfg.get("qkv_e4m3", 0)
    c.dtype = {"fp32": 0, "bf16": 1}.get(cfg["dtype"], cfg["dtype"])
    c.criterion = 0
    c.ln_eps = 1e-6
    c.select_rule = cfg.get("select_rule", 0)
    w = lm.lazymar_weights()
    blocks = (lm.lazymar_block_weights * 1)()
    w.blocks = blocks
    h = ctypes.c_void_p()
    lm._check(lib.lazymar_create(ctypes.byref(c), ctypes.byref(w), ctypes.byref(h)))


def test_null_arguments_are_rejected(lib):
    assert lib.lazymar_create(None, None, None) == 1
    si = lm.lazymar_step_in()
    assert lib.lazymar_full_step(None, ctypes.byref(si), 1.0, None, None, None) == 1
    assert lib.lazymar_cached_step(None, ctypes.byref(si), 1, 0, 1.0, None, None, None, None, None) == 1
    assert lib.lazymar_sync(None, None) == 1
    assert lib.lazymar_get_stats(None, None) == 1
    assert "NULL" in lm.lib().lazymar_last_error().decode()


@pytest.mark.parametrize("args,status", [
    ((1, 0, 0, 0, 0, 0, 128, 100, 64, 0, 128), 6),      # bf16 K % 64 != 0
    ((1, 0, 0, 0, 0, 0, 100, 64, 64, 0, 128), 6),       # bf16 N % 128 != 0
    ((0, 0, 0, 0, 0, 0, 6, 4, 4, 0, 6), 6),             # f32 N % 4 != 0
    ((1, 3, 0, 0, 0, 0, 128, 256, 64, 0, 0), 6),        # QKV needs N = 3D with D % 32 == 0 ... N=256 -> D=85
    ((1, 9, 0, 0, 0, 0, 128, 256, 64, 0, 256), 1),      # unknown epilogue
])
def test_linear_rejects_unsupported_shapes(lib, args, status):
    dtype, epi, a, w, b, _, M, N, K, _, ldo = args
    assert lib.lazymar_linear(dtype, epi, a, w, b, M, N, K, None, ldo, None, None, None, 0, None) == status


def test_component_argument_checks(lib):
    assert lib.lazymar_select_tokens(1, None, None, 2, 10, 12, 3, None, None) == 1      # D % 8
    assert lib.lazymar_select_tokens(1, None, None, 2, 10, 16, 11, None, None) == 1     # N > T
    assert lib.lazymar_select_tokens(5, None, None, 2, 10, 16, 3, None, None) == 1      # dtype
    assert lib.lazymar_select_tokens_ex(1, None, None, 2, 10, 16, 3, 3, None, None, None, None) == 1  # rule
    assert lib.lazymar_selftest_wait(0, None) == 1                                      # limit
    assert lib.lazymar_select_tokens_ex(1, None, None, 2, 10, 16, 11, 0, None, None, None, None) == 1  # N > T
    assert lib.lazymar_cfg_combine(1, 3, None, None, None, 1.0, 8, None, None, None) == 1
    assert lib.lazymar_attention(1, None, None, None, None, 1, 1, 1, 2, 96, None) == 6  # head width 96
    assert lib.lazymar_layernorm(1, None, None, None, None, None, 4, 200, 1e-6, None) == 6


def _head_cfg(**kw):
    c = dict(token_dim=16, cond_dim=768, z_dtype=lm.LAZYMAR_BF16, width=1024, depth=6, freq_dim=256, n_train=1000,
             n_steps=100, max_tokens=64, ln_eps=1e-6)
    c.update(kw)
    return lm.lazymar_head_config(*[c[n] for n, _ in lm.lazymar_head_config._fields_])


@pytest.mark.parametrize("bad,status", [
    (dict(width=1000), 6), (dict(width=0), 6), (dict(cond_dim=100), 6), (dict(freq_dim=200), 6),
    (dict(token_dim=0), 1), (dict(token_dim=65), 1), (dict(depth=0), 1), (dict(n_steps=0), 1),
    (dict(n_steps=1001), 1), (dict(max_tokens=0), 1), (dict(z_dtype=7), 1), (dict(ln_eps=0.0), 1),
])
def test_head_create_rejects_bad_configs_before_touching_the_device(lib, bad, status):
    w = lm.lazymar_head_weights()
    w.blocks = (lm.lazymar_head_block_weights * 1)()
    h = ctypes.c_void_p()
    assert lib.lazymar_head_create(ctypes.byref(_head_cfg(**bad)), ctypes.byref(w), ctypes.byref(h)) == status
    assert h.value is None


def test_head_null_arguments_are_rejected(lib):
    h = ctypes.c_void_p()
    assert lib.lazymar_head_create(None, None, ctypes.byref(h)) == 1
    assert lib.lazymar_head_sample(None, None, 1, 1, None, 1, None, 1.0, 1.0, None, None) == 1
    assert lib.lazymar_head_eval(None, None, 1, 1, None, 1, None, 0, None, None) == 1
    assert lib.lazymar_head_counters(None, None, None) == 1
    assert lib.lazymar_head_sync(None, None) == 1
    lib.lazymar_head_destroy(None)


@pytest.mark.parametrize("n_train,n_steps", [(1000, 100), (1000, 10), (1000, 1), (50, 50), (1001, 11), (4, 3), (6, 5)])
def test_head_schedule_matches_the_oracle(lib, n_train, n_steps):
    """The head's host-side schedule (kept steps, combined sampler constants)
    against the oracle's schedule: steps exact, constants to fp32 rounding."""
    import numpy as np
    from oracle import diffusion_head as HO
    kept, c = lm.lazymar_head_schedule(n_train, n_steps)
    s = HO.Schedule(n_train, n_steps)
    assert kept.tolist() == s.t.tolist()
    a_x = s.coef_x0 / np.sqrt(s.alpha_bar) + s.coef_xt          # mean = a_x x - a_eps eps
    a_eps = s.coef_x0 * np.sqrt(1.0 / s.alpha_bar - 1.0)
    np.testing.assert_allclose(c[:, 0], a_x, rtol=2e-6)
    np.testing.assert_allclose(c[:, 1], a_eps, rtol=2e-6)
    np.testing.assert_allclose(c[:, 2], np.log(s.beta), rtol=2e-6)
    np.testing.assert_allclose(c[:, 3], s.post_log_var, rtol=2e-6)


def test_head_schedule_rejects_bad_sizes(lib):
    assert lib.lazymar_head_schedule(10, 11, None, None) == 1
    assert lib.lazymar_head_schedule(0, 0, None, None) == 1
