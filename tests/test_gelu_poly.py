"""The GELU constants compiled into the kernels, checked on the CPU.

The polynomial in csrc/lazymar_internal.cuh is evaluated here with the
kernels' fp32 operation order (csrc/gen_gelu_poly.py) and compared with the
exact erf GELU from scipy, which is independent of both the generator's fit
and the oracle.
"""
import importlib.util
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2503_12450_gb300", "csrc")


def _header_coeffs():
    text = open(os.path.join(CSRC, "lazymar_internal.cuh")).read()
    found = dict(re.findall(r"constexpr float kGeluP(\d) = ([-+0-9.eE]+)f;", text))
    return np.array([np.float32(found[str(k)]) for k in range(len(found))], dtype=np.float32)


def _generator():
    spec = importlib.util.spec_from_file_location("gen_gelu_poly", os.path.join(CSRC, "gen_gelu_poly.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_gelu_polynomial_constants_within_bound():
    scipy_special = pytest.importorskip("scipy.special")
    c = _header_coeffs()
    assert len(c) == 6
    gen = _generator()
    x = np.linspace(-12, 12, 200001).astype(np.float32)
    ref = 0.5 * x.astype(np.float64) * (1.0 + scipy_special.erf(x.astype(np.float64) / np.sqrt(2.0)))
    got = gen.gelu_fp32(x, c)
    assert (np.abs(got - ref) <= 3e-7 * np.maximum(1.0, np.abs(x))).all()
    # special values: GELU(0) = 0, odd part, NaN propagates, large |x|
    z = gen.gelu_fp32(np.array([0.0, np.nan, 1e4, -1e4], dtype=np.float32), c)
    assert abs(z[0]) < 1e-7 and np.isnan(z[1]) and abs(z[2] - 1e4) < 1e-3 and abs(z[3]) < 1e-6
