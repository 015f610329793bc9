"""Generates the GELU polynomial of lazymar_internal.cuh (run by hand; numpy + scipy).

GELU(x) = x Phi(x) = max(x, 0) - |x| h(|x|), h(u) = Phi(-u) = erfc(u / sqrt 2) / 2.
The kernels evaluate h(u) = 2^P(u) with P a degree-5 polynomial fitted to
log2 h on u in [0, 6] (u clamped to 6 above, where h < 1e-9). The fit is a
weighted least-squares on Chebyshev nodes, reweighted towards minimax
(Lawson's iteration), with weights |x| h ln 2 / max(1, |x|): the sensitivity
of GELU(x) / max(1, |x|) to an error in P. The script prints the coefficients
and the worst error of the fp32 evaluation the kernels perform over
x in [-12, 12].
"""
import numpy as np
from scipy.special import erf, erfc

DEG, UMAX = 5, 6.0


def fit():
    n = 4000
    u = (np.cos(np.pi * (np.arange(n) + 0.5) / n) + 1.0) * UMAX / 2.0
    h = 0.5 * erfc(u / np.sqrt(2.0))
    target = np.log2(h)
    w = np.maximum(np.maximum(u, 1e-3) * h * np.log(2.0) / np.maximum(u, 1.0), 1e-12)
    V = np.vander(u, DEG + 1, increasing=True)
    ww = w.copy()
    c, *_ = np.linalg.lstsq(V * ww[:, None], target * ww, rcond=None)
    for _ in range(30):
        err = np.abs(V @ c - target) * w
        ww = ww * np.maximum(err / err.max(), 1e-3) ** 0.5
        c, *_ = np.linalg.lstsq(V * ww[:, None], target * ww, rcond=None)
    return c.astype(np.float32)


def f32(v):
    return np.float32(v)


def gelu_fp32(x, c):
    """The kernels' arithmetic, one fp32 rounding per (fused) operation."""
    u = np.minimum(np.abs(x), f32(UMAX)).astype(np.float32)
    p = np.full_like(u, c[-1])
    for k in range(DEG - 1, -1, -1):
        p = (p.astype(np.float64) * u + np.float64(c[k])).astype(np.float32)
    h = np.exp2(p.astype(np.float64)).astype(np.float32)
    relu = (f32(0.5) * (x + np.abs(x)).astype(np.float32)).astype(np.float32)
    return (relu.astype(np.float64) - u.astype(np.float64) * h).astype(np.float32)


def max_error(c):
    x = np.linspace(-12, 12, 400001).astype(np.float32)
    ref = 0.5 * x.astype(np.float64) * (1.0 + erf(x.astype(np.float64) / np.sqrt(2.0)))
    return float(np.max(np.abs(gelu_fp32(x, c) - ref) / np.maximum(1.0, np.abs(x))))


if __name__ == "__main__":
    c = fit()
    for k, v in enumerate(c):
        print("  constexpr float kGeluP%d = %.9ef;" % (k, v))
    print("max |error| / max(1, |x|) = %.2e" % max_error(c))
