"""Helpers of the GPU parity tests: device tensors, the tolerance metrics and
the configuration dict the binding takes."""
import numpy as np
import pytest

from paper_2503_12450_gb300 import build
from paper_2503_12450_gb300 import lazymar as lm

# Tolerances: max |gpu - oracle| / max |oracle| per tensor (bf16 2e-2, fp32
# 1e-4), and the per-token cosine of final features >= 0.999.
TOL = {"bf16": 2e-2, "fp32": 1e-4}
COS_MIN = 0.999
DT = {"bf16": lm.LAZYMAR_BF16, "fp32": lm.LAZYMAR_F32}

_built = False


def torch_cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.fail("a CUDA GPU is required for tests marked gpu")
    global _built
    if not _built:
        build.build()
        lm.lib()
        _built = True
    return torch


def dev(x, dtype="fp32"):
    torch = torch_cuda()
    t = torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).cuda()
    return t.to(torch.bfloat16) if dtype == "bf16" else t


def dev_int(x):
    torch = torch_cuda()
    return torch.from_numpy(np.ascontiguousarray(x)).cuda()


def empty(shape, dtype="fp32"):
    torch = torch_cuda()
    return torch.empty(shape, device="cuda", dtype=torch.bfloat16 if dtype == "bf16" else torch.float32)


def host(t):
    return t.float().cpu().numpy().astype(np.float64)


def sync():
    torch_cuda().cuda.synchronize()
    lm.lazymar_device_check()


def max_rel(gpu, ref):
    ref = np.asarray(ref, np.float64)
    return float(np.max(np.abs(np.asarray(gpu, np.float64) - ref)) / max(np.max(np.abs(ref)), 1e-30))


def guided_ok(g_gpu, g_ref, z_ref, gamma, tol):
    """The guided output u + gamma (c - u) is a linear map of the features, so
    the feature tolerance propagates to it: max |dg| <= tol * (|gamma| max|c| +
    |1 - gamma| max|u|), with z_ref = [c; u] the oracle's features of the pair."""
    c, u = np.asarray(z_ref[0], np.float64), np.asarray(z_ref[1], np.float64)
    bound = tol * (abs(gamma) * np.abs(c).max() + abs(1.0 - gamma) * np.abs(u).max())
    err = float(np.abs(np.asarray(g_gpu, np.float64) - np.asarray(g_ref, np.float64)).max())
    return err <= bound


def min_cos(gpu, ref):
    a = np.asarray(gpu, np.float64).reshape(-1, np.shape(gpu)[-1])
    b = np.asarray(ref, np.float64).reshape(-1, np.shape(ref)[-1])
    num = (a * b).sum(-1)
    den = np.sqrt((a * a).sum(-1) * (b * b).sum(-1))
    return float(np.min(num / np.maximum(den, 1e-300)))


def binding_cfg(cfg, max_batch=None):
    c = dict(cfg)
    c["max_batch"] = max_batch or cfg["batch"]
    return c
