"""ctypes binding of liblazymar.so (include/lazymar.h): same names, argument
marshalling only. Every step of the decoding path runs in the library's CUDA
kernels; there is no other implementation behind these functions.

Tensors are passed as torch tensors (device or host), numpy arrays (host) or
raw integer addresses; `None` becomes NULL. A non-OK status raises
LazymarError carrying the status and the library's message.
"""
import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "liblazymar.so")

LAZYMAR_F32, LAZYMAR_BF16, LAZYMAR_E4M3 = 0, 1, 2
LAZYMAR_CRITERION_VALUE, LAZYMAR_CRITERION_FEATURE = 0, 1
LAZYMAR_SELECT_LEAST_SIMILAR, LAZYMAR_SELECT_MOST_SIMILAR, LAZYMAR_SELECT_RANDOM = 0, 1, 2
LAZYMAR_CFG_GUIDE, LAZYMAR_CFG_REFRESH, LAZYMAR_CFG_REUSE = 0, 1, 2
LAZYMAR_EPI_BIAS, LAZYMAR_EPI_GELU, LAZYMAR_EPI_RESIDUAL, LAZYMAR_EPI_QKV, LAZYMAR_EPI_SILU = 0, 1, 2, 3, 4
KERNEL_CLASSES = ["gemm", "attention", "layernorm", "select", "embed", "cfg", "other"]
STATUS = {0: "LAZYMAR_OK", 1: "LAZYMAR_ERR_INVALID_ARG", 2: "LAZYMAR_ERR_OOM", 3: "LAZYMAR_ERR_CUDA",
          4: "LAZYMAR_ERR_STATE", 5: "LAZYMAR_ERR_TIMEOUT", 6: "LAZYMAR_ERR_UNSUPPORTED", 7: "LAZYMAR_ERR_DEVICE"}


class LazymarError(RuntimeError):
    def __init__(self, status, message):
        super().__init__("%s: %s" % (STATUS.get(status, status), message))
        self.status = status


class lazymar_config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in ("depth", "width", "heads", "mlp_ratio", "n_buffer", "n_img", "token_dim",
                                             "n_classes", "max_batch", "sel_layers", "dtype", "criterion")] + [
        ("ln_eps", ctypes.c_float), ("select_rule", ctypes.c_int), ("qkv_e4m3", ctypes.c_int)]


_FP = ctypes.c_void_p
BLOCK_FIELDS = ("ln1_g", "ln1_b", "w_qkv", "b_qkv", "w_o", "b_o", "ln2_g", "ln2_b", "w1", "b1", "w2", "b2")


class lazymar_block_weights(ctypes.Structure):
    _fields_ = [(n, _FP) for n in BLOCK_FIELDS]


class lazymar_weights(ctypes.Structure):
    _fields_ = [(n, _FP) for n in ("pos_emb", "class_emb", "mask_emb", "embed_w", "embed_b", "lnf_g", "lnf_b")] + [
        ("blocks", ctypes.POINTER(lazymar_block_weights))]


class lazymar_step_in(ctypes.Structure):
    _fields_ = [("latents", _FP), ("mask", _FP), ("labels", _FP), ("batch", ctypes.c_int),
                ("select_priority", _FP), ("select_keys", _FP)]


class lazymar_kernel_stats(ctypes.Structure):
    _fields_ = [("launches", ctypes.c_longlong), ("timed_launches", ctypes.c_longlong), ("ms", ctypes.c_double),
                ("flops", ctypes.c_double), ("bytes", ctypes.c_double)]


class lazymar_stats(ctypes.Structure):
    _fields_ = [("k", lazymar_kernel_stats * 7)]


class lazymar_head_config(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in ("token_dim", "cond_dim", "z_dtype", "width", "depth", "freq_dim",
                                            "n_train", "n_steps", "max_tokens")] + [("ln_eps", ctypes.c_float)]


HEAD_BLOCK_FIELDS = ("ada_w", "ada_b", "w1", "b1", "w2", "b2")


class lazymar_head_block_weights(ctypes.Structure):
    _fields_ = [(n, _FP) for n in HEAD_BLOCK_FIELDS]


HEAD_FIELDS_A = ("t_w1", "t_b1", "t_w2", "t_b2", "c_w", "c_b", "in_w", "in_b")
HEAD_FIELDS_B = ("f_ada_w", "f_ada_b", "out_w", "out_b")


class lazymar_head_weights(ctypes.Structure):
    _fields_ = [(n, _FP) for n in HEAD_FIELDS_A] + [("blocks", ctypes.POINTER(lazymar_head_block_weights))] + [
        (n, _FP) for n in HEAD_FIELDS_B]


_lib = None


def lib():
    """Load liblazymar.so (built in-tree by build.py). Fails loudly if absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError("liblazymar.so is not built (%s); run paper_2503_12450_gb300/build.py" % LIB_PATH)
    L = ctypes.CDLL(LIB_PATH)
    st, vp, i, f, sz = ctypes.c_int, ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
    sig = {
        "lazymar_create": (st, [ctypes.POINTER(lazymar_config), ctypes.POINTER(lazymar_weights),
                                ctypes.POINTER(vp)]),
        "lazymar_destroy": (None, [vp]),
        "lazymar_full_step": (st, [vp, ctypes.POINTER(lazymar_step_in), f, vp, vp, vp]),
        "lazymar_cached_step": (st, [vp, ctypes.POINTER(lazymar_step_in), i, i, f, vp, vp, vp, vp, vp]),
        "lazymar_select_tokens": (st, [i, vp, vp, i, i, i, i, vp, vp]),
        "lazymar_select_tokens_noalloc": (st, [i, vp, vp, i, i, i, i, vp, vp]),
        "lazymar_select_tokens_ex": (st, [i, vp, vp, i, i, i, i, i, vp, vp, vp, vp]),
        "lazymar_cfg_combine": (st, [i, i, vp, vp, vp, f, sz, vp, vp, vp]),
        "lazymar_linear": (st, [i, i, vp, vp, vp, i, i, i, vp, i, vp, vp, vp, i, vp]),
        "lazymar_attention": (st, [i, vp, vp, vp, vp, i, i, i, i, i, vp]),
        "lazymar_linear_e4m3": (st, [i, vp, vp, vp, vp, i, i, i, vp, i, vp, vp, vp, i, vp]),
        "lazymar_quantize_e4m3": (st, [vp, i, i, vp, vp, vp]),
        "lazymar_layernorm": (st, [i, vp, vp, vp, vp, vp, i, i, f, vp]),
        "lazymar_plan_step": (i, [i, i, i, i, i]),
        "lazymar_sync": (st, [vp, vp]),
        "lazymar_read_reference": (st, [vp, i, vp, vp]),
        "lazymar_device_check": (st, [vp]),
        "lazymar_selftest_wait": (st, [i, vp]),
        "lazymar_set_profiling": (st, [vp, i]),
        "lazymar_set_graphs": (st, [vp, i]),
        "lazymar_get_stats": (st, [vp, ctypes.POINTER(lazymar_stats)]),
        "lazymar_reset_stats": (st, [vp]),
        "lazymar_status_string": (ctypes.c_char_p, [i]),
        "lazymar_last_error": (ctypes.c_char_p, []),
        "lazymar_head_create": (st, [ctypes.POINTER(lazymar_head_config), ctypes.POINTER(lazymar_head_weights),
                                     ctypes.POINTER(vp)]),
        "lazymar_head_destroy": (None, [vp]),
        "lazymar_head_sample": (st, [vp, vp, i, i, vp, i, vp, f, f, vp, vp]),
        "lazymar_head_eval": (st, [vp, vp, i, i, vp, i, vp, i, vp, vp]),
        "lazymar_head_counters": (st, [vp, ctypes.POINTER(ctypes.c_longlong), ctypes.POINTER(ctypes.c_double)]),
        "lazymar_head_sync": (st, [vp, vp]),
        "lazymar_head_schedule": (st, [i, i, vp, vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    _lib = L
    return L


def _check(status):
    if status != 0:
        raise LazymarError(status, lib().lazymar_last_error().decode())


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    if hasattr(x, "ctypes"):
        return x.ctypes.data
    raise TypeError("cannot take the address of %r" % type(x))


def _stream(stream):
    if stream is None:
        try:
            import torch
            if torch.cuda.is_available():
                return torch.cuda.current_stream().cuda_stream
        except ImportError:
            pass
        return None
    return stream if isinstance(stream, int) else stream.cuda_stream


# ---------------------------------------------------------------------------
# Entry points (same names as the C ABI)
# ---------------------------------------------------------------------------

def lazymar_create(cfg, weights):
    """cfg: dict with the lazymar_config fields (dtype 'fp32'/'bf16' or int,
    criterion 'value'/'feature' or int, max_batch); weights: dict of fp32 numpy
    arrays or torch tensors as produced by synth.make_weights. Returns a Handle."""
    c = lazymar_config()
    for n, _ in lazymar_config._fields_:
        if n in ("dtype", "criterion", "ln_eps", "select_rule", "qkv_e4m3"):
            continue
        setattr(c, n, int(cfg[n] if n != "max_batch" else cfg.get("max_batch", cfg.get("batch"))))
    dt = cfg["dtype"]
    c.dtype = {"fp32": LAZYMAR_F32, "bf16": LAZYMAR_BF16}.get(dt, dt)
    cr = cfg.get("criterion", "value")
    c.criterion = {"value": LAZYMAR_CRITERION_VALUE, "feature": LAZYMAR_CRITERION_FEATURE}.get(cr, cr)
    c.ln_eps = float(cfg.get("ln_eps", 1e-6))
    sr = cfg.get("select_rule", LAZYMAR_SELECT_LEAST_SIMILAR)
    c.select_rule = {"least_similar": LAZYMAR_SELECT_LEAST_SIMILAR, "most_similar": LAZYMAR_SELECT_MOST_SIMILAR,
                     "random": LAZYMAR_SELECT_RANDOM}.get(sr, sr)
    c.qkv_e4m3 = int(bool(cfg.get("qkv_e4m3", 0)))
    keep = []

    def p(a):
        if hasattr(a, "data_ptr"):
            keep.append(a)
            return a.data_ptr()
        import numpy as np
        a = np.ascontiguousarray(a, dtype=np.float32)
        keep.append(a)
        return a.ctypes.data

    w = lazymar_weights()
    for n in ("pos_emb", "class_emb", "mask_emb", "embed_w", "embed_b", "lnf_g", "lnf_b"):
        setattr(w, n, p(weights[n]))
    blocks = (lazymar_block_weights * len(weights["blocks"]))()
    for i, bw in enumerate(weights["blocks"]):
        for n in BLOCK_FIELDS:
            setattr(blocks[i], n, p(bw[n]))
    w.blocks = blocks
    h = ctypes.c_void_p()
    _check(lib().lazymar_create(ctypes.byref(c), ctypes.byref(w), ctypes.byref(h)))
    return Handle(h.value, c)


def _step_in(latents, mask, labels, batch, select_priority=None, select_keys=None):
    return lazymar_step_in(_ptr(latents), _ptr(mask), _ptr(labels), int(batch), _ptr(select_priority),
                           _ptr(select_keys))


def lazymar_full_step(h, latents, mask, labels, batch, gamma, z_out=None, guided_out=None, stream=None):
    si = _step_in(latents, mask, labels, batch)
    _check(lib().lazymar_full_step(h.ptr, ctypes.byref(si), float(gamma), _ptr(z_out), _ptr(guided_out),
                                   _stream(stream)))


def lazymar_cached_step(h, latents, mask, labels, batch, n_compute, use_cond_cache, gamma, idx_in=None, idx_out=None,
                        z_out=None, guided_out=None, stream=None, select_priority=None, select_keys=None):
    si = _step_in(latents, mask, labels, batch, select_priority, select_keys)
    _check(lib().lazymar_cached_step(h.ptr, ctypes.byref(si), int(n_compute), int(bool(use_cond_cache)),
                                     float(gamma), _ptr(idx_in), _ptr(idx_out), _ptr(z_out), _ptr(guided_out),
                                     _stream(stream)))


def lazymar_select_tokens(dtype, v_cur, v_cache, rows, T, D, n_compute, idx_out, stream=None):
    _check(lib().lazymar_select_tokens(int(dtype), _ptr(v_cur), _ptr(v_cache), int(rows), int(T), int(D),
                                       int(n_compute), _ptr(idx_out), _stream(stream)))


def lazymar_select_tokens_ex(dtype, v_cur, v_cache, rows, T, D, n_compute, rule, priority, keys, idx_out,
                             stream=None):
    _check(lib().lazymar_select_tokens_ex(int(dtype), _ptr(v_cur), _ptr(v_cache), int(rows), int(T), int(D),
                                          int(n_compute), int(rule), _ptr(priority), _ptr(keys), _ptr(idx_out),
                                          _stream(stream)))


def lazymar_select_tokens_noalloc(dtype, v_cur, v_cache, rows, T, D, n_compute, idx_out, stream=None):
    _check(lib().lazymar_select_tokens_noalloc(int(dtype), _ptr(v_cur), _ptr(v_cache), int(rows), int(T), int(D),
                                               int(n_compute), _ptr(idx_out), _stream(stream)))


def lazymar_cfg_combine(dtype, mode, z_cond, z_uncond, delta, gamma, n, z_uncond_out=None, guided_out=None,
                        stream=None):
    _check(lib().lazymar_cfg_combine(int(dtype), int(mode), _ptr(z_cond), _ptr(z_uncond), _ptr(delta), float(gamma),
                                     int(n), _ptr(z_uncond_out), _ptr(guided_out), _stream(stream)))


def lazymar_linear(dtype, epilogue, a, w, bias, M, N, K, out, ldo, k_out=None, v_out=None, row_map=None, flags=0,
                   stream=None):
    _check(lib().lazymar_linear(int(dtype), int(epilogue), _ptr(a), _ptr(w), _ptr(bias), int(M), int(N), int(K),
                                _ptr(out), int(ldo), _ptr(k_out), _ptr(v_out), _ptr(row_map), int(flags),
                                _stream(stream)))


def lazymar_linear_e4m3(epilogue, a, w, wscale, bias, M, N, K, out, ldo, k_out=None, v_out=None, row_map=None,
                        flags=0, stream=None):
    _check(lib().lazymar_linear_e4m3(int(epilogue), _ptr(a), _ptr(w), _ptr(wscale), _ptr(bias), int(M), int(N),
                                     int(K), _ptr(out), int(ldo), _ptr(k_out), _ptr(v_out), _ptr(row_map), int(flags),
                                     _stream(stream)))


def lazymar_quantize_e4m3(w, rows, cols, q, scale, stream=None):
    _check(lib().lazymar_quantize_e4m3(_ptr(w), int(rows), int(cols), _ptr(q), _ptr(scale), _stream(stream)))


def lazymar_attention(dtype, q, k, v, o, rows, n_q, T, heads, head_dim, stream=None):
    _check(lib().lazymar_attention(int(dtype), _ptr(q), _ptr(k), _ptr(v), _ptr(o), int(rows), int(n_q), int(T),
                                   int(heads), int(head_dim), _stream(stream)))


def lazymar_layernorm(dtype, x, row_map, g, b, y, M, D, eps, stream=None):
    _check(lib().lazymar_layernorm(int(dtype), _ptr(x), _ptr(row_map), _ptr(g), _ptr(b), _ptr(y), int(M), int(D),
                                   float(eps), _stream(stream)))


def lazymar_plan_step(k, k0, tau, tau_cfg, use_cond_cache=True):
    """Returns (full, cond_reuse) for decoding step k."""
    r = lib().lazymar_plan_step(int(k), int(k0), int(tau), int(tau_cfg), int(bool(use_cond_cache)))
    if r < 0:
        raise LazymarError(1, "invalid schedule arguments")
    return bool(r & 1), bool(r & 2)


def lazymar_sync(h, stream=None):
    _check(lib().lazymar_sync(h.ptr, _stream(stream)))


def lazymar_read_reference(h, rows, dst, stream=None):
    _check(lib().lazymar_read_reference(h.ptr, int(rows), _ptr(dst), _stream(stream)))


def lazymar_selftest_wait(limit_us, stream=None):
    _check(lib().lazymar_selftest_wait(int(limit_us), _stream(stream)))


def lazymar_device_check(stream=None):
    _check(lib().lazymar_device_check(_stream(stream)))


def lazymar_set_profiling(h, enable):
    _check(lib().lazymar_set_profiling(h.ptr, int(bool(enable))))


def lazymar_set_graphs(h, enable):
    _check(lib().lazymar_set_graphs(h.ptr, int(bool(enable))))


def lazymar_get_stats(h):
    s = lazymar_stats()
    _check(lib().lazymar_get_stats(h.ptr, ctypes.byref(s)))
    return {name: dict(launches=s.k[i].launches, timed_launches=s.k[i].timed_launches, ms=s.k[i].ms,
                       flops=s.k[i].flops, bytes=s.k[i].bytes) for i, name in enumerate(KERNEL_CLASSES)}


def lazymar_reset_stats(h):
    _check(lib().lazymar_reset_stats(h.ptr))


def lazymar_head_create(hc, cond_dim, token_dim, weights, max_tokens, z_dtype="bf16"):
    """hc: dict with width, depth, freq_dim, n_train, n_steps (synth.head_config);
    weights: dict as produced by synth.make_head_weights. Returns a HeadHandle."""
    c = lazymar_head_config(int(token_dim), int(cond_dim),
                            {"fp32": LAZYMAR_F32, "bf16": LAZYMAR_BF16}.get(z_dtype, z_dtype), int(hc["width"]),
                            int(hc["depth"]), int(hc["freq_dim"]), int(hc["n_train"]), int(hc["n_steps"]),
                            int(max_tokens), float(hc.get("ln_eps", 1e-6)))
    keep = []

    def p(a):
        if hasattr(a, "data_ptr"):
            keep.append(a)
            return a.data_ptr()
        import numpy as np
        a = np.ascontiguousarray(a, dtype=np.float32)
        keep.append(a)
        return a.ctypes.data

    w = lazymar_head_weights()
    for n in HEAD_FIELDS_A + HEAD_FIELDS_B:
        setattr(w, n, p(weights[n]))
    blocks = (lazymar_head_block_weights * len(weights["blocks"]))()
    for i, bw in enumerate(weights["blocks"]):
        for n in HEAD_BLOCK_FIELDS:
            setattr(blocks[i], n, p(bw[n]))
    w.blocks = blocks
    h = ctypes.c_void_p()
    _check(lib().lazymar_head_create(ctypes.byref(c), ctypes.byref(w), ctypes.byref(h)))
    return HeadHandle(h.value, c)


def lazymar_head_sample(hd, z, B, n_img, pos, n_new, noise, gamma, temperature, x_out, stream=None):
    _check(lib().lazymar_head_sample(hd.ptr, _ptr(z), int(B), int(n_img), _ptr(pos), int(n_new), _ptr(noise),
                                     float(gamma), float(temperature), _ptr(x_out), _stream(stream)))


def lazymar_head_eval(hd, z, B, n_img, pos, n_new, x, j, out, stream=None):
    _check(lib().lazymar_head_eval(hd.ptr, _ptr(z), int(B), int(n_img), _ptr(pos), int(n_new), _ptr(x), int(j),
                                   _ptr(out), _stream(stream)))


def lazymar_head_counters(hd):
    n, f = ctypes.c_longlong(), ctypes.c_double()
    _check(lib().lazymar_head_counters(hd.ptr, ctypes.byref(n), ctypes.byref(f)))
    return n.value, f.value


def lazymar_head_schedule(n_train, n_steps):
    """(kept steps int32 [n_steps], constants float32 [n_steps, 4]) as the head computes them."""
    import numpy as np
    kept = np.zeros(n_steps, np.int32)
    consts = np.zeros((n_steps, 4), np.float32)
    _check(lib().lazymar_head_schedule(int(n_train), int(n_steps), kept.ctypes.data, consts.ctypes.data))
    return kept, consts


def lazymar_head_sync(hd, stream=None):
    _check(lib().lazymar_head_sync(hd.ptr, _stream(stream)))


class HeadHandle:
    """Owns a lazymar_head; destroyed with the object or by close()."""

    def __init__(self, ptr, cfg):
        self.ptr = ptr
        self.cfg = cfg

    def close(self):
        if self.ptr:
            lib().lazymar_head_destroy(self.ptr)
            self.ptr = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def lazymar_status_string(status):
    return lib().lazymar_status_string(int(status)).decode()


class Handle:
    """Owns a lazymar_handle; destroyed with the object or by close()."""

    def __init__(self, ptr, cfg):
        self.ptr = ptr
        self.cfg = cfg

    def close(self):
        if self.ptr:
            lib().lazymar_destroy(self.ptr)
            self.ptr = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
