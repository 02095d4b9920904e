"""Python binding of the FeatFix C ABI (include/featfix.h, include/featfix_ops.h).

Argument marshalling only: every computation runs in libfeatfix.so's CUDA
kernels.  Functions carry the C names (``featfix_create``, ``featfix_step``,
...); tensors are passed as device pointers (``tensor.data_ptr()``), so
PyTorch serves for device memory and streams.  The library is loaded on first
use and a missing build raises: there is no fallback path.
"""

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libfeatfix.so")

# enums of featfix.h
OK, ERR_INVALID_ARG, ERR_SCHEDULE, ERR_STATE, ERR_OOM, ERR_CUDA, ERR_UNSUPPORTED = range(7)
MODES = {"featfix": 0, "verify": 1, "exact_only": 2, "vanilla": 3}
ARCH = {"dit": 0, "mmdit": 1}
DTYPE = {"f32": 0, "bf16": 1}
SAMPLER = {"euler": 0, "ddim": 1}
PLAN_EXACT, PLAN_DRAFT, PLAN_SITE = 0, 1, 2
FLAG_TAYLOR_RECURSIVE = 1
FLAG_PER_BLOCK_DRAFT = 2
FLAG_SITE_UPDATES_HISTORY = 4
FLAG_FUSED_LN = 8
MASK_NONE, MASK_TOKENS, MASK_CHANNELS = 0, 1, 2
KCLASS = {"gemm": 0, "attention": 1, "draft": 2, "verify": 3, "other": 4}


class FeatFixError(RuntimeError):
    def __init__(self, status, msg):
        super().__init__("featfix status %d: %s" % (status, msg))
        self.status = status


class ModelDesc(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in (
        "arch", "n_dual", "n_single", "hidden", "heads", "head_dim", "mlp", "in_ch", "out_ch", "patch",
        "patch_t", "lat_f", "lat_h", "lat_w", "txt_tokens", "n_classes", "batch", "cfg")] + [
        ("cfg_scale", ctypes.c_float), ("rope_dims", ctypes.c_int), ("dtype", ctypes.c_int),
        ("sampler", ctypes.c_int)]


class Site(ctypes.Structure):
    _fields_ = [("step", ctypes.c_int), ("layer", ctypes.c_int)]


class SiteLog(ctypes.Structure):
    _fields_ = [("step", ctypes.c_int), ("layer", ctypes.c_int), ("rel_l1", ctypes.c_double),
                ("rel_l2", ctypes.c_double), ("norm_l1_f", ctypes.c_double), ("norm_l2_f", ctypes.c_double)]


class Counters(ctypes.Structure):
    _fields_ = [("refresh_steps", ctypes.c_int), ("paid_checks", ctypes.c_int), ("forwarded", ctypes.c_int),
                ("steps_done", ctypes.c_int)]


_VP = ctypes.c_void_p
_I = ctypes.c_int
_LL = ctypes.c_longlong
_D = ctypes.c_double
_P = ctypes.POINTER

# name -> (restype, argtypes); every symbol declared in include/*.h
SIGNATURES = {
    "featfix_weight_count": (_I, [_P(ModelDesc)]),
    "featfix_create": (_I, [_P(ModelDesc), _P(_VP), _I, _VP, _P(_VP)]),
    "featfix_set_schedule": (_I, [_VP, _I, _P(_I), _I, _I, _P(Site), _I, _I, ctypes.c_uint]),
    "featfix_step": (_I, [_VP, _VP, _I, _VP]),
    "featfix_sample": (_I, [_VP, ctypes.c_ulonglong, _I, _VP, _VP]),
    "featfix_sample_host": (_I, [_VP, ctypes.c_ulonglong, _I, _VP, _VP]),
    "featfix_get_log": (_I, [_VP, _P(SiteLog), _I, _P(_I), _P(Counters)]),
    "featfix_get_plan": (_I, [_VP, _P(ctypes.c_ubyte), _P(_I), _P(_D)]),
    "featfix_plan_build": (_I, [_I, _I, _P(_I), _I, _I, _P(Site), _I, _I, ctypes.c_uint, _P(ctypes.c_ubyte),
                                _P(_I), _P(_D)]),
    "featfix_set_forward_mask": (_I, [_VP, _I, _P(ctypes.c_ubyte), _I]),
    "featfix_plan_build_blocks": (_I, [_I, _I, _P(_I), _I, _I, _P(Site), _I, _I, ctypes.c_uint, _P(_I), _P(_D)]),
    "featfix_debug_capture": (_I, [_VP, _I, _I, _VP, _VP]),
    "featfix_debug_block": (_I, [_VP, _I, _I, _VP, _VP, _VP]),
    "featfix_debug_capture_history": (_I, [_VP, _I, _I, _P(_VP), _I]),
    "featfix_debug_watchdog_probe": (_I, [_VP, ctypes.c_ulonglong]),
    "featfix_token_row": (_LL, [_P(ModelDesc), _I, _I]),
    "featfix_kernel_timing": (_I, [_VP, _I, _I]),
    "featfix_kernel_time": (_I, [_VP, _I, _P(_D), _P(_LL), _P(_D)]),
    "featfix_launch_count": (_LL, []),
    "featfix_last_error": (ctypes.c_char_p, [_VP]),
    "featfix_status_string": (ctypes.c_char_p, [_I]),
    "featfix_destroy": (None, [_VP]),
    "featfix_op_draft": (_I, [_I, _VP, _P(_VP), _P(_D), _I, _LL, _VP]),
    "featfix_op_verify_workspace": (ctypes.c_size_t, [_LL]),
    "featfix_op_verify": (_I, [_I, _VP, _P(_VP), _P(_D), _I, _VP, _LL, _I, _VP, _VP, ctypes.c_size_t, _VP]),
    "featfix_op_verify_noalloc": (_I, [_I, _VP, _P(_VP), _P(_D), _I, _VP, _LL, _I, _VP, _VP]),
    "featfix_op_ln_modulate": (_I, [_I, _VP, _VP, _LL, _I, _VP, _VP, _I, _I, _VP]),
    "featfix_op_gemm": (_I, [_I, _I, _I, _I, _VP, _VP, _VP, _I, _VP, _I, _I, _VP, _VP, _VP, _VP, _VP]),
    "featfix_op_attention": (_I, [_I, _VP, _I, _VP, _I, _I, _I, _I, _I, _I, _VP]),
}

_lib = None


def lib():
    """The loaded library (raises when it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise FeatFixError(ERR_UNSUPPORTED, "libfeatfix.so is not built; run __graft_entry__.build()")
        L = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            fn = getattr(L, name)
            fn.restype = res
            fn.argtypes = args
        _lib = L
    return _lib


def _ptr(t):
    """Device (or host) address of a tensor / ndarray / int; None -> NULL."""
    if t is None:
        return None
    if isinstance(t, int):
        return t
    if hasattr(t, "data_ptr"):
        return t.data_ptr()
    if hasattr(t, "ctypes"):
        return t.ctypes.data
    raise TypeError("cannot take the address of %r" % type(t))


def _stream_ptr(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(status, ctx=None):
    if status != OK:
        msg = lib().featfix_status_string(status).decode()
        if ctx is not None:
            detail = lib().featfix_last_error(ctx).decode()
            if detail:
                msg += ": " + detail
        raise FeatFixError(status, msg)


# ----------------------------------------------------------------------------
# model description and weight order
# ----------------------------------------------------------------------------

def model_desc(shape):
    """featfix_model_desc for a ``synthetic.ModelShape``-like object."""
    return ModelDesc(
        arch=ARCH[shape.arch], n_dual=shape.n_dual, n_single=shape.n_single, hidden=shape.hidden,
        heads=shape.heads, head_dim=shape.head_dim, mlp=shape.mlp, in_ch=shape.in_ch, out_ch=shape.out_ch,
        patch=shape.patch, patch_t=shape.patch_t, lat_f=shape.lat_f, lat_h=shape.lat_h, lat_w=shape.lat_w,
        txt_tokens=shape.txt_tokens, n_classes=shape.n_classes, batch=shape.batch, cfg=int(shape.cfg),
        cfg_scale=shape.cfg_scale, rope_dims=shape.rope_dims, dtype=DTYPE[shape.dtype],
        sampler=SAMPLER[shape.sampler])


def weight_spec(shape):
    """(name, dims) of every weight tensor in the order featfix_create takes them."""
    C, M = shape.hidden, shape.mlp
    P = (shape.patch_t if shape.lat_f > 0 else 1) * shape.patch * shape.patch
    spec = [("t_fc1.w", (C, 256)), ("t_fc1.b", (C,)), ("t_fc2.w", (C, C)), ("t_fc2.b", (C,))]
    if shape.arch == "dit":
        spec += [("y_emb", (shape.n_classes + 1, C)), ("x_emb.w", (C, shape.in_ch * P)), ("x_emb.b", (C,))]
    else:
        spec += [("img_in.w", (C, shape.in_ch * P)), ("img_in.b", (C,))]
    spec += [("final.mod.w", (2 * C, C)), ("final.mod.b", (2 * C,)),
             ("final.lin.w", (P * shape.out_ch, C)), ("final.lin.b", (P * shape.out_ch,))]
    if shape.arch == "dit":
        for l in range(shape.n_dual):
            p = "blk%d." % l
            spec += [(p + "mod.w", (6 * C, C)), (p + "mod.b", (6 * C,)), (p + "qkv.w", (3 * C, C)),
                     (p + "qkv.b", (3 * C,)), (p + "proj.w", (C, C)), (p + "proj.b", (C,)),
                     (p + "fc1.w", (M, C)), (p + "fc1.b", (M,)), (p + "fc2.w", (C, M)), (p + "fc2.b", (C,))]
        return spec
    for l in range(shape.n_dual):
        p = "dual%d." % l
        for s in ("img", "txt"):
            spec += [(p + s + "_mod.w", (6 * C, C)), (p + s + "_mod.b", (6 * C,))]
        for s in ("img", "txt"):
            spec += [(p + s + "_qkv.w", (3 * C, C)), (p + s + "_qkv.b", (3 * C,))]
        for s in ("img", "txt"):
            spec += [(p + s + "_proj.w", (C, C)), (p + s + "_proj.b", (C,))]
        for s in ("img", "txt"):
            spec += [(p + s + "_fc1.w", (M, C)), (p + s + "_fc1.b", (M,)),
                     (p + s + "_fc2.w", (C, M)), (p + s + "_fc2.b", (C,))]
    for j in range(shape.n_single):
        p = "single%d." % j
        spec += [(p + "mod.w", (3 * C, C)), (p + "mod.b", (3 * C,)), (p + "lin1.w", (3 * C + M, C)),
                 (p + "lin1.b", (3 * C + M,)), (p + "lin2.w", (C, C + M)), (p + "lin2.b", (C,))]
    return spec


def featfix_weight_count(shape):
    d = model_desc(shape)
    return lib().featfix_weight_count(ctypes.byref(d))


def featfix_token_row(shape, b, n):
    d = model_desc(shape)
    return lib().featfix_token_row(ctypes.byref(d), b, n)


# ----------------------------------------------------------------------------
# context API (same names as the C ABI)
# ----------------------------------------------------------------------------

def featfix_create(shape, weights, stream=None):
    """weights: dict name -> device tensor (or a list in weight_spec order)."""
    spec = weight_spec(shape)
    if isinstance(weights, dict):
        tensors = [weights[name] for name, _ in spec]
    else:
        tensors = list(weights)
    arr = (_VP * len(tensors))(*[_ptr(t) for t in tensors])
    d = model_desc(shape)
    out = _VP()
    _check(lib().featfix_create(ctypes.byref(d), arr, len(tensors), _stream_ptr(stream), ctypes.byref(out)))
    return out.value


def _sites_arr(sites):
    sites = list(sites)
    arr = (Site * max(len(sites), 1))(*[Site(int(i), int(l)) for (i, l) in sites])
    return arr, len(sites)


def featfix_set_schedule(ctx, steps, refresh, draft_order, sites, mode="featfix", flags=0):
    ref = (_I * len(refresh))(*[int(r) for r in refresh])
    sa, ns = _sites_arr(sites)
    m = MODES[mode] if isinstance(mode, str) else int(mode)
    _check(lib().featfix_set_schedule(ctx, int(steps), ref, len(refresh), int(draft_order), sa, ns, m, int(flags)),
           ctx)


def featfix_step(ctx, latent, step, cond):
    _check(lib().featfix_step(ctx, _ptr(latent), int(step), _ptr(cond)), ctx)


def featfix_sample(ctx, seed, steps, cond, latent_out):
    _check(lib().featfix_sample(ctx, int(seed), int(steps), _ptr(cond), _ptr(latent_out)), ctx)


def featfix_sample_host(ctx, seed, steps, cond_host, latent_out_host):
    _check(lib().featfix_sample_host(ctx, int(seed), int(steps), _ptr(cond_host), _ptr(latent_out_host)), ctx)


def featfix_get_log(ctx):
    """(list of dicts, counters dict)."""
    n = _I(0)
    cnt = Counters()
    _check(lib().featfix_get_log(ctx, None, 0, ctypes.byref(n), ctypes.byref(cnt)), ctx)
    logs = (SiteLog * max(n.value, 1))()
    _check(lib().featfix_get_log(ctx, logs, n.value, ctypes.byref(n), ctypes.byref(cnt)), ctx)
    out = [{"step": e.step, "layer": e.layer, "rel_l1": e.rel_l1, "rel_l2": e.rel_l2,
            "norm_l1_f": e.norm_l1_f, "norm_l2_f": e.norm_l2_f} for e in logs[:n.value]]
    return out, {"refresh_steps": cnt.refresh_steps, "paid_checks": cnt.paid_checks,
                 "forwarded": cnt.forwarded, "steps_done": cnt.steps_done}


def featfix_get_plan(ctx, steps, n_layers):
    import numpy as np
    kinds = np.zeros(steps * n_layers, dtype=np.uint8)
    keff = np.zeros(steps, dtype=np.int32)
    w = np.zeros(steps * 4, dtype=np.float64)
    _check(lib().featfix_get_plan(ctx, kinds.ctypes.data_as(_P(ctypes.c_ubyte)), keff.ctypes.data_as(_P(_I)),
                                  w.ctypes.data_as(_P(_D))), ctx)
    return kinds.reshape(steps, n_layers), keff, w.reshape(steps, 4)


def featfix_set_forward_mask(ctx, axis, mask=None):
    """Partial forwarding at FeatFix sites: axis MASK_TOKENS / MASK_CHANNELS
    with a 0/1 mask, or MASK_NONE (whole-block forwarding)."""
    import numpy as np
    if mask is None:
        _check(lib().featfix_set_forward_mask(ctx, int(axis), None, 0), ctx)
        return
    m = np.ascontiguousarray(np.asarray(mask, dtype=np.uint8))
    _check(lib().featfix_set_forward_mask(ctx, int(axis), m.ctypes.data_as(_P(ctypes.c_ubyte)), int(m.size)), ctx)


def featfix_plan_build_blocks(steps, n_layers, refresh, draft_order, sites, mode="featfix", flags=0):
    """Host-only per-block draft plan: (k_eff [steps, L], weights [steps, L, 4])."""
    import numpy as np
    ref = (_I * max(len(refresh), 1))(*[int(r) for r in refresh])
    sa, ns = _sites_arr(sites)
    keff = np.zeros(steps * n_layers, dtype=np.int32)
    w = np.zeros(steps * n_layers * 4, dtype=np.float64)
    m = MODES[mode] if isinstance(mode, str) else int(mode)
    _check(lib().featfix_plan_build_blocks(int(steps), int(n_layers), ref, len(refresh), int(draft_order), sa, ns, m,
                                           int(flags), keff.ctypes.data_as(_P(_I)), w.ctypes.data_as(_P(_D))))
    return keff.reshape(steps, n_layers), w.reshape(steps, n_layers, 4)


def featfix_plan_build(steps, n_layers, refresh, draft_order, sites, mode="featfix", flags=0):
    """Host-only plan: (kinds [steps, L] uint8, k_eff [steps], weights [steps, 4])."""
    import numpy as np
    ref = (_I * max(len(refresh), 1))(*[int(r) for r in refresh])
    sa, ns = _sites_arr(sites)
    kinds = np.zeros(steps * n_layers, dtype=np.uint8)
    keff = np.zeros(steps, dtype=np.int32)
    w = np.zeros(steps * 4, dtype=np.float64)
    m = MODES[mode] if isinstance(mode, str) else int(mode)
    _check(lib().featfix_plan_build(int(steps), int(n_layers), ref, len(refresh), int(draft_order), sa, ns, m,
                                    int(flags), kinds.ctypes.data_as(_P(ctypes.c_ubyte)),
                                    keff.ctypes.data_as(_P(_I)), w.ctypes.data_as(_P(_D))))
    return kinds.reshape(steps, n_layers), keff, w.reshape(steps, 4)


def featfix_debug_capture(ctx, step, layer, dev_in, dev_out):
    _check(lib().featfix_debug_capture(ctx, int(step), int(layer), _ptr(dev_in), _ptr(dev_out)), ctx)


def featfix_debug_capture_history(ctx, step, layer, dev_slots):
    arr = (_VP * len(dev_slots))(*[_ptr(t) for t in dev_slots])
    _check(lib().featfix_debug_capture_history(ctx, int(step), int(layer), arr, len(dev_slots)), ctx)


def featfix_debug_watchdog_probe(ctx, limit_ns):
    _check(lib().featfix_debug_watchdog_probe(ctx, int(limit_ns)), ctx)


def featfix_debug_block(ctx, step, layer, dev_in, dev_out, cond):
    _check(lib().featfix_debug_block(ctx, int(step), int(layer), _ptr(dev_in), _ptr(dev_out), _ptr(cond)), ctx)


def featfix_kernel_timing(ctx, kclass, on):
    k = KCLASS[kclass] if isinstance(kclass, str) else int(kclass)
    _check(lib().featfix_kernel_timing(ctx, k, int(bool(on))), ctx)


def featfix_kernel_time(ctx, kclass):
    """(total ms, launches, algorithmic work) since timing was switched on."""
    k = KCLASS[kclass] if isinstance(kclass, str) else int(kclass)
    ms, n, work = _D(0), _LL(0), _D(0)
    _check(lib().featfix_kernel_time(ctx, k, ctypes.byref(ms), ctypes.byref(n), ctypes.byref(work)), ctx)
    return ms.value, n.value, work.value


def featfix_launch_count():
    return int(lib().featfix_launch_count())


def featfix_destroy(ctx):
    if ctx:
        lib().featfix_destroy(ctx)


# ----------------------------------------------------------------------------
# kernels on caller buffers (featfix_ops.h)
# ----------------------------------------------------------------------------

def _dt(dtype):
    return DTYPE[dtype] if isinstance(dtype, str) else int(dtype)


def featfix_op_draft(dtype, x, hist, w, stream=None):
    hp = (_VP * len(hist))(*[_ptr(h) for h in hist])
    wa = (_D * len(hist))(*[float(v) for v in w])
    _check(lib().featfix_op_draft(_dt(dtype), _ptr(x), hp, wa, len(hist), x.numel(), _stream_ptr(stream)))


def featfix_op_verify_workspace(n):
    return int(lib().featfix_op_verify_workspace(int(n)))


def featfix_op_verify(dtype, u, hist, w, hf, sums, workspace, write_draft=False, stream=None):
    hp = (_VP * len(hist))(*[_ptr(h) for h in hist])
    wa = (_D * len(hist))(*[float(v) for v in w])
    _check(lib().featfix_op_verify(_dt(dtype), _ptr(u), hp, wa, len(hist), _ptr(hf), u.numel(), int(write_draft),
                                   _ptr(sums), _ptr(workspace), workspace.numel() * workspace.element_size(),
                                   _stream_ptr(stream)))


def featfix_op_verify_noalloc(dtype, u, hist, w, hf, sums, write_draft=False, stream=None):
    """featfix_op_verify with the library's fixed scratch array (no device
    allocation by anyone); see include/featfix_ops.h."""
    hp = (_VP * len(hist))(*[_ptr(h) for h in hist])
    wa = (_D * len(hist))(*[float(v) for v in w])
    _check(lib().featfix_op_verify_noalloc(_dt(dtype), _ptr(u), hp, wa, len(hist), _ptr(hf), u.numel(),
                                           int(write_draft), _ptr(sums), _stream_ptr(stream)))


def featfix_op_ln_modulate(dtype, x, out, rows, C, shift, scale, mod_stride, rows_per_batch, stream=None):
    _check(lib().featfix_op_ln_modulate(_dt(dtype), _ptr(x), _ptr(out), int(rows), int(C), _ptr(shift), _ptr(scale),
                                        int(mod_stride), int(rows_per_batch), _stream_ptr(stream)))


def featfix_op_gemm(dtype, a, w, out, bias=None, act=0, gate=None, gate_stride=0, rows_per_batch=0, resid=None,
                    hist_base=None, hist_out=None, stream=None):
    M, K = a.shape
    N = w.shape[0]
    _check(lib().featfix_op_gemm(_dt(dtype), int(M), int(N), int(K), _ptr(a), _ptr(w), _ptr(bias), int(act),
                                 _ptr(gate), int(gate_stride), int(rows_per_batch), _ptr(resid), _ptr(out),
                                 _ptr(hist_base), _ptr(hist_out), _stream_ptr(stream)))


def featfix_op_attention(dtype, qkv, out, batch, n_txt, n_img, heads, head_dim, stream=None):
    _check(lib().featfix_op_attention(_dt(dtype), _ptr(qkv), qkv.shape[-1], _ptr(out), out.shape[-1], int(batch),
                                      int(n_txt), int(n_img), int(heads), int(head_dim), _stream_ptr(stream)))


class FeatFix:
    """Owner of one featfix_ctx (convenience wrapper over the functions above)."""

    def __init__(self, shape, weights, stream=None):
        self.shape = shape
        self._weights = weights  # keep the borrowed device tensors alive
        self.ctx = featfix_create(shape, weights, stream)

    def set_schedule(self, steps, refresh, draft_order, sites, mode="featfix", flags=0):
        featfix_set_schedule(self.ctx, steps, refresh, draft_order, sites, mode, flags)

    def step(self, latent, i, cond):
        featfix_step(self.ctx, latent, i, cond)

    def sample(self, seed, steps, cond, latent_out):
        featfix_sample(self.ctx, seed, steps, cond, latent_out)

    def sample_host(self, seed, steps, cond_host, latent_out_host):
        featfix_sample_host(self.ctx, seed, steps, cond_host, latent_out_host)

    def log(self):
        return featfix_get_log(self.ctx)

    def close(self):
        if self.ctx:
            featfix_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
