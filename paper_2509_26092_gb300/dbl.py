"""ctypes binding of ``libdbl.so`` and ``libdbl_f16.so`` (see ``include/dbl.h``).

Argument marshalling only: every function here calls the C entry point of
the same name, passing device pointers, sizes and the CUDA stream.  Tensors
may be given as torch tensors (their ``data_ptr()`` is passed) or as raw
integer addresses.  A nonzero status raises ``DblError`` with the library's
error text.  There is no fallback: if the library is not built, importing
the functions fails.

The two libraries differ only in the 16-bit storage format (bfloat16, or
IEEE binary16); calls go to the bfloat16 one unless made inside
``with precision("f16"):``.
"""
import contextlib
import contextvars
import ctypes
import os

from . import build_lib

DBL_OK, DBL_ERR_INVALID, DBL_ERR_UNSUPPORTED, DBL_ERR_CUDA, DBL_ERR_TIMEOUT, DBL_ERR_WORKSPACE = 0, -1, -2, -3, -4, -5
DBL_F32, DBL_BF16 = 0, 1
DBL_PASS_FWD, DBL_PASS_DGRAD, DBL_PASS_WGRAD = 0, 1, 2


class DblError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__(f"libdbl error {code}: {msg}")
        self.code = code


class ConvShape(ctypes.Structure):
    _fields_ = [(f, ctypes.c_int32) for f in ("n", "h", "w", "c", "k", "r", "s", "stride", "pad", "stride_w", "pad_w")]


class ConvPlanInfo(ctypes.Structure):
    _fields_ = [("kernel", ctypes.c_int32), ("tile_cols", ctypes.c_int32), ("ctas_per_mma", ctypes.c_int32),
                ("tiles", ctypes.c_int32), ("zdim", ctypes.c_int32), ("grid", ctypes.c_int32),
                ("smem_bytes", ctypes.c_int64)]


DBL_KERNEL_IGEMM, DBL_KERNEL_WINDOW, DBL_KERNEL_WINDOW_WGRAD = 0, 1, 2


class BnShape(ctypes.Structure):
    _fields_ = [("count", ctypes.c_int64), ("c", ctypes.c_int32), ("eps", ctypes.c_float), ("relu", ctypes.c_int32)]


class HeadOpts(ctypes.Structure):
    _fields_ = [("drop_rate", ctypes.c_float), ("seed", ctypes.c_uint64), ("step", ctypes.c_void_p),
                ("loss_scale", ctypes.c_void_p)]


class LossScale(ctypes.Structure):
    """dbl_loss_scale: its device copy is a 4-element tensor (fp32 scale, int32 good, found_inf, skipped)."""
    _fields_ = [("scale", ctypes.c_float), ("good_steps", ctypes.c_int32), ("found_inf", ctypes.c_int32),
                ("skipped", ctypes.c_int32)]


class MergeParams(ctypes.Structure):
    _fields_ = [("lr", ctypes.c_float), ("momentum", ctypes.c_float), ("f_large", ctypes.c_float),
                ("f_small", ctypes.c_float), ("order", ctypes.c_int32)]


_libs = {}
_precision = contextvars.ContextVar("dbl_precision", default="bf16")
PRECISIONS = ("bf16", "f16")
_V = ctypes.c_void_p
_I32 = ctypes.c_int32
_I64 = ctypes.c_int64
_SZ = ctypes.c_size_t
_D = ctypes.c_double


def lib_path(p=None):
    return build_lib.library_path(p or _precision.get())


@contextlib.contextmanager
def precision(p):
    """Route the calls made inside the block to the library of storage format p ("bf16" or "f16")."""
    if p not in PRECISIONS:
        raise ValueError(f"precision must be one of {PRECISIONS}, not {p!r}")
    tok = _precision.set(p)
    try:
        yield
    finally:
        _precision.reset(tok)


def current_precision():
    return _precision.get()


def lib(p=None):
    """Load the library of storage format p (default: the current one); it must have been built
    by ``build_lib.build()``."""
    p = p or _precision.get()
    if p not in _libs:
        path = build_lib.library_path(p)
        if not os.path.exists(path):
            raise ImportError(f"{path} is missing: build it with paper_2509_26092_gb300.build_lib.build()")
        L = ctypes.CDLL(path)
        sig = {
            "dbl_last_error": (ctypes.c_char_p, []),
            "dbl_version": (ctypes.c_int, []),
            "dbl_kernel_launches": (_I64, []),
            "dbl_device_status": (ctypes.c_int, [ctypes.POINTER(_I32)]),
            "dbl_conv_workspace_bytes": (_SZ, [ctypes.POINTER(ConvShape), ctypes.c_int]),
            "dbl_conv_plan": (ctypes.c_int, [ctypes.POINTER(ConvShape), ctypes.c_int, ctypes.POINTER(ConvPlanInfo)]),
            "dbl_conv_fwd": (ctypes.c_int, [ctypes.POINTER(ConvShape), _V, _V, _V, _V, _V, _V, _SZ, _V]),
            "dbl_conv_dgrad": (ctypes.c_int, [ctypes.POINTER(ConvShape), _V, _V, _V, _V, _SZ, _V]),
            "dbl_conv_wgrad": (ctypes.c_int, [ctypes.POINTER(ConvShape), _V, _V, _V, ctypes.c_int, _V, _SZ, _V]),
            "dbl_conv_dgrad_proj": (ctypes.c_int, [ctypes.POINTER(ConvShape), _V, _V, _I32, _V, _V, _V, _V, _SZ, _V]),
            "dbl_conv_stats_parts_bytes": (_SZ, [ctypes.POINTER(ConvShape)]),
            "dbl_conv_fwd_parts": (ctypes.c_int, [ctypes.POINTER(ConvShape), _V, _V, _V, _V, _SZ,
                                                  ctypes.POINTER(_I32), _V]),
            "dbl_bn_relu_fused_parts": (ctypes.c_int, [ctypes.POINTER(BnShape), _V, _V, _I32] + [_V] * 7),
            "dbl_bn_stats": (ctypes.c_int, [ctypes.POINTER(BnShape), _V, _V, _V, _V]),
            "dbl_bn_relu_fused": (ctypes.c_int, [ctypes.POINTER(BnShape)] + [_V] * 10),
            "dbl_bn_workspace_bytes": (_SZ, [ctypes.POINTER(BnShape)]),
            "dbl_bn_relu_fused_bwd": (ctypes.c_int, [ctypes.POINTER(BnShape)] + [_V] * 13 + [_SZ, _V]),
            "dbl_bn_relu_fused_bwd_noalloc": (ctypes.c_int, [ctypes.POINTER(BnShape)] + [_V] * 13),
            "dbl_maxpool_fwd": (ctypes.c_int, [_I32] * 4 + [_V, _V, _V, _V]),
            "dbl_maxpool_bwd": (ctypes.c_int, [_I32] * 4 + [_V, _V, _V, _V, _V]),
            "dbl_bn_relu_maxpool_fwd": (ctypes.c_int, [ctypes.POINTER(BnShape), _I32, _I32, _I32] + [_V] * 10),
            "dbl_head_workspace_bytes": (_SZ, [_I32, _I32, _I32]),
            "dbl_head_fwd_bwd": (ctypes.c_int, [_I32] * 4 + [_V] * 8 + [_V, _SZ, _V]),
            "dbl_head_fwd_bwd_ex": (ctypes.c_int, [_I32] * 4 + [_V] * 4 + [ctypes.POINTER(HeadOpts)] + [_V] * 5
                                    + [_SZ, _V]),
            "dbl_ps_dual_batch_merge_scaled": (ctypes.c_int, [_V, _V, _V, _V, _V, _I64, ctypes.POINTER(MergeParams),
                                                              _V, _V, _V, _V]),
            "dbl_grads_finite": (ctypes.c_int, [_V, _I64, _V, _V]),
            "dbl_loss_scale_update": (ctypes.c_int, [_V, _I32, _V]),
            "dbl_dropout_mask": (ctypes.c_int, [_I32, _I32, ctypes.c_float, ctypes.c_uint64, _V, _V, _V]),
            "dbl_event_wait": (ctypes.c_int, [_V, _D]),
            "dbl_set_conv_pdl": (ctypes.c_int, [_I32]),
            "dbl_conv_test_stall_next": (ctypes.c_int, []),
            "dbl_hold": (ctypes.c_int, [_V, _D, _V, _V]),
            "dbl_ps_dual_batch_merge": (ctypes.c_int, [_V, _V, _V, _V, _V, _I64, ctypes.POINTER(MergeParams), _V]),
            "dbl_progressive_resize": (ctypes.c_int, [_V, ctypes.c_int, _I32, _I32, _I32, _I32, _V, ctypes.c_int,
                                                      _I32, _I32, _I32, _V]),
            "dbl_resize_taps": (ctypes.c_int, [_I32, _I32, _V, _V, _V]),
            "dbl_progressive_resize_stem": (ctypes.c_int, [_V, _I32, _I32, _I32, _I32, _V, _I32, _I32, _I32, _I32,
                                                           _I32, _I32, _I32, _I32, _V]),
            "dbl_zero_f32_2d": (ctypes.c_int, [_V, _I64, _I64, _I64, _V]),
            "dbl_progressive_resize_stem_u8": (ctypes.c_int, [_V, _I32, _I32, _I32, _I32, ctypes.POINTER(ctypes.c_float),
                                                              ctypes.POINTER(ctypes.c_float), _V, _I32, _I32, _I32,
                                                              _I32, _I32, _I32, _I32, _I32, _V]),
            "dbl_update_factor": (_D, [_D, _D, ctypes.c_int]),
            "dbl_plan": (ctypes.c_int, [_D, _D, _I32, _I32, _D, _D, _D, ctypes.c_int] + [ctypes.POINTER(_D)] * 4),
        }
        for name, (res, args) in sig.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _libs[p] = L
    return _libs[p]


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(rc):
    if rc != DBL_OK:
        raise DblError(rc, lib().dbl_last_error().decode(errors="replace"))


def dbl_last_error():
    return lib().dbl_last_error().decode(errors="replace")


def dbl_version():
    return lib().dbl_version()


def dbl_kernel_launches():
    """Kernel launches issued so far by the libraries loaded in this process (both formats)."""
    lib()
    return sum(L.dbl_kernel_launches() for L in _libs.values())


def dbl_device_status():
    """Synchronous: the device-side status words of the loaded libraries (DBL_OK, or the first
    DBL_ERR_TIMEOUT), then cleared."""
    lib()
    out = DBL_OK
    for p, L in _libs.items():
        v = _I32(0)
        rc = L.dbl_device_status(ctypes.byref(v))
        if rc != DBL_OK:
            raise DblError(rc, L.dbl_last_error().decode(errors="replace"))
        out = out if out != DBL_OK else v.value
    return out


def conv_shape(n, h, w, c, k, r, stride, pad, s=None, stride_w=0, pad_w=0):
    """dbl_conv_shape; s defaults to r, stride_w == 0 means the same stride and pad along W."""
    return ConvShape(n, h, w, c, k, r, r if s is None else s, stride, pad, stride_w, pad_w)


def dbl_conv_test_stall_next():
    """Test hook: the next implicit-GEMM convolution launch's block 0 never loads its first
    K-block, so its bounded MMA wait runs out and the device status reports DBL_ERR_TIMEOUT."""
    _check(lib().dbl_conv_test_stall_next())


def dbl_conv_workspace_bytes(shape, pass_):
    return lib().dbl_conv_workspace_bytes(ctypes.byref(shape), pass_)


def dbl_conv_plan(shape, pass_):
    """How the pass runs on the current device (host): a ConvPlanInfo."""
    info = ConvPlanInfo()
    _check(lib().dbl_conv_plan(ctypes.byref(shape), pass_, ctypes.byref(info)))
    return info


def dbl_conv_fwd(shape, x, w, y, ch_sum=None, ch_sumsq=None, ws=None, ws_bytes=0, stream=None):
    _check(lib().dbl_conv_fwd(ctypes.byref(shape), _ptr(x), _ptr(w), _ptr(y), _ptr(ch_sum), _ptr(ch_sumsq), _ptr(ws),
                              ws_bytes, _stream(stream)))


def dbl_conv_stats_parts_bytes(shape):
    return lib().dbl_conv_stats_parts_bytes(ctypes.byref(shape))


def dbl_conv_fwd_parts(shape, x, w, y, parts, parts_bytes, stream=None):
    """Returns the number of partial rows written to parts (see dbl_bn_relu_fused_parts)."""
    n = _I32(0)
    _check(lib().dbl_conv_fwd_parts(ctypes.byref(shape), _ptr(x), _ptr(w), _ptr(y), _ptr(parts), parts_bytes,
                                    ctypes.byref(n), _stream(stream)))
    return n.value


def dbl_bn_relu_fused_parts(shape, y, parts, nparts, gamma, beta, residual, out, save_mean, save_invstd,
                            stream=None):
    _check(lib().dbl_bn_relu_fused_parts(ctypes.byref(shape), _ptr(y), _ptr(parts), int(nparts), _ptr(gamma),
                                         _ptr(beta), _ptr(residual), _ptr(out), _ptr(save_mean), _ptr(save_invstd),
                                         _stream(stream)))


def dbl_conv_dgrad(shape, dy, w, dx, ws=None, ws_bytes=0, stream=None):
    _check(lib().dbl_conv_dgrad(ctypes.byref(shape), _ptr(dy), _ptr(w), _ptr(dx), _ptr(ws), ws_bytes,
                                _stream(stream)))


def dbl_conv_dgrad_proj(shape, dy, w, k2, dy2, w2, dx, ws=None, ws_bytes=0, stream=None):
    _check(lib().dbl_conv_dgrad_proj(ctypes.byref(shape), _ptr(dy), _ptr(w), int(k2), _ptr(dy2), _ptr(w2), _ptr(dx),
                                     _ptr(ws), ws_bytes, _stream(stream)))


def dbl_conv_wgrad(shape, x, dy, dw, accumulate=False, ws=None, ws_bytes=0, stream=None):
    _check(lib().dbl_conv_wgrad(ctypes.byref(shape), _ptr(x), _ptr(dy), _ptr(dw), int(bool(accumulate)), _ptr(ws),
                                ws_bytes, _stream(stream)))


def bn_shape(count, c, eps=1e-5, relu=True):
    return BnShape(count, c, eps, int(bool(relu)))


def dbl_bn_stats(shape, y, ch_sum, ch_sumsq, stream=None):
    _check(lib().dbl_bn_stats(ctypes.byref(shape), _ptr(y), _ptr(ch_sum), _ptr(ch_sumsq), _stream(stream)))


def dbl_bn_relu_fused(shape, y, ch_sum, ch_sumsq, gamma, beta, residual, out, save_mean, save_invstd, stream=None):
    _check(lib().dbl_bn_relu_fused(ctypes.byref(shape), _ptr(y), _ptr(ch_sum), _ptr(ch_sumsq), _ptr(gamma),
                                   _ptr(beta), _ptr(residual), _ptr(out), _ptr(save_mean), _ptr(save_invstd),
                                   _stream(stream)))


def dbl_bn_workspace_bytes(shape):
    return lib().dbl_bn_workspace_bytes(ctypes.byref(shape))


def dbl_bn_relu_fused_bwd(shape, dout, dout2, y, out, gamma, save_mean, save_invstd, dy, dresidual, dgamma, dbeta,
                          ws, ws_bytes, stream=None, beta=None):
    """out=None with shape.relu: the ReLU mask is recomputed from y (needs beta)."""
    _check(lib().dbl_bn_relu_fused_bwd(ctypes.byref(shape), _ptr(dout), _ptr(dout2), _ptr(y), _ptr(out), _ptr(gamma),
                                       _ptr(beta), _ptr(save_mean), _ptr(save_invstd), _ptr(dy), _ptr(dresidual),
                                       _ptr(dgamma), _ptr(dbeta), _ptr(ws), ws_bytes, _stream(stream)))


def dbl_bn_relu_fused_bwd_noalloc(shape, dout, dout2, y, out, gamma, save_mean, save_invstd, dy, dresidual, dgamma,
                                  dbeta, stream=None, beta=None):
    """dbl_bn_relu_fused_bwd without a workspace argument: the scratch is a fixed array inside
    the library (channels <= 512; calls must not overlap on the GPU)."""
    _check(lib().dbl_bn_relu_fused_bwd_noalloc(ctypes.byref(shape), _ptr(dout), _ptr(dout2), _ptr(y), _ptr(out),
                                               _ptr(gamma), _ptr(beta), _ptr(save_mean), _ptr(save_invstd), _ptr(dy),
                                               _ptr(dresidual), _ptr(dgamma), _ptr(dbeta), _stream(stream)))


def dbl_bn_relu_maxpool_fwd(shape, n, h, w, x, ch_sum, ch_sumsq, gamma, beta, save_mean, save_invstd, y, argmax,
                            stream=None):
    _check(lib().dbl_bn_relu_maxpool_fwd(ctypes.byref(shape), n, h, w, _ptr(x), _ptr(ch_sum), _ptr(ch_sumsq),
                                         _ptr(gamma), _ptr(beta), _ptr(save_mean), _ptr(save_invstd), _ptr(y),
                                         _ptr(argmax), _stream(stream)))


def dbl_maxpool_fwd(n, h, w, c, x, y, argmax, stream=None):
    _check(lib().dbl_maxpool_fwd(n, h, w, c, _ptr(x), _ptr(y), _ptr(argmax), _stream(stream)))


def dbl_maxpool_bwd(n, h, w, c, dy, dy2, argmax, dx, stream=None):
    _check(lib().dbl_maxpool_bwd(n, h, w, c, _ptr(dy), _ptr(dy2), _ptr(argmax), _ptr(dx), _stream(stream)))


def dbl_head_workspace_bytes(n, c, classes):
    return lib().dbl_head_workspace_bytes(n, c, classes)


def dbl_head_fwd_bwd(n, hw, c, classes, x, fc_w, fc_b, labels, loss, dfc_w, dfc_b, dx, ws, ws_bytes, stream=None):
    _check(lib().dbl_head_fwd_bwd(n, hw, c, classes, _ptr(x), _ptr(fc_w), _ptr(fc_b), _ptr(labels), _ptr(loss),
                                  _ptr(dfc_w), _ptr(dfc_b), _ptr(dx), _ptr(ws), ws_bytes, _stream(stream)))


def head_opts(drop_rate=0.0, seed=0, step=None, loss_scale=None):
    """dbl_head_opts: dropout of rate drop_rate (step: device uint64 counter, incremented by one on
    the stream after each call) and loss_scale (device fp32 pointer/tensor, or None)."""
    return HeadOpts(float(drop_rate), int(seed) & (2**64 - 1), _ptr(step), _ptr(loss_scale))


def dbl_head_fwd_bwd_ex(n, hw, c, classes, x, fc_w, fc_b, labels, opts, loss, dfc_w, dfc_b, dx, ws, ws_bytes,
                        stream=None):
    _check(lib().dbl_head_fwd_bwd_ex(n, hw, c, classes, _ptr(x), _ptr(fc_w), _ptr(fc_b), _ptr(labels),
                                     ctypes.byref(opts), _ptr(loss), _ptr(dfc_w), _ptr(dfc_b), _ptr(dx), _ptr(ws),
                                     ws_bytes, _stream(stream)))


def dbl_ps_dual_batch_merge_scaled(w, u, w16_out, g_large, g_small, n, lr, momentum, f_large, f_small, order,
                                   scale_large, scale_small, found_inf, stream=None):
    p = MergeParams(lr, momentum, f_large, f_small, order)
    _check(lib().dbl_ps_dual_batch_merge_scaled(_ptr(w), _ptr(u), _ptr(w16_out), _ptr(g_large), _ptr(g_small), n,
                                                ctypes.byref(p), _ptr(scale_large), _ptr(scale_small),
                                                _ptr(found_inf), _stream(stream)))


def dbl_grads_finite(g, n, found_inf, stream=None):
    _check(lib().dbl_grads_finite(_ptr(g), n, _ptr(found_inf), _stream(stream)))


def dbl_loss_scale_update(state, growth_interval, stream=None):
    _check(lib().dbl_loss_scale_update(_ptr(state), growth_interval, _stream(stream)))


def dbl_dropout_mask(n, c, drop_rate, seed, step, keep, stream=None):
    """keep [n, c] uint8: the mask dbl_head_fwd_bwd_ex draws for (drop_rate, seed, *step)."""
    _check(lib().dbl_dropout_mask(n, c, float(drop_rate), int(seed) & (2**64 - 1), _ptr(step), _ptr(keep),
                                  _stream(stream)))


def dbl_set_conv_pdl(mode):
    """Programmatic dependent launch of the convolutions that follow: 1 on, 0 off, -1 the
    environment's choice (DBL_CONV_PDL), in both storage formats' libraries."""
    for p in PRECISIONS:
        _check_lib(lib(p), lib(p).dbl_set_conv_pdl(int(mode)))


def _check_lib(L, rc):
    if rc != DBL_OK:
        raise DblError(rc, L.dbl_last_error().decode(errors="replace"))


def dbl_event_wait(event, timeout_s):
    """DBL_OK once the torch.cuda.Event (or raw cudaEvent_t) has completed, DBL_ERR_TIMEOUT if it
    has not after timeout_s seconds; other failures raise DblError."""
    handle = event.cuda_event if hasattr(event, "cuda_event") else event
    rc = lib().dbl_event_wait(ctypes.c_void_p(handle), float(timeout_s))
    if rc not in (DBL_OK, DBL_ERR_TIMEOUT):
        _check(rc)
    return rc


def dbl_hold(flag, timeout_s, status=None, stream=None):
    """Hold the stream until the pinned host uint32 `flag` is non-zero or timeout_s passes."""
    _check(lib().dbl_hold(_ptr(flag), float(timeout_s), _ptr(status), _stream(stream)))


def dbl_ps_dual_batch_merge(w, u, w16_out, g_large, g_small, n, lr, momentum, f_large, f_small, order=0,
                            stream=None):
    p = MergeParams(lr, momentum, f_large, f_small, order)
    _check(lib().dbl_ps_dual_batch_merge(_ptr(w), _ptr(u), _ptr(w16_out), _ptr(g_large), _ptr(g_small), n,
                                         ctypes.byref(p), _stream(stream)))


def dbl_progressive_resize(inp, in_dtype, n, h_in, w_in, c, out, out_dtype, h_out, w_out, c_out_stride, stream=None):
    _check(lib().dbl_progressive_resize(_ptr(inp), in_dtype, n, h_in, w_in, c, _ptr(out), out_dtype, h_out, w_out,
                                        c_out_stride, _stream(stream)))


def dbl_progressive_resize_stem(inp, n, h_in, w_in, c, out, h_out, w_out, taps, stride_w, pad_w, row_group=1,
                                pad_h=0, rows_out=None, stream=None):
    if rows_out is None:
        rows_out = h_out
    _check(lib().dbl_progressive_resize_stem(_ptr(inp), n, h_in, w_in, c, _ptr(out), h_out, w_out, taps, stride_w, pad_w,
                                             row_group, pad_h, rows_out, _stream(stream)))


def dbl_progressive_resize_stem_u8(inp, n, h_in, w_in, c, scale, bias, out, h_out, w_out, taps, stride_w, pad_w,
                                   row_group=1, pad_h=0, rows_out=None, stream=None):
    """8-bit images, standardized per channel as p*scale + bias (scale, bias: c floats)."""
    if rows_out is None:
        rows_out = h_out
    sc = (ctypes.c_float * c)(*[float(v) for v in scale])
    bi = (ctypes.c_float * c)(*[float(v) for v in bias])
    _check(lib().dbl_progressive_resize_stem_u8(_ptr(inp), n, h_in, w_in, c, sc, bi, _ptr(out), h_out, w_out, taps,
                                                stride_w, pad_w, row_group, pad_h, rows_out, _stream(stream)))


def dbl_zero_f32_2d(base, rows, cols, ld, stream=None):
    _check(lib().dbl_zero_f32_2d(_ptr(base), rows, cols, ld, _stream(stream)))


def dbl_resize_taps(n_in, n_out):
    import numpy as np
    i0 = np.empty(n_out, np.int32)
    i1 = np.empty(n_out, np.int32)
    lam = np.empty(n_out, np.float32)
    _check(lib().dbl_resize_taps(n_in, n_out, i0.ctypes.data, i1.ctypes.data, lam.ctypes.data))
    return i0, i1, lam


def dbl_update_factor(d_small, d_large, sqrt_scheme=False):
    return lib().dbl_update_factor(d_small, d_large, int(bool(sqrt_scheme)))


def dbl_plan(k, d, n_small, n_large, a, b, batch_large, sqrt_scheme=False):
    out = [_D(0) for _ in range(4)]
    _check(lib().dbl_plan(k, d, n_small, n_large, a, b, batch_large, int(bool(sqrt_scheme)),
                          *[ctypes.byref(o) for o in out]))
    return tuple(o.value for o in out)
