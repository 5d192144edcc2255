"""fp64 CPU oracle for the ResNet-18 dual-batch training step (arXiv 2509.26092).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  It shares no code
with the CUDA library and never imports it.

The functions here are thin numpy wrappers over ``dbl_oracle.c`` (plain loops
in double precision); see that file for the definitions and the paper passage
each one follows.
"""
import ctypes
import os

import numpy as np

from . import build as _build

_lib = None

_D = ctypes.POINTER(ctypes.c_double)
_I32 = ctypes.POINTER(ctypes.c_int32)
_i = ctypes.c_int
_i64 = ctypes.c_int64
_d = ctypes.c_double


def lib():
    """Load (building on first use) the oracle shared library."""
    global _lib
    if _lib is None:
        path = _build.build()
        L = ctypes.CDLL(path)
        conv = [_D, _D, _D] + [_i] * 9
        for name in ("orc_conv2d_fwd", "orc_conv2d_dgrad", "orc_conv2d_wgrad"):
            getattr(L, name).argtypes = conv
            getattr(L, name).restype = None
        for name in ("orc_conv2d_fwd_at", "orc_conv2d_dgrad_at", "orc_conv2d_wgrad_at"):
            getattr(L, name).argtypes = [_D, _D] + [_i] * 13
            getattr(L, name).restype = _d
        L.orc_round_bf16.argtypes = [_d]
        L.orc_round_bf16.restype = _d
        L.orc_round_bf16_array.argtypes = [_D, _i64]
        L.orc_round_f16.argtypes = [_d]
        L.orc_round_f16.restype = _d
        L.orc_round_f16_array.argtypes = [_D, _i64]
        L.orc_ps_merge_scaled.argtypes = [_D, _D, _D, _D, _i64, _d, _d, _d, _d, _i, _d, _d]
        L.orc_ps_merge_scaled.restype = _i
        L.orc_loss_scale_update.argtypes = [_D, ctypes.POINTER(ctypes.c_int), _i, _i]
        L.orc_loss_scale_update.restype = None
        L.orc_bn_fwd.argtypes = [_D, _i64, _i, _D, _D, _d, _D, _i, _D, _D, _D]
        L.orc_bn_bwd.argtypes = [_D, _D, _D, _i, _D, _i64, _i, _D, _D, _D, _D, _D, _D, _D]
        L.orc_maxpool_fwd.argtypes = [_D, _i, _i, _i, _i, _i, _i, _i, _D, _I32]
        L.orc_maxpool_bwd.argtypes = [_D, _I32, _i, _i, _i, _i, _i, _i, _i, _D]
        L.orc_avgpool_fwd.argtypes = [_D, _i, _i, _i, _D]
        L.orc_avgpool_bwd.argtypes = [_D, _i, _i, _i, _D]
        L.orc_fc_fwd.argtypes = [_D, _D, _D, _i, _i, _i, _D]
        L.orc_fc_bwd.argtypes = [_D, _D, _D, _i, _i, _i, _D, _D, _D]
        L.orc_softmax_ce.argtypes = [_D, _I32, _i, _i, _D]
        L.orc_softmax_ce.restype = _d
        L.orc_ps_merge.argtypes = [_D, _D, _D, _D, _i64, _d, _d, _d, _d, _i]
        _U64 = ctypes.POINTER(ctypes.c_uint64)
        L.orc_philox4x64_10.argtypes = [_U64, _U64, _U64]
        L.orc_philox4x64_10.restype = None
        L.orc_dropout_mask.argtypes = [_i, _i, _d, ctypes.c_uint64, ctypes.c_uint64, ctypes.POINTER(ctypes.c_uint8)]
        L.orc_dropout_mask.restype = None
        L.orc_dropout_apply.argtypes = [_D, ctypes.POINTER(ctypes.c_uint8), _i64, _d, _D]
        L.orc_dropout_apply.restype = None
        L.orc_resize_taps.argtypes = [_i, _i, _I32, _I32, _D]
        L.orc_resize_taps.restype = _i
        L.orc_bilinear_resize.argtypes = [_D, _i, _i, _i, _i, _D, _i, _i]
        L.orc_bilinear_resize.restype = _i
        _lib = L
    return _lib


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


def _p(a):
    return None if a is None else a.ctypes.data_as(_D)


def _pi(a):
    return None if a is None else a.ctypes.data_as(_I32)


def out_dim(n, k, stride, pad):
    return (n + 2 * pad - k) // stride + 1


# --------------------------------------------------------------------------- bf16
def round_bf16(a):
    """Round-to-nearest-even onto the bfloat16 grid (returned as float64)."""
    a = _f64(a).copy()
    lib().orc_round_bf16_array(_p(a), a.size)
    return a


def round_f16(a):
    """Round-to-nearest-even onto the IEEE binary16 grid (returned as float64)."""
    a = _f64(a).copy()
    lib().orc_round_f16_array(_p(a), a.size)
    return a


# --------------------------------------------------------------------------- conv
def conv2d_fwd(x, w, stride, pad):
    """x [N,H,W,C], w [K,R,S,C] -> y [N,P,Q,K] (cross-correlation, zero padding)."""
    x, w = _f64(x), _f64(w)
    N, H, W, C = x.shape
    K, R, S, C2 = w.shape
    assert C == C2
    y = np.empty((N, out_dim(H, R, stride, pad), out_dim(W, S, stride, pad), K))
    lib().orc_conv2d_fwd(_p(x), _p(w), _p(y), N, H, W, C, K, R, S, stride, pad)
    return y


def conv2d_dgrad(dy, w, x_shape, stride, pad):
    """Adjoint of conv2d_fwd in its input: dy [N,P,Q,K] -> dx [N,H,W,C]."""
    dy, w = _f64(dy), _f64(w)
    N, H, W, C = x_shape
    K, R, S, _ = w.shape
    dx = np.empty((N, H, W, C))
    lib().orc_conv2d_dgrad(_p(dy), _p(w), _p(dx), N, H, W, C, K, R, S, stride, pad)
    return dx


def conv2d_wgrad(x, dy, w_shape, stride, pad):
    """Adjoint of conv2d_fwd in its weights: -> dw [K,R,S,C]."""
    x, dy = _f64(x), _f64(dy)
    N, H, W, C = x.shape
    K, R, S, _ = w_shape
    dw = np.empty((K, R, S, C))
    lib().orc_conv2d_wgrad(_p(x), _p(dy), _p(dw), N, H, W, C, K, R, S, stride, pad)
    return dw


def conv2d_fwd_at(x, w, stride, pad, n, p, q, k):
    N, H, W, C = x.shape
    K, R, S, _ = w.shape
    return lib().orc_conv2d_fwd_at(_p(x), _p(w), N, H, W, C, K, R, S, stride, pad, n, p, q, k)


def conv2d_dgrad_at(dy, w, x_shape, stride, pad, n, h, ww, c):
    N, H, W, C = x_shape
    K, R, S, _ = w.shape
    return lib().orc_conv2d_dgrad_at(_p(dy), _p(w), N, H, W, C, K, R, S, stride, pad, n, h, ww, c)


def conv2d_wgrad_at(x, dy, w_shape, stride, pad, k, r, s, c):
    N, H, W, C = x.shape
    K, R, S, _ = w_shape
    return lib().orc_conv2d_wgrad_at(_p(x), _p(dy), N, H, W, C, K, R, S, stride, pad, k, r, s, c)


# --------------------------------------------------------------------------- BN
def bn_fwd(y, gamma, beta, eps=1e-5, res=None, relu=True):
    """Training-mode BatchNorm over all rows of y [..., C]; returns (out, mean, invstd)."""
    y = _f64(y)
    C = y.shape[-1]
    M = y.size // C
    out = np.empty_like(y)
    mean, invstd = np.empty(C), np.empty(C)
    res = None if res is None else _f64(res)
    lib().orc_bn_fwd(_p(y), M, C, _p(_f64(gamma)), _p(_f64(beta)), eps, _p(res), int(relu), _p(out), _p(mean),
                     _p(invstd))
    return out, mean, invstd


def bn_bwd(dout, out, y, gamma, mean, invstd, relu=True, dout2=None, want_dres=False):
    """Backward of bn_fwd; returns (dy, dgamma, dbeta, dres or None)."""
    dout, out, y = _f64(dout), _f64(out), _f64(y)
    C = y.shape[-1]
    M = y.size // C
    dy = np.empty_like(y)
    dres = np.empty_like(y) if want_dres else None
    dg, db = np.empty(C), np.empty(C)
    d2 = None if dout2 is None else _f64(dout2)
    lib().orc_bn_bwd(_p(dout), _p(d2), _p(out), int(relu), _p(y), M, C, _p(_f64(gamma)), _p(_f64(mean)),
                     _p(_f64(invstd)), _p(dy), _p(dres), _p(dg), _p(db))
    return dy, dg, db, dres


# --------------------------------------------------------------------------- pooling / head
def maxpool_fwd(x, k=3, stride=2, pad=1):
    x = _f64(x)
    N, H, W, C = x.shape
    P, Q = out_dim(H, k, stride, pad), out_dim(W, k, stride, pad)
    y = np.empty((N, P, Q, C))
    arg = np.empty((N, P, Q, C), dtype=np.int32)
    lib().orc_maxpool_fwd(_p(x), N, H, W, C, k, stride, pad, _p(y), _pi(arg))
    return y, arg


def maxpool_bwd(dy, arg, x_shape, k=3, stride=2, pad=1):
    dy = _f64(dy)
    arg = np.ascontiguousarray(arg, dtype=np.int32)
    N, H, W, C = x_shape
    dx = np.empty((N, H, W, C))
    lib().orc_maxpool_bwd(_p(dy), _pi(arg), N, H, W, C, k, stride, pad, _p(dx))
    return dx


def avgpool_fwd(x):
    x = _f64(x)
    N, H, W, C = x.shape
    f = np.empty((N, C))
    lib().orc_avgpool_fwd(_p(x), N, H * W, C, _p(f))
    return f


def avgpool_bwd(df, x_shape):
    df = _f64(df)
    N, H, W, C = x_shape
    dx = np.empty((N, H, W, C))
    lib().orc_avgpool_bwd(_p(df), N, H * W, C, _p(dx))
    return dx


def philox4x64_10(counter, key):
    """Philox4x64-10 of a 4-word counter and 2-word key (uint64 words) -> 4 uint64 words."""
    c = np.ascontiguousarray(counter, dtype=np.uint64)
    k = np.ascontiguousarray(key, dtype=np.uint64)
    out = np.empty(4, dtype=np.uint64)
    U = ctypes.POINTER(ctypes.c_uint64)
    lib().orc_philox4x64_10(c.ctypes.data_as(U), k.ctypes.data_as(U), out.ctypes.data_as(U))
    return out


def dropout_mask(N, C, d, seed, step):
    """keep [N, C] uint8 (1 = kept) of the dropout before the FC layer (see dbl_oracle.c)."""
    keep = np.empty((N, C), dtype=np.uint8)
    lib().orc_dropout_mask(N, C, float(d), int(seed), int(step), keep.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8)))
    return keep


def dropout_apply(x, keep, d):
    """keep * x / (1 - d), elementwise (forward of the features, backward of their gradient)."""
    x = _f64(x)
    keep = np.ascontiguousarray(keep, dtype=np.uint8)
    assert keep.shape == x.shape
    out = np.empty_like(x)
    lib().orc_dropout_apply(_p(x), keep.ctypes.data_as(ctypes.POINTER(ctypes.c_uint8)), x.size, float(d), _p(out))
    return out


def fc_fwd(f, Wt, b):
    f, Wt, b = _f64(f), _f64(Wt), _f64(b)
    N, C = f.shape
    J = Wt.shape[0]
    out = np.empty((N, J))
    lib().orc_fc_fwd(_p(f), _p(Wt), _p(b), N, C, J, _p(out))
    return out


def fc_bwd(dl, f, Wt):
    dl, f, Wt = _f64(dl), _f64(f), _f64(Wt)
    N, C = f.shape
    J = Wt.shape[0]
    dW, db, df = np.empty((J, C)), np.empty(J), np.empty((N, C))
    lib().orc_fc_bwd(_p(dl), _p(f), _p(Wt), N, C, J, _p(dW), _p(db), _p(df))
    return dW, db, df


def softmax_ce(logits, labels):
    """Mean softmax cross-entropy and its gradient (already divided by the batch)."""
    logits = _f64(logits)
    labels = np.ascontiguousarray(labels, dtype=np.int32)
    N, J = logits.shape
    dl = np.empty_like(logits)
    loss = lib().orc_softmax_ce(_p(logits), _pi(labels), N, J, _p(dl))
    return loss, dl


# --------------------------------------------------------------------------- merge
def ps_merge(w, u, g_large, g_small, lr, momentum, f_large, f_small, order=0):
    """Dual-batch parameter-server merge; returns new (w, u).  See orc_ps_merge."""
    w, u = _f64(w).copy(), _f64(u).copy()
    gl = None if g_large is None else _f64(g_large)
    gs = None if g_small is None else _f64(g_small)
    lib().orc_ps_merge(_p(w), _p(u), _p(gl), _p(gs), w.size, lr, momentum, f_large, f_small, order)
    return w, u


def ps_merge_scaled(w, u, g_large, g_small, lr, momentum, f_large, f_small, order, scale_large, scale_small):
    """The merge of pushes made under loss scaling (see orc_ps_merge_scaled): returns new
    (w, u, applied); applied is False (and w, u unchanged) when a pushed value is not finite."""
    w, u = _f64(w).copy(), _f64(u).copy()
    gl = None if g_large is None else _f64(g_large)
    gs = None if g_small is None else _f64(g_small)
    ok = lib().orc_ps_merge_scaled(_p(w), _p(u), _p(gl), _p(gs), w.size, lr, momentum, f_large, f_small, order,
                                   float(scale_large), float(scale_small))
    return w, u, bool(ok)


def loss_scale_update(scale, good, found_inf, interval):
    """One step of the dynamic loss scale; returns (scale, good)."""
    s_ = ctypes.c_double(scale)
    g_ = ctypes.c_int(good)
    lib().orc_loss_scale_update(ctypes.byref(s_), ctypes.byref(g_), int(bool(found_inf)), int(interval))
    return s_.value, g_.value


# --------------------------------------------------------------------------- resize
def resize_taps(n_in, n_out):
    i0 = np.empty(n_out, dtype=np.int32)
    i1 = np.empty(n_out, dtype=np.int32)
    lam = np.empty(n_out)
    rc = lib().orc_resize_taps(n_in, n_out, _pi(i0), _pi(i1), _p(lam))
    if rc != 0:
        raise ValueError("bad resize sizes")
    return i0, i1, lam


def bilinear_resize(x, h_out, w_out):
    x = _f64(x)
    N, H, W, C = x.shape
    out = np.empty((N, h_out, w_out, C))
    if lib().orc_bilinear_resize(_p(x), N, H, W, C, _p(out), h_out, w_out) != 0:
        raise MemoryError("oracle resize")
    return out


def threads():
    """Number of OpenMP threads the oracle library uses."""
    return int(os.environ.get("OMP_NUM_THREADS", os.cpu_count() or 1))
