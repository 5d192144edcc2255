"""Pins for the oracle's convolution passes (forward, data and weight gradient).

The forward pass is pinned to a library routine (torch's fp64 CPU conv2d) and
to the unit-impulse closed form; the two gradients are pinned as the exact
adjoints of the forward map, by finite differences and by torch autograd.
"""
import numpy as np
import pytest
import torch

import oracle as orc

SHAPES = [  # N, H, W, C, K, R, stride, pad
    (2, 5, 5, 3, 4, 3, 1, 1),
    (1, 6, 7, 2, 3, 3, 2, 1),
    (2, 8, 8, 3, 2, 7, 2, 3),
    (2, 6, 6, 4, 5, 1, 2, 0),
    (1, 4, 4, 8, 8, 3, 1, 1),
]


def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


def _torch_conv(x, w, st, pad):
    xt = torch.from_numpy(x).permute(0, 3, 1, 2)
    wt = torch.from_numpy(w).permute(0, 3, 1, 2)
    return torch.nn.functional.conv2d(xt, wt, stride=st, padding=pad).permute(0, 2, 3, 1).numpy()


@pytest.mark.parametrize("shape", SHAPES)
def test_fwd_matches_torch(shape):
    N, H, W, C, K, R, st, pad = shape
    x, w = _rand((N, H, W, C), 1), _rand((K, R, R, C), 2)
    np.testing.assert_allclose(orc.conv2d_fwd(x, w, st, pad), _torch_conv(x, w, st, pad), rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("shape", SHAPES)
def test_grads_match_torch_autograd(shape):
    N, H, W, C, K, R, st, pad = shape
    x, w = _rand((N, H, W, C), 3), _rand((K, R, R, C), 4)
    xt = torch.from_numpy(x).permute(0, 3, 1, 2).requires_grad_()
    wt = torch.from_numpy(w).permute(0, 3, 1, 2).requires_grad_()
    yt = torch.nn.functional.conv2d(xt, wt, stride=st, padding=pad)
    dy = _rand(tuple(yt.permute(0, 2, 3, 1).shape), 5)
    yt.backward(torch.from_numpy(dy).permute(0, 3, 1, 2))
    np.testing.assert_allclose(orc.conv2d_dgrad(dy, w, x.shape, st, pad), xt.grad.permute(0, 2, 3, 1).numpy(),
                               rtol=1e-11, atol=1e-11)
    np.testing.assert_allclose(orc.conv2d_wgrad(x, dy, w.shape, st, pad), wt.grad.permute(0, 2, 3, 1).numpy(),
                               rtol=1e-11, atol=1e-11)


def test_unit_impulse_returns_kernel():
    # x = e_(n0,h0,w0,c0)  =>  y[n0,p,q,k] = w[k, h0 - p*st + pad, w0 - q*st + pad, c0] where in range
    N, H, W, C, K, R, st, pad = 2, 7, 6, 3, 4, 3, 1, 1
    w = _rand((K, R, R, C), 7)
    n0, h0, w0, c0 = 1, 3, 2, 2
    x = np.zeros((N, H, W, C))
    x[n0, h0, w0, c0] = 1.0
    y = orc.conv2d_fwd(x, w, st, pad)
    expect = np.zeros_like(y)
    for p in range(y.shape[1]):
        for q in range(y.shape[2]):
            r, s = h0 - p * st + pad, w0 - q * st + pad
            if 0 <= r < R and 0 <= s < R:
                expect[n0, p, q, :] = w[:, r, s, c0]
    np.testing.assert_array_equal(y, expect)
    # the patch around (h0, w0) is the kernel flipped in space
    np.testing.assert_array_equal(y[n0, h0 - 1:h0 + 2, w0 - 1:w0 + 2, :], w[:, ::-1, ::-1, c0].transpose(1, 2, 0))


@pytest.mark.parametrize("shape", SHAPES)
def test_adjoint_identities(shape):
    # <conv(x,w), y> = <x, dgrad(y,w)> = <w, wgrad(x,y)>
    N, H, W, C, K, R, st, pad = shape
    x, w = _rand((N, H, W, C), 8), _rand((K, R, R, C), 9)
    fx = orc.conv2d_fwd(x, w, st, pad)
    y = _rand(fx.shape, 10)
    a = np.sum(fx * y)
    b = np.sum(x * orc.conv2d_dgrad(y, w, x.shape, st, pad))
    c = np.sum(w * orc.conv2d_wgrad(x, y, w.shape, st, pad))
    assert abs(a - b) <= 1e-11 * max(1.0, abs(a))
    assert abs(a - c) <= 1e-11 * max(1.0, abs(a))


def test_wgrad_central_difference():
    # L(w) = <conv(x,w), y> is linear in w, so the central difference is exact up to rounding
    N, H, W, C, K, R, st, pad = 2, 6, 6, 3, 2, 3, 2, 1
    x, w = _rand((N, H, W, C), 11), _rand((K, R, R, C), 12)
    y = _rand(orc.conv2d_fwd(x, w, st, pad).shape, 13)
    dw = orc.conv2d_wgrad(x, y, w.shape, st, pad)
    eps = 1e-3
    for idx in [(0, 0, 0, 0), (1, 2, 1, 2), (0, 1, 2, 1), (1, 0, 2, 0)]:
        wp, wm = w.copy(), w.copy()
        wp[idx] += eps
        wm[idx] -= eps
        fd = (np.sum(orc.conv2d_fwd(x, wp, st, pad) * y) - np.sum(orc.conv2d_fwd(x, wm, st, pad) * y)) / (2 * eps)
        assert abs(fd - dw[idx]) <= 1e-9 * max(1.0, abs(dw[idx]))


def test_linearity():
    x1, x2, w = _rand((2, 5, 5, 3), 14), _rand((2, 5, 5, 3), 15), _rand((4, 3, 3, 3), 16)
    lhs = orc.conv2d_fwd(2.0 * x1 - 3.0 * x2, w, 1, 1)
    rhs = 2.0 * orc.conv2d_fwd(x1, w, 1, 1) - 3.0 * orc.conv2d_fwd(x2, w, 1, 1)
    np.testing.assert_allclose(lhs, rhs, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("shape", SHAPES)
def test_single_element_evaluators(shape):
    # gather-form dgrad and the point evaluators agree with the full passes
    N, H, W, C, K, R, st, pad = shape
    x, w = _rand((N, H, W, C), 17), _rand((K, R, R, C), 18)
    y = orc.conv2d_fwd(x, w, st, pad)
    dy = _rand(y.shape, 19)
    dx = orc.conv2d_dgrad(dy, w, x.shape, st, pad)
    dw = orc.conv2d_wgrad(x, dy, w.shape, st, pad)
    g = np.random.default_rng(20)
    for _ in range(12):
        n, p, q, k = (int(g.integers(0, d)) for d in y.shape)
        assert abs(orc.conv2d_fwd_at(x, w, st, pad, n, p, q, k) - y[n, p, q, k]) <= 1e-12 * (1 + abs(y[n, p, q, k]))
        n, h, ww, c = (int(g.integers(0, d)) for d in x.shape)
        v = orc.conv2d_dgrad_at(dy, w, x.shape, st, pad, n, h, ww, c)
        assert abs(v - dx[n, h, ww, c]) <= 1e-12 * (1 + abs(v))
        k, r, s, c = (int(g.integers(0, d)) for d in w.shape)
        v = orc.conv2d_wgrad_at(x, dy, w.shape, st, pad, k, r, s, c)
        assert abs(v - dw[k, r, s, c]) <= 1e-12 * (1 + abs(v))
