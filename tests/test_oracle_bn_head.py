"""Pins for the oracle's BatchNorm, pooling, head and bf16-rounding routines."""
import math

import numpy as np
import pytest
import torch

import oracle as orc


def _rand(shape, seed):
    return np.random.default_rng(seed).standard_normal(shape)


# ----------------------------------------------------------------------------- BatchNorm
def test_bn_normalised_output_has_zero_mean_unit_variance():
    y = _rand((4, 5, 5, 6), 1) * 3.0 + 2.0
    out, mean, invstd = orc.bn_fwd(y, np.ones(6), np.zeros(6), eps=0.0, relu=False)
    flat = out.reshape(-1, 6)
    np.testing.assert_allclose(flat.mean(0), 0.0, atol=1e-12)
    np.testing.assert_allclose(flat.var(0), 1.0, rtol=1e-12)


@pytest.mark.parametrize("relu,res", [(False, False), (True, False), (True, True)])
def test_bn_fwd_bwd_match_torch(relu, res):
    N, H, W, C = 3, 4, 5, 6
    y = _rand((N, H, W, C), 2)
    g, b = 1.0 + 0.3 * _rand(C, 3), 0.2 * _rand(C, 4)
    r = _rand((N, H, W, C), 5) if res else None
    out, mean, invstd = orc.bn_fwd(y, g, b, eps=1e-5, res=r, relu=relu)
    yt = torch.from_numpy(y).permute(0, 3, 1, 2).requires_grad_()
    gt = torch.from_numpy(g).requires_grad_()
    bt = torch.from_numpy(b).requires_grad_()
    ot = torch.nn.functional.batch_norm(yt, None, None, gt, bt, training=True, eps=1e-5)
    if res:
        ot = ot + torch.from_numpy(r).permute(0, 3, 1, 2)
    if relu:
        ot = torch.relu(ot)
    np.testing.assert_allclose(out, ot.detach().permute(0, 2, 3, 1).numpy(), rtol=1e-11, atol=1e-11)
    dout = _rand((N, H, W, C), 6)
    dout2 = _rand((N, H, W, C), 7)
    ot.backward(torch.from_numpy(dout + dout2).permute(0, 3, 1, 2))
    dy, dg, db, dres = orc.bn_bwd(dout, out, y, g, mean, invstd, relu=relu, dout2=dout2, want_dres=True)
    np.testing.assert_allclose(dy, yt.grad.permute(0, 2, 3, 1).numpy(), rtol=1e-10, atol=1e-11)
    np.testing.assert_allclose(dg, gt.grad.numpy(), rtol=1e-10, atol=1e-11)
    np.testing.assert_allclose(db, bt.grad.numpy(), rtol=1e-10, atol=1e-11)
    mask = (out > 0) if relu else np.ones_like(out, bool)
    np.testing.assert_allclose(dres, (dout + dout2) * mask, rtol=0, atol=0)


def test_bn_bwd_central_difference():
    y = _rand((2, 3, 3, 2), 8)
    g, b = np.array([1.3, 0.7]), np.array([0.1, -0.2])
    dout = _rand(y.shape, 9)
    out, mean, invstd = orc.bn_fwd(y, g, b, eps=1e-5, relu=False)
    dy, _, _, _ = orc.bn_bwd(dout, out, y, g, mean, invstd, relu=False)
    eps = 1e-6
    for idx in [(0, 0, 0, 0), (1, 2, 1, 1), (0, 1, 2, 0)]:
        yp, ym = y.copy(), y.copy()
        yp[idx] += eps
        ym[idx] -= eps
        lp = np.sum(orc.bn_fwd(yp, g, b, 1e-5, relu=False)[0] * dout)
        lm = np.sum(orc.bn_fwd(ym, g, b, 1e-5, relu=False)[0] * dout)
        assert abs((lp - lm) / (2 * eps) - dy[idx]) < 1e-7


# ----------------------------------------------------------------------------- pooling
def test_maxpool_matches_torch_and_conserves_gradient():
    x = _rand((2, 9, 8, 3), 10)
    y, arg = orc.maxpool_fwd(x, 3, 2, 1)
    xt = torch.from_numpy(x).permute(0, 3, 1, 2).requires_grad_()
    yt = torch.nn.functional.max_pool2d(xt, 3, 2, 1)
    np.testing.assert_array_equal(y, yt.detach().permute(0, 2, 3, 1).numpy())
    dy = _rand(y.shape, 11)
    yt.backward(torch.from_numpy(dy).permute(0, 3, 1, 2))
    dx = orc.maxpool_bwd(dy, arg, x.shape, 3, 2, 1)
    np.testing.assert_allclose(dx, xt.grad.permute(0, 2, 3, 1).numpy(), rtol=1e-14, atol=1e-14)
    assert abs(dx.sum() - dy.sum()) < 1e-10


def test_maxpool_tie_goes_to_first_in_window_order():
    # an all-equal window (post-ReLU zeros): the gradient lands on the first in-bounds tap
    x = np.zeros((1, 4, 4, 1))
    y, arg = orc.maxpool_fwd(x, 3, 2, 1)
    # output (0,0) covers rows -1..1, cols -1..1 -> first in-bounds tap is (r=1, s=1)
    assert arg[0, 0, 0, 0] == 1 * 3 + 1
    # output (1,1) covers rows 1..3, cols 1..3 -> first tap (0,0)
    assert arg[0, 1, 1, 0] == 0
    dx = orc.maxpool_bwd(np.ones(y.shape), arg, x.shape, 3, 2, 1)
    assert dx[0, 0, 0, 0] == 1.0 and dx[0, 1, 1, 0] == 1.0 and dx.sum() == y.size


# ----------------------------------------------------------------------------- head
def test_softmax_ce_closed_forms():
    for classes in (100, 1000):
        loss, dl = orc.softmax_ce(np.zeros((3, classes)), np.array([0, 5, 7]))
        assert abs(loss - math.log(classes)) < 1e-12
    logits = _rand((5, 10), 12) * 4
    labels = np.array([1, 3, 3, 9, 0])
    loss, dl = orc.softmax_ce(logits, labels)
    np.testing.assert_allclose(dl.sum(1), 0.0, atol=1e-15)
    # softmax rows sum to one: N*dl + onehot
    p = dl * 5 + np.eye(10)[labels]
    np.testing.assert_allclose(p.sum(1), 1.0, rtol=1e-14)
    lt = torch.from_numpy(logits).requires_grad_()
    lref = torch.nn.functional.cross_entropy(lt, torch.from_numpy(labels).long())
    lref.backward()
    assert abs(loss - lref.item()) < 1e-12
    np.testing.assert_allclose(dl, lt.grad.numpy(), rtol=1e-12, atol=1e-15)


def test_fc_and_avgpool_match_library():
    x = _rand((3, 4, 4, 8), 13)
    f = orc.avgpool_fwd(x)
    np.testing.assert_allclose(f, x.mean(axis=(1, 2)), rtol=1e-14)
    Wt, b = _rand((5, 8), 14), _rand(5, 15)
    logits = orc.fc_fwd(f, Wt, b)
    np.testing.assert_allclose(logits, f @ Wt.T + b, rtol=1e-13)
    dl = _rand((3, 5), 16)
    dW, db, df = orc.fc_bwd(dl, f, Wt)
    np.testing.assert_allclose(dW, dl.T @ f, rtol=1e-13)
    np.testing.assert_allclose(db, dl.sum(0), rtol=1e-13)
    np.testing.assert_allclose(df, dl @ Wt, rtol=1e-13)
    dx = orc.avgpool_bwd(df, x.shape)
    np.testing.assert_allclose(dx.sum(axis=(1, 2)), df, rtol=1e-13)


# ----------------------------------------------------------------------------- bf16
def test_round_bf16_matches_torch_rne():
    g = np.random.default_rng(17)
    v = np.concatenate([g.standard_normal(20000) * 10.0 ** g.integers(-6, 6, 20000),
                        np.array([1 + 2 ** -8, 1 + 3 * 2 ** -8, -(1 + 2 ** -8), 2 ** -130, 3 * 2 ** -134, 0.0,
                                  1e38, -3.3e38])]).astype(np.float32)
    ref = torch.from_numpy(v).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(orc.round_bf16(v.astype(np.float64)), ref)
