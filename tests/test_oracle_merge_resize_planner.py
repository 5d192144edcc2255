"""Pins for the oracle's parameter-server merge, bilinear resize and planner.

* Merge (Sec. 3.4 with Eq. 1): each push is one momentum-SGD step on the
  factor-scaled gradient, so a push sequence equals torch.optim.SGD steps, and
  exact rational arithmetic of the PyTorch momentum form gives the same values.
* Resize (Sec. 4.1): half-pixel bilinear equals torch's interpolate
  (align_corners=False, no antialias); 32->16 is 2x2 average pooling; affine
  images are reproduced exactly; the integer taps follow closed forms.
* Planner (Sec. 3.3, Eqs. 4-8; factor Sec. 3.4): the values printed in
  Tables 2, 3 and 6 of the paper.
"""
import math
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle as orc
from oracle import planner

GOLD = os.path.join(os.path.dirname(__file__), "golden")


def _rows(name):
    with open(os.path.join(GOLD, name)) as f:
        return [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]


# ----------------------------------------------------------------------------- merge
def _torch_sgd(w0, u0, pushes, lr, mu):
    """Apply pushes [(factor, grad)] with torch's momentum SGD (v <- mu v + g; w <- w - lr v).

    The oracle's form u <- mu u - lr f g ; w <- w + u is the same map with u = -lr v.
    """
    w = torch.tensor(w0, dtype=torch.float64, requires_grad=True)
    opt = torch.optim.SGD([w], lr=lr, momentum=mu, dampening=0.0)
    opt.state[w]["momentum_buffer"] = torch.tensor(-np.asarray(u0) / lr, dtype=torch.float64)
    for f, g in pushes:
        w.grad = torch.tensor(f * np.asarray(g), dtype=torch.float64)
        opt.step()
    return w.detach().numpy(), -lr * opt.state[w]["momentum_buffer"].numpy()


@pytest.mark.parametrize("order", [0, 1, 2])
@pytest.mark.parametrize("mu", [0.0, 0.9])
def test_merge_equals_torch_sgd_pushes(order, mu):
    g = np.random.default_rng(1)
    n = 257
    w0, u0 = g.standard_normal(n), 0.01 * g.standard_normal(n)
    gl, gs = g.standard_normal(n), g.standard_normal(n)
    lr, fL, fS = 0.2, 1.0, 19.0 / 21.0
    w, u = orc.ps_merge(w0, u0, gl, gs, lr, mu, fL, fS, order)
    if order == 0:
        pushes = [(fL, gl), (fS, gs)]
    elif order == 1:
        pushes = [(fS, gs), (fL, gl)]
    else:
        pushes = [(1.0, fL * gl + fS * gs)]
    wr, ur = _torch_sgd(w0, u0, pushes, lr, mu)
    if mu == 0.0:  # torch keeps no momentum buffer without momentum; u is the last step taken
        ur = -lr * pushes[-1][0] * pushes[-1][1]
    np.testing.assert_allclose(w, wr, rtol=1e-14, atol=1e-15)
    np.testing.assert_allclose(u, ur, rtol=1e-13, atol=1e-15)


def test_merge_exact_rationals_pytorch_form():
    # Two pushes, large then small, worked in exact rationals in the v-form of momentum SGD.
    w0 = [Fraction(1), Fraction(-2), Fraction(1, 2), Fraction(0)]
    u0 = [Fraction(1, 100), Fraction(-2, 100), Fraction(0), Fraction(5, 100)]
    gl = [Fraction(1, 10), Fraction(2, 10), Fraction(-3, 10), Fraction(4, 10)]
    gs = [Fraction(1), Fraction(-1), Fraction(1, 2), Fraction(0)]
    lr, mu, fS = Fraction(1, 5), Fraction(9, 10), Fraction(19, 21)
    ew, eu = [], []
    for i in range(4):
        v = -u0[i] / lr
        w = w0[i]
        for f, gr in ((Fraction(1), gl[i]), (fS, gs[i])):
            v = mu * v + f * gr
            w = w - lr * v
        ew.append(float(w))
        eu.append(float(-lr * v))
    w, u = orc.ps_merge(np.array([float(a) for a in w0]), np.array([float(a) for a in u0]),
                        np.array([float(a) for a in gl]), np.array([float(a) for a in gs]), 0.2, 0.9, 1.0,
                        19.0 / 21.0, 0)
    np.testing.assert_allclose(w, ew, rtol=1e-15, atol=1e-16)
    np.testing.assert_allclose(u, eu, rtol=1e-14, atol=1e-16)


def test_merge_special_cases():
    g = np.random.default_rng(2)
    n = 64
    w0, u0, gl, gs = (g.standard_normal(n) for _ in range(4))
    # f_S = 0: the small push is a pure momentum decay step
    w, u = orc.ps_merge(w0, u0, gl, gs, 0.1, 0.9, 1.0, 0.0, 0)
    u1 = 0.9 * u0 - 0.1 * gl
    np.testing.assert_allclose(u, 0.9 * u1, rtol=1e-14)
    np.testing.assert_allclose(w, w0 + u1 + 0.9 * u1, rtol=1e-13, atol=1e-14)
    # a missing push is a single step
    w, u = orc.ps_merge(w0, u0, gl, None, 0.1, 0.9, 1.0, 0.5, 0)
    np.testing.assert_allclose(u, 0.9 * u0 - 0.1 * gl, rtol=1e-14)
    w2, u2 = orc.ps_merge(w0, u0, None, gl, 0.1, 0.9, 0.5, 1.0, 0)
    np.testing.assert_array_equal(w, w2)
    # without momentum the three orders agree on w (plain SGD, Eq. 1)
    ws = [orc.ps_merge(w0, np.zeros(n), gl, gs, 0.2, 0.0, 1.0, 0.8, o)[0] for o in (0, 1, 2)]
    np.testing.assert_allclose(ws[0], ws[1], rtol=1e-14)
    np.testing.assert_allclose(ws[0], ws[2], rtol=1e-14)
    np.testing.assert_allclose(ws[0], w0 - 0.2 * (gl + 0.8 * gs), rtol=1e-13, atol=1e-14)


# ----------------------------------------------------------------------------- resize
@pytest.mark.parametrize("hin,hout", [(32, 16), (32, 24), (224, 128), (224, 160), (224, 224), (17, 5)])
def test_resize_matches_torch_interpolate(hin, hout):
    x = np.random.default_rng(3).standard_normal((2, hin, hin, 3))
    got = orc.bilinear_resize(x, hout, hout)
    ref = torch.nn.functional.interpolate(torch.from_numpy(x).permute(0, 3, 1, 2), size=(hout, hout),
                                          mode="bilinear", align_corners=False, antialias=False)
    np.testing.assert_allclose(got, ref.permute(0, 2, 3, 1).numpy(), rtol=1e-12, atol=1e-12)


def test_resize_half_is_2x2_average():
    x = np.random.default_rng(4).standard_normal((1, 32, 32, 3))
    got = orc.bilinear_resize(x, 16, 16)
    ref = x.reshape(1, 16, 2, 16, 2, 3).mean(axis=(2, 4))
    np.testing.assert_allclose(got, ref, rtol=1e-14, atol=1e-15)


def test_resize_reproduces_affine_images():
    h = np.arange(224)[:, None] * 0.5 - np.arange(224)[None, :] * 0.25 + 3.0
    x = np.broadcast_to(h[None, :, :, None], (1, 224, 224, 1))
    for out in (128, 160):
        got = orc.bilinear_resize(x, out, out)[0, :, :, 0]
        src = (np.arange(out) + 0.5) * 224 / out - 0.5
        ref = src[:, None] * 0.5 - src[None, :] * 0.25 + 3.0
        np.testing.assert_allclose(got, ref, rtol=0, atol=1e-12)


def test_resize_tap_closed_forms():
    i0, i1, lam = orc.resize_taps(32, 24)
    # src = (4j - 1)/6: floor and fraction repeat with period 3
    assert list(i0[:6]) == [0, 1, 2, 4, 5, 6]
    np.testing.assert_allclose(lam[:6], [1 / 6, 1 / 2, 5 / 6] * 2, rtol=1e-15)
    i0, i1, lam = orc.resize_taps(224, 128)  # src = (14j + 3)/8
    j = np.arange(128)
    np.testing.assert_array_equal(i0, (14 * j + 3) // 8)
    np.testing.assert_allclose(lam, ((14 * j + 3) % 8) / 8, rtol=0, atol=0)
    i0, i1, lam = orc.resize_taps(224, 160)  # src = (7j + 1)/5, an integer when j = 2 mod 5
    j = np.arange(160)
    np.testing.assert_array_equal(i0, (7 * j + 1) // 5)
    np.testing.assert_array_equal(lam[j % 5 == 2], 0.0)
    assert int(np.sum(lam == 0.0)) == 32
    i0, i1, lam = orc.resize_taps(50, 50)  # identity
    np.testing.assert_array_equal(i0, np.arange(50))
    np.testing.assert_array_equal(lam, 0.0)
    assert np.all(i1 <= 49)


# ----------------------------------------------------------------------------- planner
def test_table2_data_amounts_and_factor():
    d, n = 50000, 4
    for k, ns, nl, bs, ds, bl, dl, fac in _rows("planner_table2.txt"):
        k, ns, nl = float(k), int(ns), int(nl)
        if nl == 0:
            # all workers small: each gets the even share d/n
            assert planner.data_small(d, 0, ns, 0.0) == float(ds)
            continue
        dL = planner.data_large(k, d, n)
        assert round(dL) == int(dl)
        dS = planner.data_small(d, nl, ns, dL)
        dS_printed = math.floor(dS + 1e-9)  # the table truncates 12291.67 and 12083.33
        assert dS_printed == int(ds)
        # the printed factor is taken from the truncated d_S (12291/13125 = 0.93646 -> 0.936)
        assert round(planner.update_factor(dS_printed, dL), 3) == float(fac)


def test_table2_small_batch_from_eq8():
    # Eq. 8 depends on a and b only through c = b/a, which the paper does not print.
    # One c reproduces all eight printed B_S values with the floor.
    c = 24.8
    d, n = 50000, 4
    for k, ns, nl, bs, ds, bl, dl, fac in _rows("planner_table2.txt"):
        k, ns, nl = float(k), int(ns), int(nl)
        dL = planner.data_large(k, d, n)
        dS = planner.data_small(d, nl, ns, dL) if nl else d / n
        assert math.floor(planner.small_batch(1.0, c, 500.0, dL, dS)) == int(bs)


def test_table3_sqrt_factor():
    # The printed scheme-2 values are the square roots of the printed 3-place scheme-1 values
    # (sqrt(0.879) = 0.93755 -> 0.938, while sqrt(12083/13750) = 0.93742).
    for ns, nl, ds, f1, f2 in _rows("factor_table3.txt"):
        f1_printed = round(planner.update_factor(float(ds), 13750.0), 3)
        assert f1_printed == float(f1)
        assert round(planner.update_factor(f1_printed, 1.0, sqrt_scheme=True), 3) == float(f2)
        assert abs(planner.update_factor(float(ds), 13750.0, sqrt_scheme=True) - float(f2)) < 1e-3


def test_table6_data_amounts():
    for ds_name, d, ns, dS, dL in _rows("hybrid_table6.txt"):
        d, ns = int(d), int(ns)
        if ns == 0:
            assert round(d / 4) == int(dL)
            continue
        if ns == 4:
            assert round(d / 4) == int(dS)
            continue
        dLr = round(planner.data_large(1.05, d, 4))
        assert dLr == int(dL)
        assert round(planner.data_small(d, 4 - ns, ns, dLr)) == int(dS)


def test_emulation_factor_two_workers():
    # n = 2, one large and one small worker, k = 1.05 (Sec. 5.2.1): f_S = 0.95/1.05 = 19/21
    dL = planner.data_large(1.05, 1.0, 2)
    dS = planner.data_small(1.0, 1, 1, dL)
    assert abs(planner.update_factor(dS, dL) - 19.0 / 21.0) < 1e-15


def test_time_model_simplification():
    # Eq. 3 is Eq. 2 with ceil(d/x) replaced by d/x
    for x, d in ((500, 50000), (83, 10625)):
        assert abs(planner.epoch_time(0.3, 7.4, x, d) - planner.epoch_time_simplified(0.3, 7.4, x, d)) < \
            (0.3 * x + 7.4)
