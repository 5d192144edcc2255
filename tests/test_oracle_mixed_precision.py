"""Pins for the oracle's fp16 mixed precision with loss scaling (the paper's ImageNet runs used
mixed-precision training, Sec. 5.2.3, citing Micikevicius et al.).

binary16 rounding is checked against numpy's float16 conversion; loss scaling by a power of
two against exactness (it commutes with every fp64 operation of the step); the scaled merge
against the unscaled one and its skip rule; the dynamic scale against its closed-form sequence.
"""
import numpy as np
import pytest

import oracle as orc
from oracle import resnet18 as R
from paper_2509_26092_gb300 import synth


def test_round_f16_matches_numpy():
    g = np.random.default_rng(0)
    x = np.concatenate([
        g.standard_normal(8000) * np.exp2(g.integers(-30, 17, 8000)),   # normals, subnormals, overflow
        (np.arange(-2000, 2000) + 0.5) * 2.0**-10,                         # ties at quantum 2^-10 (|x| in [1, 2))
        (np.arange(1, 2000) + 0.5) * 2.0**-24,                             # subnormal ties
        [65504.0, 65519.99, 65520.0, -65520.0, 2.0**-25, 2.0**-25 * 1.0001, 0.0, -0.0, np.inf, -np.inf],
    ])
    ref = x.astype(np.float16).astype(np.float64)
    got = orc.round_f16(x)
    assert np.array_equal(got, ref) and np.array_equal(np.signbit(got), np.signbit(ref))


def test_round_f16_edges():
    assert orc.round_f16(np.array([65519.0]))[0] == 65504.0
    assert orc.round_f16(np.array([65520.0]))[0] == np.inf
    assert orc.round_f16(np.array([2.0**-25]))[0] == 0.0           # a tie below the smallest subnormal: to even (0)
    assert orc.round_f16(np.array([3 * 2.0**-25]))[0] == 2.0**-23  # a tie between 1 and 2 quanta: to even (2)


@pytest.mark.parametrize("order", [0, 1, 2])
def test_scaled_merge_equals_unscaled_for_power_of_two_scales(order):
    g = np.random.default_rng(order)
    n = 1000
    w, u, gl, gs = (g.standard_normal(n) for _ in range(4))
    rw, ru = orc.ps_merge(w, u, gl, gs, 0.2, 0.9, 1.0, 19 / 21, order)
    sw, su, ok = orc.ps_merge_scaled(w, u, gl * 2.0**15, gs * 2.0**9, 0.2, 0.9, 1.0, 19 / 21, order, 2.0**15, 2.0**9)
    assert ok and np.array_equal(sw, rw) and np.array_equal(su, ru)
    # a single push
    rw, ru = orc.ps_merge(w, u, gl, None, 0.2, 0.9, 1.0, 19 / 21, order)
    sw, su, ok = orc.ps_merge_scaled(w, u, gl * 1024.0, None, 0.2, 0.9, 1.0, 19 / 21, order, 1024.0, 1.0)
    assert ok and np.array_equal(sw, rw) and np.array_equal(su, ru)


@pytest.mark.parametrize("bad", [np.inf, -np.inf, np.nan])
def test_scaled_merge_skips_a_non_finite_push(bad):
    g = np.random.default_rng(1)
    w, u, gl, gs = (g.standard_normal(64) for _ in range(4))
    gs[17] = bad
    sw, su, ok = orc.ps_merge_scaled(w, u, gl, gs, 0.2, 0.9, 1.0, 0.5, 0, 8.0, 8.0)
    assert not ok and np.array_equal(sw, w) and np.array_equal(su, u)


def test_loss_scale_sequence():
    s, good = 2.0**15, 0
    seq = []
    for found_inf in (False, False, True, False, False, False, False):
        s, good = orc.loss_scale_update(s, good, found_inf, 3)
        seq.append((s, good))
    assert seq == [(2.0**15, 1), (2.0**15, 2), (2.0**14, 0), (2.0**14, 1), (2.0**14, 2), (2.0**15, 0),
                   (2.0**15, 1)]


def test_loss_scaling_commutes_with_the_fp64_step():
    widths = (4, 4, 8, 8)
    table = R.layer_table("imagenet", 5, widths)
    params = {k: v.astype(np.float64) for k, v in synth.params(table, 0, random_bn=True).items()}
    img = synth.images(3, 32, 32, 3, 0).astype(np.float64)
    lab = synth.labels(3, 5, 0)
    a = R.train_step(params, img, lab, "imagenet", storage=None, widths=widths)
    b = R.train_step(params, img, lab, "imagenet", storage=None, widths=widths, loss_scale=2.0**12)
    assert a["loss"] == b["loss"]
    for k in a["grads"]:
        assert np.array_equal(b["grads"][k], a["grads"][k] * 2.0**12), k
