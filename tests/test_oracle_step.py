"""Pins for the oracle's whole ResNet-18 step and dual-batch iteration.

The composed backward pass is pinned by central finite differences of the
fp64 loss (no bf16 rounding) on narrow networks of the same topology, and the
parameter counts by the known ResNet-18 totals.
"""
import numpy as np
import pytest

import oracle as orc
from oracle import resnet18 as R
from paper_2509_26092_gb300 import synth


def test_parameter_counts():
    assert R.n_params("cifar", 100) == 11_220_132
    assert R.n_params("imagenet", 1000) == 11_689_512


def _small_setup(variant, widths, res, batch, classes, seed=0):
    table = R.layer_table(variant, classes, widths)
    params = {k: v.astype(np.float64) for k, v in synth.params(table, seed, random_bn=True).items()}
    img = synth.images(batch, res, res, 3, seed).astype(np.float64)
    lab = synth.labels(batch, classes, seed)
    return table, params, img, lab


@pytest.mark.parametrize("variant,res", [("cifar", 12), ("imagenet", 32)])
def test_full_step_central_difference(variant, res):
    widths = (4, 4, 8, 8)
    table, params, img, lab = _small_setup(variant, widths, res, 3, 5)
    base = R.train_step(params, img, lab, variant, bf16_storage=False, widths=widths)
    g = np.random.default_rng(1)
    eps = 1e-6
    checked = 0
    for name, shape, _ in table:
        if not (name.endswith(".w") or name.endswith(".g") or name.endswith(".b")):
            continue
        # one element per tensor, a few tensors per layer kind
        idx = tuple(int(g.integers(0, s)) for s in shape)
        p = {k: v.copy() for k, v in params.items()}
        p[name][idx] += eps
        lp = R.train_step(p, img, lab, variant, bf16_storage=False, widths=widths)["loss"]
        p[name][idx] -= 2 * eps
        lm = R.train_step(p, img, lab, variant, bf16_storage=False, widths=widths)["loss"]
        fd = (lp - lm) / (2 * eps)
        an = base["grads"][name][idx]
        assert abs(fd - an) <= 1e-6 + 1e-4 * abs(an), (name, idx, fd, an)
        checked += 1
    assert checked == len(table)


def test_bf16_storage_changes_loss_little():
    # Gradients are not compared here: BatchNorm over a handful of rows amplifies
    # storage rounding far beyond what full-size groups do.
    widths = (4, 4, 8, 8)
    table, params, img, lab = _small_setup("cifar", widths, 12, 4, 5)
    a = R.train_step(params, img, lab, "cifar", bf16_storage=False, widths=widths)
    b = R.train_step(params, img, lab, "cifar", bf16_storage=True, widths=widths)
    assert abs(a["loss"] - b["loss"]) < 2e-2 * abs(a["loss"])


def test_dual_batch_iteration_composes_merge():
    widths = (4, 4, 8, 8)
    table, params, img, lab = _small_setup("cifar", widths, 16, 4, 5)
    u = {k: np.zeros_like(v) for k, v in params.items()}
    # large worker: samples 2..3, small worker: samples 0..1, both resized to 12x12
    nw, nu, lL, lS, gL, gS = R.dual_batch_iteration(params, u, img[2:], lab[2:], img[:2], lab[:2], 12, "cifar",
                                                     lr=0.2, momentum=0.9, f_large=1.0, f_small=19 / 21, order=2,
                                                     bf16_storage=False, widths=widths)
    for k in params:
        np.testing.assert_allclose(nu[k], -0.2 * (gL[k] + 19 / 21 * gS[k]), rtol=1e-12, atol=1e-15)
        np.testing.assert_allclose(nw[k], params[k] + nu[k], rtol=1e-12, atol=1e-15)
    # a worker's gradient does not depend on the other worker's batch
    xs = orc.bilinear_resize(img[:2], 12, 12)
    one = R.train_step(params, xs, lab[:2], "cifar", bf16_storage=False, widths=widths)
    for k in params:
        np.testing.assert_array_equal(one["grads"][k], gS[k])


def test_conv_flop_count_per_image():
    # 2*M*N*K per pass over the unpadded problem; fwd + dgrad (not the stem) + wgrad: 10.65 GFLOP per
    # 224 px ImageNet image and 3.33 per 32 px CIFAR image
    assert abs(R.conv_flops("imagenet", 256, 224) / 256 / 1e9 - 10.65) < 0.01
    assert abs(R.conv_flops("cifar", 256, 32) / 256 / 1e9 - 3.33) < 0.01
