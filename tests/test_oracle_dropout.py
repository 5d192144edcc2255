"""Pins for the oracle's dropout before the FC layer (Sec. 4.1; rates in Tables 7 and 9).

The counter-based generator (Philox4x64-10) is checked against numpy's
independent implementation of the same published generator, the mask rule
against its special cases and its binomial statistics, the scaling against
its closed form, and the whole step with dropout by central differences.
"""
import numpy as np
import pytest

import oracle as orc
from oracle import resnet18 as R
from paper_2509_26092_gb300 import synth


def _numpy_philox(counter, key):
    """numpy.random.Philox advances its counter by one before each block of four
    words, so starting it one below gives the block at `counter`."""
    v = sum(int(w) << (64 * i) for i, w in enumerate(counter))
    v = (v - 1) % (1 << 256)  # numpy's counter is one 256-bit integer, word 0 lowest
    c = [(v >> (64 * i)) & (2**64 - 1) for i in range(4)]
    bg = np.random.Philox(counter=np.array(c, dtype=np.uint64), key=np.array(key, dtype=np.uint64))
    return bg.random_raw(4).astype(np.uint64)


@pytest.mark.parametrize("counter,key", [
    ([1, 0, 0, 0], [0, 0]),
    ([7, 3, 0, 0], [12345, 0]),
    ([2**40 + 17, 2**63 + 5, 11, 2**64 - 1], [2**64 - 1, 2**32 + 3]),
    ([2**64 - 1, 9, 0, 0], [42, 0]),
])
def test_philox_matches_numpy(counter, key):
    assert np.array_equal(orc.philox4x64_10(counter, key), _numpy_philox(counter, key))


def test_philox_counter_zero():
    # counter 0 is reached from the wrapped counter 2^256 - 1
    assert np.array_equal(orc.philox4x64_10([0, 0, 0, 0], [0, 0]), _numpy_philox([0, 0, 0, 0], [0, 0]))


def test_mask_special_cases():
    assert orc.dropout_mask(8, 64, 0.0, 5, 0).all()  # d = 0 keeps everything
    # d = 1/2: the threshold is 2^31, so a feature is kept exactly when the top bit of its word is set
    N, C, seed, step = 5, 16, 77, 3
    keep = orc.dropout_mask(N, C, 0.5, seed, step)
    for n in range(N):
        for g in range(C // 4):
            words = _numpy_philox([n * (C // 4) + g, step, 0, 0], [seed, 0])
            assert np.array_equal(keep[n, 4 * g:4 * g + 4], (words >> np.uint64(63)).astype(np.uint8))


@pytest.mark.parametrize("d", [0.1, 0.2, 0.3])
def test_mask_keeps_one_minus_d(d):
    N, C = 128, 512
    keep = orc.dropout_mask(N, C, d, 2024, 1)
    n = N * C
    kept = int(keep.sum())
    sd = np.sqrt(n * d * (1 - d))
    assert abs(kept - n * (1 - d)) < 6 * sd
    # every channel position and every sample sees drops (no stuck word or lane)
    assert keep.min(axis=0).max() <= 1 and (keep.sum(axis=0) < N).all() and (keep.sum(axis=1) < C).all()


def test_masks_differ_by_step_and_seed():
    a = orc.dropout_mask(16, 512, 0.3, 1, 0)
    assert not np.array_equal(a, orc.dropout_mask(16, 512, 0.3, 1, 1))
    assert not np.array_equal(a, orc.dropout_mask(16, 512, 0.3, 2, 0))
    assert np.array_equal(a, orc.dropout_mask(16, 512, 0.3, 1, 0))


def test_apply_closed_form_and_expectation():
    g = np.random.default_rng(0)
    x = g.standard_normal((64, 512))
    d = 0.2
    keep = orc.dropout_mask(64, 512, d, 9, 4)
    y = orc.dropout_apply(x, keep, d)
    assert np.all(y[keep == 0] == 0.0)
    assert np.array_equal(y[keep == 1], x[keep == 1] / (1 - d))
    # inverted dropout leaves the expectation unchanged: the mean over many steps' masks tends to x
    ones = np.ones((8, 512))
    acc = np.zeros_like(ones)
    steps = 400
    for s in range(steps):
        acc += orc.dropout_apply(ones, orc.dropout_mask(8, 512, d, 9, s), d)
    mean = acc / steps
    sd = np.sqrt(d / (1 - d) / steps)  # standard deviation of the mean of keep/(1-d)
    assert np.abs(mean - 1.0).max() < 6 * sd


@pytest.mark.parametrize("variant,res", [("cifar", 12), ("imagenet", 32)])
def test_step_with_dropout_central_difference(variant, res):
    widths = (4, 4, 8, 8)
    table = R.layer_table(variant, 5, widths)
    params = {k: v.astype(np.float64) for k, v in synth.params(table, 0, random_bn=True).items()}
    img = synth.images(3, res, res, 3, 0).astype(np.float64)
    lab = synth.labels(3, 5, 0)
    drop = (0.3, 11, 2)
    base = R.train_step(params, img, lab, variant, bf16_storage=False, widths=widths, dropout=drop, keep=True)
    keep = base["acts"]["dropout_keep"]
    assert keep is not None and 0 < keep.sum() < keep.size
    nodrop = R.train_step(params, img, lab, variant, bf16_storage=False, widths=widths)
    assert base["loss"] != nodrop["loss"]
    g = np.random.default_rng(2)
    eps = 1e-6
    for name in ("fc.w", "fc.b", "layer4.1.conv2.w", "layer4.1.bn2.g", "layer1.0.conv1.w", "conv1.w"):
        shape = params[name].shape
        idx = tuple(int(g.integers(0, s)) for s in shape)
        p = {k: v.copy() for k, v in params.items()}
        p[name][idx] += eps
        lp = R.train_step(p, img, lab, variant, bf16_storage=False, widths=widths, dropout=drop)["loss"]
        p[name][idx] -= 2 * eps
        lm = R.train_step(p, img, lab, variant, bf16_storage=False, widths=widths, dropout=drop)["loss"]
        fd = (lp - lm) / (2 * eps)
        an = base["grads"][name][idx]
        assert abs(fd - an) <= 1e-6 + 1e-4 * abs(an), (name, idx, fd, an)
    # the FC weight gradient of a dropped feature is exactly zero for every class
    dropped = np.where(keep.sum(axis=0) == 0)[0]
    for c in dropped:
        assert np.all(base["grads"]["fc.w"][:, c] == 0.0)
