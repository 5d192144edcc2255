"""Seeded synthetic inputs shaped like the paper's CIFAR-100 and ImageNet
ResNet-18 workloads.

Neither dataset is available, so every input is drawn here: images are
i.i.d. N(0, 1) fp32 NHWC, labels are uniform integers, weights are
Kaiming-normal with fan-in scaling, and BatchNorm starts at gamma = 1,
beta = 0 (or a seeded perturbation for tests).  This module holds no
arithmetic of the training step itself; both the CUDA path and the CPU
reference draw their inputs from it.

Every array has its own generator, seeded from (seed, a stable hash of its
name), so adding or reordering tensors never changes another tensor's values.
"""
import math
import zlib

import numpy as np


def rng(seed, name=""):
    return np.random.default_rng([int(seed) & 0xFFFFFFFF, zlib.crc32(name.encode())])


def images(n, h, w, c=3, seed=0, name="images"):
    """[n, h, w, c] float32, i.i.d. N(0, 1)."""
    return rng(seed, name).standard_normal((n, h, w, c), dtype=np.float32)


def images_u8(n, h, w, c=3, seed=0, name="images_u8"):
    """[n, h, w, c] uint8, i.i.d. uniform in 0..255 (decoded 8-bit pixels)."""
    return rng(seed, name).integers(0, 256, size=(n, h, w, c), dtype=np.uint8)


def labels(n, classes, seed=0, name="labels"):
    """[n] int32, uniform in [0, classes)."""
    return rng(seed, name).integers(0, classes, size=n, dtype=np.int32)


def normal(shape, std, seed=0, name="normal"):
    return (rng(seed, name).standard_normal(shape) * std).astype(np.float32)


def kaiming_normal(shape, fan_in, seed=0, name="w"):
    """N(0, 2/fan_in) float32."""
    return normal(shape, math.sqrt(2.0 / fan_in), seed, name)


def params(table, seed=0, random_bn=False):
    """Draw every tensor of a parameter table.

    table: iterable of (name, shape, fan_in); names ending in '.g'/'.b' with a
    None fan_in are BatchNorm gamma/beta or a bias.  Returns {name: float32 array}.
    """
    out = {}
    for name, shape, fan_in in table:
        if fan_in is not None:
            out[name] = kaiming_normal(shape, fan_in, seed, name)
        elif name.endswith(".g"):
            out[name] = (rng(seed, name).uniform(0.5, 1.5, shape).astype(np.float32) if random_bn
                         else np.ones(shape, np.float32))
        else:
            out[name] = (normal(shape, 0.1, seed, name) if random_bn else np.zeros(shape, np.float32))
    return out


def momentum_state(table, std=0.01, seed=0):
    """A seeded nonzero momentum buffer u, so the momentum term is exercised."""
    return {name: normal(shape, std, seed, "u/" + name) for name, shape, _ in table}
