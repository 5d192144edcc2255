"""The memory model of Eq. 9 as calibrated by paper_2509_26092_gb300.memory_model:
the least-squares fit M(B) = P + B*A and the largest batch that fits."""
import numpy as np
import pytest

from paper_2509_26092_gb300 import build_lib
from paper_2509_26092_gb300 import memory_model as MM


def test_fit_recovers_an_exact_line():
    p, a = 1.9e9, 1.37e7  # bytes, bytes per sample
    bs = [64, 128, 192, 256, 320, 384, 448, 512]
    fp, fa, r2 = MM.fit_memory(bs, [p + a * b for b in bs])
    assert abs(fp - p) / p < 1e-12 and abs(fa - a) / a < 1e-12 and abs(r2 - 1.0) < 1e-12


def test_fit_is_the_least_squares_line():
    g = np.random.default_rng(9)
    bs = np.array([64, 128, 192, 256, 320, 384, 448, 512], dtype=float)
    m = 2e9 + 1.1e7 * bs + g.normal(0.0, 2e7, bs.size)
    fp, fa, _ = MM.fit_memory(list(bs), list(m))
    ref, *_ = np.linalg.lstsq(np.stack([bs, np.ones_like(bs)], 1), m, rcond=None)
    assert abs(fa - ref[0]) / ref[0] < 1e-10 and abs(fp - ref[1]) / ref[1] < 1e-10


def test_max_batch_is_the_largest_that_fits():
    p, a, m = 2.0e9, 1.0e7, 24.0e9
    b = MM.max_batch(p, a, m)
    assert p + a * b <= m < p + a * (b + 1)
    assert b == 2200
    assert MM.max_batch(30e9, 1e7, 24e9) == 0  # not even one sample fits
    with pytest.raises(ValueError):
        MM.max_batch(1e9, 0.0, 24e9)


@pytest.mark.gpu
def test_measured_memory_is_linear_in_the_batch():
    """On the GPU: the step's peak memory at four CIFAR-shaped batch sizes grows with the
    batch, and the fitted line predicts a held-out batch twice the largest within 10%."""
    build_lib.build()
    bs = [64, 128, 192, 256]
    peaks = MM.measure("cifar", 100, 32, 32, bs)
    assert all(peaks[i] < peaks[i + 1] for i in range(len(bs) - 1))
    p, a, r2 = MM.fit_memory(bs, peaks)
    assert p > 0.0 and a > 0.0 and r2 > 0.99
    got = MM.measure("cifar", 100, 32, 32, [512])[0]
    assert abs(p + a * 512 - got) / got < 0.10
