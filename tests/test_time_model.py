"""The training-time model of Sec. 3.2 (Eq. 2) as calibrated by
paper_2509_26092_gb300.time_model: the least-squares fit, Eq. 2's epoch time, and
the chain into the planner (Eqs. 4-8)."""
import math

import numpy as np
import pytest

from oracle import planner
from paper_2509_26092_gb300 import build_lib
from paper_2509_26092_gb300 import time_model as TM


@pytest.fixture(scope="module")
def D():
    build_lib.build()
    from paper_2509_26092_gb300 import dbl
    return dbl


def test_fit_recovers_an_exact_line():
    a, b = 3.1e-4, 7.4e-3  # seconds per image, per batch
    xs = [16, 32, 64, 128, 256, 500]
    fa, fb, r2 = TM.fit_linear(xs, [a * x + b for x in xs])
    assert abs(fa - a) < 1e-15 and abs(fb - b) < 1e-14 and abs(r2 - 1.0) < 1e-12


def test_fit_is_the_least_squares_line():
    g = np.random.default_rng(5)
    xs = np.array([64, 128, 192, 256, 384, 512], dtype=float)
    ts = 2e-5 * xs + 1.5e-3 + g.normal(0.0, 5e-5, xs.size)
    fa, fb, r2 = TM.fit_linear(list(xs), list(ts))
    # the normal equations of min ||A [a b] - t||, solved by an independent routine
    ref, *_ = np.linalg.lstsq(np.stack([xs, np.ones_like(xs)], 1), ts, rcond=None)
    assert abs(fa - ref[0]) < 1e-12 and abs(fb - ref[1]) < 1e-12
    assert 0.9 < r2 < 1.0


def test_fit_rejects_degenerate_input():
    with pytest.raises(ValueError):
        TM.fit_linear([64], [1.0])
    with pytest.raises(ValueError):
        TM.fit_linear([64, 64], [1.0, 2.0])


def test_epoch_time_is_eq2():
    for x in (1, 7, 100, 500):
        assert TM.epoch_time(0.3, 7.4, x, 50000) == planner.epoch_time(0.3, 7.4, x, 50000)
    assert TM.epoch_time(0.3, 7.4, 500, 50000) == (0.3 * 500 + 7.4) * 100


def test_plan_from_fit_matches_eq8(D):
    a, b = 1.0, 24.8  # the paper's b/a for its GPU (Table 2)
    p = TM.plan(a, b, 1.05, 50000, 1, 3, 500)
    d_l = planner.data_large(1.05, 50000, 4)
    d_s = planner.data_small(50000, 3, 1, d_l)
    assert p["d_large"] == pytest.approx(d_l, rel=1e-15) and p["d_small"] == pytest.approx(d_s, rel=1e-15)
    assert p["batch_small"] == pytest.approx(planner.small_batch(a, b, 500.0, d_l, d_s), rel=1e-12)
    assert p["batch_small_floor"] == math.floor(p["batch_small"])
    assert p["f_small"] == pytest.approx(d_s / d_l, rel=1e-15)


@pytest.mark.gpu
def test_measured_batch_times_grow_with_the_batch(D):
    """On the GPU: single-worker iterations of the CIFAR-shaped step at three batch sizes
    take longer for larger batches, and the fitted per-image cost is positive."""
    times = TM.measure("cifar", 100, 32, 32, [64, 128, 256], reps=3, warmup=2)
    assert all(t > 0.0 for t in times) and times[0] < times[2]
    a, b, r2 = TM.fit_linear([64, 128, 256], times)
    assert a > 0.0 and math.isfinite(b) and r2 > 0.5
