"""fp64 reference of the dual-batch planner (Sec. 3.3, Eqs. 3-8) and the
model-update factor (Sec. 3.4).

TEST INFRASTRUCTURE ONLY (see the package docstring).
"""
import math


def data_large(k, d, n):
    """d_L = k*d/n (from Eq. 4: the large-batch workers' share at time k*t)."""
    return k * d / n


def data_small(d, n_large, n_small, d_large):
    """d_S from Eq. 6: d = n_L*d_L + n_S*d_S."""
    return (d - n_large * d_large) / n_small


def small_batch(a, b, B_large, d_large, d_small):
    """B_S of Eq. 8: B_S = b / ((a + b/B_L) * d_L/d_S - a)."""
    return b / ((a + b / B_large) * d_large / d_small - a)


def update_factor(d_small, d_large, sqrt_scheme=False):
    """Model-update factor of a small-batch worker (Sec. 3.4): d_S/d_L, or its square root."""
    r = d_small / d_large
    return math.sqrt(r) if sqrt_scheme else r


def epoch_time(a, b, x, d):
    """Eq. 2: t = (a*x + b) * ceil(d/x)."""
    return (a * x + b) * math.ceil(d / x)


def epoch_time_simplified(a, b, x, d):
    """Eq. 3: t ~ (a + b/x) * d."""
    return (a + b / x) * d
