"""Host logic of the asynchronous dual-batch driver and the hybrid schedule
(paper_2509_26092_gb300.schedule): the ASP push order, the paper's schedule tables
and the per-sub-stage plan."""
import math

import pytest

from oracle import planner
from paper_2509_26092_gb300 import build_lib
from paper_2509_26092_gb300 import schedule as S


@pytest.fixture(scope="module")
def D():
    build_lib.build()
    from paper_2509_26092_gb300 import dbl
    return dbl


def test_push_order_merges_arrival_times():
    order = S.push_order(3.0, 1.0, 2, 6)
    assert "".join(t for _, t, _ in order) == "SSLSSSLS"  # ties at 3 and 6 go to the large worker
    assert [x[0] for x in order] == sorted(x[0] for x in order)
    assert [k for _, t, k in order if t == "L"] == [1, 2] and [k for _, t, k in order if t == "S"] == list(range(1, 7))


def test_push_order_counts_and_edges():
    order = S.push_order(2.5, 1.0, 4, 10)
    assert sum(t == "L" for _, t, _ in order) == 4 and sum(t == "S" for _, t, _ in order) == 10
    # within the first 10 time units the small worker pushes 2.5 times as often
    assert sum(1 for tm, t, _ in order if t == "S" and tm <= 10.0) == 10
    assert sum(1 for tm, t, _ in order if t == "L" and tm <= 10.0) == 4
    assert S.push_order(1.0, 1.0, 0, 2) == [(1.0, "S", 1), (2.0, "S", 2)]
    with pytest.raises(ValueError):
        S.push_order(0.0, 1.0, 1, 1)


def test_hybrid_schedules_are_the_papers():
    c = S.hybrid_schedule("cifar")
    assert sum(s.epochs for s in c) == 140
    assert [s.res for s in c] == [24, 32] * 3 and [s.batch_large for s in c] == [600, 560] * 3
    assert [s.lr for s in c] == [0.2, 0.2, 0.02, 0.02, 0.002, 0.002]
    assert [s.epochs for s in c] == [40, 40, 20, 20, 10, 10]
    i = S.hybrid_schedule("imagenet")
    assert sum(s.epochs for s in i) == 105
    assert [s.res for s in i] == [160, 224, 288] * 3 and [s.batch_large for s in i] == [2330, 1110, 740] * 3
    assert [s.dropout for s in i] == [0.1, 0.2, 0.3] * 3
    with pytest.raises(ValueError):
        S.hybrid_schedule("mnist")


def test_substage_plan_follows_eqs_4_to_8(D):
    sub = S.hybrid_schedule("cifar")[1]  # 40 epochs at 32 px, B_L 560
    a, b = 4.0e-6, 1.26e-3  # seconds per image and per batch
    p = S.substage_pushes(sub, 50000, 1.05, a, b, data_fraction=0.01)
    d_l = planner.data_large(1.05, 50000, 2)
    d_s = planner.data_small(50000, 1, 1, d_l)
    assert p["batch_small"] == math.floor(planner.small_batch(a, b, 560.0, d_l, d_s))
    assert p["f_small"] == pytest.approx(d_s / d_l, rel=1e-15)
    assert p["pushes_large"] == 40 * math.ceil(d_l * 0.01 / 560)
    assert p["pushes_small"] == 40 * math.ceil(d_s * 0.01 / p["batch_small"])
    assert p["t_large"] == pytest.approx(a * 560 + b) and p["t_small"] == pytest.approx(a * p["batch_small"] + b)
