"""Host-side detection of a worker that does not push (ASP, Sec. 2.4: the server applies
what arrives and does not wait for a stopped worker).  The server's deadline logic runs on
the host and is tested here without a GPU, with fake events, a fake wait and a fake clock."""
import pytest

from paper_2509_26092_gb300 import dbl as D
from paper_2509_26092_gb300.resnet18 import collect_pushes


class FakeClock:
    def __init__(self):
        self.t = 0.0

    def __call__(self):
        return self.t


def _waiter(clock, finish_at, log):
    """wait(event, seconds): an event completes at finish_at[event] on the fake clock (None: never)."""
    def wait(ev, seconds):
        log.append((ev, round(seconds, 6)))
        t_done = finish_at[ev]
        if t_done is not None and t_done <= clock.t + seconds:
            clock.t = max(clock.t, t_done)
            return D.DBL_OK
        clock.t += seconds
        return D.DBL_ERR_TIMEOUT
    return wait


def test_both_workers_push():
    clock, log = FakeClock(), []
    wait = _waiter(clock, {"eL": 0.2, "eS": 0.5}, log)
    assert collect_pushes({"L": "eL", "S": "eS"}, 1.0, wait, clock) == (["L", "S"], [])
    # the second wait gets what is left of the one deadline
    assert log == [("eL", 1.0), ("eS", 0.8)]


def test_a_worker_that_never_pushes_is_left_out():
    clock, log = FakeClock(), []
    wait = _waiter(clock, {"eL": 0.1, "eS": None}, log)
    assert collect_pushes({"L": "eL", "S": "eS"}, 0.5, wait, clock) == (["L"], ["S"])
    assert clock.t == pytest.approx(0.5)


def test_deadline_is_shared_not_per_worker():
    clock, log = FakeClock(), []
    wait = _waiter(clock, {"eL": None, "eS": 0.3}, log)
    # the large worker eats the whole deadline; the small one, done at 0.3, is still checked (with 0 s left)
    assert collect_pushes({"L": "eL", "S": "eS"}, 0.5, wait, clock) == (["S"], ["L"])
    assert log == [("eL", 0.5), ("eS", 0.0)]


def test_no_worker_pushes():
    clock, log = FakeClock(), []
    wait = _waiter(clock, {"eL": None, "eS": None}, log)
    assert collect_pushes({"L": "eL", "S": "eS"}, 0.2, wait, clock) == ([], ["L", "S"])


def test_a_failed_query_is_an_error_not_a_timeout():
    with pytest.raises(D.DblError):
        collect_pushes({"L": "eL"}, 1.0, lambda ev, s: D.DBL_ERR_CUDA, FakeClock())
