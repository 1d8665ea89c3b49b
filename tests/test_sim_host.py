"""The product's simulator (host code, no GPU): its schedules equal the oracle's, written
independently from the same published generator definition, and its segments are maximal
runs of distinct workers."""
import numpy as np
import pytest

import oracle
from paper_1805_08469_gb300 import sim
from paper_1805_08469_gb300._build import build_library


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build_library()


@pytest.mark.parametrize("seed,n,T", [(1, 4, 200), (2, 20, 5000), (4, 100, 5000), (9, 1, 10)])
def test_uniform_schedule_matches_oracle(seed, n, T):
    o1, t1 = sim.gem_schedule_uniform(seed, n, T)
    o2, t2 = oracle.schedule_uniform(seed, n, T)
    assert np.array_equal(o1, o2) and np.array_equal(t1, t2)


@pytest.mark.parametrize("seed,n,T,rate", [(3, 30, 2000, 1.0), (5, 7, 3000, 0.5)])
def test_queue_schedule_matches_oracle(seed, n, T, rate):
    o1, t1 = sim.gem_schedule_queue(seed, n, T, rate)
    o2, t2 = oracle.schedule_queue(seed, n, T, rate)
    assert np.array_equal(o1, o2) and np.array_equal(t1, t2)


@pytest.mark.parametrize("n", [1, 4, 30, 100])
def test_segments_are_maximal_runs_of_distinct_workers(n):
    order, _ = sim.gem_schedule_uniform(11, n, 3000)
    seg = sim.gem_plan_segments(order, n)
    assert seg[0] == 0 and seg[-1] == len(order)
    assert np.all(np.diff(seg) > 0)
    for a, b in zip(seg[:-1], seg[1:]):
        ws = order[a:b]
        assert len(set(ws.tolist())) == len(ws)            # distinct workers
        if b < len(order):
            assert order[b] in set(ws.tolist())           # maximal
    if n == 1:
        assert len(seg) == len(order) + 1


def test_simulator_rejects_bad_arguments():
    with pytest.raises(ValueError):
        sim.gem_schedule_uniform(1, 0, 5)
    with pytest.raises(ValueError):
        sim.gem_schedule_queue(1, 3, 5, -1.0)
    with pytest.raises(ValueError):
        sim.gem_plan_segments(np.array([0, 5, 1]), 3)
