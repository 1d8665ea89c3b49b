"""Pins of the oracle's commit schedules (Introduction, Eq. staleness).

The generator is checked against SplitMix64's published outputs; the schedules against
the expected staleness n - 1 of a homogeneous queueing model and the geometric law of
the gap between two commits of the same worker.
"""
import numpy as np
import pytest

import oracle
from conftest import GOLDEN
from paper_1805_08469_gb300 import synth


def _golden_splitmix():
    lines = (GOLDEN / "splitmix64_state0.txt").read_text().splitlines()
    return [int(l.strip(), 16) for l in lines if l.strip() and not l.startswith("#")]


def test_splitmix64_published_outputs():
    gold = _golden_splitmix()
    assert len(gold) == 3
    assert [oracle.splitmix64_raw(0, c) for c in range(3)] == gold
    # the input generators follow the same definition
    assert synth.splitmix64_sequence(0, 3) == gold
    assert [int(synth.draw(0, c)) for c in range(3)] == gold


def test_keyed_streams_agree_with_generator_module():
    for seed, stream, c in ((1, 10, 0), (7, 11, 123456789), (2**63 + 5, 3, 2**40 + 17)):
        assert oracle.splitmix64_draw(seed, stream, c) == int(synth.draw(synth.key(seed, stream), c))


def _check_staleness(order, tau, n):
    T = len(order)
    assert order.min() >= 0 and order.max() < n
    # staleness recount from its definition: commits since the worker's last commit
    last = {}
    for t in range(T):
        w = int(order[t])
        assert tau[t] == t - last.get(w, -1) - 1
        last[w] = t
    # E[tau] = n - 1 (geometric gaps with p = 1/n), after the first round
    body = tau[T // 10:]
    se = np.sqrt((1 - 1 / n) * n * n / len(body))
    assert abs(body.mean() - (n - 1)) < 5 * se, (body.mean(), n - 1, se)
    # P(tau = 0) = 1/n
    p0 = (body == 0).mean()
    assert abs(p0 - 1 / n) < 5 * np.sqrt(p0 * (1 - p0) / len(body)) + 1e-3
    counts = np.bincount(order, minlength=n)
    expect = T / n
    chi2 = ((counts - expect) ** 2 / expect).sum()
    assert chi2 < n + 6 * np.sqrt(2 * n), chi2


@pytest.mark.parametrize("n", [1, 4, 30, 100])
def test_uniform_tick_schedule(n):
    T = 100_000
    order, tau = oracle.schedule_uniform(1 + n, n, T)
    if n == 1:
        assert np.all(order == 0) and np.all(tau == 0)
        return
    _check_staleness(order, tau, n)
    order2, _ = oracle.schedule_uniform(1 + n, n, T)
    assert np.array_equal(order, order2)


@pytest.mark.parametrize("n", [4, 30])
def test_exponential_queue_schedule(n):
    # Memorylessness of exponential service makes the next committer uniform, so the
    # staleness law is again geometric with mean n - 1.
    T = 60_000
    order, tau = oracle.schedule_queue(3 + n, n, T, 1.0)
    _check_staleness(order, tau, n)
    # the rate only rescales time: same order at rate 2
    order2, _ = oracle.schedule_queue(3 + n, n, T, 2.0)
    assert np.array_equal(order, order2)


def test_schedule_rejects_bad_arguments():
    with pytest.raises(ValueError):
        oracle.schedule_uniform(1, 0, 10)
    with pytest.raises(ValueError):
        oracle.schedule_queue(1, 4, 10, 0.0)
