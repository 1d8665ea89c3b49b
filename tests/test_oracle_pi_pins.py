"""Pins of the oracle's scaling-factor record and of its per-segment median.

The experiments section reports the median per-parameter value of pi over time, and the
ImageNet figures its median per tensor.  The oracle records pi as each commit applies it
(Algorithm 1, Psi_GEM, clamped at zero) and takes medians by sorting.  These tests tie
both to facts that do not come from the oracle:

* a single worker without momentum has no drift (its snapshot is the central variable)
  and m = dtheta, so pi reduces to |dtheta| / (|dtheta| + eps);
* the recorded pi is the factor the commit applied: theta_{t+1} - theta_t = pi dtheta;
* pi = 0 exactly where the proxy energy does not exceed the drift (the clamp);
* DOWNPOUR applies pi = 1 and adaptive staleness pi = 1 / (tau + 1);
* the kappa forms coincide with GEM at kappa = 1, and with each other when sqrt(kappa)
  is exact;
* the medians of hand-sorted cases, rank-count properties and numpy's median.
"""
import numpy as np
import pytest

import oracle


def _rand(P, n, T, seed, dtype):
    rng = np.random.default_rng(seed)
    theta0 = (0.05 * rng.standard_normal(P)).astype(dtype)
    grads = (rng.standard_normal((T, P)) * 10.0 ** rng.uniform(-4, -1, P)).astype(dtype)
    grads[:, ::9] = 0.0
    order, tau = oracle.schedule_uniform(seed, n, T)
    return theta0, grads, order, tau


def _fresh(theta0, n):
    return theta0.copy(), np.zeros((n, theta0.size), theta0.dtype), np.tile(theta0, (n, 1))


def test_single_worker_without_momentum_closed_form():
    P, T, eta, eps = 257, 12, 0.05, 1e-8
    theta0, grads, _o, _t = _rand(P, 1, T, 3, np.float64)
    th, m, s = _fresh(theta0, 1)
    pi = oracle.gem_run(th, m, s, grads, [0] * T, eta=eta, mu=0.0, eps=eps, record_pi=True)
    d = np.abs(eta * grads)
    assert np.array_equal(pi, d / (d + eps))
    assert np.all(pi[:, ::9] == 0.0)                      # zero gradient: pi = 0 / eps


@pytest.mark.parametrize("mode", [oracle.MODE_GEM, oracle.MODE_KAPPA_LINEAR, oracle.MODE_ADAPTIVE])
def test_recorded_pi_is_the_applied_factor(mode):
    """theta after minus theta before equals pi * dtheta up to one rounding of theta."""
    P, n, T, eta = 300, 4, 40, 0.01
    theta0, grads, order, tau = _rand(P, n, T, 5, np.float64)
    th, m, s = _fresh(theta0, n)
    before = th.copy()
    for t in range(T):
        pi = oracle.gem_run(th, m, s, grads[t:t + 1], order[t:t + 1], eta=eta, mu=0.9, eps=1e-8,
                            tau=tau[t:t + 1], mode=mode, kappa=1.7, record_pi=True)[0]
        step = pi * -(eta * grads[t])
        assert np.all(np.abs((th - before) - step) <= 2 * np.spacing(np.abs(th)) + 1e-300), t
        before = th.copy()


def test_pi_is_zero_exactly_where_the_proxy_does_not_exceed_the_drift():
    P, n, T, eta, mu = 500, 5, 60, 0.01, 0.9
    theta0, grads, order, _tau = _rand(P, n, T, 9, np.float64)
    th, m, s = _fresh(theta0, n)
    zeros = 0
    for t in range(T):
        w = int(order[t])
        drift = np.abs(th - s[w])
        pi = oracle.gem_run(th, m, s, grads[t:t + 1], [w], eta=eta, mu=mu, eps=1e-8,
                            record_pi=True)[0]
        assert np.all(pi >= 0.0)
        assert np.array_equal(pi == 0.0, np.abs(m[w]) <= drift), t     # m[w] is the new moment
        zeros += int((pi == 0.0).sum())
    assert 0 < zeros < T * P                              # both branches exercised


def test_fixed_rules_record_their_factor():
    P, n, T = 64, 6, 50
    theta0, grads, order, tau = _rand(P, n, T, 11, np.float32)
    th, m, s = _fresh(theta0, n)
    pi = oracle.gem_run(th, m, s, grads, order, eta=0.01, mu=0.9, eps=1e-8,
                        mode=oracle.MODE_DOWNPOUR, record_pi=True)
    assert np.all(pi == 1.0)
    th, m, s = _fresh(theta0, n)
    pi = oracle.gem_run(th, m, s, grads, order, eta=0.01, mu=0.9, eps=1e-8, tau=tau,
                        mode=oracle.MODE_ADAPTIVE, record_pi=True)
    want = (np.float32(1.0) / (tau.astype(np.float32) + np.float32(1.0))).astype(np.float32)
    assert np.array_equal(pi, np.repeat(want[:, None], P, axis=1))
    assert tau.max() > 5                                  # a range of staleness values


def test_kappa_forms_against_gem_and_each_other():
    P, n, T = 200, 3, 30
    theta0, grads, order, _tau = _rand(P, n, T, 13, np.float32)
    runs = {}
    for key, mode, kappa in [("gem", oracle.MODE_GEM, 1.0), ("lin1", oracle.MODE_KAPPA_LINEAR, 1.0),
                             ("sqrt4", oracle.MODE_KAPPA_SQRT, 4.0), ("lin2", oracle.MODE_KAPPA_LINEAR, 2.0),
                             ("sqrt1", oracle.MODE_KAPPA_SQRT, 1.0)]:
        th, m, s = _fresh(theta0, n)
        runs[key] = oracle.gem_run(th, m, s, grads, order, eta=0.01, mu=0.9, eps=1e-8, mode=mode,
                                   kappa=kappa, record_pi=True)
    assert np.array_equal(runs["gem"], runs["lin1"]) and np.array_equal(runs["gem"], runs["sqrt1"])
    assert np.array_equal(runs["sqrt4"], runs["lin2"])
    assert not np.array_equal(runs["gem"], runs["lin2"])
    assert np.median(runs["lin2"]) >= np.median(runs["gem"])       # more energy, larger factors


@pytest.mark.parametrize("x,lo,hi", [
    ([3.0, 1.0, 2.0], 2.0, 2.0),
    ([4.0, 1.0, 3.0, 2.0], 2.0, 3.0),
    ([7.5], 7.5, 7.5),
    ([0.0, 0.0, 0.0, 1.0], 0.0, 0.0),
    ([0.0, 1.0, 1.0, 1.0], 1.0, 1.0),
    ([np.inf, 0.5], 0.5, np.inf),
    ([-1.0, -0.0, 0.0, 2.0, -3.0], -0.0, -0.0),
])
def test_median_hand_cases(x, lo, hi):
    a = np.array(x, np.float32)
    got_lo, got_hi = oracle.pi_median(a, [0, a.size])
    assert got_lo[0] == lo and got_hi[0] == hi


def test_median_segments_empty_and_rank_counts():
    rng = np.random.default_rng(17)
    x = rng.exponential(size=1001).astype(np.float32)
    x[rng.integers(0, 1001, 300)] = 0.0                   # ties, as clamped factors give
    seg = [0, 0, 1, 2, 10, 11, 500, 1001]
    lo, hi = oracle.pi_median(x, seg)
    assert np.isnan(lo[0]) and np.isnan(hi[0])
    for i in range(1, len(seg) - 1):
        v = x[seg[i]:seg[i + 1]]
        N = v.size
        for val, r in ((lo[i], (N - 1) // 2), (hi[i], N // 2)):
            assert (v < val).sum() <= r < (v <= val).sum()
        assert np.float64(lo[i]) / 2 + np.float64(hi[i]) / 2 == pytest.approx(np.median(v), rel=1e-15)


def test_mlp_simulator_records_the_factors_of_its_commits():
    """The simulator's first commit applies the gradient at theta_0 (every snapshot is
    theta_0); its recorded factors equal those of a flat commit of that gradient, which the
    tests above pin."""
    from paper_1805_08469_gb300 import synth
    dims, n, b, seed = [12, 7, 3], 3, 5, 21
    P = synth.mlp_param_count(dims)
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((40, dims[0])).astype(np.float32)
    y = rng.integers(0, dims[-1], 40).astype(np.int32)
    rows = rng.integers(0, 40, (4, b)).astype(np.int32)
    theta0 = (0.3 * rng.standard_normal(P)).astype(np.float32)
    order = np.array([2, 0, 2, 1], np.int32)
    th, m, s = theta0.copy(), np.zeros((n, P), np.float32), np.tile(theta0, (n, 1))
    _r, _l, pi = oracle.mlp_sim_run(dims, th, m, s, order, X, y, rows, eta=0.05, mu=0.9, eps=1e-8,
                                    record_pi=True)
    _loss, g = oracle.mlp_loss_grad(dims, theta0.astype(np.float64), X[rows[0]].astype(np.float64), y[rows[0]])
    th2, m2, s2 = theta0.copy(), np.zeros((n, P), np.float32), np.tile(theta0, (n, 1))
    ref = oracle.gem_run(th2, m2, s2, g.astype(np.float32)[None, :], [2], eta=0.05, mu=0.9, eps=1e-8,
                         record_pi=True)
    assert np.array_equal(pi[0], ref[0])
    assert pi.shape == (4, P) and np.all(pi >= 0)


def test_momentum_proxy_rule_closed_form_and_identities():
    """The proxy rule (Eq. momentum_update committed as is): with one worker and a constant
    gradient g, theta_t = theta_0 - eta g sum_{k=1..t} (1 - mu^k) / (1 - mu); with mu = 0 it
    is DOWNPOUR bit for bit; with one worker it is the textbook recursion v <- mu v - eta g,
    theta <- theta + v."""
    P, T, eta, mu = 50, 25, 0.05, 0.9
    rng = np.random.default_rng(2)
    theta0 = rng.standard_normal(P)
    g = rng.standard_normal(P)
    th, m, s = _fresh(theta0, 1)
    oracle.gem_run(th, m, s, np.tile(g, (T, 1)), [0] * T, eta=eta, mu=mu, eps=1e-8,
                   mode=oracle.MODE_MOMENTUM)
    want = theta0 - eta * g * sum((1 - mu ** k) / (1 - mu) for k in range(1, T + 1))
    np.testing.assert_allclose(th, want, rtol=1e-12, atol=1e-12)
    theta0, grads, order, _tau = _rand(64, 3, 40, 4, np.float32)
    a = _fresh(theta0, 3)
    b = _fresh(theta0, 3)
    oracle.gem_run(*a, grads, order, eta=0.01, mu=0.0, eps=1e-8, mode=oracle.MODE_MOMENTUM)
    oracle.gem_run(*b, grads, order, eta=0.01, mu=0.0, eps=1e-8, mode=oracle.MODE_DOWNPOUR)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[2], b[2])
    theta0, grads, _o, _t = _rand(32, 1, 30, 6, np.float64)
    th, m, s = _fresh(theta0, 1)
    oracle.gem_run(th, m, s, grads, [0] * 30, eta=0.02, mu=0.8, eps=1e-8, mode=oracle.MODE_MOMENTUM)
    v, ref = np.zeros(32), theta0.copy()
    for t in range(30):
        v = 0.8 * v - 0.02 * grads[t]
        ref = ref + v
    np.testing.assert_allclose(th, ref, rtol=1e-13, atol=1e-15)
