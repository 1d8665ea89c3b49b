"""Pins of the oracle's GEM commit against what the paper and the mathematics fix.

Each test ties the oracle to something other than itself: hand-derived commits, special
cases that reduce to plain SGD or to a closed form, invariants of the energy argument
(Eqs. stability, stability_preferred, central_variable_energy_ideal) and an independent
history-based restatement of the asynchronous system on tiny inputs.
"""
import math

import numpy as np
import pytest

import oracle
from conftest import GOLDEN


def _fresh(theta0, n, dtype):
    theta = np.array(theta0, dtype=dtype)
    m = np.zeros((n, theta.shape[0]), dtype=dtype)
    s = np.tile(theta, (n, 1)).astype(dtype)
    return theta, m, s


def _hand_cases():
    rows = []
    for line in (GOLDEN / "gem_hand_commits.txt").read_text().splitlines():
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        lhs, rhs = line.split("|")
        rows.append((list(map(float, lhs.split())), list(map(float, rhs.split()))))
    return rows


@pytest.mark.parametrize("dtype", [np.float32, np.float64])
def test_hand_derived_commits(dtype):
    cases = _hand_cases()
    assert len(cases) == 6
    for (theta, s, m, mu, eta, eps, g), (theta1, m1, s1) in cases:
        th = np.array([theta], dtype=dtype)
        mm = np.array([[m]], dtype=dtype)
        ss = np.array([[s]], dtype=dtype)
        gg = np.array([[g]], dtype=dtype)
        oracle.gem_run(th, mm, ss, gg, [0], eta=eta, mu=mu, eps=eps)
        assert th[0] == theta1 and mm[0, 0] == m1 and ss[0, 0] == s1, (theta, s, m, g)


@pytest.mark.parametrize("dtype", [np.float32, np.float64])
def test_single_worker_without_momentum_is_sgd(dtype):
    # n = 1 and post-commit pull: theta - s = 0, so pi = |dtheta| / |dtheta| = 1 exactly
    # once eps is below half an ulp of |dtheta|; the commit is then plain SGD, bit for bit.
    rng = np.random.default_rng(11)
    P, T, eta = 257, 60, 0.01
    theta0 = rng.standard_normal(P)
    g = rng.uniform(1e-3, 1.0, (T, P)) * rng.choice([-1.0, 1.0], (T, P))
    g[:, :5] = 0.0  # zero gradients leave theta unchanged in both rules
    g = g.astype(dtype)
    theta, m, s = _fresh(theta0, 1, dtype)
    oracle.gem_run(theta, m, s, g, np.zeros(T), eta=eta, mu=0.0, eps=1e-30)
    ref = np.array(theta0, dtype=dtype)
    e = dtype(eta)
    for t in range(T):
        ref = ref - e * g[t]
    assert np.array_equal(theta, ref)
    assert np.array_equal(s[0], theta)


def test_single_worker_with_momentum_closed_form():
    # n = 1, mu > 0: theta - s = 0 and pi = |m| / |dtheta| (eps -> 0), so each commit adds
    # |m_t| sign(dtheta_t) with m_t = sum_i mu^(t-i) dtheta_i (Eq. moment_estimate unrolled).
    rng = np.random.default_rng(12)
    P, T, eta, mu = 64, 40, 0.05, 0.9
    theta0 = rng.standard_normal(P)
    g = rng.standard_normal((T, P))
    theta, m, s = _fresh(theta0, 1, np.float64)
    oracle.gem_run(theta, m, s, g, np.zeros(T), eta=eta, mu=mu, eps=1e-300)
    dth = -eta * g
    expect = np.array(theta0, dtype=np.float64)
    for t in range(T):
        mt = sum(mu ** (t - i) * dth[i] for i in range(t + 1))
        expect = expect + np.abs(mt) * np.sign(dth[t])
    np.testing.assert_allclose(theta, expect, rtol=1e-12, atol=1e-12)


def test_eps_sits_outside_the_absolute_value():
    # n = 1, mu = 0: pi = |dtheta| / (|dtheta| + eps) exactly as printed in Psi_GEM.
    rng = np.random.default_rng(13)
    P, eta, eps = 50, 1.0, 0.3
    theta0 = rng.standard_normal(P)
    g = rng.standard_normal((1, P))
    theta, m, s = _fresh(theta0, 1, np.float64)
    oracle.gem_run(theta, m, s, g, [0], eta=eta, mu=0.0, eps=eps)
    d = -eta * g[0]
    np.testing.assert_allclose(theta, theta0 + d * np.abs(d) / (np.abs(d) + eps), rtol=1e-14)


def _random_run_states(dtype, n=4, P=400, T=300, seed=14, eps=1e-8):
    rng = np.random.default_rng(seed)
    theta0 = (0.05 * rng.standard_normal(P)).astype(dtype)
    g = (rng.standard_normal((T, P)) * 10.0 ** rng.uniform(-4, -1, P)).astype(dtype)
    order = rng.integers(0, n, T)
    theta, m, s = _fresh(theta0, n, dtype)
    for t in range(T):
        w = order[t]
        before = (theta.copy(), m[w].copy(), s[w].copy())
        oracle.gem_run(theta, m, s, g[t:t + 1], [w], eta=0.01, mu=0.9, eps=eps)
        yield before, (theta.copy(), m[w].copy(), s[w].copy()), g[t], w


@pytest.mark.parametrize("dtype", [np.float32, np.float64])
def test_energy_bound_nonnegative_pi_and_compliance(dtype):
    # Stability (Eq. stability): the central variable's energy seen by the committing
    # worker, 1/2 (theta_{t+1} - s)^2, stays below the proxy energy 1/2 m^2 unless the
    # drift alone already exceeded it, in which case the commit adds nothing (pi = 0).
    # Compliance (Eq. stability_preferred) holds with equality when the drift and the
    # update share a sign and pi is not clamped (eps negligible here).
    u = np.finfo(dtype).eps
    n_same = n_clamped = 0
    for (th0, m0, s0), (th1, m1, s1), g, _w in _random_run_states(dtype, eps=1e-30):
        dth = -(dtype(0.01) * g)
        drift0 = np.abs(th0 - s0)
        step = th1 - th0
        scale = np.abs(th1) + np.abs(s0) + np.abs(m1)
        # pi >= 0: the applied step never opposes the update
        assert np.all((step == 0) | (np.sign(step) == np.sign(dth)))
        # energy bound
        lhs = np.abs(th1 - s0)
        assert np.all(lhs <= np.maximum(np.abs(m1), drift0) + 16 * u * scale)
        # clamped coordinates are left unchanged
        clamped = np.abs(m1) < drift0
        n_clamped += int(clamped.sum())
        assert np.array_equal(th1[clamped], th0[clamped])
        # compliance in the same-sign, unclamped case
        same = (np.sign(th0 - s0) == np.sign(dth)) & (np.abs(m1) > drift0)
        n_same += int(same.sum())
        assert np.all(np.abs(lhs[same] - np.abs(m1[same])) <= 16 * u * scale[same])
        # the worker's snapshot after its commit is the new central variable
        assert np.array_equal(s1, th1)
    assert n_same > 1000 and n_clamped > 1000


def test_history_restatement_on_tiny_inputs():
    # An independent statement of the asynchronous system, straight from the equations:
    # s_t = theta_{t - tau_t} looked up in the history of the central variable (Eq.
    # staleness) with tau_t counted from the schedule, m_t as the power sum of the
    # worker's own raw updates (Eq. moment_estimate unrolled), the proxy energy
    # E_k = 1/2 m_t^2 (Eq. proxy_estimate) and pi from Eq. new_pi with its square roots.
    rng = np.random.default_rng(15)
    for n, P, T in ((1, 3, 25), (2, 5, 40), (3, 8, 60)):
        eta, mu, eps = 0.1, 0.8, 1e-9
        theta0 = rng.standard_normal(P)
        g = rng.standard_normal((T, P))
        order = rng.integers(0, n, T)
        theta, m, s = _fresh(theta0, n, np.float64)
        traj = oracle.gem_run(theta, m, s, g, order, eta=eta, mu=mu, eps=eps,
                              record_cols=np.arange(P))
        hist = [list(theta0)]
        last = {}
        mine = {w: [] for w in range(n)}
        for t in range(T):
            w = int(order[t])
            tau = t - last.get(w, -1) - 1
            last[w] = t
            snap = hist[t - tau]
            cur = hist[t]
            nxt = []
            mine[w].append([-eta * g[t][j] for j in range(P)])
            k = len(mine[w]) - 1
            for j in range(P):
                dth = mine[w][k][j]
                mt = sum(mu ** (k - i) * mine[w][i][j] for i in range(k + 1))
                ek = 0.5 * mt * mt
                pi = (math.sqrt(2.0) * math.sqrt(ek) - abs(cur[j] - snap[j])) / (abs(dth) + eps)
                pi = max(pi, 0.0)
                nxt.append(cur[j] + pi * dth)
            hist.append(nxt)
        np.testing.assert_allclose(traj, np.array(hist[1:]), rtol=1e-9, atol=1e-11)


def test_round_robin_drift_is_the_other_workers_updates():
    # Eq. central_variable_energy_ideal: with round-robin commits, theta_t - s_t is the
    # sum of the n - 1 updates committed since the worker's last commit, so the energy is
    # 1/2 (pi_t dtheta_t + sum_{i=1}^{n-1} pi_{t-i} dtheta_{t-i})^2.
    rng = np.random.default_rng(16)
    n, P, T = 5, 32, 40
    theta0 = rng.standard_normal(P)
    g = rng.standard_normal((T, P))
    order = np.arange(T) % n
    theta, m, s = _fresh(theta0, n, np.float64)
    traj = oracle.gem_run(theta, m, s, g, order, eta=0.05, mu=0.9, eps=1e-12,
                          record_cols=np.arange(P))
    full = np.vstack([theta0, traj])
    applied = np.diff(full, axis=0)  # pi_t dtheta_t
    for t in range(n, T):
        snap = full[t - (n - 1)]     # worker pulled right after its commit at t - n
        np.testing.assert_allclose(full[t] - snap, applied[t - n + 1:t].sum(axis=0),
                                   rtol=1e-12, atol=1e-13)


def test_worker_drop_out_freezes_its_state():
    """A worker that stops committing (it dropped out, or stalled for good) keeps m_w and
    s_w exactly as its last commit left them, and from then on the run is that of the
    remaining workers alone, started from the same theta and the same per-worker state: a
    commit reads and writes only theta and its own worker's row."""
    rng = np.random.default_rng(17)
    n, P, T, gone, after = 3, 64, 60, 2, 12
    theta0 = rng.standard_normal(P).astype(np.float32)
    g = (0.3 * rng.standard_normal((T, P))).astype(np.float32)
    base = rng.integers(0, n, 4 * T)
    order = np.array([w for t, w in enumerate(base) if not (w == gone and t >= after)][:T], np.int32)
    last = max(t for t in range(T) if order[t] == gone)
    theta, m, s = _fresh(theta0, n, np.float32)
    oracle.gem_run(theta, m, s, g[:last + 1], order[:last + 1], eta=0.05, mu=0.9, eps=1e-8)
    m_gone, s_gone = m[gone].copy(), s[gone].copy()
    keep = [w for w in range(n) if w != gone]
    th_b, m_b, s_b = theta.copy(), m[keep].copy(), s[keep].copy()
    oracle.gem_run(theta, m, s, g[last + 1:], order[last + 1:], eta=0.05, mu=0.9, eps=1e-8)
    assert np.array_equal(m[gone], m_gone) and np.array_equal(s[gone], s_gone)
    remap = {w: i for i, w in enumerate(keep)}
    oracle.gem_run(th_b, m_b, s_b, g[last + 1:], np.array([remap[w] for w in order[last + 1:]], np.int32),
                   eta=0.05, mu=0.9, eps=1e-8)
    assert np.array_equal(theta, th_b)
    assert np.array_equal(m[keep], m_b) and np.array_equal(s[keep], s_b)
    assert not np.array_equal(theta, s_gone)              # the others did move theta


def test_literal_precommit_snapshot_reading_differs():
    # Contrast: taking s as the value pulled before the own commit breaks the reduction
    # of a single worker to SGD (its drift is then its own previous update).
    rng = np.random.default_rng(17)
    P, T = 16, 10
    theta0 = rng.standard_normal(P)
    g = rng.uniform(0.1, 1.0, (T, P))
    a = _fresh(theta0, 1, np.float64)
    b = _fresh(theta0, 1, np.float64)
    oracle.gem_run(*a, g, np.zeros(T), eta=0.1, mu=0.0, eps=1e-300)
    oracle.gem_run(*b, g, np.zeros(T), eta=0.1, mu=0.0, eps=1e-300, precommit_snapshot=True)
    np.testing.assert_allclose(a[0], theta0 - 0.1 * g.sum(axis=0), rtol=1e-12)
    assert not np.allclose(b[0], a[0])


def test_downpour_is_plain_asynchronous_sgd():
    # DOWNPOUR commits dtheta unscaled: theta_T = theta_0 - eta sum_t g_t, in commit order.
    rng = np.random.default_rng(18)
    n, P, T = 3, 100, 50
    theta0 = rng.standard_normal(P).astype(np.float32)
    g = rng.standard_normal((T, P)).astype(np.float32)
    theta, m, s = _fresh(theta0, n, np.float32)
    oracle.gem_run(theta, m, s, g, rng.integers(0, n, T), eta=0.01, mu=0.9, eps=1e-8,
                   mode=oracle.MODE_DOWNPOUR)
    ref = theta0.copy()
    for t in range(T):
        ref = ref - np.float32(0.01) * g[t]
    assert np.array_equal(theta, ref)


def test_adaptive_staleness_round_robin_divides_by_n():
    # Round robin gives tau = n - 1 after the first round, so each update is dtheta / n.
    rng = np.random.default_rng(19)
    n, P, T = 4, 20, 24
    theta0 = rng.standard_normal(P)
    g = rng.standard_normal((T, P))
    order = np.arange(T) % n
    tau = np.array([t if t < n else n - 1 for t in range(T)])
    theta, m, s = _fresh(theta0, n, np.float64)
    oracle.gem_run(theta, m, s, g, order, tau=tau, eta=0.1, mu=0.9, eps=1e-8,
                   mode=oracle.MODE_ADAPTIVE)
    expect = theta0 - 0.1 * sum(g[t] / (tau[t] + 1) for t in range(T))
    np.testing.assert_allclose(theta, expect, rtol=1e-12, atol=1e-12)


def test_kappa_variants():
    # App. B: kappa = 1 is GEM under both forms; sqrt(kappa) with kappa = 4 equals the
    # linear form with kappa = 2; a single worker without momentum commits kappa dtheta.
    rng = np.random.default_rng(20)
    n, P, T = 3, 64, 30
    theta0 = (0.05 * rng.standard_normal(P)).astype(np.float32)
    g = (0.1 * rng.standard_normal((T, P))).astype(np.float32)
    order = rng.integers(0, n, T)

    def run(mode, kappa):
        st = _fresh(theta0, n, np.float32)
        oracle.gem_run(*st, g, order, eta=0.01, mu=0.9, eps=1e-8, mode=mode, kappa=kappa)
        return st[0]

    base = run(oracle.MODE_GEM, 1.0)
    assert np.array_equal(run(oracle.MODE_KAPPA_SQRT, 1.0), base)
    assert np.array_equal(run(oracle.MODE_KAPPA_LINEAR, 1.0), base)
    assert np.array_equal(run(oracle.MODE_KAPPA_SQRT, 4.0), run(oracle.MODE_KAPPA_LINEAR, 2.0))
    th, m, s = _fresh(theta0.astype(np.float64), 1, np.float64)
    oracle.gem_run(th, m, s, g[:1].astype(np.float64), [0], eta=0.01, mu=0.0, eps=1e-300,
                   mode=oracle.MODE_KAPPA_LINEAR, kappa=2.0)
    nz = g[0] != 0
    np.testing.assert_allclose(th[nz], theta0[nz] - 2 * 0.01 * g[0][nz].astype(np.float64), rtol=1e-12)


def test_commit_threads_change_no_bit():
    # Psi_GEM and the update are elementwise (Algorithm 1), so splitting each commit's
    # coordinates across threads (the CPU baseline's multi-core run) must leave every bit
    # of theta, m, s and the recorded factors unchanged, for every commit rule.
    rng = np.random.default_rng(31)
    n, P, T = 5, 10_007, 40
    theta0 = (0.05 * rng.standard_normal(P)).astype(np.float32)
    g = (0.1 * rng.standard_normal((T, P))).astype(np.float32)
    order = rng.integers(0, n, T)
    tau = rng.integers(0, 7, T)
    for mode in (oracle.MODE_GEM, oracle.MODE_ADAPTIVE, oracle.MODE_KAPPA_LINEAR,
                 oracle.MODE_MOMENTUM):
        out = []
        for threads in (1, 4):
            prev = oracle.set_commit_threads(threads)
            try:
                st = _fresh(theta0, n, np.float32)
                pi = oracle.gem_run(*st, g, order, tau=tau, eta=0.01, mu=0.9, eps=1e-8,
                                    mode=mode, kappa=2.0, record_pi=True)
            finally:
                oracle.set_commit_threads(prev)
            out.append((*st, pi))
        for a, b in zip(*out):
            assert np.array_equal(a, b, equal_nan=True), mode
