"""GPU parity of the other commit rules against the oracle, through the C ABI.

Besides Algorithm 1 the library applies the comparison rules of the paper's experiments
(DOWNPOUR: pi = 1; adaptive staleness: the update divided by tau + 1), the high-energy
proxies of Appendix B (sqrt(kappa) |m| and kappa |m|), and the momentum proxy itself
(Eq. momentum_update) as a reference run.  Each is one IEEE fp32 operation per
step on both sides, so the bar is bit-for-bit equality, as for the GEM rule.  The staleness
of the adaptive rule comes from the library's own commit clock; the oracle takes the tau
that its schedule generator computes, so the two are counted independently.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_1805_08469_gb300 import gem, sim, synth
from paper_1805_08469_gb300._build import build_library
from paper_1805_08469_gb300._lib import GemError

from test_gpu_mlp import device_data, host_rows, rel_l2

pytestmark = pytest.mark.gpu

ETA, MU, EPS = 0.01, 0.9, 1e-8

# (library mode, oracle mode, kappa)
RULES = [
    (gem.GEM_MODE_DOWNPOUR, oracle.MODE_DOWNPOUR, 1.0),
    (gem.GEM_MODE_ADAPTIVE, oracle.MODE_ADAPTIVE, 1.0),
    (gem.GEM_MODE_KAPPA_SQRT, oracle.MODE_KAPPA_SQRT, 2.0),     # sqrt(2) is inexact in fp32
    (gem.GEM_MODE_KAPPA_SQRT, oracle.MODE_KAPPA_SQRT, 4.0),
    (gem.GEM_MODE_KAPPA_LINEAR, oracle.MODE_KAPPA_LINEAR, 1.5),
    (gem.GEM_MODE_KAPPA_LINEAR, oracle.MODE_KAPPA_LINEAR, 0.3),
    (gem.GEM_MODE_MOMENTUM, oracle.MODE_MOMENTUM, 1.0),
]


@pytest.fixture(scope="module", autouse=True)
def _setup():
    build_library()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    torch.cuda.set_device(0)


def _padded(a: np.ndarray) -> torch.Tensor:
    T, P = a.shape
    d = torch.zeros((T, (P + 3) // 4 * 4), dtype=torch.float32, device="cuda")
    d[:, :P] = torch.from_numpy(a).cuda()
    return d


def _inputs(P, n, T, seed):
    rng = np.random.default_rng(seed)
    theta0 = (0.05 * rng.standard_normal(P)).astype(np.float32)
    grads = (rng.standard_normal((T, P)) * 10.0 ** rng.uniform(-4, -1, P)).astype(np.float32)
    grads[:, ::11] = 0.0                          # dtheta = 0: pi = 0 / eps, theta unchanged
    order, tau = oracle.schedule_uniform(seed, n, T)
    return theta0, grads, order, tau


def _state(G, n):
    return (G.theta().cpu().numpy(), [G.moment(w).cpu().numpy() for w in range(n)],
            [G.snapshot(w).cpu().numpy() for w in range(n)])


def _assert_bitwise(G, th, m, s, n, what):
    gth, gm, gs = _state(G, n)
    assert np.array_equal(gth, th), f"{what}: theta differs in {int((gth != th).sum())} elements"
    for w in range(n):
        assert np.array_equal(gm[w], m[w]), f"{what}: m_{w} differs"
        assert np.array_equal(gs[w], s[w]), f"{what}: s_{w} differs"


@pytest.mark.parametrize("mode,omode,kappa", RULES)
@pytest.mark.parametrize("P,n", [(5, 6), (4099, 6), (262_147, 6), (262_147, 40)])
def test_rule_batches_bitwise(mode, omode, kappa, P, n):
    """450 commits (three launches of at most 200) with repeated workers, against the
    oracle's run of the same rule.  With 40 workers a launch has more repeats open at once
    than it has on-chip slots, so every slot (shared memory and registers) is in use, next
    to repeats that go through global memory."""
    T = 450
    theta0, grads, order, tau = _inputs(P, n, T, 1000 + P)
    th, m, s = theta0.copy(), np.zeros((n, P), np.float32), np.tile(theta0, (n, 1))
    oracle.gem_run(th, m, s, grads, order, eta=ETA, mu=MU, eps=EPS, tau=tau, mode=omode, kappa=kappa)
    g_dev = _padded(grads)
    with gem.Gem(P, n, ETA, MU, EPS) as G:
        G.set_mode(mode, kappa)
        G.set_theta(torch.from_numpy(theta0).cuda())
        G.commit_batch(order.tolist(), [g_dev[k, :P] for k in range(T)])
        G.sync()
        _assert_bitwise(G, th, m, s, n, f"mode {mode} kappa {kappa}")
        clock, last = G.clock()
        assert clock == T
        for w in range(n):
            hits = np.nonzero(order == w)[0]
            assert last[w] == (int(hits[-1]) if hits.size else -1)


@pytest.mark.parametrize("mode,omode,kappa", RULES)
def test_rule_single_commits_and_staleness(mode, omode, kappa):
    """Commit by commit, with the staleness the library reports before each commit equal to
    the oracle schedule's tau."""
    P, n, T = 1003, 3, 30
    theta0, grads, order, tau = _inputs(P, n, T, 7)
    th, m, s = theta0.copy(), np.zeros((n, P), np.float32), np.tile(theta0, (n, 1))
    g_dev = _padded(grads)
    with gem.Gem(P, n, ETA, MU, EPS) as G:
        G.set_theta(torch.from_numpy(theta0).cuda())
        G.set_mode(mode, kappa)
        assert gem.gem_get_mode(G.h)[0] == mode
        for t in range(T):
            w = int(order[t])
            assert G.staleness(w) == int(tau[t]), t
            G.commit(w, g_dev[t, :P])
            oracle.gem_run(th, m, s, grads[t:t + 1], [w], eta=ETA, mu=MU, eps=EPS,
                           tau=tau[t:t + 1], mode=omode, kappa=kappa)
        G.sync()
        _assert_bitwise(G, th, m, s, n, f"mode {mode}")


def test_switching_rules_mid_run():
    """GEM, then DOWNPOUR and adaptive (which leave m alone), then kappa, then GEM again on
    the moments GEM left: the same chunks through the oracle give the same bits."""
    P, n, T = 70_001, 5, 300
    theta0, grads, order, tau = _inputs(P, n, T, 11)
    plan = [(0, 100, gem.GEM_MODE_GEM, oracle.MODE_GEM, 1.0),
            (100, 150, gem.GEM_MODE_DOWNPOUR, oracle.MODE_DOWNPOUR, 1.0),
            (150, 200, gem.GEM_MODE_ADAPTIVE, oracle.MODE_ADAPTIVE, 1.0),
            (200, 250, gem.GEM_MODE_KAPPA_LINEAR, oracle.MODE_KAPPA_LINEAR, 2.0),
            (250, 300, gem.GEM_MODE_GEM, oracle.MODE_GEM, 1.0)]
    th, m, s = theta0.copy(), np.zeros((n, P), np.float32), np.tile(theta0, (n, 1))
    g_dev = _padded(grads)
    with gem.Gem(P, n, ETA, MU, EPS) as G:
        G.set_theta(torch.from_numpy(theta0).cuda())
        for a, e, mode, omode, kappa in plan:
            G.set_mode(mode, kappa)
            G.commit_batch(order[a:e].tolist(), [g_dev[k, :P] for k in range(a, e)])
            oracle.gem_run(th, m, s, grads[a:e], order[a:e], eta=ETA, mu=MU, eps=EPS,
                           tau=tau[a:e], mode=omode, kappa=kappa)
        G.sync()
        _assert_bitwise(G, th, m, s, n, "mode switches")


def test_clock_checkpoint_resume():
    """An adaptive run interrupted after 120 commits and resumed in a new handle from the
    saved state and clock ends bit-identical to the uninterrupted run."""
    P, n, T, cut = 9_999, 4, 200, 120
    theta0, grads, order, _tau = _inputs(P, n, T, 13)
    g_dev = _padded(grads)
    gl = [g_dev[k, :P] for k in range(T)]
    with gem.Gem(P, n, ETA, MU, EPS) as A:
        A.set_mode(gem.GEM_MODE_ADAPTIVE)
        A.set_theta(torch.from_numpy(theta0).cuda())
        A.commit_batch(order.tolist(), gl)
        A.sync()
        ref = _state(A, n)
    with gem.Gem(P, n, ETA, MU, EPS) as B:
        B.set_mode(gem.GEM_MODE_ADAPTIVE)
        B.set_theta(torch.from_numpy(theta0).cuda())
        B.commit_batch(order[:cut].tolist(), gl[:cut])
        th = np.empty(P, np.float32)
        m = np.empty((n, P), np.float32)
        s = np.empty((n, P), np.float32)
        gem.gem_save_state(B.h, th, m, s)
        B.sync()
        clock, last = B.clock()
    assert clock == cut
    with gem.Gem(P, n, ETA, MU, EPS) as C:
        C.set_mode(gem.GEM_MODE_ADAPTIVE)
        gem.gem_load_state(C.h, th, m, s)
        C.set_clock(clock, last)
        C.commit_batch(order[cut:].tolist(), gl[cut:])
        C.sync()
        got = _state(C, n)
    assert np.array_equal(got[0], ref[0])
    for w in range(n):
        assert np.array_equal(got[1][w], ref[1][w]) and np.array_equal(got[2][w], ref[2][w])


def test_mode_and_clock_argument_checks():
    with gem.Gem(100, 3, ETA, MU, EPS) as G:
        for mode, kappa in [(-1, 1.0), (6, 1.0), (gem.GEM_MODE_KAPPA_SQRT, 0.0),
                            (gem.GEM_MODE_KAPPA_LINEAR, -2.0), (gem.GEM_MODE_KAPPA_LINEAR, float("nan")),
                            (gem.GEM_MODE_KAPPA_SQRT, float("inf"))]:
            with pytest.raises(GemError) as e:
                G.set_mode(mode, kappa)
            assert e.value.status == gem.GEM_EINVAL
        assert gem.gem_get_mode(G.h) == (gem.GEM_MODE_GEM, 1.0)    # unchanged by the failures
        G.set_mode(gem.GEM_MODE_DOWNPOUR, 7.0)                        # kappa ignored
        assert gem.gem_get_mode(G.h) == (gem.GEM_MODE_DOWNPOUR, 1.0)
        for clock, last in [(-1, None), (5, [0, 5, 1]), (5, [0, -2, 1])]:
            with pytest.raises(GemError):
                G.set_clock(clock, last)
        assert G.clock() == (0, [-1, -1, -1])
        with pytest.raises(GemError):
            G.staleness(3)
        G.set_clock(10, [3, -1, 9])
        assert [G.staleness(w) for w in range(3)] == [6, 10, 0]
        G.set_theta(torch.zeros(100, device="cuda"))                  # a new run: clock reset
        assert G.clock() == (0, [-1, -1, -1])


@pytest.mark.parametrize("mode,omode,kappa", [RULES[0], RULES[1], RULES[3], RULES[4]])
def test_mlp_runs_under_each_rule(mode, omode, kappa):
    """MLP 784-64-10, n = 4, b = 32, 40 uniform-tick commits from theta_0 under each rule,
    against the oracle's simulator with the same rule and the schedule's tau (fp32
    products: 1e-4, the trajectory bar)."""
    dims, n, b, T, seed = [784, 64, 10], 4, 32, 40, 1
    P = synth.mlp_param_count(dims)
    order, tau = oracle.schedule_uniform(seed, n, T)
    batches = synth.schedule_batches(seed, order, b)
    theta0 = synth.xavier_theta0(seed, dims)
    X, y = device_data(seed)
    with gem.Gem(P, n, ETA, MU, EPS) as G:
        G.set_mode(mode, kappa)
        G.set_theta(torch.from_numpy(theta0).cuda())
        M = sim.gem_mlp_create(G.h, dims, b)
        try:
            sim.gem_mlp_set_data(M, X, y)
            losses = torch.empty(T, device="cuda")
            sim.gem_mlp_run(M, order, batches, losses)
            G.sync()
            got = G.theta().cpu().numpy()
            got_losses = losses.cpu().numpy()
        finally:
            sim.gem_mlp_destroy(M)
    Xh, yh, local = host_rows(seed, batches)
    th, m, s = theta0.copy(), np.zeros((n, P), np.float32), np.tile(theta0, (n, 1))
    _rec, ref_losses = oracle.mlp_sim_run(dims, th, m, s, order, Xh, yh, local, eta=ETA, mu=MU,
                                          eps=EPS, tau=tau, mode=omode, kappa=kappa,
                                          want_losses=True)
    assert rel_l2(got, th) < 1e-4, rel_l2(got, th)
    np.testing.assert_allclose(got_losses, ref_losses, rtol=1e-4)
