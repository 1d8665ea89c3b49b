"""GPU parity of the scaling-factor statistics against the oracle, through the C ABI.

gem_commit_batch_pi records the factor pi each commit applied to each coordinate; the
oracle records the same quantity (bit for bit, as the commit arithmetic is identical).
gem_pi_median selects, per row and segment, the lower and upper middle elements; the
oracle sorts.  Selection is exact, so the bar is equality of the selected values.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_1805_08469_gb300 import gem, synth, synth_gpu
from paper_1805_08469_gb300._build import build_library
from paper_1805_08469_gb300._lib import GemError

pytestmark = pytest.mark.gpu

ETA, MU, EPS = 0.01, 0.9, 1e-8


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
    grads[:, ::13] = 0.0
    order, tau = oracle.schedule_uniform(seed, n, T)
    return theta0, grads, order, tau


@pytest.mark.parametrize("mode,omode,kappa", [
    (gem.GEM_MODE_GEM, oracle.MODE_GEM, 1.0),
    (gem.GEM_MODE_KAPPA_LINEAR, oracle.MODE_KAPPA_LINEAR, 2.0),
    (gem.GEM_MODE_ADAPTIVE, oracle.MODE_ADAPTIVE, 1.0),
])
@pytest.mark.parametrize("P", [5, 4099, 100_003])
def test_recorded_factors_bitwise_and_commits_unchanged(mode, omode, kappa, P):
    """Every third commit recorded (the others pass None); the recorded rows equal the
    oracle's, and theta, m, s equal a run without recording."""
    n, T = 5, 230
    theta0, grads, order, tau = _inputs(P, n, T, 300 + P)
    th, m, s = theta0.copy(), np.zeros((n, P), np.float32), np.tile(theta0, (n, 1))
    ref_pi = oracle.gem_run(th, m, s, grads, order, eta=ETA, mu=MU, eps=EPS, tau=tau, mode=omode,
                            kappa=kappa, record_pi=True)
    g_dev = _padded(grads)
    pi_dev = torch.full((T, (P + 3) // 4 * 4), -1.0, device="cuda")
    rec = [pi_dev[k, :P] if k % 3 == 0 else None for k in range(T)]
    with gem.Gem(P, n, ETA, MU, EPS) as A, gem.Gem(P, n, ETA, MU, EPS) as B:
        for G in (A, B):
            G.set_mode(mode, kappa)
            G.set_theta(torch.from_numpy(theta0).cuda())
        A.commit_batch_pi(order.tolist(), [g_dev[k, :P] for k in range(T)], rec)
        B.commit_batch(order.tolist(), [g_dev[k, :P] for k in range(T)])
        A.sync()
        B.sync()
        assert torch.equal(A.theta(), B.theta())
        for w in range(n):
            assert torch.equal(A.moment(w), B.moment(w)) and torch.equal(A.snapshot(w), B.snapshot(w))
        assert np.array_equal(A.theta().cpu().numpy(), th)
    got = pi_dev.cpu().numpy()
    for k in range(T):
        if k % 3 == 0:
            assert np.array_equal(got[k, :P], ref_pi[k]), k
        else:
            assert np.all(got[k, :P] == -1.0), k           # not recorded: untouched


def _check_medians(rows: np.ndarray, seg, K_dev=None):
    """Upload rows [K, P], select on the GPU, compare with the oracle's sorted medians."""
    K, P = rows.shape
    nseg = len(seg) - 1
    dev = _padded(rows)
    lo = torch.empty((K, nseg), device="cuda")
    hi = torch.empty((K, nseg), device="cuda")
    with gem.Gem(P, 1, ETA, MU, EPS) as G:
        G.pi_median([dev[k, :P] for k in range(K)], seg, lo, hi)
        G.sync()
    glo, ghi = lo.cpu().numpy(), hi.cpu().numpy()
    for k in range(K):
        rlo, rhi = oracle.pi_median(rows[k], seg)
        both_nan = np.isnan(rlo) & np.isnan(glo[k])
        assert np.all(both_nan | (glo[k] == rlo)), (k, glo[k], rlo)
        assert np.all(np.isnan(rhi) & np.isnan(ghi[k]) | (ghi[k] == rhi)), (k, ghi[k], rhi)


def test_medians_of_ties_signs_and_infinities():
    rng = np.random.default_rng(1)
    K, P = 7, 50_001
    rows = rng.exponential(size=(K, P)).astype(np.float32)
    rows[0, :] = 0.0                                      # all equal
    rows[1, rng.random(P) < 0.7] = 0.0                    # most clamped
    rows[2] = -rows[2]                                    # negatives
    rows[3, ::2] = -0.0
    rows[4, rng.integers(0, P, 100)] = np.inf
    rows[5] = np.float32(1.0) / (rng.integers(0, 40, P).astype(np.float32) + 1)   # adaptive-like
    rows[6] = (rng.standard_normal(P) * 1e-40).astype(np.float32)                 # subnormals
    _check_medians(rows, [0, P])


def test_medians_per_tensor_of_the_mlp_layout_and_odd_segments():
    dims = [784, 1000, 1000, 10]
    P = synth.mlp_param_count(dims)
    seg = [0]
    for (wo, bo, fo, fi) in synth.mlp_layout(dims):
        seg += [wo + fo * fi, bo + fo]
    assert seg[-1] == P
    rng = np.random.default_rng(2)
    rows = (rng.exponential(size=(3, P)) * (rng.random((3, P)) < 0.6)).astype(np.float32)
    _check_medians(rows, seg)
    # empty, length-1, length-2 and unaligned segments
    _check_medians(rows[:, :100_000], [0, 0, 1, 3, 3, 40_001, 99_999, 100_000])


def test_more_rows_than_one_select_launch():
    rng = np.random.default_rng(3)
    rows = rng.standard_normal((250, 3001)).astype(np.float32)
    _check_medians(rows, [0, 1000, 3001])


def test_full_size_rows_of_the_benchmark_workload():
    """P = 25M, four commits of the heavy-tailed workload (n = 100, seed 5): factors
    recorded on the GPU and compared with the oracle's factors for a sample of coordinates
    (every coordinate's factor depends only on that coordinate), then medians of the full
    rows against a host sort of the GPU's rows."""
    P, n, K, seed = 25_000_000, 100, 4, 5
    order, tau = oracle.schedule_uniform(seed, n, K)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream), gem.Gem(P, n, ETA, MU, EPS, stream=stream) as G:
        theta0 = synth_gpu.theta0_flat(seed, torch.empty(P, device="cuda"), stream=stream)
        G.set_theta(theta0)
        pool = torch.empty((K, P), device="cuda")
        synth_gpu.grad_heavytail(seed, 0, pool, P, stream=stream)
        pi = torch.empty((K, P), device="cuda")
        G.commit_batch_pi(order.tolist(), [pool[k] for k in range(K)], [pi[k] for k in range(K)])
        lo = torch.empty((K, 1), device="cuda")
        hi = torch.empty((K, 1), device="cuda")
        G.pi_median([pi[k] for k in range(K)], [0, P], lo, hi)
        G.sync()
        cols = np.sort(np.random.default_rng(4).choice(P, 20_000, replace=False))
        cols_dev = torch.from_numpy(cols).cuda()
        g_host = pool[:, cols_dev].cpu().numpy()
        th0 = theta0[cols_dev].cpu().numpy()
        rows = pi.cpu().numpy()
        glo, ghi = lo.cpu().numpy()[:, 0], hi.cpu().numpy()[:, 0]
    th, m, s = th0.copy(), np.zeros((n, cols.size), np.float32), np.tile(th0, (n, 1))
    ref = oracle.gem_run(th, m, s, np.ascontiguousarray(g_host), order, eta=ETA, mu=MU, eps=EPS,
                         record_pi=True)
    assert np.array_equal(rows[:, cols], ref)
    for k in range(K):
        rlo, rhi = oracle.pi_median(rows[k], [0, P])
        assert glo[k] == rlo[0] and ghi[k] == rhi[0], (k, glo[k], rlo, ghi[k], rhi)


def test_argument_checks():
    P = 1000
    with gem.Gem(P, 2, ETA, MU, EPS) as G:
        row = torch.zeros(P, device="cuda")
        lo = torch.empty(4, device="cuda")
        hi = torch.empty(4, device="cuda")
        for seg in ([0], [0, P + 1], [10, 5], [-1, 5], list(range(66))):
            with pytest.raises(GemError) as e:
                G.pi_median([row], seg, lo, hi)
            assert e.value.status == gem.GEM_EINVAL
        G.pi_median([], [0, P], lo, hi)                   # K = 0: no-op
        g = torch.zeros(P + 8, device="cuda")
        with pytest.raises(GemError):
            G.commit_batch_pi([0], [g[:P]], [g[1:P + 1]])  # unaligned pi row
        G.sync()
