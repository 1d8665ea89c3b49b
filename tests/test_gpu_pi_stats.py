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


def test_medians_at_the_edges_of_a_zero_run():
    """Runs of exact +0 (the clamp of the factor) next to negatives, -0, positives and
    positive subnormals, with the run ending between the lower and the upper middle element
    or just before both; compared bit for bit, so a -0 returned for +0 (or the reverse), or
    a subnormal ranked as if the zeros were not counted, fails."""
    rng = np.random.default_rng(4)
    P = 50_000
    pos = lambda n: (rng.exponential(size=n) + 1e-3).astype(np.float32)
    sub = lambda n: rng.integers(1, 0x200000, n).astype(np.uint32).view(np.float32)
    parts = [
        [np.zeros(25_000), pos(25_000)],                                  # lo = +0, hi > 0
        [-pos(25_000), np.zeros(25_000)],                                 # lo < 0, hi = +0
        [-pos(10_000), np.zeros(30_000), pos(10_000)],                    # both +0 after negatives
        [-pos(20_000), np.full(10_000, -0.0), np.zeros(10_000), pos(10_000)],   # both -0
        [np.full(25_000, -0.0), np.zeros(25_000)],                        # lo = -0, hi = +0
        # positive subnormals (bit patterns 1 .. 0x1FFFFF) share the first pass's bin with
        # +0: middle elements just past the zeros must be ranked among the subnormals
        [np.zeros(24_990), sub(25_010)],                                  # both subnormal
        [np.zeros(25_000), sub(25_000)],                                  # lo = +0, hi subnormal
        [-pos(1_000), np.zeros(23_998), sub(25_002)],                     # both just past the zeros
        [-pos(1_000), np.full(500, -0.0), np.zeros(22_000), sub(26_500)],
    ]
    rows = np.stack([rng.permutation(np.concatenate(p).astype(np.float32)) for p in parts])
    dev = _padded(rows)
    lo = torch.empty((len(parts), 1), device="cuda")
    hi = torch.empty((len(parts), 1), device="cuda")
    with gem.Gem(P, 1, ETA, MU, EPS) as G:
        G.pi_median([dev[k, :P] for k in range(len(parts))], [0, P], lo, hi)
        G.sync()
    glo, ghi = lo.cpu().numpy(), hi.cpu().numpy()
    for k in range(len(parts)):
        # values as the oracle's sort gives them (IEEE order: -0 and +0 compare equal) ...
        rlo, rhi = oracle.pi_median(rows[k], [0, P])
        assert glo[k, 0] == rlo[0] and ghi[k, 0] == rhi[0], (k, glo[k], ghi[k], rlo, rhi)
        # ... and the exact bits of the total order the library documents (-0 below +0)
        u = rows[k].view(np.uint32)
        keys = np.sort(np.where(u >> 31, ~u, u | np.uint32(0x80000000)))
        back = lambda key: np.where(key >> 31, key & np.uint32(0x7FFFFFFF), ~key).astype(np.uint32)
        assert np.float32(glo[k, 0]).view(np.uint32) == back(keys[(P - 1) // 2]), k
        assert np.float32(ghi[k, 0]).view(np.uint32) == back(keys[P // 2]), k


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


def _mlp_setup(dims, n, b, T, seed):
    from test_gpu_mlp import device_data
    order, tau = oracle.schedule_uniform(seed, n, T)
    batches = synth.schedule_batches(seed, order, b)
    theta0 = synth.xavier_theta0(seed, dims)
    X, y = device_data(seed)
    tensors = [0]
    for (wo, bo, fo, fi) in synth.mlp_layout(dims):
        tensors += [wo + fo * fi, bo + fo]
    return order, tau, batches, theta0, X, y, tensors


def test_mlp_run_pi_equals_the_flat_calls_bitwise():
    """gem_mlp_run_pi against the same segments replayed through the public flat calls
    (gem_mlp_grad for the segment's workers, gem_commit_batch_pi, gem_pi_median over the
    tensors of the flat layout): identical medians and theta, bit for bit."""
    from paper_1805_08469_gb300 import sim
    dims, n, b, T, seed = [784, 64, 10], 4, 32, 60, 1
    order, _tau, batches, theta0, X, y, tensors = _mlp_setup(dims, n, b, T, seed)
    P = synth.mlp_param_count(dims)
    nseg = len(tensors) - 1
    lo_a = torch.empty((T, nseg), device="cuda")
    hi_a = torch.empty((T, nseg), device="cuda")
    with gem.Gem(P, n, ETA, MU, EPS) as A:
        A.set_theta(torch.from_numpy(theta0).cuda())
        M = sim.gem_mlp_create(A.h, dims, b)
        try:
            sim.gem_mlp_set_data(M, X, y)
            sim.gem_mlp_run_pi(M, order, batches, lo_a, hi_a)
            A.sync()
            theta_a = A.theta().clone()
        finally:
            sim.gem_mlp_destroy(M)
    segs = sim.gem_plan_segments(order, n)
    lo_b = torch.empty((T, nseg), device="cuda")
    hi_b = torch.empty((T, nseg), device="cuda")
    ld = (P + 3) // 4 * 4                                 # 16-byte aligned rows
    grads = torch.empty((n, ld), device="cuda")
    pis = torch.empty((n, ld), device="cuda")
    with gem.Gem(P, n, ETA, MU, EPS) as B:
        B.set_theta(torch.from_numpy(theta0).cuda())
        M = sim.gem_mlp_create(B.h, dims, b)
        try:
            sim.gem_mlp_set_data(M, X, y)
            for a, e in zip(segs[:-1], segs[1:]):
                k = e - a
                sim.gem_mlp_grad(M, order[a:e], batches[a:e], [grads[i, :P] for i in range(k)])
                B.commit_batch_pi(order[a:e].tolist(), [grads[i, :P] for i in range(k)],
                                  [pis[i, :P] for i in range(k)])
                B.pi_median([pis[i, :P] for i in range(k)], tensors, lo_b[a:e], hi_b[a:e])
            B.sync()
            theta_b = B.theta().clone()
        finally:
            sim.gem_mlp_destroy(M)
    assert torch.equal(theta_a, theta_b)
    assert torch.equal(lo_a, lo_b) and torch.equal(hi_a, hi_b)


def test_mlp_run_pi_against_the_oracle_simulator():
    """Per-tensor medians of the factors of every commit against the oracle simulator's
    recorded factors (sorted on the host), n = 4, 40 commits from theta_0.  The two
    trajectories agree to rounding (1e-4 relative over this horizon); a factor's numerator
    |m| - |theta - s| subtracts close numbers, which amplifies that difference, and a
    median moves by at most the largest change of the factors around it, so the bar is
    1e-3 relative."""
    n, T = 4, 40
    from paper_1805_08469_gb300 import sim
    from test_gpu_mlp import host_rows
    dims, b, seed = [784, 64, 10], 32, 1
    order, _tau, batches, theta0, X, y, tensors = _mlp_setup(dims, n, b, T, seed)
    P = synth.mlp_param_count(dims)
    nseg = len(tensors) - 1
    lo = torch.empty((T, nseg), device="cuda")
    hi = torch.empty((T, nseg), device="cuda")
    with gem.Gem(P, n, ETA, MU, EPS) as G:
        G.set_theta(torch.from_numpy(theta0).cuda())
        M = sim.gem_mlp_create(G.h, dims, b)
        try:
            sim.gem_mlp_set_data(M, X, y)
            sim.gem_mlp_run_pi(M, order, batches, lo, hi)
            G.sync()
        finally:
            sim.gem_mlp_destroy(M)
    glo, ghi = lo.cpu().numpy(), hi.cpu().numpy()
    Xh, yh, local = host_rows(seed, batches)
    th, m, s = theta0.copy(), np.zeros((n, P), np.float32), np.tile(theta0, (n, 1))
    _r, _l, pi = oracle.mlp_sim_run(dims, th, m, s, order, Xh, yh, local, eta=ETA, mu=MU, eps=EPS,
                                    record_pi=True)
    for t in range(T):
        rlo, rhi = oracle.pi_median(pi[t], tensors)
        np.testing.assert_allclose(glo[t], rlo, rtol=1e-3, atol=1e-7, err_msg=f"commit {t} lower")
        np.testing.assert_allclose(ghi[t], rhi, rtol=1e-3, atol=1e-7, err_msg=f"commit {t} upper")
    assert np.any(glo > 0) and np.any(glo < 1)          # the factors vary over the run


def test_mlp_run_pi_windows_resumed_from_the_oracle():
    """n = 16, where the drift |theta - s| is larger and the factors more sensitive: windows
    of 4 commits resumed from the oracle's state (gem_load_state) at commits 0, 16, 32 and
    48, so the two sides differ only by the rounding of this window's gradients; medians
    within 1e-3 relative."""
    from paper_1805_08469_gb300 import sim
    from test_gpu_mlp import host_rows
    dims, n, b, seed, W = [784, 64, 10], 16, 32, 1, 4
    starts = [0, 16, 32, 48]
    T = starts[-1] + W
    order, _tau, batches, theta0, X, y, tensors = _mlp_setup(dims, n, b, T, seed)
    P = synth.mlp_param_count(dims)
    nseg = len(tensors) - 1
    Xh, yh, local = host_rows(seed, batches)
    th, m, s = theta0.copy(), np.zeros((n, P), np.float32), np.tile(theta0, (n, 1))
    states, t = {}, 0
    ref_pi = np.empty((T, P), np.float32)
    for c in starts + [T]:
        if c > t:
            _r, _l, pi = oracle.mlp_sim_run(dims, th, m, s, order[t:c], Xh, yh, local[t:c], eta=ETA,
                                            mu=MU, eps=EPS, record_pi=True)
            ref_pi[t:c] = pi
        states[c] = (th.copy(), m.copy(), s.copy())
        t = c
    lo = torch.empty((W, nseg), device="cuda")
    hi = torch.empty((W, nseg), device="cuda")
    with gem.Gem(P, n, ETA, MU, EPS) as G:
        M = sim.gem_mlp_create(G.h, dims, b)
        try:
            sim.gem_mlp_set_data(M, X, y)
            for c in starts:
                gem.gem_load_state(G.h, *states[c])
                sim.gem_mlp_run_pi(M, order[c:c + W], batches[c:c + W], lo, hi)
                G.sync()
                glo, ghi = lo.cpu().numpy(), hi.cpu().numpy()
                for i in range(W):
                    rlo, rhi = oracle.pi_median(ref_pi[c + i], tensors)
                    np.testing.assert_allclose(glo[i], rlo, rtol=1e-3, atol=1e-7, err_msg=f"commit {c + i}")
                    np.testing.assert_allclose(ghi[i], rhi, rtol=1e-3, atol=1e-7, err_msg=f"commit {c + i}")
        finally:
            sim.gem_mlp_destroy(M)


def _segments(P, kind):
    if kind == "one":
        return [0, P]
    # empty segments, a segment of one coordinate, boundaries inside float4 groups
    a, b = max(1, P // 3), max(2, P - 2)
    return sorted({0, 1, a, b, P} | {1}) if P > 4 else [0, 1, 1, 2, 2, P]


@pytest.mark.parametrize("mode,omode,kappa", [
    (gem.GEM_MODE_GEM, oracle.MODE_GEM, 1.0),
    (gem.GEM_MODE_KAPPA_LINEAR, oracle.MODE_KAPPA_LINEAR, 2.0),
    (gem.GEM_MODE_ADAPTIVE, oracle.MODE_ADAPTIVE, 1.0),
    (gem.GEM_MODE_MOMENTUM, oracle.MODE_MOMENTUM, 1.0),
])
@pytest.mark.parametrize("P,kind", [(5, "one"), (5, "many"), (4099, "many"), (100_003, "one"),
                                    (100_003, "many")])
def test_fused_commit_medians_equal_separate_calls_and_oracle(mode, omode, kappa, P, kind):
    """gem_commit_batch_pi_median against gem_commit_batch_pi + gem_pi_median on a second
    handle: theta, m, s, the recorded rows and both medians bit for bit; the medians also
    bit for bit against the oracle's sorted factors.  230 commits (two chunks)."""
    n, T = 5, 230
    seg = _segments(P, kind)
    nseg = len(seg) - 1
    theta0, grads, order, tau = _inputs(P, n, T, 700 + P)
    th, m, s = theta0.copy(), np.zeros((n, P), np.float32), np.tile(theta0, (n, 1))
    ref_pi = oracle.gem_run(th, m, s, grads, order, eta=ETA, mu=MU, eps=EPS, tau=tau, mode=omode,
                            kappa=kappa, record_pi=True)
    g_dev = _padded(grads)
    Pp = (P + 3) // 4 * 4
    pa = torch.full((T, Pp), -1.0, device="cuda")
    pb = torch.full((T, Pp), -1.0, device="cuda")
    lo_a, hi_a = (torch.full((T, nseg), -2.0, device="cuda") for _ in range(2))
    lo_b, hi_b = (torch.full((T, nseg), -2.0, device="cuda") for _ in range(2))
    gl = [g_dev[k, :P] for k in range(T)]
    with gem.Gem(P, n, ETA, MU, EPS) as A, gem.Gem(P, n, ETA, MU, EPS) as B:
        for G in (A, B):
            G.set_mode(mode, kappa)
            G.set_theta(torch.from_numpy(theta0).cuda())
        A.commit_batch_pi_median(order.tolist(), gl, [pa[k, :P] for k in range(T)], seg, lo_a, hi_a)
        B.commit_batch_pi(order.tolist(), gl, [pb[k, :P] for k in range(T)])
        B.pi_median([pb[k, :P] for k in range(T)], seg, lo_b, hi_b)
        A.sync()
        B.sync()
        assert torch.equal(A.theta(), B.theta())
        for w in range(n):
            assert torch.equal(A.moment(w), B.moment(w)) and torch.equal(A.snapshot(w), B.snapshot(w))
        assert np.array_equal(A.theta().cpu().numpy(), th)
    bits = lambda t: t.cpu().numpy().view(np.uint32)
    assert np.array_equal(bits(pa), bits(pb))
    assert np.array_equal(pa.cpu().numpy()[:, :P], ref_pi, equal_nan=True)
    for x, y in ((lo_a, lo_b), (hi_a, hi_b)):
        assert np.array_equal(bits(x), bits(y))
    glo, ghi = lo_a.cpu().numpy(), hi_a.cpu().numpy()
    for k in range(T):
        rlo, rhi = oracle.pi_median(ref_pi[k], seg)
        assert np.array_equal(glo[k], rlo, equal_nan=True), (k, glo[k], rlo)
        assert np.array_equal(ghi[k], rhi, equal_nan=True), (k, ghi[k], rhi)


@pytest.mark.parametrize("P", [1000, 40_002])
def test_fused_counts_at_the_edges_of_the_zero_run(P):
    """One worker without momentum: the factor of a coordinate is exactly +0 where its
    gradient is 0 and positive elsewhere (no drift, m = dtheta), so each row's run of zeros
    can be set exactly.  Rows whose zeros end just before the lower middle element, between
    the two middle elements, and just after the upper one, in two segments and over all of
    P: the targets that the commit kernel's counts resolve and the ones a selection pass
    finds must together equal the oracle's sorted medians bit for bit."""
    rng = np.random.default_rng(P)
    half = P // 2
    seg = [0, half, P]
    rows = []
    for zl, zr in ((half // 2 - 1, half // 2), (half // 2, (P - half) // 2 + 1), (half // 2 + 1, 0),
                   (0, P - half), (half, (P - half) // 2 - 1), (3, 5)):
        g = (0.1 * rng.standard_normal(P) + 0.3).astype(np.float32)
        g[g == 0] = 0.5
        g[rng.choice(half, zl, replace=False)] = 0.0
        g[half + rng.choice(P - half, zr, replace=False)] = 0.0
        rows.append(g)
    grads = np.stack(rows)
    T = grads.shape[0]
    order = np.zeros(T, np.int32)
    theta0 = (0.05 * rng.standard_normal(P)).astype(np.float32)
    th, m, s = theta0.copy(), np.zeros((1, P), np.float32), theta0.copy()[None, :]
    ref_pi = oracle.gem_run(th, m, s, grads, order, eta=ETA, mu=0.0, eps=EPS, record_pi=True)
    for k in range(T):                    # the construction holds in the oracle
        assert np.array_equal(ref_pi[k] == 0, grads[k] == 0) and np.all(ref_pi[k] >= 0)
    g_dev = _padded(grads)
    pi = torch.empty((T, (P + 3) // 4 * 4), device="cuda")
    for sg in (seg, [0, P]):
        nseg = len(sg) - 1
        lo, hi = torch.empty((T, nseg), device="cuda"), torch.empty((T, nseg), device="cuda")
        with gem.Gem(P, 1, ETA, 0.0, EPS) as G:
            G.set_theta(torch.from_numpy(theta0).cuda())
            G.commit_batch_pi_median(order.tolist(), [g_dev[k, :P] for k in range(T)],
                                     [pi[k, :P] for k in range(T)], sg, lo, hi)
            G.sync()
            assert np.array_equal(G.theta().cpu().numpy(), th)
        glo, ghi = lo.cpu().numpy(), hi.cpu().numpy()
        for k in range(T):
            rlo, rhi = oracle.pi_median(ref_pi[k], sg)
            assert np.array_equal(glo[k].view(np.uint32), rlo.view(np.uint32)), (sg, k, glo[k], rlo)
            assert np.array_equal(ghi[k].view(np.uint32), rhi.view(np.uint32)), (sg, k, ghi[k], rhi)


def test_fused_medians_with_64_segments_in_chunks():
    """64 segments allow 32 commits per chunk (the counters of a launch live in shared
    memory): 100 commits in four chunks, medians bit for bit against the oracle."""
    P, n, T = 70_001, 7, 100
    theta0, grads, order, tau = _inputs(P, n, T, 64)
    seg = np.linspace(0, P, 65).astype(np.int64).tolist()
    th, m, s = theta0.copy(), np.zeros((n, P), np.float32), np.tile(theta0, (n, 1))
    ref_pi = oracle.gem_run(th, m, s, grads, order, eta=ETA, mu=MU, eps=EPS, record_pi=True)
    g_dev = _padded(grads)
    pi = torch.empty((T, (P + 3) // 4 * 4), device="cuda")
    lo, hi = torch.empty((T, 64), device="cuda"), torch.empty((T, 64), device="cuda")
    with gem.Gem(P, n, ETA, MU, EPS) as G:
        G.set_theta(torch.from_numpy(theta0).cuda())
        G.commit_batch_pi_median(order.tolist(), [g_dev[k, :P] for k in range(T)],
                                 [pi[k, :P] for k in range(T)], seg, lo, hi)
        G.sync()
        assert np.array_equal(G.theta().cpu().numpy(), th)
    glo, ghi = lo.cpu().numpy(), hi.cpu().numpy()
    for k in range(T):
        rlo, rhi = oracle.pi_median(ref_pi[k], seg)
        assert np.array_equal(glo[k], rlo) and np.array_equal(ghi[k], rhi), k
