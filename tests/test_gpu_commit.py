"""GPU parity of the GEM commit path against the oracle, through the C ABI.

The commit (Algorithm 1, Psi_GEM then Commit) is evaluated with one IEEE fp32 operation per
step on both sides, so the bar is the benchmark spec's tolerance of 1e-6 relative per element,
and the tests also assert the stronger bit-for-bit equality that this order gives.  Every
coordinate's trajectory depends only on that coordinate's inputs (pi is elementwise), so
at full size the oracle reruns a sample of coordinates over the whole schedule.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_1805_08469_gb300 import gem, sim, synth, synth_gpu
from paper_1805_08469_gb300._build import build_library
from paper_1805_08469_gb300._lib import GemError

pytestmark = pytest.mark.gpu

ETA, MU, EPS = 0.01, 0.9, 1e-8


@pytest.fixture(scope="module", autouse=True)
def _setup():
    build_library()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    torch.cuda.set_device(0)


def _close(gpu, cpu, what):
    """North-star single-commit bar (1e-6 relative per element), then bitwise equality."""
    gpu = np.asarray(gpu)
    cpu = np.asarray(cpu)
    bad = np.abs(gpu.astype(np.float64) - cpu) > 1e-6 * np.abs(cpu.astype(np.float64)) + 1e-30
    assert not bad.any(), f"{what}: {int(bad.sum())} elements beyond 1e-6 relative"
    assert np.array_equal(gpu, cpu), f"{what}: {int((gpu != cpu).sum())} elements not bit-identical"


def _padded(a: np.ndarray) -> torch.Tensor:
    """[T, P] host array -> device array with rows padded to 16 bytes (aligned row starts)."""
    T, P = a.shape
    ld = (P + 3) // 4 * 4
    d = torch.zeros((T, ld), dtype=torch.float32, device="cuda")
    d[:, :P] = torch.from_numpy(a).cuda()
    return d


def _fresh_cpu(theta0, n):
    return theta0.copy(), np.zeros((n, theta0.size), np.float32), np.tile(theta0, (n, 1))


@pytest.mark.parametrize("P", [1, 2, 3, 4, 5, 17, 1000, 4099, 65539, 1_000_003])
def test_single_commits_bitwise(P):
    n, T = 3, 10
    rng = np.random.default_rng(P)
    theta0 = (0.05 * rng.standard_normal(P)).astype(np.float32)
    grads = (rng.standard_normal((T, P)) * 10.0 ** rng.uniform(-4, -1, P)).astype(np.float32)
    grads[:, ::7] = 0.0                       # zero updates: pi = 0 / eps
    order = rng.integers(0, n, T)
    th, m, s = _fresh_cpu(theta0, n)
    g_dev = _padded(grads)
    with gem.Gem(P, n, ETA, MU, EPS) as G:
        G.set_theta(torch.from_numpy(theta0).cuda())
        for t in range(T):
            w = int(order[t])
            G.commit(w, g_dev[t, :P])
            oracle.gem_run(th, m, s, grads[t:t + 1], [w], eta=ETA, mu=MU, eps=EPS)
            G.sync()
            _close(G.theta().cpu().numpy(), th, f"theta after commit {t}")
            _close(G.moment(w).cpu().numpy(), m[w], f"m_w after commit {t}")
            _close(G.snapshot(w).cpu().numpy(), s[w], f"s_w after commit {t}")
        assert G.launches() == T


# (250_003, 40, 200): more repeats open at once than on-chip slots (every slot in use), and a
# last warp whose lanes run past the coordinates
@pytest.mark.parametrize("P,n,K", [(4099, 5, 450), (64, 2, 37), (1_048_579, 16, 64), (250_003, 40, 200)])
def test_batch_equals_sequence_bitwise(P, n, K):
    rng = np.random.default_rng(K)
    theta0 = (0.05 * rng.standard_normal(P)).astype(np.float32)
    grads = (0.05 * rng.standard_normal((K, P))).astype(np.float32)
    order = rng.integers(0, n, K)                 # many repeated workers
    th, m, s = _fresh_cpu(theta0, n)
    oracle.gem_run(th, m, s, grads, order, eta=ETA, mu=MU, eps=EPS)
    g_dev = _padded(grads)
    with gem.Gem(P, n, ETA, MU, EPS) as G:
        G.set_theta(torch.from_numpy(theta0).cuda())
        G.commit_batch([], [])                    # K = 0 is a no-op
        G.commit_batch(order.tolist(), [g_dev[k, :P] for k in range(K)])
        G.sync()
        assert G.launches() == (K + 199) // 200
        _close(G.theta().cpu().numpy(), th, "theta")
        for w in range(n):
            _close(G.moment(w).cpu().numpy(), m[w], f"m_{w}")
            _close(G.snapshot(w).cpu().numpy(), s[w], f"s_{w}")


def test_host_gradient_batch_equals_device_batch():
    P, n, K = 100_003, 7, 43
    rng = np.random.default_rng(5)
    theta0 = (0.05 * rng.standard_normal(P)).astype(np.float32)
    grads = (0.05 * rng.standard_normal((K, P))).astype(np.float32)
    order = rng.integers(0, n, K).tolist()
    host = [torch.from_numpy(grads[k].copy()).pin_memory() if k % 2 else torch.from_numpy(grads[k].copy())
            for k in range(K)]
    g_dev = _padded(grads)
    pinned = [torch.from_numpy(grads[k].copy()).pin_memory() for k in range(K)]
    with gem.Gem(P, n, ETA, MU, EPS) as A, gem.Gem(P, n, ETA, MU, EPS) as B, \
            gem.Gem(P, n, ETA, MU, EPS) as Z:
        for H in (A, B, Z):
            H.set_theta(torch.from_numpy(theta0).cuda())
        A.commit_batch(order, [g_dev[k, :P] for k in range(K)])
        B.commit_batch_host(order, host)      # some pageable: staged copies
        Z.commit_batch_host(order, pinned)    # all page-locked: read in place
        for H in (A, B, Z):
            H.sync()
        for H in (B, Z):
            assert torch.equal(A.theta(), H.theta())
            for w in range(n):
                assert torch.equal(A.moment(w), H.moment(w))
                assert torch.equal(A.snapshot(w), H.snapshot(w))
        out = torch.empty(P, dtype=torch.float32).pin_memory()
        gem.gem_read_theta(B.h, out)
        B.sync()
        assert torch.equal(out, B.theta().cpu())


def test_host_gradient_batches_back_to_back():
    """Five gem_commit_batch_host calls issued without waiting, pageable gradients (each
    call stages its chunks through the same two halves of the staging buffer, so a call
    must not overwrite a half the previous one is still reading); the same as the device
    path, bit for bit."""
    P, n, K, calls = 50_001, 5, 11, 5
    rng = np.random.default_rng(9)
    theta0 = (0.05 * rng.standard_normal(P)).astype(np.float32)
    grads = (0.05 * rng.standard_normal((calls * K, P))).astype(np.float32)
    order = rng.integers(0, n, calls * K).tolist()
    g_dev = _padded(grads)
    with gem.Gem(P, n, ETA, MU, EPS) as A, gem.Gem(P, n, ETA, MU, EPS) as B:
        for H in (A, B):
            H.set_theta(torch.from_numpy(theta0).cuda())
        for c in range(calls):
            ks = range(c * K, (c + 1) * K)
            A.commit_batch([order[k] for k in ks], [g_dev[k, :P] for k in ks])
            B.commit_batch_host([order[k] for k in ks], [torch.from_numpy(grads[k].copy()) for k in ks])
        A.sync()
        B.sync()
        assert torch.equal(A.theta(), B.theta())
        for w in range(n):
            assert torch.equal(A.moment(w), B.moment(w)) and torch.equal(A.snapshot(w), B.snapshot(w))


def test_invalid_arguments_leave_the_handle_usable():
    P, n = 1000, 2
    g = torch.zeros(P + 4, dtype=torch.float32, device="cuda")
    with gem.Gem(P, n, ETA, MU, EPS) as G:
        G.set_theta(torch.ones(P, device="cuda"))
        with pytest.raises(GemError) as e:
            G.commit(2, g[:P])                        # worker out of range
        assert e.value.status == gem.GEM_EINVAL
        with pytest.raises(GemError):
            G.commit(0, g[1:P + 1])                   # not 16-byte aligned
        with pytest.raises(GemError):
            G.commit_batch([0, -1], [g[:P], g[:P]])
        before = gem.gem_launch_count(G.h)
        assert before == 0
        G.commit(1, g[:P])
        G.sync()
        assert gem.gem_launch_count(G.h) == 1
        assert torch.equal(G.theta(), torch.ones(P, device="cuda"))  # zero gradient


# ----------------------------------------------------------------- input generators

def test_device_generators_match_host_generators():
    seed = 77
    cols = np.array([0, 1, 2, 3, 5, 1023, 4096, 99_999, 123_457, 199_999])
    P = 200_000
    th = synth_gpu.theta0_flat(seed, torch.empty(P, device="cuda"))
    assert np.array_equal(th.cpu().numpy()[cols], synth.theta0_flat(seed, cols))
    pool = torch.empty((3, P + 4), device="cuda")
    synth_gpu.grad_heavytail(seed, 5, pool, P)
    for r in range(3):
        assert np.array_equal(pool[r, :P].cpu().numpy()[cols], synth.grad_heavytail(seed, 5 + r, cols))
    # full rows too (covers both branches of the mask everywhere)
    assert np.array_equal(pool[1, :P].cpu().numpy(), synth.grad_heavytail(seed, 6, np.arange(P)))
    sig = synth.sigma_loguniform(seed, np.arange(P))
    g = synth_gpu.grad_loguniform(seed, 41, torch.from_numpy(sig).cuda(), torch.empty(P, device="cuda"))
    assert np.array_equal(g.cpu().numpy(), synth.grad_loguniform(seed, 41, np.arange(P), sig))
    X = torch.empty((3000, 784), device="cuda")
    y = torch.empty(3000, dtype=torch.int32, device="cuda")
    synth_gpu.data(seed, X, y, 10)
    rows = np.array([0, 1, 17, 2999])
    assert np.array_equal(X.cpu().numpy()[rows], synth.data_rows(seed, rows, 784))
    assert np.array_equal(y.cpu().numpy(), synth.teacher_labels(seed, np.arange(3000), 784, 10))
    dims = [784, 64, 10]
    t = synth_gpu.xavier(seed, dims, torch.empty(synth.mlp_param_count(dims), device="cuda"))
    assert np.array_equal(t.cpu().numpy(), synth.xavier_theta0(seed, dims))


# ----------------------------------------------------------------- workload-sized runs

def _sample_cols(P, S, seed):
    rng = np.random.default_rng(seed)
    cols = np.unique(np.concatenate([rng.choice(P, S, replace=False), np.arange(8), P - 1 - np.arange(8)]))
    return cols.astype(np.int64)


@pytest.mark.slow
def test_config2_flat_commit_by_commit_sampled():
    """P = 1.2M, n = 20, 5,000 uniform-tick commits of fresh log-uniform gradients;
    theta compared after every commit on a sample of coordinates, and everything at the end."""
    seed, P, n, T = 2, 1_200_000, 20, 5000
    order, _ = sim.gem_schedule_uniform(seed, n, T)
    cols = _sample_cols(P, 4096, seed)
    S = cols.size
    sigma = synth.sigma_loguniform(seed, np.arange(P))
    theta0 = synth.theta0_flat(seed, np.arange(P))
    # oracle on the sampled coordinates
    c = (np.arange(T, dtype=np.uint64)[:, None] << np.uint64(32)) | cols.astype(np.uint64)[None, :]
    z = synth.normal(synth.key(seed, synth.STREAM_GRAD_Z), c)
    g_cpu = (sigma[cols][None, :] * z).astype(np.float32)
    th, m, s = _fresh_cpu(theta0[cols], n)
    traj_cpu = oracle.gem_run(th, m, s, g_cpu, order, eta=ETA, mu=MU, eps=EPS, record_cols=np.arange(S))
    # GPU
    stream = torch.cuda.Stream()
    idx = torch.from_numpy(cols).cuda()
    traj = torch.empty((T, S), device="cuda")
    with torch.cuda.stream(stream), gem.Gem(P, n, ETA, MU, EPS, stream=stream) as G:
        G.set_theta(torch.from_numpy(theta0).cuda())
        sig_d = torch.from_numpy(sigma).cuda()
        gbuf = torch.empty(P, device="cuda")
        theta_v = G.theta()
        for t in range(T):
            synth_gpu.grad_loguniform(seed, t, sig_d, gbuf, stream=stream)
            G.commit(int(order[t]), gbuf)
            torch.index_select(theta_v, 0, idx, out=traj[t])
        G.sync()
        _close(traj.cpu().numpy(), traj_cpu, "theta trajectory (sampled)")
        for w in range(n):
            _close(G.moment(w).cpu().numpy()[cols], m[w], f"m_{w} (sampled)")
            _close(G.snapshot(w).cpu().numpy()[cols], s[w], f"s_{w} (sampled)")


@pytest.mark.slow
def test_config2_full_vectors_first_commits():
    seed, P, n, T = 2, 1_200_000, 20, 12
    order, _ = sim.gem_schedule_uniform(seed, n, T)
    sigma = synth.sigma_loguniform(seed, np.arange(P))
    theta0 = synth.theta0_flat(seed, np.arange(P))
    grads = np.stack([synth.grad_loguniform(seed, t, np.arange(P), sigma) for t in range(T)])
    th, m, s = _fresh_cpu(theta0, n)
    oracle.gem_run(th, m, s, grads, order, eta=ETA, mu=MU, eps=EPS)
    with gem.Gem(P, n, ETA, MU, EPS) as G:
        G.set_theta(torch.from_numpy(theta0).cuda())
        g_dev = torch.from_numpy(grads).cuda()
        for t in range(T):
            G.commit(int(order[t]), g_dev[t])
        G.sync()
        _close(G.theta().cpu().numpy(), th, "theta")
        for w in set(order.tolist()):
            _close(G.moment(w).cpu().numpy(), m[w], f"m_{w}")
            _close(G.snapshot(w).cpu().numpy(), s[w], f"s_{w}")


@pytest.mark.slow
def test_config5_batched_commits_sampled():
    """P = 25M, n = 100, a 10 GB pool of 100 heavy-tailed gradients reused cyclically,
    10 batches of 100 commits in uniform-tick order (the benchmark's launch configuration)."""
    seed, P, n, K, batches, pool_rows = 5, 25_000_000, 100, 100, 10, 100
    T = K * batches
    order, _ = sim.gem_schedule_uniform(seed, n, T)
    cols = _sample_cols(P, 8192, seed)
    S = cols.size
    theta0 = synth.theta0_flat(seed, cols)
    pool_cpu = np.stack([synth.grad_heavytail(seed, r, cols) for r in range(pool_rows)])
    th, m, s = _fresh_cpu(theta0, n)
    gidx = np.arange(T) % pool_rows
    oracle.gem_run(th, m, s, pool_cpu, order, grad_index=gidx, eta=ETA, mu=MU, eps=EPS)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream), gem.Gem(P, n, ETA, MU, EPS, stream=stream) as G:
        th0 = synth_gpu.theta0_flat(seed, torch.empty(P, device="cuda"), stream=stream)
        G.set_theta(th0)
        pool = torch.empty((pool_rows, P), device="cuda")
        synth_gpu.grad_heavytail(seed, 0, pool, P, stream=stream)
        for b in range(batches):
            ks = range(b * K, (b + 1) * K)
            G.commit_batch([int(order[k]) for k in ks], [pool[gidx[k]] for k in ks])
        G.sync()
        assert G.launches() == batches
        idx = torch.from_numpy(cols).cuda()
        _close(G.theta()[idx].cpu().numpy(), th, "theta (sampled)")
        for w in range(0, n, 7):
            _close(G.moment(w)[idx].cpu().numpy(), m[w], f"m_{w} (sampled)")
            _close(G.snapshot(w)[idx].cpu().numpy(), s[w], f"s_{w} (sampled)")


def test_parameter_vector_beyond_two_to_the_31():
    """P = 2^31 + 5 coordinates (about 34 GB of state and gradient): every index of theta,
    m, s and the gradient needs 64 bits, and P mod 4 = 1 leaves a ragged tail.  Three
    commits by one worker (its own moment and snapshot), checked on coordinates on both
    sides of 2^31, the tail, and a random sample."""
    seed, n = 5, 1
    P = (1 << 31) + 5
    order = [0, 0, 0]
    rng = np.random.default_rng(31)
    edge = np.concatenate([np.arange(8), (1 << 31) - 4 + np.arange(9), P - 1 - np.arange(8)])
    cols = np.unique(np.concatenate([edge, rng.integers(0, P, 4096)])).astype(np.int64)
    theta0 = synth.theta0_flat(seed, cols)
    g_cpu = synth.grad_heavytail(seed, 0, cols)[None, :]
    th, m, s = _fresh_cpu(theta0, n)
    oracle.gem_run(th, m, s, g_cpu, np.asarray(order, np.int32), grad_index=np.zeros(3, np.int64),
                   eta=ETA, mu=MU, eps=EPS)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream), gem.Gem(P, n, ETA, MU, EPS, stream=stream) as G:
        th0 = synth_gpu.theta0_flat(seed, torch.empty(P, device="cuda"), stream=stream)
        G.set_theta(th0)
        del th0
        grad = torch.empty((1, P), device="cuda")
        synth_gpu.grad_heavytail(seed, 0, grad, P, stream=stream)
        G.commit(0, grad[0])                              # a single commit
        G.commit_batch([0, 0], [grad[0], grad[0]])        # and a batch reusing it
        G.sync()
        idx = torch.from_numpy(cols).cuda()
        _close(G.theta()[idx].cpu().numpy(), th, "theta beyond 2^31 (sampled)")
        _close(G.moment(0)[idx].cpu().numpy(), m[0], "m beyond 2^31 (sampled)")
        _close(G.snapshot(0)[idx].cpu().numpy(), s[0], "s beyond 2^31 (sampled)")
        del grad


def test_worker_drop_out_on_the_device():
    """Worker 2 of 4 stops committing after commit 40 of 300; batches before and after.
    The device matches the oracle bit for bit, and the dropped worker's m_w and s_w on the
    device do not change after its last commit."""
    P, n, T, gone, after = 70_001, 4, 300, 2, 40
    rng = np.random.default_rng(23)
    theta0 = (0.05 * rng.standard_normal(P)).astype(np.float32)
    grads = (0.1 * rng.standard_normal((T, P))).astype(np.float32)
    base = rng.integers(0, n, 2 * T)
    order = [int(w) for t, w in enumerate(base) if not (w == gone and t >= after)][:T]
    last = max(t for t in range(T) if order[t] == gone)
    th, m, s = _fresh_cpu(theta0, n)
    oracle.gem_run(th, m, s, grads, np.asarray(order, np.int32), eta=ETA, mu=MU, eps=EPS)
    g_dev = _padded(grads)
    with gem.Gem(P, n, ETA, MU, EPS) as G:
        G.set_theta(torch.from_numpy(theta0).cuda())
        G.commit_batch(order[:last + 1], [g_dev[t, :P] for t in range(last + 1)])
        G.sync()
        m_gone, s_gone = G.moment(gone).clone(), G.snapshot(gone).clone()
        for t0 in range(last + 1, T, 37):
            t1 = min(T, t0 + 37)
            G.commit_batch(order[t0:t1], [g_dev[t, :P] for t in range(t0, t1)])
        G.sync()
        assert torch.equal(G.moment(gone), m_gone) and torch.equal(G.snapshot(gone), s_gone)
        _close(G.theta().cpu().numpy(), th, "theta")
        for w in range(n):
            _close(G.moment(w).cpu().numpy(), m[w], f"m_{w}")
            _close(G.snapshot(w).cpu().numpy(), s[w], f"s_{w}")


def test_commits_read_gradients_written_by_the_kernel_just_before():
    """Every commit launch is a programmatic dependent of the previous kernel in its
    stream and waits for it at entry.  Here each gradient is written by a PyTorch kernel on
    the same stream immediately before the commit that reads it, into a buffer that held
    NaN: a commit that started reading early would see NaN or the previous gradient."""
    P, n, T = 4_000_003, 3, 12
    rng = np.random.default_rng(21)
    theta0 = (0.05 * rng.standard_normal(P)).astype(np.float32)
    base = (0.1 * rng.standard_normal((T, P))).astype(np.float32)
    grads = base * np.float32(3.0)                       # what the device kernel writes
    order = [int(w) for w in rng.integers(0, n, T)]
    th, m, s = _fresh_cpu(theta0, n)
    oracle.gem_run(th, m, s, grads, np.asarray(order, np.int32), eta=ETA, mu=MU, eps=EPS)

    stream = torch.cuda.Stream()
    src = _padded(base)
    buf = torch.full_like(src[0], float("nan"))
    with torch.cuda.stream(stream), gem.Gem(P, n, ETA, MU, EPS, stream=stream) as G:
        G.set_theta(torch.from_numpy(theta0).cuda())
        for t in range(T):
            torch.mul(src[t], 3.0, out=buf)              # kernel on the commit's stream
            G.commit(order[t], buf[:P])                  # single commit
            buf.fill_(float("nan"))                      # and a kernel right after it
        for t in range(0, T, 4):                         # batches of 4, fresh buffers
            bufs = [torch.mul(src[t + k], 3.0) for k in range(4)]
            G.commit_batch(order[t:t + 4], [b[:P] for b in bufs])
        G.sync()
        got = G.theta().cpu().numpy()
    th2, m2, s2 = th.copy(), m.copy(), s.copy()
    oracle.gem_run(th2, m2, s2, grads, np.asarray(order, np.int32), eta=ETA, mu=MU, eps=EPS)
    assert np.isfinite(got).all()
    _close(got, th2, "theta after single commits and batches fed by the previous kernel")


def test_checkpoint_save_and_load_state():
    """gem_save_state / gem_load_state round trip (host and device buffers), then the
    resumed handle continues bit for bit like the original."""
    P, n, K = 10_007, 4, 30
    rng = np.random.default_rng(8)
    theta0 = (0.05 * rng.standard_normal(P)).astype(np.float32)
    grads = _padded((0.05 * rng.standard_normal((2 * K, P))).astype(np.float32))
    order = rng.integers(0, n, 2 * K).tolist()
    with gem.Gem(P, n, ETA, MU, EPS) as A, gem.Gem(P, n, ETA, MU, EPS) as B:
        A.set_theta(torch.from_numpy(theta0).cuda())
        A.commit_batch(order[:K], [grads[k, :P] for k in range(K)])
        th = np.empty(P, np.float32)
        m = np.empty((n, P), np.float32)
        s = torch.empty((n, P), device="cuda")
        gem.gem_save_state(A.h, th, m, s)
        A.sync()
        gem.gem_load_state(B.h, th, m, s)
        A.commit_batch(order[K:], [grads[k, :P] for k in range(K, 2 * K)])
        B.commit_batch(order[K:], [grads[k, :P] for k in range(K, 2 * K)])
        A.sync()
        B.sync()
        assert torch.equal(A.theta(), B.theta())
        for w in range(n):
            assert torch.equal(A.moment(w), B.moment(w)) and torch.equal(A.snapshot(w), B.snapshot(w))
