"""GPU parity of the MNIST convolutional network (include/gem_cnn.h) against the oracle.

The network's gradient at a worker's snapshot is fp32 on the GPU and double in the oracle
(rounded once to fp32), so the bar is the MLP's: 1e-5 relative L2 per parameter tensor.
The asynchronous runs are compared as the MLP's are: in windows resumed from the oracle's
state, and free-running over a horizon.  The dropout scales and initial parameters come
from the seeded generators, whose device and host twins must agree bit for bit.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_1805_08469_gb300 import cnn, gem, synth, synth_gpu
from paper_1805_08469_gb300._build import build_library
from paper_1805_08469_gb300._lib import GemError

from test_gpu_mlp import device_data, host_rows, rel_l2

pytestmark = pytest.mark.gpu

ETA, MU, EPS = 0.05, 0.9, 1e-8          # the paper's MNIST settings


@pytest.fixture(scope="module", autouse=True)
def _setup():
    build_library()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    torch.cuda.set_device(0)


def test_device_generators_match_host_generators():
    for shape in (cnn.CNN_MNIST, (16, 3, 4, 5, 4, 3)):
        P = synth.cnn_param_count(shape)
        dev = synth_gpu.cnn_theta0(9, shape, torch.empty(P, device="cuda"))
        assert np.array_equal(dev.cpu().numpy(), synth.cnn_theta0(9, shape))
    dev = synth_gpu.dropout(4, 17, torch.empty((5, 64, 20), device="cuda"))
    host = synth.dropout_scales(4, 17, 5, 64, 20)
    assert np.array_equal(dev.cpu().numpy(), host)
    assert 0.4 < (host == 0).mean() < 0.6 and set(np.unique(host)) == {0.0, 2.0}


def _blocks(shape):
    names = [t[0] for t in synth.cnn_layout(shape)]
    return [(nm, off, cnt) for nm, off, cnt, _f in synth.cnn_layout(shape)], names


@pytest.mark.parametrize("shape,b,G", [(cnn.CNN_MNIST, 64, 3), ((16, 3, 4, 5, 4, 3), 7, 2),
                                       ((20, 2, 3, 7, 6, 4), 5, 3)])
def test_gradients_match_the_oracle(shape, b, G):
    """G workers with different snapshots, in one batched call; every parameter tensor of
    every worker's gradient within 1e-5 relative L2 of the oracle's double gradient."""
    seed = 11
    P = synth.cnn_param_count(shape)
    H = shape[0]
    rows_total = 300
    X = torch.from_numpy(synth.data_rows(seed, np.arange(rows_total), H * H)).cuda()
    y = torch.from_numpy(synth.teacher_labels(seed, np.arange(rows_total), H * H, shape[5])).cuda()
    theta0 = synth.cnn_theta0(seed, shape)
    rng = np.random.default_rng(3)
    snaps = np.stack([theta0 + (0.02 * rng.standard_normal(P)).astype(np.float32) for _ in range(G)])
    rows = rng.integers(0, rows_total, (G, b)).astype(np.int32)
    drop_host = synth.dropout_scales(seed, 0, G, b, shape[2])
    drop = torch.from_numpy(drop_host).cuda()
    with gem.Gem(P, G, ETA, MU, EPS) as Gh:
        gem.gem_load_state(Gh.h, theta0, np.zeros((G, P), np.float32), snaps)
        net = cnn.gem_cnn_create(Gh.h, shape, b)
        try:
            cnn.gem_cnn_set_data(net, X, y)
            ld = (P + 3) // 4 * 4
            out = torch.empty((G, ld), device="cuda")
            losses = torch.empty(G, device="cuda")
            cnn.gem_cnn_grad(net, list(range(G)), rows, drop, [out[g, :P] for g in range(G)], losses)
            cnn.gem_cnn_status(net)
            got = out[:, :P].cpu().numpy()
            got_loss = losses.cpu().numpy()
        finally:
            cnn.gem_cnn_destroy(net)
    Xh = synth.data_rows(seed, np.arange(rows_total), H * H)
    yh = synth.teacher_labels(seed, np.arange(rows_total), H * H, shape[5])
    blocks, _names = _blocks(shape)
    for g in range(G):
        loss, ref = oracle.cnn_loss_grad(shape, snaps[g].astype(np.float64), Xh[rows[g]], yh[rows[g]],
                                         drop_host[g])
        assert abs(got_loss[g] - loss) <= 1e-5 * abs(loss), (g, got_loss[g], loss)
        for nm, off, cnt in blocks:
            err = rel_l2(got[g, off:off + cnt], ref[off:off + cnt])
            assert err < 1e-5, (g, nm, err)


def _cnn_inputs(shape, n, b, T, seed):
    order, tau = oracle.schedule_uniform(seed, n, T)
    batches = synth.schedule_batches(seed, order, b)
    drop = synth.dropout_scales(seed, 0, T, b, shape[2])
    return order, tau, batches, drop


def test_windows_and_free_run_match_the_oracle():
    """The paper's network, n = 4 workers, b = 64, 60 uniform-tick commits (seed 1):
    windows of 10 commits resumed from the oracle's state at commits 0, 20 and 40 within
    1e-4, and the free-running first 30 commits within 1e-4."""
    shape, n, b, seed, W = cnn.CNN_MNIST, 4, 64, 1, 10
    starts = [0, 20, 40]
    T = starts[-1] + W
    P = synth.cnn_param_count(shape)
    order, _tau, batches, drop_host = _cnn_inputs(shape, n, b, T, seed)
    theta0 = synth.cnn_theta0(seed, shape)
    Xh, yh, local = host_rows(seed, batches)
    # oracle states at the window boundaries
    th, m, s = theta0.copy(), np.zeros((n, P), np.float32), np.tile(theta0, (n, 1))
    states, ref_losses, t = {}, np.empty(T), 0
    for c in sorted(set(starts + [c + W for c in starts])):
        if c > t:
            _r, ls = oracle.cnn_sim_run(shape, th, m, s, order[t:c], Xh, yh, local[t:c], drop_host[t:c],
                                        eta=ETA, mu=MU, eps=EPS, want_losses=True)
            ref_losses[t:c] = ls
        states[c] = (th.copy(), m.copy(), s.copy())
        t = c
    X, y = device_data(seed)
    drop = torch.from_numpy(drop_host).cuda()
    with gem.Gem(P, n, ETA, MU, EPS) as G:
        net = cnn.gem_cnn_create(G.h, shape, b)
        try:
            cnn.gem_cnn_set_data(net, X, y)
            losses = torch.empty(W, device="cuda")
            for c in starts:
                gem.gem_load_state(G.h, *states[c])
                cnn.gem_cnn_run(net, order[c:c + W], batches[c:c + W], drop[c:c + W], losses)
                G.sync()
                err = rel_l2(G.theta().cpu().numpy(), states[c + W][0])
                assert err < 1e-4, (c, err)
                np.testing.assert_allclose(losses.cpu().numpy(), ref_losses[c:c + W], rtol=1e-4)
            # free-running from theta_0
            G.set_theta(torch.from_numpy(theta0).cuda())
            cnn.gem_cnn_run(net, order[:30], batches[:30], drop[:30])
            G.sync()
            free = G.theta().cpu().numpy()
        finally:
            cnn.gem_cnn_destroy(net)
    th, m, s = theta0.copy(), np.zeros((n, P), np.float32), np.tile(theta0, (n, 1))
    oracle.cnn_sim_run(shape, th, m, s, order[:30], Xh, yh, local[:30], drop_host[:30], eta=ETA, mu=MU,
                       eps=EPS)
    assert rel_l2(free, th) < 1e-4, rel_l2(free, th)


def test_argument_checks():
    shape = (16, 3, 4, 5, 4, 3)
    P = synth.cnn_param_count(shape)
    assert cnn.gem_cnn_param_count((17, 3, 4, 5, 4, 3)) == -1      # H - 4 odd
    assert cnn.gem_cnn_param_count((12, 3, 4, 5, 4, 3)) == -1      # conv2 output too small
    with gem.Gem(P + 1, 2, ETA, MU, EPS) as G:
        with pytest.raises(GemError):
            cnn.gem_cnn_create(G.h, shape, 4)                       # P does not match
    X = torch.zeros((10, 256), device="cuda")
    y = torch.zeros(10, dtype=torch.int32, device="cuda")
    drop = torch.ones((1, 4, 4), device="cuda")
    with gem.Gem(P, 2, ETA, MU, EPS) as G:
        net = cnn.gem_cnn_create(G.h, shape, 4)
        try:
            cnn.gem_cnn_set_data(net, X, y)
            with pytest.raises(GemError):
                cnn.gem_cnn_run(net, [0], np.full((1, 4), 10, np.int32), drop)   # row outside
            with pytest.raises(GemError):
                cnn.gem_cnn_run(net, [2], np.zeros((1, 4), np.int32), drop)      # worker outside
            cnn.gem_cnn_run(net, [1], np.zeros((1, 4), np.int32), drop)          # still usable
            cnn.gem_cnn_status(net)
            assert cnn.gem_cnn_launch_count(net) > 0
        finally:
            cnn.gem_cnn_destroy(net)
