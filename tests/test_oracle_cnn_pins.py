"""Pins of the oracle's convolutional network (the MNIST model of Appendix A).

The oracle's forward and backward passes are plain loops in double.  They are tied to:
* PyTorch's CPU operators (conv2d, max_pool2d, linear, log_softmax, nll_loss) and its
  autograd, in double, on the same network: losses, logits and every gradient block;
* central finite differences of the oracle's own loss on a small network, all parameters;
* closed forms: zero parameters give loss ln C and a gradient only in the last bias,
  mean(1/C - onehot);
* the place of dropout: scaling every channel of conv2 by 2 equals doubling conv2's
  weights and bias;
* the simulation: one worker without momentum is minibatch SGD scaled by
  |dtheta| / (|dtheta| + eps) (no drift), with the same gradients.
"""
import math

import numpy as np
import pytest

import oracle

torch = pytest.importorskip("torch")
F = torch.nn.functional


def _layout(shape):
    H, c1, c2, f1, f2, C = shape
    P2 = ((H - 4) // 2 - 4) // 2
    Fe = c2 * P2 * P2
    sizes = [("w1", (c1, 1, 5, 5)), ("b1", (c1,)), ("w2", (c2, c1, 5, 5)), ("b2", (c2,)),
             ("wf1", (f1, Fe)), ("bf1", (f1,)), ("wf2", (f2, f1)), ("bf2", (f2,)),
             ("wf3", (C, f2)), ("bf3", (C,))]
    out, off = {}, 0
    for name, shp in sizes:
        cnt = int(np.prod(shp))
        out[name] = (off, shp)
        off += cnt
    return out, off


def _torch_reference(shape, theta, X, y, drop):
    """Loss, logits and gradient from PyTorch's operators and autograd (double)."""
    H = shape[0]
    lay, P = _layout(shape)
    th = torch.tensor(theta, dtype=torch.float64, requires_grad=True)
    prm = {k: th[o:o + int(np.prod(s))].view(*s) for k, (o, s) in lay.items()}
    x = torch.tensor(X, dtype=torch.float64).view(-1, 1, H, H)
    z = F.relu(F.max_pool2d(F.conv2d(x, prm["w1"], prm["b1"]), 2))
    z = F.conv2d(z, prm["w2"], prm["b2"]) * torch.tensor(drop, dtype=torch.float64)[:, :, None, None]
    z = F.relu(F.max_pool2d(z, 2)).flatten(1)
    z = F.relu(F.linear(z, prm["wf1"], prm["bf1"]))
    z = F.relu(F.linear(z, prm["wf2"], prm["bf2"]))
    logits = F.linear(z, prm["wf3"], prm["bf3"])
    loss = F.nll_loss(F.log_softmax(logits, dim=1), torch.tensor(y, dtype=torch.int64))
    loss.backward()
    return float(loss.detach()), logits.detach().numpy(), th.grad.numpy()


def _inputs(shape, b, seed, scale=0.2):
    rng = np.random.default_rng(seed)
    P = oracle.cnn_param_count(shape)
    theta = rng.standard_normal(P) * scale
    X = rng.standard_normal((b, shape[0] * shape[0]))
    y = rng.integers(0, shape[5], b).astype(np.int32)
    drop = np.where(rng.random((b, shape[2])) < 0.5, 0.0, 2.0)
    return theta, X, y, drop


@pytest.mark.parametrize("shape,b", [((28, 10, 20, 128, 64, 10), 4), ((16, 3, 4, 5, 4, 3), 5),
                                     ((20, 2, 3, 7, 6, 4), 3)])
def test_against_pytorch_autograd(shape, b):
    theta, X, y, drop = _inputs(shape, b, sum(shape))
    loss, grad, logits = oracle.cnn_loss_grad(shape, theta, X, y, drop, want_logits=True)
    rloss, rlogits, rgrad = _torch_reference(shape, theta, X, y, drop)
    assert loss == pytest.approx(rloss, rel=1e-12)
    np.testing.assert_allclose(logits, rlogits, rtol=1e-11, atol=1e-13)
    lay, _P = _layout(shape)
    for name, (o, s) in lay.items():
        n = int(np.prod(s))
        np.testing.assert_allclose(grad[o:o + n], rgrad[o:o + n], rtol=1e-9, atol=1e-13, err_msg=name)
    o, s1 = lay["w1"]
    assert np.abs(grad[o:o + int(np.prod(s1))]).max() > 0       # the first layer is reached


def test_finite_differences_every_parameter():
    shape, b = (16, 3, 4, 5, 4, 3), 3
    theta, X, y, drop = _inputs(shape, b, 7, scale=0.4)
    _l, grad = oracle.cnn_loss_grad(shape, theta, X, y, drop)
    h = 1e-6
    fd = np.empty_like(theta)
    for j in range(theta.size):
        tp, tm = theta.copy(), theta.copy()
        tp[j] += h
        tm[j] -= h
        fd[j] = (oracle.cnn_loss_grad(shape, tp, X, y, drop)[0] -
                 oracle.cnn_loss_grad(shape, tm, X, y, drop)[0]) / (2 * h)
    np.testing.assert_allclose(grad, fd, rtol=1e-5, atol=1e-8)


def test_zero_parameters_closed_form():
    shape, b = (28, 10, 20, 128, 64, 10), 6
    _t, X, y, drop = _inputs(shape, b, 3)
    P = oracle.cnn_param_count(shape)
    loss, grad = oracle.cnn_loss_grad(shape, np.zeros(P), X, y, drop)
    assert loss == pytest.approx(math.log(10), rel=1e-15)
    want = np.full(10, 1.0 / 10)
    for c in y:
        want[c] -= 1.0 / b
    np.testing.assert_allclose(grad[-10:], want, rtol=1e-14, atol=1e-16)
    assert np.all(grad[:-10] == 0.0)


def test_dropout_sits_on_conv2_output():
    shape, b = (28, 10, 20, 128, 64, 10), 3
    theta, X, y, _d = _inputs(shape, b, 11)
    lay, _P = _layout(shape)
    twice = theta.copy()
    o, s = lay["w2"]
    twice[o:o + int(np.prod(s))] *= 2
    o, s = lay["b2"]
    twice[o:o + int(np.prod(s))] *= 2
    l2, _g, z2 = oracle.cnn_loss_grad(shape, theta, X, y, np.full((b, 20), 2.0), want_logits=True)
    l1, _g, z1 = oracle.cnn_loss_grad(shape, twice, X, y, np.ones((b, 20)), want_logits=True)
    np.testing.assert_allclose(z2, z1, rtol=1e-13)
    assert l2 == pytest.approx(l1, rel=1e-13)


def test_simulation_with_one_worker_is_scaled_minibatch_sgd():
    shape, b, T, eta = (16, 3, 4, 5, 4, 3), 4, 5, 0.05
    rng = np.random.default_rng(5)
    P = oracle.cnn_param_count(shape)
    theta0 = (rng.standard_normal(P) * 0.3).astype(np.float32)
    X = rng.standard_normal((30, 256)).astype(np.float32)
    labels = rng.integers(0, 3, 30).astype(np.int32)
    rows = rng.integers(0, 30, (T, b)).astype(np.int32)
    drop = np.where(rng.random((T, b, 4)) < 0.5, 0.0, 2.0).astype(np.float32)
    th, m, s = theta0.copy(), np.zeros((1, P), np.float32), theta0[None, :].copy()
    oracle.cnn_sim_run(shape, th, m, s, np.zeros(T, np.int32), X, labels, rows, drop, eta=eta, mu=0.0,
                       eps=1e-8)
    ref = theta0.copy()
    for t in range(T):
        _l, g = oracle.cnn_loss_grad(shape, ref.astype(np.float64), X[rows[t]], labels[rows[t]], drop[t])
        dtheta = -(np.float32(eta) * g.astype(np.float32))
        ref = (ref + (np.abs(dtheta) / (np.abs(dtheta) + np.float32(1e-8))).astype(np.float32) * dtheta).astype(np.float32)
    # GEM with one worker and mu = 0: pi = |dtheta| / (|dtheta| + eps) (no drift), so the
    # step is dtheta scaled by that factor, in fp32 with one rounding per operation
    np.testing.assert_allclose(th, ref, rtol=1e-6, atol=1e-9)
