"""Sanity of the seeded input generators (shapes, ranges and the distributions that the
workloads ask for).  These are inputs, not GEM: they are checked against their stated
laws, not against the oracle."""
import numpy as np
import pytest

from paper_1805_08469_gb300 import synth


def test_normal_moments_and_support():
    z = synth.normal(synth.key(1, synth.STREAM_GRAD_Z), np.arange(400_000))
    assert z.dtype == np.float32
    assert abs(z.mean()) < 5 / np.sqrt(len(z))
    assert abs(z.var() - 1.0) < 0.01
    assert z.min() >= -6.0 and z.max() < 6.0
    # exact multiples of 2**-20
    assert np.all(z * np.float32(2 ** 20) == np.round(z * np.float32(2 ** 20)))


def test_student_t3_tails():
    t = synth.student_t3(synth.key(2, synth.STREAM_GRAD_T), np.arange(300_000))
    # P(|T| > 3) for 3 degrees of freedom is 0.0577
    frac = np.mean(np.abs(t) > 3.0)
    assert abs(frac - 0.0577) < 0.004, frac
    assert abs(np.median(t)) < 0.01


def test_heavy_tail_gradient_workload():
    j = np.arange(200_000)
    mask = synth.heavy_mask(5, j)
    assert abs(mask.mean() - 0.1) < 0.005
    g0 = synth.grad_heavytail(5, 0, j)
    g1 = synth.grad_heavytail(5, 1, j)
    assert g0.dtype == np.float32 and not np.array_equal(g0, g1)
    assert abs(g0[~mask].std() - 0.01) < 2e-4
    assert np.abs(g0[mask]).max() > 10 * np.abs(g0[~mask]).max() / 6


def test_loguniform_sigma_and_gradients():
    j = np.arange(100_000)
    sig = synth.sigma_loguniform(2, j)
    lg = np.log10(sig.astype(np.float64))
    assert lg.min() >= -4.0 - 1e-6 and lg.max() <= -1.0 + 1e-6
    assert abs(lg.mean() + 2.5) < 0.02
    g = synth.grad_loguniform(2, 3, j, sig)
    assert abs(np.std(g / sig) - 1.0) < 0.02


def test_mlp_layout_and_xavier():
    dims = [784, 1000, 1000, 10]
    assert synth.mlp_param_count(dims) == 1_796_010
    assert synth.mlp_param_count([784, 64, 10]) == 50_890
    lay = synth.mlp_layout([784, 64, 10])
    assert lay[0] == (0, 50176, 64, 784) and lay[1] == (50240, 50880, 10, 64)
    th = synth.xavier_theta0(3, [784, 64, 10])
    a0 = np.sqrt(6 / (784 + 64))
    w0 = th[:50176]
    assert np.abs(w0).max() <= a0 and np.abs(w0).max() > 0.99 * a0
    assert np.all(th[50176:50240] == 0) and np.all(th[50880:] == 0)


def test_teacher_labels_and_batches():
    rows = np.arange(2000)
    y = synth.teacher_labels(4, rows, 784, 10)
    assert y.min() >= 0 and y.max() <= 9
    counts = np.bincount(y, minlength=10)
    assert counts.min() > 100
    # labels are the argmax of the float inputs against the float teacher too
    X = synth.data_rows(4, rows[:50], 784).astype(np.float64)
    T = synth.teacher_int(4, 784, 10).astype(np.float64) * 2.0 ** -20
    assert np.array_equal(np.argmax(X @ T, axis=1), y[:50])
    b = synth.batch_indices(4, 3, 7, 128)
    assert b.min() >= 0 and b.max() < synth.DATA_ROWS and b.shape == (128,)
    order = np.array([0, 1, 0, 2, 1, 0])
    sb = synth.schedule_batches(4, order, 16)
    assert np.array_equal(sb[2], synth.batch_indices(4, 0, 1, 16))
    assert np.array_equal(sb[5], synth.batch_indices(4, 0, 2, 16))
    assert np.array_equal(sb[4], synth.batch_indices(4, 1, 1, 16))
