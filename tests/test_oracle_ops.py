"""Pins of the oracle's primitive ops against brute force, closed forms,
invariants and independent library routines (CPU only)."""
import itertools
import json
import os

import numpy as np
import pytest
import scipy.special
import torch
import torch.nn.functional as F

from oracle import pnn_oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
rng = np.random.default_rng(7)


def brute_conv(x, w, stride, pad):
    B, C, H, W = x.shape
    K, _, R, S = w.shape
    P = (H + 2 * pad - R) // stride + 1
    Q = (W + 2 * pad - S) // stride + 1
    y = np.zeros((B, K, P, Q))
    for b, k, p, q in itertools.product(range(B), range(K), range(P), range(Q)):
        acc = 0.0
        for c, r, s in itertools.product(range(C), range(R), range(S)):
            h, ww = p * stride + r - pad, q * stride + s - pad
            if 0 <= h < H and 0 <= ww < W:
                acc += x[b, c, h, ww] * w[k, c, r, s]
        y[b, k, p, q] = acc
    return y


@pytest.mark.parametrize("C,K,H,W,R,stride", [(3, 4, 5, 5, 3, 1), (2, 3, 6, 7, 3, 2),
                                              (4, 5, 6, 6, 1, 2), (3, 2, 1, 1, 3, 1)])
def test_conv_brute_force(C, K, H, W, R, stride):
    x = rng.standard_normal((2, C, H, W))
    w = rng.standard_normal((K, C, R, R))
    pad = R // 2
    np.testing.assert_allclose(O.conv2d(x, w, stride, pad), brute_conv(x, w, stride, pad), rtol=1e-12, atol=1e-12)


def test_conv_matches_torch_functional():
    x = rng.standard_normal((3, 5, 9, 8))
    w = rng.standard_normal((6, 5, 3, 3))
    for stride in (1, 2):
        ref = F.conv2d(torch.from_numpy(x), torch.from_numpy(w), stride=stride, padding=1).numpy()
        np.testing.assert_allclose(O.conv2d(x, w, stride, 1), ref, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("R,stride", [(3, 1), (3, 2), (1, 2), (1, 1)])
def test_conv_backward_is_adjoint(R, stride):
    """<conv(x), dy> = <x, dx(dy)> and d<conv(x),dy>/dw = dw, both exact for a
    bilinear map; checked against the brute-force forward."""
    x = rng.standard_normal((2, 3, 5, 6))
    w = rng.standard_normal((4, 3, R, R))
    pad = R // 2
    y = brute_conv(x, w, stride, pad)
    dy = rng.standard_normal(y.shape)
    dx, dw = O.conv2d_backward(x, w, stride, pad, dy)
    assert np.isclose((y * dy).sum(), (x * dx).sum(), rtol=1e-12)
    assert np.isclose((y * dy).sum(), (w * dw).sum(), rtol=1e-12)
    # and elementwise against a perturbation of single entries
    for idx in [(0, 1, 2, 3), (1, 2, 4, 5), (0, 0, 0, 0)]:
        e = np.zeros_like(x)
        e[idx] = 1.0
        assert np.isclose((brute_conv(e, w, stride, pad) * dy).sum(), dx[idx], rtol=1e-10, atol=1e-12)


def test_batchnorm_normalises():
    h = rng.standard_normal((4, 3, 5, 5)) * 3 + 2
    z, _ = O.batchnorm(h, np.ones(3), np.zeros(3))
    np.testing.assert_allclose(z.mean(axis=(0, 2, 3)), 0, atol=1e-12)
    var = z.var(axis=(0, 2, 3))
    expect = h.var(axis=(0, 2, 3)) / (h.var(axis=(0, 2, 3)) + O.BN_EPS)
    np.testing.assert_allclose(var, expect, rtol=1e-12)
    g, b = rng.standard_normal(3), rng.standard_normal(3)
    z2, _ = O.batchnorm(h, g, b)
    np.testing.assert_allclose(z2, z * g.reshape(1, 3, 1, 1) + b.reshape(1, 3, 1, 1), rtol=1e-12, atol=1e-12)


def test_batchnorm_backward_finite_difference():
    h = rng.standard_normal((3, 2, 4, 4))
    g, b = rng.standard_normal(2), rng.standard_normal(2)
    G = rng.standard_normal(h.shape)

    def f(hh, gg, bb):
        return (O.batchnorm(hh, gg, bb)[0] * G).sum()

    _, cache = O.batchnorm(h, g, b)
    dh, dg, db = O.batchnorm_backward(G, g, cache)
    eps = 1e-6
    for idx in [(0, 0, 1, 2), (2, 1, 3, 3), (1, 1, 0, 0)]:
        e = np.zeros_like(h)
        e[idx] = eps
        fd = (f(h + e, g, b) - f(h - e, g, b)) / (2 * eps)
        assert abs(fd - dh[idx]) < 1e-7 * max(1, abs(fd))
    for c in range(2):
        e = np.zeros(2)
        e[c] = eps
        assert abs((f(h, g + e, b) - f(h, g - e, b)) / (2 * eps) - dg[c]) < 1e-6
        assert abs((f(h, g, b + e) - f(h, g, b - e)) / (2 * eps) - db[c]) < 1e-6


def test_maxpool_brute_force_and_first_max_routing():
    x = rng.standard_normal((2, 2, 7, 6))
    y, arg = O.maxpool(x, 3, 2, 1)
    P, Q = y.shape[2:]
    for b, c, p, q in itertools.product(range(2), range(2), range(P), range(Q)):
        vals = [x[b, c, p * 2 + r - 1, q * 2 + s - 1] for r in range(3) for s in range(3)
                if 0 <= p * 2 + r - 1 < 7 and 0 <= q * 2 + s - 1 < 6]
        assert y[b, c, p, q] == max(vals)
    # ties: a constant window routes its gradient to the first element in row-major order
    t = np.zeros((1, 1, 2, 2))
    yt, at = O.maxpool(t, 2, 2, 0)
    dx = O.maxpool_backward(np.ones_like(yt), at, t.shape, 2, 2, 0)
    assert dx[0, 0, 0, 0] == 1 and dx.sum() == 1
    # gradient check on distinct values
    dy = rng.standard_normal(y.shape)
    dx = O.maxpool_backward(dy, arg, x.shape, 3, 2, 1)
    tx = torch.from_numpy(x).requires_grad_()
    F.max_pool2d(tx, 3, 2, 1).backward(torch.from_numpy(dy))
    np.testing.assert_allclose(dx, tx.grad.numpy(), rtol=1e-12)


def test_softmax_cross_entropy_closed_form():
    z = rng.standard_normal((5, 7)) * 4
    labels = np.array([0, 6, 3, 3, 1])
    loss, dz = O.softmax_cross_entropy(z, labels)
    expect = np.mean(scipy.special.logsumexp(z, axis=1) - z[np.arange(5), labels])
    assert np.isclose(loss, expect, rtol=1e-13)
    np.testing.assert_allclose(dz.sum(axis=1), 0, atol=1e-15)
    # uniform logits: loss = log(m)
    assert np.isclose(O.softmax_cross_entropy(np.zeros((3, 7)), np.array([1, 2, 3]))[0], np.log(7))
    eps = 1e-6
    for idx in [(0, 0), (2, 3), (4, 6)]:
        e = np.zeros_like(z)
        e[idx] = eps
        fd = (O.softmax_cross_entropy(z + e, labels)[0] - O.softmax_cross_entropy(z - e, labels)[0]) / (2 * eps)
        assert abs(fd - dz[idx]) < 1e-8


def test_sgd_nesterov_hand_example():
    g = json.load(open(os.path.join(GOLDEN, "sgd_nesterov_hand.json")))
    th1, b1 = O.sgd_step(np.array(g["theta0"]), np.array(g["grad1"]), None, g["lr"], g["momentum"],
                         g["weight_decay"], True)
    np.testing.assert_allclose(th1, g["theta1"], rtol=1e-12)
    np.testing.assert_allclose(b1, g["buf1"], rtol=1e-12)
    th2, b2 = O.sgd_step(th1, np.array(g["grad2"]), b1, g["lr"], g["momentum"], g["weight_decay"], True)
    np.testing.assert_allclose(th2, g["theta2"], rtol=1e-10)
    np.testing.assert_allclose(b2, g["buf2"], rtol=1e-10, atol=1e-15)


def test_round_bf16_matches_torch_and_ties_to_even():
    x = (rng.standard_normal(20000) * 10.0 ** rng.integers(-6, 6, 20000)).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(O.round_bf16(x.astype(np.float64)), ref)
    # exact halfway cases round to the even neighbour
    assert O.round_bf16(1 + 2.0 ** -8) == 1.0
    assert O.round_bf16(1 + 3 * 2.0 ** -8) == 1 + 2.0 ** -6
    assert O.round_bf16(-(1 + 2.0 ** -8)) == -1.0
    assert O.round_bf16(np.inf) == np.inf


def test_bf16_precision_model_rounds_conv_operands():
    """With precision='bf16' every convolution input the oracle contracts is
    bf16-representable; with the default precision nothing is rounded."""
    import workloads as W
    d = W.tiny_resnet(batch=2)
    d["in_h"] = d["in_w"] = 8
    seen = []
    orig = O.conv2d

    def spy(x, w, stride, pad):
        seen.append(np.array_equal(O.round_bf16(x), x) and np.array_equal(O.round_bf16(w), w))
        return orig(x, w, stride, pad)

    O.conv2d = spy
    try:
        net = O.ParaNet(d, precision="bf16")
        theta = W.init_params(net.spec, seed=1, bf16=True)
        x, labels = W.make_batch(d, seed=2)
        net.forward(theta, x, labels)
        assert seen and all(seen)
        seen.clear()
        O.ParaNet(d).forward(theta, x.astype(np.float64) + 1e-3, labels)
        assert not all(seen)
    finally:
        O.conv2d = orig
