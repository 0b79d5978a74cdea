"""BN running statistics and the eval-mode forward (pnn_infer) against the
oracle, through the C ABI.

* After a training-mode forward every BN's running mean and variance (momentum 0.1,
  unbiased batch variance) match the oracle's: fp32 check mode within 1e-4
  (the fp32 target bound), bf16 within 2e-2 max-relative (the forward bound;
  the statistics are forward quantities).
* An inference net (opts.inference = 1: forward only, activations sharing
  buffers) given the same parameters and running statistics returns the
  oracle's eval-mode logits within the same bounds; in bf16 the oracle runs
  its bf16 forward model.
"""
import numpy as np
import pytest

import workloads as W
from oracle import pnn_oracle as O
from parity import inputs, max_rel

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2103_08802_gb300 import build
    build.build()


def _cuda(x, labels):
    import torch
    return torch.from_numpy(x).cuda(), torch.from_numpy(labels).cuda()


def _reduced(idx, precision):
    if idx == 0:
        d = W.config(0)
    elif idx == 1:
        d = W.parareal_vgg16(batch=32)
    elif idx == 4:
        d = W.parareal_resnet1001(n_seg=8, batch=32, classes=200, hw=64, per_stage=3,
                                  segments=[2, 1, 1, 1, 1, 1, 1, 1])
    else:
        d = W.paper_parareal_resnet(3, batch=32, per_stage=2)
    d["precision"] = precision
    return d


CASES = [(0, "fp32", "residual"), (0, "fp32", "delta"), (4, "fp32", "residual"), (1, "bf16", "residual"),
         (4, "bf16", "residual"), (4, "bf16", "delta"), ("paper3", "bf16", "residual")]


@pytest.mark.parametrize("idx,precision,mode", CASES)
def test_running_statistics_after_a_training_forward(idx, precision, mode):
    from paper_2103_08802_gb300 import pnn
    d = _reduced(idx, precision)
    d["correction"] = mode
    onet, theta, x, labels = inputs(d)
    r0 = O.RunningStats(onet.spec)
    rng = np.random.default_rng(3)
    for o, c in r0.layers:
        r0.mean[o] = 0.2 * rng.standard_normal(c)
        r0.var[o] = rng.uniform(0.5, 2.0, c)
    start = r0.flat().astype(np.float32)
    net = pnn.ParaNet(d)
    net.set_params(theta)
    net.set_running_stats(start)
    np.testing.assert_array_equal(net.running_stats(), start)
    xd, ld = _cuda(x, labels)
    net.forward(xd, ld)
    net.sync()
    got = net.running_stats()
    onet_p = O.ParaNet(d, precision="bf16" if precision == "bf16" else "fp64")
    rs = O.RunningStats(onet_p.spec).from_flat(start.astype(np.float64))
    onet_p.forward(theta.astype(np.float64), x.astype(np.float64), labels, rs)
    want = rs.flat()
    tol = 1e-4 if precision == "fp32" else 2e-2
    # per BN layer, means and variances separately
    i = 0
    for _, c in r0.layers:
        for part in (slice(i, i + c), slice(i + c, i + 2 * c)):
            assert max_rel(got[part], want[part]) <= tol, (i, max_rel(got[part], want[part]))
        i += 2 * c
    assert not np.allclose(got, start)


@pytest.mark.parametrize("idx,precision,mode", CASES)
def test_inference_logits(idx, precision, mode):
    import torch
    from paper_2103_08802_gb300 import pnn
    d = _reduced(idx, precision)
    d["correction"] = mode
    onet, theta, x, labels = inputs(d)
    rs = O.RunningStats(onet.spec)
    rng = np.random.default_rng(4)
    for o, c in rs.layers:
        rs.mean[o] = 0.2 * rng.standard_normal(c)
        rs.var[o] = rng.uniform(0.5, 2.0, c)
    run = rs.flat().astype(np.float32)
    net = pnn.ParaNet(d, inference=True)
    net.set_params(theta)
    net.set_running_stats(run)
    xd, _ = _cuda(x, labels)
    logits = torch.empty(d["batch"] * d["classes"], dtype=torch.float32, device="cuda")
    net.infer(xd, logits)
    net.sync()
    got = logits.cpu().numpy().reshape(d["batch"], d["classes"])
    np.testing.assert_array_equal(net.get_tensor("logits").reshape(got.shape), got)
    want = O.ParaNet(d, precision="bf16" if precision == "bf16" else "fp64").infer(
        theta.astype(np.float64), x.astype(np.float64), run.astype(np.float64))
    tol = 1e-4 if precision == "fp32" else 2e-2
    err = max_rel(got.ravel(), want.ravel())
    print(d["name"], precision, mode, "inference logits max-rel", err)
    assert err <= tol
    # a replay of the captured graph gives the same logits
    logits.zero_()
    net.infer(xd, logits)
    net.sync()
    np.testing.assert_array_equal(logits.cpu().numpy().reshape(got.shape), got)


def test_inference_net_refuses_training_calls():
    import torch
    from paper_2103_08802_gb300 import pnn
    d = W.config(0)
    onet, theta, x, labels = inputs(d)
    net = pnn.ParaNet(d, inference=True)
    xd, ld = _cuda(x, labels)
    for call in (lambda: net.forward(xd, ld), lambda: net.train_step(xd, ld), lambda: net.get_grads(),
                 lambda: net.get_tensor("x", 1)):
        with pytest.raises(pnn.PnnError):
            call()
    train = pnn.ParaNet(d)
    with pytest.raises(pnn.PnnError):
        train.infer(xd, torch.empty(d["batch"] * d["classes"], device="cuda"))
