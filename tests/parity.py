"""Shared helpers of the GPU parity tests: run one training step through the
C ABI and through the oracle on the same seeded inputs and compare.

Metrics (the target tolerances; the formulas are these):
  forward tensors  max|a - r| / max|r|            <= 2e-2 (bf16), 1e-4 (fp32 check)
  gradients        ||g - r||_2 / ||r||_2 per tensor <= 5e-2 (bf16), 1e-4 (fp32 check)
"""
from __future__ import annotations

import numpy as np

import workloads as W
from oracle import pnn_oracle as O

TOL = {"bf16": {"fwd": 2e-2, "grad": 5e-2}, "fp32": {"fwd": 1e-4, "grad": 1e-4}}


def max_rel(a, r):
    r = np.asarray(r, np.float64)
    den = np.abs(r).max()
    return float(np.abs(np.asarray(a, np.float64) - r).max() / (den if den > 0 else 1.0))


def norm_rel(a, r):
    r = np.asarray(r, np.float64)
    den = np.linalg.norm(r)
    return float(np.linalg.norm(np.asarray(a, np.float64) - r) / (den if den > 0 else 1.0))


def inputs(desc, seed=None):
    onet = O.ParaNet(desc)
    theta = W.init_params(onet.spec, seed=0, bf16=desc["precision"] == "bf16")
    x, labels = W.make_batch(desc, seed=seed)
    return onet, theta, x, labels


def run_gpu(desc, theta, x, labels, **kw):
    import torch
    from paper_2103_08802_gb300 import pnn
    net = pnn.ParaNet(desc, **kw)
    net.set_params(theta)
    xd = torch.from_numpy(x).cuda()
    ld = torch.from_numpy(labels).cuda()
    loss = torch.zeros(1, dtype=torch.float32, device="cuda")
    net.forward(xd, ld, loss)
    net.backward()
    net.sync()
    N = len(desc["segments"])
    out = {"loss": float(loss.cpu()), "grad": net.get_grads(), "logits": net.get_tensor("logits"),
           "ytilde": net.get_tensor("ytilde")}
    for j in range(1, N + 1):
        out[f"x{j}"] = net.get_tensor("x", j)
        out[f"y{j}"] = net.get_tensor("y", j)
        out[f"rt{j}"] = net.get_tensor("rtilde", j)
        out[f"D{j}"] = net.get_tensor("D", j)
        if j < N:
            out[f"r{j}"] = net.get_tensor("r", j)
    net.sgd_step()
    net.sync()
    out["theta_new"] = net.get_params()
    out["momentum"] = net.get_momentum()
    out["net"] = net
    out["onet"] = O.ParaNet(desc)
    return out


def run_oracle(desc, theta, x, labels, precision=None):
    """The oracle step.  bf16 workloads use the oracle's bf16 forward model
    (decisions such as ReLU masks and maxpool argmax taken in the kernel's
    precision) unless precision="fp64" is asked for."""
    if precision is None:
        precision = "bf16" if desc["precision"] == "bf16" else "fp64"
    res = O.train_step(desc, theta.astype(np.float64), x.astype(np.float64), labels, precision=precision)
    st = res["state"]
    N = len(desc["segments"])
    out = {"loss": res["loss"], "grad": res["grad"], "logits": st["logits"], "ytilde": st["ytilde"],
           "theta_new": res["theta_new"], "momentum": res["buf_new"], "onet": res["net"]}
    for j in range(1, N + 1):
        out[f"x{j}"] = st["xs"][j - 1]
        out[f"y{j}"] = st["ys"][j - 1]
        out[f"rt{j}"] = st["rt"][j - 1]
        out[f"D{j}"] = st["D"][j - 1]
        if j < N:
            out[f"r{j}"] = st["r"][j - 1]
    return out


def compare(desc, g, o, tol=None):
    """Returns a dict of metric -> value and the list of failures."""
    tol = tol or TOL[desc["precision"]]
    report, fails = {}, []
    N = len(desc["segments"])
    names = ["logits", "ytilde"] + [f"{p}{j}" for j in range(1, N + 1) for p in ("x", "y", "rt")] \
        + [f"r{j}" for j in range(1, N)]
    for k in names:
        e = max_rel(g[k].ravel(), o[k].ravel())
        report[k] = e
        if not e <= tol["fwd"]:
            fails.append((k, e))
    for j in range(1, N + 1):
        e = norm_rel(g[f"D{j}"].ravel(), o[f"D{j}"].ravel())
        report[f"D{j}"] = e
        if not e <= tol["grad"]:
            fails.append((f"D{j}", e))
    le = abs(g["loss"] - o["loss"]) / max(1.0, abs(o["loss"]))
    report["loss"] = le
    if not le <= tol["fwd"]:
        fails.append(("loss", le))
    onet = o.get("onet") or g.get("onet")
    if onet is None:  # two GPU runs: no parameter table at hand
        return report, fails
    off = 0
    worst = 0.0
    for i, (kind, shape) in enumerate(onet.spec):
        n = int(np.prod(shape))
        e = norm_rel(g["grad"][off:off + n], o["grad"][off:off + n])
        worst = max(worst, e)
        if not e <= tol["grad"]:
            fails.append((f"grad[{i}] kind {kind} {shape}", e))
        off += n
    report["grad_worst"] = worst
    return report, fails
