"""An independent float64 PyTorch-CPU evaluation of the same networks, used
only by the tests to pin the oracle.  It is written with torch.nn.functional
and autograd, shares no code with oracle/ and reads only the description
dict and the flat parameter vector (ordered as in eq:barf)."""
from __future__ import annotations

import math
import torch
import torch.nn.functional as F

F64 = torch.float64


class _Params:
    def __init__(self, theta):
        self.t = theta
        self.i = 0

    def take(self, *shape):
        n = math.prod(shape)
        v = self.t[self.i:self.i + n].view(*shape)
        self.i += n
        return v


# Running statistics: None, or {"train": bool, "stats": {gamma offset: (mean, var)}}.
# torch.nn.functional.batch_norm moves the buffers itself in training mode
# (momentum 0.1, unbiased variance) and normalises with them in eval mode.
RUNNING = None


def _bn(h, p, linear=False):
    off = p.i
    g = p.take(h.shape[1])
    b = p.take(h.shape[1])
    if linear:
        return h
    if RUNNING is None:
        return F.batch_norm(h, None, None, g, b, training=True, momentum=0.0, eps=1e-5)
    rm, rv = RUNNING["stats"].setdefault(
        off, (torch.zeros(h.shape[1], dtype=F64), torch.ones(h.shape[1], dtype=F64)))
    return F.batch_norm(h, rm, rv, g, b, training=RUNNING["train"], momentum=0.1, eps=1e-5)


def _act(z, linear=False):
    return z if linear else F.relu(z)


def layer(spec, x, p, linear=False):
    op = spec["op"]
    cin = x.shape[1]
    if op == "conv":
        k, s = spec.get("k", 3), spec.get("stride", 1)
        return F.conv2d(x, p.take(spec["cout"], cin, k, k), stride=s, padding=k // 2)
    if op == "conv_bn_relu":
        k, s = spec.get("k", 3), spec.get("stride", 1)
        h = F.conv2d(x, p.take(spec["cout"], cin, k, k), stride=s, padding=k // 2)
        a = _act(_bn(h, p, linear), linear)
        if spec.get("pool", 0):
            a = F.avg_pool2d(a, 2, 2) if linear else F.max_pool2d(a, 2, 2)
        return a
    if op == "basic":
        c = spec["cout"]
        h1 = F.conv2d(x, p.take(c, cin, 3, 3), padding=1)
        a1 = _act(_bn(h1, p, linear), linear)
        h2 = F.conv2d(a1, p.take(c, c, 3, 3), padding=1)
        return _act(_bn(h2, p, linear) + x, linear)
    if op == "bottleneck":
        c, m, s = spec["cout"], spec["mid"], spec.get("stride", 1)
        a1 = _act(_bn(x, p, linear), linear)
        h1 = F.conv2d(a1, p.take(m, cin, 1, 1))
        a2 = _act(_bn(h1, p, linear), linear)
        h2 = F.conv2d(a2, p.take(m, m, 3, 3), stride=s, padding=1)
        a3 = _act(_bn(h2, p, linear), linear)
        h3 = F.conv2d(a3, p.take(c, m, 1, 1))
        if cin != c or s != 1:
            return h3 + F.conv2d(a1, p.take(c, cin, 1, 1), stride=s)
        return h3 + x
    if op == "coarse_ru":
        c, s = spec["cout"], spec.get("stride", 1)
        a1 = _act(_bn(x, p, linear), linear)
        h1 = F.conv2d(a1, p.take(c, cin, 3, 3), stride=s, padding=1)
        a2 = _act(_bn(h1, p, linear), linear)
        h2 = F.conv2d(a2, p.take(c, c, 3, 3), padding=1)
        if cin != c or s != 1:
            return h2 + F.conv2d(a1, p.take(c, cin, 1, 1), stride=s)
        return h2 + x
    raise ValueError(op)


def stack(specs, x, p, linear=False):
    for s in specs:
        x = layer(s, x, p, linear)
    return x


def preprocess(x, target, post, p):
    c, h, w = target
    while x.shape[2] > h:
        x = F.max_pool2d(x, 3, 2, 1)
    assert x.shape[2] == h
    y = F.conv2d(x, p.take(c, x.shape[1], 1, 1))
    if post == "bn_relu":
        y = F.relu(_bn(y, p))
    return y


def head(desc, y, p):
    hd = desc["head"]
    if hd["kind"] == "bn_relu_gap_fc":
        y = F.relu(_bn(y, p))
    f = y.mean(dim=(2, 3))
    widths = [f.shape[1]] + list(hd.get("hidden", [])) + [desc["classes"]]
    for i in range(len(widths) - 1):
        W = p.take(widths[i + 1], widths[i])
        b = p.take(widths[i + 1])
        f = F.linear(f, W, b)
        if i < len(widths) - 2:
            f = F.relu(f)
    return f


def _shapes(desc, x):
    """Output shapes X_0..X_N found by a dry run with zero parameters (which
    leaves running statistics alone)."""
    global RUNNING
    saved, RUNNING = RUNNING, None
    try:
        return _dry_shapes(desc, x)
    finally:
        RUNNING = saved


def _dry_shapes(desc, x):
    with torch.no_grad():
        p = _Params(torch.zeros(10 ** 8, dtype=F64))
        h = stack(desc["stem"], x[:2], p)
        out = [tuple(h.shape[1:])]
        i = 0
        for n in desc["segments"]:
            h = stack(desc["body"][i:i + n], h, p)
            out.append(tuple(h.shape[1:]))
            i += n
    return out


def parareal_loss(desc, theta, x, labels, linear_body=False, return_parts=False):
    """Loss of the parareal network (eq:correct or its delta form)."""
    x = torch.as_tensor(x, dtype=torch.float64)
    labels = torch.as_tensor(labels, dtype=torch.long)
    X = _shapes(desc, x)
    p = _Params(theta)
    N = len(desc["segments"])
    xs, ys = [], []
    i = 0
    for j, n in enumerate(desc["segments"]):
        xj = stack(desc["stem"], x, p) if j == 0 else preprocess(x, X[j], desc["cj_post"], p)
        ys.append(stack(desc["body"][i:i + n], xj, p, linear_body))
        xs.append(xj)
        i += n
    r = [ys[j] - xs[j + 1] for j in range(N - 1)] + [torch.zeros_like(ys[-1])]
    rt = r[0]
    mode = desc.get("correction", "residual")
    for j in range(N - 1):
        start = p.i
        if mode == "residual":
            rt = r[j + 1] + stack(desc["coarse"][j], rt, p, linear_body)
        else:
            f0 = stack(desc["coarse"][j], xs[j + 1], p, linear_body)
            p.i = start
            f1 = stack(desc["coarse"][j], xs[j + 1] + rt, p, linear_body)
            rt = r[j + 1] + f1 - f0
    ytilde = ys[-1] + rt
    z = head(desc, ytilde, p)
    assert p.i == theta.numel(), (p.i, theta.numel())
    loss = F.cross_entropy(z, labels)
    if return_parts:
        return loss, {"xs": xs, "ys": ys, "ytilde": ytilde, "logits": z}
    return loss


def sequential_loss(desc, theta_seq, x, labels, linear_body=False):
    """The untorn network f = h o g o C_delta (stem, all body layers, head)."""
    x = torch.as_tensor(x, dtype=torch.float64)
    labels = torch.as_tensor(labels, dtype=torch.long)
    p = _Params(theta_seq)
    h = stack(desc["stem"], x, p)
    h = stack(desc["body"], h, p, linear_body)
    z = head(desc, h, p)
    assert p.i == theta_seq.numel()
    return F.cross_entropy(z, labels), z


def grad_of(desc, theta, x, labels, linear_body=False):
    t = torch.tensor(theta, dtype=torch.float64, requires_grad=True)
    loss = parareal_loss(desc, t, x, labels, linear_body)
    loss.backward()
    return float(loss.detach()), t.grad.numpy().copy()
