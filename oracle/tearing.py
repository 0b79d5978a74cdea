"""Plain reference for cost-balanced tearing (test infrastructure only).

TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and the
cpu_baseline / reference legs of bench.py may import it; it shares no code
with the library.

Section 4.2 (the remark after Table grad): cutting the block-repetitive part
into subnetworks with equal numbers of RUs is not optimal because RUs differ in
cost; a cut into subnetworks of equal computational cost should shorten the
virtual wall-clock time of the parallel phase, which is the largest subnetwork's
time.  Written out here:

  * the cost of a layer as the number of multiply-adds of its convolutions,
    from the layer's shapes (forward; the backward of a conv is a data-gradient
    and a weight-gradient convolution of the same size, so training costs three
    times the forward);
  * the best cut by exhaustive search: every placement of n_seg - 1 cuts between
    n layers, keeping the smallest largest segment sum.
"""
from __future__ import annotations

import itertools


def _conv_macs(cin, h, w, cout, k, stride):
    """Multiply-adds of a k x k conv with zero padding k // 2 on a cin x h x w map."""
    p = (h + 2 * (k // 2) - k) // stride + 1
    q = (w + 2 * (k // 2) - k) // stride + 1
    return p * q * cout * cin * k * k, (cout, p, q)


def layer_forward_macs(spec, shape):
    """Forward multiply-adds of one layer of a description on one image, and
    its output shape (C, H, W)."""
    c, h, w = shape
    op = spec["op"]
    if op in ("conv", "conv_bn_relu"):
        m, out = _conv_macs(c, h, w, spec["cout"], spec.get("k", 3), spec.get("stride", 1))
        if spec.get("pool", 0):
            out = (out[0], out[1] // 2, out[2] // 2)
        return m, out
    if op == "basic":
        m1, out = _conv_macs(c, h, w, spec["cout"], 3, 1)
        m2, out = _conv_macs(spec["cout"], out[1], out[2], spec["cout"], 3, 1)
        return m1 + m2, out
    if op == "bottleneck":
        k, mid, s = spec["cout"], spec["mid"], spec.get("stride", 1)
        m1, o1 = _conv_macs(c, h, w, mid, 1, 1)
        m2, o2 = _conv_macs(mid, h, w, mid, 3, s)
        m3, out = _conv_macs(mid, o2[1], o2[2], k, 1, 1)
        mp = _conv_macs(c, h, w, k, 1, s)[0] if (c != k or s != 1) else 0
        return m1 + m2 + m3 + mp, out
    if op == "coarse_ru":
        k, s = spec["cout"], spec.get("stride", 1)
        m1, o1 = _conv_macs(c, h, w, k, 3, s)
        m2, out = _conv_macs(k, o1[1], o1[2], k, 3, 1)
        mp = _conv_macs(c, h, w, k, 1, s)[0] if (c != k or s != 1) else 0
        return m1 + m2 + mp, out
    raise ValueError(op)


def body_training_flops(desc, body_in_shape):
    """Per body layer: FLOPs of its forward, data-gradient and weight-gradient
    convolutions for the whole batch (3 x 2 x forward multiply-adds)."""
    out, shape = [], tuple(body_in_shape)
    for spec in desc["body"]:
        m, shape = layer_forward_macs(spec, shape)
        out.append(3 * 2 * m * desc["batch"])
    return out


def best_cut(costs, n_seg):
    """Smallest possible largest segment sum over all cuts of `costs` into
    n_seg consecutive non-empty segments (exhaustive)."""
    n = len(costs)
    best = None
    for cuts in itertools.combinations(range(1, n), n_seg - 1):
        bounds = (0,) + cuts + (n,)
        worst = max(sum(costs[bounds[i]:bounds[i + 1]]) for i in range(n_seg))
        best = worst if best is None else min(best, worst)
    return best
