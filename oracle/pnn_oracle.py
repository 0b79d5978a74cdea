"""Plain CPU fp64 oracle of the parareal neural network training step.

TEST INFRASTRUCTURE ONLY.  This module exists to check the CUDA library.  Only
tests/, __graft_entry__.smoke() and the cpu_baseline / reference legs of
bench.py may import it.  It shares no code with the CUDA path and never calls
it; the product path does not import it.

What it computes (Lee, Lee & Park, "Parareal Neural Networks Emulating a
Parallel-in-time Algorithm"):

  * Section 3.1, eq:xjyj:  x_j = C^j(x),  y_j = g^j(x_j)            (fine, parallel)
  * Section 3.1, eq:correct (default "residual" mode):
        r_N = 0,  r_j = y_j - x_{j+1}                                 (j < N)
        rt_1 = r_1,  rt_{j+1} = r_{j+1} + F^j(rt_j)
        ytilde = y_N + rt_N
    "delta" mode (the classic parareal update of Section 2):
        rt_{j+1} = r_{j+1} + F^j(x_{j+1} + rt_j) - F^j(x_{j+1})
  * eq:barf: output h(ytilde), parameters ordered
        (delta_1, phi_1, ..., delta_N, phi_N, eta_1, ..., eta_{N-1}, eps)
  * Algorithm 2 / Section 3.2 (eq:etak, eq:phij, eq:deltaj): D_N = dL/dytilde,
    the coarse chain backwards for D_j and the eta_j gradients, then every
    subnetwork with seed dL/dy_j = D_j and dL/dx_j -= D_{j-1}.
  * Section 4: SGD with Nesterov momentum and weight decay.
  * BN running statistics and the eval-mode forward (the paper states no rule;
    the reading is PyTorch's BatchNorm2d, see RunningStats): ParaNet.forward
    with a RunningStats moves them, ParaNet.infer normalises with them.
  * Section 4.2's coarse RU (two 3x3 convs and a skip, CoarseRU).

Layout is NCHW, every value float64.  Each primitive is the textbook
definition written out; numpy's tensordot (a library matmul) serves as the
inner contraction of the convolution.  Readings of points the paper leaves
open (BN eps, pooling padding, block layout, loss) are the module constants
and the layer classes below.

Precision model.  The paper fixes no precision.  By default everything is
float64.  With precision="bf16" the pass rounds to bfloat16 exactly the
values a bf16 tensor-core implementation holds in bf16: every convolution
operand (input activation, weight, and in the backward pass the output
gradient), and every stored convolution / pooling output that is not
followed by a residual add.  This makes the floating-point decisions of the
forward pass (ReLU masks, maxpool argmax) use the kernel's precision; all
arithmetic stays float64.  A description with "residual_stream": "bf16" also
rounds the residual-stream values the library then stores in bf16: every
residual block's output, r_j, rt_j, the delta form's x_{j+1} + rt_j, and
ytilde.
"""
from __future__ import annotations

import math
import numpy as np

BN_EPS = 1e-5
KIND_CONV_W, KIND_BN_G, KIND_BN_B, KIND_FC_W, KIND_FC_B = 0, 1, 2, 3, 4


# ====================================================================== ops
def round_bf16(a):
    """Round float64 values to the nearest bfloat16 value (8 significant bits,
    ties to even), returned as float64.  Operates on the float64 bit pattern:
    drop the low 45 of the 52 mantissa bits with round-half-to-even."""
    a = np.asarray(a, dtype=np.float64)
    u = a.view(np.uint64)
    lsb = (u >> np.uint64(45)) & np.uint64(1)
    r = (u + np.uint64((1 << 44) - 1) + lsb) & ~np.uint64((1 << 45) - 1)
    out = r.view(np.float64)
    return np.where(np.isfinite(a), out, a)


def conv2d(x, w, stride, pad):
    """y[b,k,p,q] = sum_{c,r,s} x[b,c,p*stride+r-pad,q*stride+s-pad] w[k,c,r,s]
    with zero padding."""
    B, C, H, W = x.shape
    K, C2, R, S = w.shape
    assert C == C2
    P = (H + 2 * pad - R) // stride + 1
    Q = (W + 2 * pad - S) // stride + 1
    xp = np.pad(x, ((0, 0), (0, 0), (pad, pad), (pad, pad)))
    y = np.zeros((B, K, P, Q))
    for r in range(R):
        for s in range(S):
            patch = xp[:, :, r:r + stride * (P - 1) + 1:stride, s:s + stride * (Q - 1) + 1:stride]
            # sum over c of patch[b,c,p,q] * w[k,c,r,s]
            y += np.tensordot(patch, w[:, :, r, s], axes=([1], [1])).transpose(0, 3, 1, 2)
    return y


def conv2d_backward(x, w, stride, pad, dy, need_dx=True):
    """Adjoint of conv2d: dw[k,c,r,s] = sum_{b,p,q} dy[b,k,p,q] x[b,c,p*s+r-pad,...]
    and dx = the transpose scatter of dy through w."""
    B, C, H, W = x.shape
    K, _, R, S = w.shape
    P, Q = dy.shape[2], dy.shape[3]
    xp = np.pad(x, ((0, 0), (0, 0), (pad, pad), (pad, pad)))
    dxp = np.zeros_like(xp) if need_dx else None
    dw = np.zeros_like(w)
    for r in range(R):
        for s in range(S):
            sl = (slice(None), slice(None),
                  slice(r, r + stride * (P - 1) + 1, stride),
                  slice(s, s + stride * (Q - 1) + 1, stride))
            patch = xp[sl]
            dw[:, :, r, s] = np.tensordot(dy, patch, axes=([0, 2, 3], [0, 2, 3]))
            if need_dx:
                dxp[sl] += np.tensordot(dy, w[:, :, r, s], axes=([1], [0])).transpose(0, 3, 1, 2)
    dx = dxp[:, :, pad:pad + H, pad:pad + W] if need_dx else None
    return dx, dw


BN_MOMENTUM = 0.1


class RunningStats:
    """Running statistics of every BN layer.  The paper trains with BN and
    states no rule for them; the reading is PyTorch's BatchNorm2d: per layer a
    running mean (initially 0) and variance (initially 1); every training-mode
    evaluation moves them the fraction `momentum` towards the batch mean and
    the unbiased batch variance (n / (n - 1) times the biased one, n values
    per channel); an evaluation in eval mode normalises with them instead of
    the batch's statistics.  A layer is identified by the offset of its gamma
    in the parameter vector, so the delta form's two evaluations of F^j move
    the same statistics, in the order they run.

    Flat layout (`flat`, `from_flat`): for every BN layer in parameter order,
    its C running means, then its C running variances."""

    def __init__(self, spec, momentum=BN_MOMENTUM, eval_mode=False):
        self.momentum, self.eval = momentum, eval_mode
        self.layers, off = [], 0
        for kind, shape in spec:
            if kind == KIND_BN_G:
                self.layers.append((off, int(shape[0])))
            off += int(np.prod(shape))
        self.mean = {o: np.zeros(c) for o, c in self.layers}
        self.var = {o: np.ones(c) for o, c in self.layers}
        self.base = None

    def flat(self):
        return np.concatenate([np.concatenate([self.mean[o], self.var[o]]) for o, _ in self.layers]) \
            if self.layers else np.zeros(0)

    def from_flat(self, a):
        a = np.asarray(a, np.float64)
        i = 0
        for o, c in self.layers:
            self.mean[o] = a[i:i + c].copy()
            self.var[o] = a[i + c:i + 2 * c].copy()
            i += 2 * c
        return self

    def key(self, gamma):
        return (gamma.__array_interface__["data"][0] - self.base) // 8


_RUNNING = None   # the RunningStats batchnorm() consults during a forward, if any


def batchnorm(h, gamma, beta):
    """Batch normalisation over (batch, H, W), eps = 1e-5.  Training mode
    (the default) normalises with the batch mean and biased variance and, when
    running statistics are attached, moves them; eval mode normalises with the
    running statistics.  Returns (z, cache)."""
    if _RUNNING is not None and _RUNNING.eval:
        k = _RUNNING.key(gamma)
        rstd = 1.0 / np.sqrt(_RUNNING.var[k] + BN_EPS)
        xhat = (h - _RUNNING.mean[k].reshape(1, -1, 1, 1)) * rstd.reshape(1, -1, 1, 1)
        return gamma.reshape(1, -1, 1, 1) * xhat + beta.reshape(1, -1, 1, 1), None
    mean = h.mean(axis=(0, 2, 3), keepdims=True)
    var = ((h - mean) ** 2).mean(axis=(0, 2, 3), keepdims=True)
    if _RUNNING is not None:
        k = _RUNNING.key(gamma)
        n = h.shape[0] * h.shape[2] * h.shape[3]
        m = _RUNNING.momentum
        _RUNNING.mean[k] = (1 - m) * _RUNNING.mean[k] + m * mean.ravel()
        _RUNNING.var[k] = (1 - m) * _RUNNING.var[k] + m * var.ravel() * (n / max(n - 1, 1))
    rstd = 1.0 / np.sqrt(var + BN_EPS)
    xhat = (h - mean) * rstd
    z = gamma.reshape(1, -1, 1, 1) * xhat + beta.reshape(1, -1, 1, 1)
    return z, (xhat, rstd)


def batchnorm_backward(dz, gamma, cache):
    xhat, rstd = cache
    m = dz.shape[0] * dz.shape[2] * dz.shape[3]
    dbeta = dz.sum(axis=(0, 2, 3))
    dgamma = (dz * xhat).sum(axis=(0, 2, 3))
    dh = (gamma.reshape(1, -1, 1, 1) * rstd) * (
        dz - dbeta.reshape(1, -1, 1, 1) / m - xhat * dgamma.reshape(1, -1, 1, 1) / m)
    return dh, dgamma, dbeta


def relu(z):
    return np.maximum(z, 0.0)


def relu_backward(da, z):
    """ReLU'(0) = 0."""
    return da * (z > 0)


def maxpool(x, k, stride, pad):
    """Max over k x k windows (padding never wins).  Returns (y, arg) where
    arg is the row-major index in the window of the first maximum."""
    B, C, H, W = x.shape
    P = (H + 2 * pad - k) // stride + 1
    Q = (W + 2 * pad - k) // stride + 1
    xp = np.pad(x, ((0, 0), (0, 0), (pad, pad), (pad, pad)), constant_values=-np.inf)
    wins = np.stack([xp[:, :, r:r + stride * (P - 1) + 1:stride, s:s + stride * (Q - 1) + 1:stride]
                     for r in range(k) for s in range(k)], axis=0)
    arg = np.argmax(wins, axis=0)
    y = np.take_along_axis(wins, arg[None], axis=0)[0]
    return y, arg


def maxpool_backward(dy, arg, in_shape, k, stride, pad):
    B, C, H, W = in_shape
    P, Q = dy.shape[2], dy.shape[3]
    dxp = np.zeros((B, C, H + 2 * pad, W + 2 * pad))
    for r in range(k):
        for s in range(k):
            sel = (arg == r * k + s)
            dxp[:, :, r:r + stride * (P - 1) + 1:stride, s:s + stride * (Q - 1) + 1:stride] += dy * sel
    return dxp[:, :, pad:pad + H, pad:pad + W]


def avgpool(x, k, stride, pad):
    """Average over k x k windows, zero padding counted (linear stand-in for
    maxpool in the linearised network of Prop:equiv)."""
    B, C, H, W = x.shape
    P = (H + 2 * pad - k) // stride + 1
    Q = (W + 2 * pad - k) // stride + 1
    xp = np.pad(x, ((0, 0), (0, 0), (pad, pad), (pad, pad)))
    y = np.zeros((B, C, P, Q))
    for r in range(k):
        for s in range(k):
            y += xp[:, :, r:r + stride * (P - 1) + 1:stride, s:s + stride * (Q - 1) + 1:stride]
    return y / (k * k)


def avgpool_backward(dy, in_shape, k, stride, pad):
    B, C, H, W = in_shape
    P, Q = dy.shape[2], dy.shape[3]
    dxp = np.zeros((B, C, H + 2 * pad, W + 2 * pad))
    for r in range(k):
        for s in range(k):
            dxp[:, :, r:r + stride * (P - 1) + 1:stride, s:s + stride * (Q - 1) + 1:stride] += dy / (k * k)
    return dxp[:, :, pad:pad + H, pad:pad + W]


def softmax_cross_entropy(z, labels):
    """loss = mean_b ( log sum_i exp z[b,i] - z[b,label_b] );
    dz = (softmax(z) - onehot) / B."""
    B = z.shape[0]
    zmax = z.max(axis=1, keepdims=True)
    e = np.exp(z - zmax)
    lse = np.log(e.sum(axis=1, keepdims=True)) + zmax
    loss = float(np.mean(lse[:, 0] - z[np.arange(B), labels]))
    p = e / e.sum(axis=1, keepdims=True)
    p[np.arange(B), labels] -= 1.0
    return loss, p / B


def sgd_step(theta, grad, buf, lr, momentum, weight_decay, nesterov):
    """One SGD step with weight decay and (Nesterov) momentum, dampening 0;
    the momentum buffer starts as the first step's direction.
    Returns (theta_new, buf_new)."""
    d = grad + weight_decay * theta
    buf = d.copy() if buf is None else momentum * buf + d
    step = d + momentum * buf if nesterov else buf
    return theta - lr * step, buf


# =================================================================== layers
# Test hook (never set by the oracle itself): while a `perturbed` context is
# active every convolution output is multiplied by (1 + rel * N(0, 1)) before
# any rounding.  Tests use it to measure how far the oracle's own result moves
# under differences of the size an fp32 accumulation order leaves in a
# convolution, which bounds how far any correct implementation can be from it.
_PERTURB = None


class perturbed:
    """Context manager: conv outputs perturbed by a relative `rel`, normal
    draws from numpy Generator `rng` (see _PERTURB)."""

    def __init__(self, rng, rel):
        self.rng, self.rel = rng, rel

    def __enter__(self):
        global _PERTURB
        _PERTURB = (self.rng, self.rel)
        return self

    def __exit__(self, *a):
        global _PERTURB
        _PERTURB = None


class _Layer:
    """A layer maps (C,H,W) -> (C',H',W'); it lists its parameters as
    (kind, shape) and implements forward / backward on numpy arrays."""

    linear = False
    bf16 = False      # precision model (see the module docstring)
    store_q = True    # this conv's output is stored (rounded) on its own
    stream_q = False  # residual-stream values (block outputs) are stored in bf16

    def _q(self, a):
        return round_bf16(a) if self.bf16 else a

    def _sq(self, a):
        return round_bf16(a) if self.stream_q else a

    def _bn(self, h, g, b):
        if self.linear:
            return h, None
        return batchnorm(h, g, b)

    def _bn_back(self, dz, g, cache):
        if self.linear:
            return dz, np.zeros_like(g), np.zeros_like(g)
        return batchnorm_backward(dz, g, cache)

    def _relu(self, z):
        return z if self.linear else relu(z)

    def _relu_back(self, da, z):
        return da if self.linear else relu_backward(da, z)


class Conv(_Layer):
    def __init__(self, cin, h, w, cout, k, stride):
        self.cin, self.cout, self.k, self.stride, self.pad = cin, cout, k, stride, k // 2
        self.in_shape = (cin, h, w)
        self.out_shape = (cout, (h + 2 * self.pad - k) // stride + 1, (w + 2 * self.pad - k) // stride + 1)
        self.spec = [(KIND_CONV_W, (cout, cin, k, k))]

    def forward(self, x, P):
        xq = self._q(x)
        y = conv2d(xq, self._q(P[0]), self.stride, self.pad)
        if _PERTURB is not None:
            y = y * (1.0 + _PERTURB[1] * _PERTURB[0].standard_normal(y.shape))
        return (self._q(y) if self.store_q else y), xq

    def backward(self, dy, P, cache, need_dx=True):
        # the bf16 model: the output gradient is a contraction operand too
        dx, dw = conv2d_backward(cache, self._q(P[0]), self.stride, self.pad, self._q(dy), need_dx)
        if _PERTURB is not None and dx is not None:
            dx = dx * (1.0 + _PERTURB[1] * _PERTURB[0].standard_normal(dx.shape))
        return dx, [dw]


class ConvBnRelu(_Layer):
    """conv k x k (pad k//2) -> BN -> ReLU (-> 2x2/s2 maxpool)."""

    def __init__(self, cin, h, w, cout, k, stride, pool):
        self.conv = Conv(cin, h, w, cout, k, stride)
        self.pool = pool
        c, ho, wo = self.conv.out_shape
        self.out_shape = (c, ho // 2, wo // 2) if pool else (c, ho, wo)
        self.spec = self.conv.spec + [(KIND_BN_G, (cout,)), (KIND_BN_B, (cout,))]

    def forward(self, x, P):
        h, cc = self.conv.forward(x, P[0:1])
        z, bc = self._bn(h, P[1], P[2])
        a = self._relu(z)
        if self.pool:
            if self.linear:
                out, arg = avgpool(a, 2, 2, 0), None
            else:
                out, arg = maxpool(a, 2, 2, 0)
                out = self._q(out)
        else:
            out, arg = a, None
        return out, (cc, z, bc, a.shape, arg)

    def backward(self, dy, P, cache, need_dx=True):
        cc, z, bc, ashape, arg = cache
        if self.pool:
            da = avgpool_backward(dy, ashape, 2, 2, 0) if self.linear else maxpool_backward(dy, arg, ashape, 2, 2, 0)
        else:
            da = dy
        dz = self._relu_back(da, z)
        dh, dg, db = self._bn_back(dz, P[1], bc)
        dx, (dw,) = self.conv.backward(dh, P[0:1], cc, need_dx)
        return dx, [dw, dg, db]


class Basic(_Layer):
    """Post-activation basic block: out = ReLU(BN2(conv2(ReLU(BN1(conv1 x)))) + x)."""

    def __init__(self, cin, h, w, cout):
        assert cin == cout
        self.c1 = Conv(cin, h, w, cout, 3, 1)
        self.c2 = Conv(cout, h, w, cout, 3, 1)
        self.out_shape = (cout, h, w)
        self.spec = (self.c1.spec + [(KIND_BN_G, (cout,)), (KIND_BN_B, (cout,))]
                     + self.c2.spec + [(KIND_BN_G, (cout,)), (KIND_BN_B, (cout,))])

    def forward(self, x, P):
        h1, k1 = self.c1.forward(x, P[0:1])
        z1, b1 = self._bn(h1, P[1], P[2])
        a1 = self._relu(z1)
        h2, k2 = self.c2.forward(a1, P[3:4])
        z2, b2 = self._bn(h2, P[4], P[5])
        s = z2 + x
        return self._sq(self._relu(s)), (k1, z1, b1, k2, b2, s)

    def backward(self, dout, P, cache, need_dx=True):
        k1, z1, b1, k2, b2, s = cache
        ds = self._relu_back(dout, s)
        dh2, dg2, db2 = self._bn_back(ds, P[4], b2)
        da1, (dw2,) = self.c2.backward(dh2, P[3:4], k2)
        dz1 = self._relu_back(da1, z1)
        dh1, dg1, db1 = self._bn_back(dz1, P[1], b1)
        dx, (dw1,) = self.c1.backward(dh1, P[0:1], k1, need_dx)
        if need_dx:
            dx = dx + ds
        return dx, [dw1, dg1, db1, dw2, dg2, db2]


class Bottleneck(_Layer):
    """Pre-activation bottleneck (He et al. 2016, identity mappings):
        a1 = ReLU(BN1(x)); h1 = conv1x1(a1); h2 = conv3x3_s(ReLU(BN2(h1)));
        h3 = conv1x1(ReLU(BN3(h2))); out = h3 + (x, or conv1x1_s(a1) when the
        shape changes).  The stride sits on the 3x3 conv."""

    def __init__(self, cin, h, w, cout, mid, stride):
        self.cin, self.cout, self.mid, self.stride = cin, cout, mid, stride
        self.proj = (cin != cout) or stride != 1
        self.c1 = Conv(cin, h, w, mid, 1, 1)
        self.c2 = Conv(mid, h, w, mid, 3, stride)
        _, ho, wo = self.c2.out_shape
        self.c3 = Conv(mid, ho, wo, cout, 1, 1)
        self.cp = Conv(cin, h, w, cout, 1, stride) if self.proj else None
        self.c3.store_q = False   # its output goes straight into the residual sum
        self.out_shape = (cout, ho, wo)
        self.spec = ([(KIND_BN_G, (cin,)), (KIND_BN_B, (cin,))] + self.c1.spec
                     + [(KIND_BN_G, (mid,)), (KIND_BN_B, (mid,))] + self.c2.spec
                     + [(KIND_BN_G, (mid,)), (KIND_BN_B, (mid,))] + self.c3.spec
                     + (self.cp.spec if self.proj else []))

    def forward(self, x, P):
        z1, b1 = self._bn(x, P[0], P[1])
        a1 = self._relu(z1)
        h1, k1 = self.c1.forward(a1, P[2:3])
        z2, b2 = self._bn(h1, P[3], P[4])
        a2 = self._relu(z2)
        h2, k2 = self.c2.forward(a2, P[5:6])
        z3, b3 = self._bn(h2, P[6], P[7])
        a3 = self._relu(z3)
        h3, k3 = self.c3.forward(a3, P[8:9])
        if self.proj:
            sc, kp = self.cp.forward(a1, P[9:10])
        else:
            sc, kp = x, None
        return self._sq(h3 + sc), (b1, z1, k1, b2, z2, k2, b3, z3, k3, kp)

    def backward(self, dout, P, cache, need_dx=True):
        b1, z1, k1, b2, z2, k2, b3, z3, k3, kp = cache
        da3, (dw3,) = self.c3.backward(dout, P[8:9], k3)
        dh2, dg3, db3 = self._bn_back(self._relu_back(da3, z3), P[6], b3)
        da2, (dw2,) = self.c2.backward(dh2, P[5:6], k2)
        dh1, dg2, db2 = self._bn_back(self._relu_back(da2, z2), P[3], b2)
        da1, (dw1,) = self.c1.backward(dh1, P[2:3], k1)
        grads_p = []
        if self.proj:
            dap, (dwp,) = self.cp.backward(dout, P[9:10], kp)
            da1 = da1 + dap
            grads_p = [dwp]
        dx, dg1, db1 = self._bn_back(self._relu_back(da1, z1), P[0], b1)
        if not self.proj:
            dx = dx + dout
        return dx, [dg1, db1, dw1, dg2, db2, dw2, dg3, db3, dw3] + grads_p


class CoarseRU(_Layer):
    """Coarse residual unit of Parareal ResNet (Section 4.2): two 3x3 convs
    and a skip connection, the first conv strided when the block downsamples.
    Written in the pre-activation order of the ResNet-1001 units it stands
    in for (the paper does not place the BNs):
        a1 = ReLU(BN1(x)); h1 = conv3x3_s(a1); a2 = ReLU(BN2(h1));
        out = conv3x3(a2) + (x, or conv1x1_s(a1) when the shape changes)."""

    def __init__(self, cin, h, w, cout, stride):
        self.proj = (cin != cout) or stride != 1
        self.c1 = Conv(cin, h, w, cout, 3, stride)
        _, ho, wo = self.c1.out_shape
        self.c2 = Conv(cout, ho, wo, cout, 3, 1)
        self.cp = Conv(cin, h, w, cout, 1, stride) if self.proj else None
        self.c2.store_q = False   # its output goes straight into the residual sum
        self.out_shape = (cout, ho, wo)
        self.spec = ([(KIND_BN_G, (cin,)), (KIND_BN_B, (cin,))] + self.c1.spec
                     + [(KIND_BN_G, (cout,)), (KIND_BN_B, (cout,))] + self.c2.spec
                     + (self.cp.spec if self.proj else []))

    def forward(self, x, P):
        z1, b1 = self._bn(x, P[0], P[1])
        a1 = self._relu(z1)
        h1, k1 = self.c1.forward(a1, P[2:3])
        z2, b2 = self._bn(h1, P[3], P[4])
        a2 = self._relu(z2)
        h2, k2 = self.c2.forward(a2, P[5:6])
        if self.proj:
            sc, kp = self.cp.forward(a1, P[6:7])
        else:
            sc, kp = x, None
        return self._sq(h2 + sc), (b1, z1, k1, b2, z2, k2, kp)

    def backward(self, dout, P, cache, need_dx=True):
        b1, z1, k1, b2, z2, k2, kp = cache
        da2, (dw2,) = self.c2.backward(dout, P[5:6], k2)
        dh1, dg2, db2 = self._bn_back(self._relu_back(da2, z2), P[3], b2)
        da1, (dw1,) = self.c1.backward(dh1, P[2:3], k1)
        grads_p = []
        if self.proj:
            dap, (dwp,) = self.cp.backward(dout, P[6:7], kp)
            da1 = da1 + dap
            grads_p = [dwp]
        dx, dg1, db1 = self._bn_back(self._relu_back(da1, z1), P[0], b1)
        if not self.proj:
            dx = dx + dout
        return dx, [dg1, db1, dw1, dg2, db2, dw2] + grads_p


def make_layer(spec, shape, linear=False, bf16=False, stream_bf16=False):
    c, h, w = shape
    op = spec["op"]
    if op == "conv":
        L = Conv(c, h, w, spec["cout"], spec.get("k", 3), spec.get("stride", 1))
    elif op == "conv_bn_relu":
        L = ConvBnRelu(c, h, w, spec["cout"], spec.get("k", 3), spec.get("stride", 1), spec.get("pool", 0))
    elif op == "basic":
        L = Basic(c, h, w, spec["cout"])
    elif op == "bottleneck":
        L = Bottleneck(c, h, w, spec["cout"], spec["mid"], spec.get("stride", 1))
    elif op == "coarse_ru":
        L = CoarseRU(c, h, w, spec["cout"], spec.get("stride", 1))
    else:
        raise ValueError(op)
    L.linear = linear
    L.bf16 = bf16
    L.stream_q = bf16 and stream_bf16
    for sub in ("conv", "c1", "c2", "c3", "cp"):
        if getattr(L, sub, None) is not None:
            getattr(L, sub).linear = linear
            getattr(L, sub).bf16 = bf16
    return L


class Stack:
    """A sequence of layers with a contiguous slice of the parameter vector."""

    def __init__(self, specs, shape, linear=False, bf16=False, stream_bf16=False):
        self.layers = []
        self.in_shape = tuple(shape)
        for s in specs:
            L = make_layer(s, shape, linear, bf16, stream_bf16)
            self.layers.append(L)
            shape = L.out_shape
        self.out_shape = tuple(shape)
        self.spec = [p for L in self.layers for p in L.spec]

    def _split(self, params):
        out, i = [], 0
        for L in self.layers:
            out.append(params[i:i + len(L.spec)])
            i += len(L.spec)
        return out

    def forward(self, x, params):
        caches = []
        for L, P in zip(self.layers, self._split(params)):
            x, c = L.forward(x, P)
            caches.append(c)
        return x, caches

    def backward(self, dy, params, caches, need_dx=True):
        grads = [None] * len(self.layers)
        Ps = self._split(params)
        for i in range(len(self.layers) - 1, -1, -1):
            dy, grads[i] = self.layers[i].backward(dy, Ps[i], caches[i], need_dx or i > 0)
        return dy, [g for gl in grads for g in gl]


class Preprocess:
    """C^j for j > 1 (Section 4): k 3x3/s2 (pad 1) maxpools taking the input
    image down to the size of X_{j-1}, then a bias-free 1x1 conv to its
    channel count, optionally followed by BN + ReLU."""

    def __init__(self, in_shape, target, post, bf16=False):
        c, h, w = in_shape
        ct, ht, wt = target
        k = int(round(math.log2(h / ht)))
        assert h == ht << k and w == wt << k, (in_shape, target)
        self.k, self.post = k, post
        self.conv = Conv(c, ht, wt, ct, 1, 1)
        self.conv.bf16 = bf16
        self.spec = self.conv.spec + ([(KIND_BN_G, (ct,)), (KIND_BN_B, (ct,))] if post == "bn_relu" else [])
        self.out_shape = tuple(target)

    def forward(self, x, P):
        for _ in range(self.k):
            x, _ = maxpool(x, 3, 2, 1)
        h, kc = self.conv.forward(x, P[0:1])
        if self.post == "bn_relu":
            z, bc = batchnorm(h, P[1], P[2])
            return relu(z), (kc, z, bc)
        return h, (kc, None, None)

    def backward(self, dy, P, cache):
        kc, z, bc = cache
        if self.post == "bn_relu":
            dh, dg, db = batchnorm_backward(relu_backward(dy, z), P[1], bc)
            _, (dw,) = self.conv.backward(dh, P[0:1], kc, need_dx=False)
            return [dw, dg, db]
        _, (dw,) = self.conv.backward(dy, P[0:1], kc, need_dx=False)
        return [dw]


class Head:
    """h_eps: gap_fc (GAP -> FC), bn_relu_gap_fc (BN -> ReLU -> GAP -> FC),
    gap_mlp (GAP -> [FC -> ReLU]* -> FC)."""

    def __init__(self, head, in_shape, classes):
        self.kind = head["kind"]
        c = in_shape[0]
        self.spec = []
        if self.kind == "bn_relu_gap_fc":
            self.spec += [(KIND_BN_G, (c,)), (KIND_BN_B, (c,))]
        widths = [c] + list(head.get("hidden", [])) + [classes]
        if self.kind != "gap_mlp":
            assert len(widths) == 2
        self.widths = widths
        for i in range(len(widths) - 1):
            self.spec += [(KIND_FC_W, (widths[i + 1], widths[i])), (KIND_FC_B, (widths[i + 1],))]

    def forward(self, y, P):
        i = 0
        cache = {}
        if self.kind == "bn_relu_gap_fc":
            z, bc = batchnorm(y, P[0], P[1])
            a = relu(z)
            cache["bn"] = (z, bc)
            i = 2
        else:
            a = y
        cache["shape"] = a.shape
        f = a.mean(axis=(2, 3))
        feats = []
        nfc = len(self.widths) - 1
        for l in range(nfc):
            W, b = P[i + 2 * l], P[i + 2 * l + 1]
            feats.append(f)
            f = f @ W.T + b
            if l < nfc - 1:
                cache.setdefault("pre", []).append(f)
                f = relu(f)
        cache["feats"] = feats
        return f, cache

    def backward(self, dz, P, cache):
        i = 2 if self.kind == "bn_relu_gap_fc" else 0
        nfc = len(self.widths) - 1
        grads = [None] * (2 * nfc)
        g = dz
        for l in range(nfc - 1, -1, -1):
            W = P[i + 2 * l]
            f = cache["feats"][l]
            grads[2 * l] = g.T @ f
            grads[2 * l + 1] = g.sum(axis=0)
            g = g @ W
            if l > 0:
                g = relu_backward(g, cache["pre"][l - 1])
        B, C, H, W_ = cache["shape"]
        da = np.broadcast_to(g[:, :, None, None] / (H * W_), (B, C, H, W_)).copy()
        if self.kind == "bn_relu_gap_fc":
            z, bc = cache["bn"]
            dy, dgam, dbet = batchnorm_backward(relu_backward(da, z), P[0], bc)
            return dy, [dgam, dbet] + grads
        return da, grads


# ================================================================= network
class ParaNet:
    """The parareal network f-bar of eq:barf built from a description."""

    def __init__(self, desc, linear_body=False, precision="fp64"):
        self.desc = desc
        self.mode = desc.get("correction", "residual")
        q = precision == "bf16"
        # the residual stream (block outputs, correction tensors) stored in
        # bf16 as well: a storage policy of the bf16 path
        sq = q and desc.get("residual_stream", "fp32") == "bf16"
        self.sq = (lambda a: round_bf16(a)) if sq else (lambda a: a)
        x_shape = (desc["in_c"], desc["in_h"], desc["in_w"])
        self.stem = Stack(desc["stem"], x_shape, bf16=q)
        segs = desc["segments"]
        assert sum(segs) == len(desc["body"]) and all(s > 0 for s in segs)
        self.N = len(segs)
        self.fine = []
        shape = self.stem.out_shape
        start = 0
        for n in segs:
            st = Stack(desc["body"][start:start + n], shape, linear_body, q, sq)
            self.fine.append(st)
            shape = st.out_shape
            start += n
        # X_0 .. X_N
        self.X = [self.stem.out_shape] + [st.out_shape for st in self.fine]
        self.pre = [None] + [Preprocess(x_shape, self.X[j], desc["cj_post"], q) for j in range(1, self.N)]
        assert len(desc["coarse"]) == self.N - 1
        self.coarse = []
        for j in range(self.N - 1):
            st = Stack(desc["coarse"][j], self.X[j + 1], linear_body, q, sq)
            assert st.out_shape == self.X[j + 2], (j, st.out_shape, self.X[j + 2])
            self.coarse.append(st)
        self.head = Head(desc["head"], self.X[self.N], desc["classes"])
        # eq:barf ordering of the parameter vector
        self.blocks = [("pre", 0, self.stem.spec), ("fine", 0, self.fine[0].spec)]
        for j in range(1, self.N):
            self.blocks += [("pre", j, self.pre[j].spec), ("fine", j, self.fine[j].spec)]
        for j in range(self.N - 1):
            self.blocks.append(("coarse", j, self.coarse[j].spec))
        self.blocks.append(("head", 0, self.head.spec))
        self.spec = [p for _, _, sp in self.blocks for p in sp]

    # ------------------------------------------------------------ params
    def num_params(self):
        return int(sum(np.prod(s) for _, s in self.spec))

    def unflatten(self, theta):
        theta = np.asarray(theta, dtype=np.float64)
        assert theta.size == self.num_params()
        out, i = {}, 0
        for name, j, sp in self.blocks:
            arrs = []
            for _, shape in sp:
                n = int(np.prod(shape))
                arrs.append(theta[i:i + n].reshape(shape))
                i += n
            out[(name, j)] = arrs
        return out

    def flatten(self, grads):
        return np.concatenate([np.asarray(g, dtype=np.float64).ravel()
                               for name, j, _ in self.blocks for g in grads[(name, j)]])

    # ------------------------------------------------------------ forward
    def forward(self, theta, x, labels, running=None):
        """Algorithm 1.  Returns the loss and a state holding every interface
        tensor (x_j, y_j, r_j, rt_j, ytilde), the logits and the caches.  With
        `running` (a RunningStats) every BN moves its running statistics, or
        normalises with them if `running` is in eval mode."""
        global _RUNNING
        theta = np.ascontiguousarray(theta, dtype=np.float64)
        if running is None:
            return self._forward(theta, x, labels)
        running.base = theta.__array_interface__["data"][0]
        _RUNNING = running
        try:
            return self._forward(theta, x, labels)
        finally:
            _RUNNING = None

    def infer(self, theta, x, running):
        """The eval-mode forward: every BN normalises with `running` (a
        RunningStats or its flat layout).  Returns the logits."""
        if not isinstance(running, RunningStats):
            running = RunningStats(self.spec).from_flat(running)
        running.eval = True
        _, st = self.forward(theta, x, np.zeros(np.asarray(x).shape[0], np.int64), running)
        return st["logits"]

    def _forward(self, theta, x, labels):
        P = self.unflatten(theta)
        x = np.asarray(x, dtype=np.float64)
        N = self.N
        st = {"P": P, "labels": np.asarray(labels)}
        # fine subnetworks (independent of each other)
        xs, ys, fc, pc = [], [], [], []
        for j in range(N):
            if j == 0:
                xj, c = self.stem.forward(x, P[("pre", 0)])
            else:
                xj, c = self.pre[j].forward(x, P[("pre", j)])
            pc.append(c)
            yj, c2 = self.fine[j].forward(xj, P[("fine", j)])
            xs.append(xj)
            ys.append(yj)
            fc.append(c2)
        # coarse network, eq:correct
        sq = self.sq  # storage rounding of residual-stream values (identity unless bf16)
        r = [sq(ys[j] - xs[j + 1]) for j in range(N - 1)] + [np.zeros_like(ys[N - 1])]
        rt = [r[0]]
        cc, ccx = [], []
        for j in range(N - 1):
            if self.mode == "residual":
                f, c = self.coarse[j].forward(rt[j], P[("coarse", j)])
                cc.append(c)
                rt.append(sq(r[j + 1] + f))
            else:
                # F^j(x_{j+1}) first: with running statistics the order of the
                # two evaluations matters, and this one does not depend on rt_j
                f0, c0 = self.coarse[j].forward(xs[j + 1], P[("coarse", j)])
                f1, c1 = self.coarse[j].forward(sq(xs[j + 1] + rt[j]), P[("coarse", j)])
                cc.append(c1)
                ccx.append(c0)
                rt.append(sq(r[j + 1] + f1 - f0))
        ytilde = sq(ys[N - 1] + rt[N - 1])
        logits, hc = self.head.forward(ytilde, P[("head", 0)])
        loss, dz = softmax_cross_entropy(logits, st["labels"])
        st.update(x=x, xs=xs, ys=ys, r=r, rt=rt, ytilde=ytilde, logits=logits, loss=loss,
                  dz=dz, fc=fc, pc=pc, cc=cc, ccx=ccx, hc=hc)
        return loss, st

    # ------------------------------------------------------------ backward
    def backward(self, st):
        """Algorithm 2 (Section 3.2).  Returns (flat gradient, D list, dy
        seeds) with D[j] = dL/drt_{j+1} (0-based)."""
        P = st["P"]
        N = self.N
        G = {}
        D = [None] * N
        D[N - 1], G[("head", 0)] = self.head.backward(st["dz"], P[("head", 0)], st["hc"])
        dx_extra = [None] * N
        for j in range(N - 2, -1, -1):
            # F^j maps rt_j -> rt_{j+1} (1-based); here index j is 0-based
            dstate, g1 = self.coarse[j].backward(D[j + 1], P[("coarse", j)], st["cc"][j])
            if self.mode == "residual":
                D[j] = dstate
                G[("coarse", j)] = g1
            else:
                dx0, g0 = self.coarse[j].backward(D[j + 1], P[("coarse", j)], st["ccx"][j])
                D[j] = dstate
                G[("coarse", j)] = [a - b for a, b in zip(g1, g0)]
                dx_extra[j + 1] = dstate - dx0
        # fine subnetworks in parallel: dL/dy_j = D_j, dL/dx_j -= D_{j-1}
        dys = list(D)
        for j in range(N):
            dxj, G[("fine", j)] = self.fine[j].backward(dys[j], P[("fine", j)], st["fc"][j], need_dx=True)
            if j > 0:
                dxj = dxj - D[j - 1]
                if dx_extra[j] is not None:
                    dxj = dxj + dx_extra[j]
            if j == 0:
                _, G[("pre", 0)] = self.stem.backward(dxj, P[("pre", 0)], st["pc"][0], need_dx=False)
            else:
                G[("pre", j)] = self.pre[j].backward(dxj, P[("pre", j)], st["pc"][j])
            st.setdefault("dx", [None] * N)[j] = dxj
        st["D"] = D
        return self.flatten(G)


def train_step(desc, theta, x, labels, lr=0.1, momentum=0.9, weight_decay=5e-4,
               nesterov=True, momentum_buf=None, linear_body=False, precision="fp64", running=None,
               bn_momentum=BN_MOMENTUM):
    """Forward, backward and one SGD step.  Returns a dict with loss, grad,
    theta_new, buf_new, the forward state and running_new, the BN running
    statistics after the step (flat layout of RunningStats; `running` gives
    them before it, default zeros / ones)."""
    net = ParaNet(desc, linear_body, precision)
    rs = RunningStats(net.spec, bn_momentum)
    if running is not None:
        rs.from_flat(running)
    loss, st = net.forward(theta, x, labels, rs)
    grad = net.backward(st)
    theta_new, buf = sgd_step(np.asarray(theta, np.float64), grad, momentum_buf, lr, momentum,
                              weight_decay, nesterov)
    return {"net": net, "loss": loss, "grad": grad, "theta_new": theta_new, "buf_new": buf, "state": st,
            "running_new": rs.flat()}
