"""Per-kernel parity of the tensor-core convolutions (forward, data gradient,
weight gradient; TMA-fed and thread-gathered) against the oracle's conv2d /
conv2d_backward, one grouped launch at a time through the C ABI
(pnn_conv_run).  A single convolution has no ReLU or maxpool decision
downstream of it, so the bound is fixed by the arithmetic alone.

Bound.  Both operands of every product are bf16 values the test builds on
the host the same way the kernel does (activations: bf16 storage, or the BN
transform act(scale * x + shift) evaluated in fp32 and rounded to bf16; data
and weight gradients: the fp32 gradient rounded to bf16; both round to
nearest even), so each product is exact in fp32 and the oracle's fp64 sum of
the same products is the exact result.  The kernel adds n products in fp32 in
some order; whatever the order, the error of each output is at most
gamma_n * sum_i |a_i b_i| (recursive-summation bound), gamma_n = n*u/(1 - n*u)
with u = 2^-24; the test allows 2u per addition (u for the sum, u for a
tensor-core adder that truncates instead of rounding) and adds the rounding
of the epilogue: the residual add (u), and for a bf16 output the rounding to
bf16 (8 significant bits: at most half an ulp, 2^-8 of the value).  Per
element:

    |got - exact| <= 2 * n * 2^-24 * (|a| conv |b|) + 2^-24 |res| + [2^-8 + 2^-24] |exact|  (bf16 y)

The norm-relative error of fp32 outputs is also held to 1e-5 (the observed
level is ~sqrt(n) * u), far inside the 5e-2 gradient bound of the training
step, and bf16 outputs to 4e-3 max-relative (one bf16 ulp).
"""
import ctypes as C

import numpy as np
import pytest

from oracle import pnn_oracle as O

pytestmark = pytest.mark.gpu
U = 2.0 ** -24


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2103_08802_gb300 import build
    build.build()


def _t(a, dtype):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).to(device="cuda", dtype=dtype)


def _nchw(a_nhwc):
    return np.ascontiguousarray(np.asarray(a_nhwc, np.float64).transpose(0, 3, 1, 2))


def _bf16_round_f32(a):
    """float32 values rounded to bf16 (nearest even), as float64."""
    return O.round_bf16(np.asarray(a, np.float32).astype(np.float64))


def _operand(x, scale, shift, relu):
    """The A operand the kernel forms from a stored activation: act(scale*x+shift)
    evaluated in fp32 (a fused multiply-add: the fp64 product of two fp32
    values is exact, one rounding to fp32), then bf16."""
    if scale is None:
        return _bf16_round_f32(x)
    v = (scale.astype(np.float64) * x.astype(np.float64) + shift.astype(np.float64)).astype(np.float32)
    if relu:
        v = np.maximum(v, np.float32(0))
    return _bf16_round_f32(v)


def _pq(g):
    pad = g["ksize"] // 2
    return ((g["h"] + 2 * pad - g["ksize"]) // g["stride"] + 1, (g["w"] + 2 * pad - g["ksize"]) // g["stride"] + 1)


class Case:
    """Host data of one instance: geometry, bf16-representable operands,
    optional BN transform of the input."""

    def __init__(self, seed, batch, h, w, c, k, ksize, stride, bn=False, relu=True, x_fp32=False):
        rng = np.random.default_rng(seed)
        self.g = dict(batch=batch, h=h, w=w, c=c, k=k, ksize=ksize, stride=stride)
        self.P, self.Q = _pq(self.g)
        self.pad = ksize // 2
        self.x = rng.standard_normal((batch, h, w, c)).astype(np.float32)
        if not x_fp32:
            self.x = _bf16_round_f32(self.x).astype(np.float32)
        self.x_fp32 = x_fp32
        self.wt = _bf16_round_f32(rng.standard_normal((k, ksize, ksize, c)) * np.sqrt(2.0 / (c * ksize * ksize)))
        self.scale = self.shift = None
        self.relu = relu
        if bn:
            self.scale = (0.5 + rng.random(c)).astype(np.float32)
            self.shift = (0.3 * rng.standard_normal(c)).astype(np.float32)
        self.a = _operand(self.x, self.scale, self.shift, relu)          # NHWC, exact bf16 values
        self.dy = rng.standard_normal((batch, self.P, self.Q, k)).astype(np.float32)
        self.dyq = _bf16_round_f32(self.dy)

    def w_kcrs(self):
        return np.ascontiguousarray(self.wt.transpose(0, 3, 1, 2))

    def dev(self):
        import torch
        d = dict(self.g)
        d["x"] = _t(self.x, torch.float32 if self.x_fp32 else torch.bfloat16)
        d["wt"] = _t(self.wt.astype(np.float32), torch.bfloat16)
        if self.scale is not None:
            d["bn_scale"] = _t(self.scale, torch.float32)
            d["bn_shift"] = _t(self.shift, torch.float32)
            d["relu"] = int(self.relu)
        return d


def _check(name, got, exact, absbound, extra_rel, norm_tol, maxrel_tol=None):
    """|got - exact| <= absbound * (1 + extra_rel) + extra_rel * |exact|: the
    final rounding (relative extra_rel) applies to the computed value, which
    is within absbound of exact."""
    got = np.asarray(got, np.float64)
    err = np.abs(got - exact)
    bound = absbound * (1 + extra_rel) + extra_rel * np.abs(exact) + 1e-30
    worst = float((err / bound).max())
    nrel = float(np.linalg.norm(got - exact) / max(np.linalg.norm(exact), 1e-30))
    mrel = float(err.max() / max(np.abs(exact).max(), 1e-30))
    print(f"{name}: worst err/bound {worst:.3f}  norm-rel {nrel:.2e} (<= {norm_tol:.0e})  max-rel {mrel:.2e}")
    assert np.isfinite(got).all(), name
    assert worst <= 1.0, (name, worst)
    assert nrel <= norm_tol, (name, nrel)
    if maxrel_tol is not None:
        assert mrel <= maxrel_tol, (name, mrel)


# ------------------------------------------------------------------ cases
# (name, constructor args); every ResNet-1001 / VGG-16 conv shape family:
# 1x1 and 3x3, stride 1 and 2, C in {8, 16, 64, 256, 512}, K up to 512, M not a
# multiple of the 128-row tile, N not a multiple of 16 (K = 24).
CASES = {
    "1x1_c64_k16_bn": dict(batch=2, h=15, w=15, c=64, k=16, ksize=1, stride=1, bn=True),
    "1x1_c16_k64_bn": dict(batch=2, h=15, w=15, c=16, k=64, ksize=1, stride=1, bn=True),
    "3x3_c16_k16_bn": dict(batch=2, h=13, w=11, c=16, k=16, ksize=3, stride=1, bn=True),
    "3x3_c64_k128_s2": dict(batch=2, h=17, w=17, c=64, k=128, ksize=3, stride=2, bn=True),
    "1x1_c64_k128_s2": dict(batch=3, h=9, w=9, c=64, k=128, ksize=1, stride=2, bn=True),
    "3x3_c256_k512": dict(batch=3, h=6, w=5, c=256, k=512, ksize=3, stride=1, bn=True),
    "1x1_c512_k256_fp32x": dict(batch=2, h=7, w=7, c=512, k=256, ksize=1, stride=1, bn=True, x_fp32=True),
    "3x3_c8_k24_raw": dict(batch=2, h=9, w=10, c=8, k=24, ksize=3, stride=1, bn=False),
    "3x3_c64_k64_norelu": dict(batch=2, h=8, w=8, c=64, k=64, ksize=3, stride=1, bn=True, relu=False),
    # halo tiles (128 | h*w, w <= 63): one tile per image, a wide image, a
    # narrow one, A sources of 16, 32 and 48 channels (forward c, data
    # gradient k); 64 channels at w = 16 exceed two stages of shared memory
    # and keep one box per tap
    "3x3_c32_k16_halo_hw128": dict(batch=3, h=16, w=8, c=32, k=16, ksize=3, stride=1, bn=True),
    "3x3_c16_k32_halo_w32": dict(batch=2, h=8, w=32, c=16, k=32, ksize=3, stride=1, bn=True),
    "3x3_c48_k16_halo_w4": dict(batch=2, h=32, w=4, c=48, k=16, ksize=3, stride=1, bn=False),
    "3x3_c64_k64_w16_tap": dict(batch=2, h=16, w=16, c=64, k=64, ksize=3, stride=1, bn=True),
}
# grouped: instances of different stages in one launch, as the N subnetworks'
# same layer in a step (stage 1 / 2 / 3 bottleneck 3x3 and 1x1 convs)
GROUPS = {
    "group_3x3": [dict(batch=2, h=16, w=16, c=16, k=16, ksize=3, stride=1, bn=True),
                  dict(batch=2, h=8, w=8, c=32, k=32, ksize=3, stride=1, bn=True),
                  dict(batch=2, h=4, w=4, c=64, k=64, ksize=3, stride=1, bn=True)],
    # halo instances (16x16, 16x8) beside per-tap ones (8x8: 128 does not divide h*w)
    "group_3x3_halo": [dict(batch=2, h=16, w=16, c=16, k=16, ksize=3, stride=1, bn=True),
                       dict(batch=2, h=16, w=8, c=32, k=32, ksize=3, stride=1, bn=True),
                       dict(batch=3, h=8, w=8, c=64, k=64, ksize=3, stride=1, bn=True)],
    "group_1x1_expand": [dict(batch=2, h=16, w=16, c=16, k=64, ksize=1, stride=1, bn=True),
                         dict(batch=2, h=8, w=8, c=32, k=128, ksize=1, stride=1, bn=True),
                         dict(batch=2, h=4, w=4, c=64, k=256, ksize=1, stride=1, bn=True)],
}


def _cases(name, seed=0):
    specs = GROUPS[name] if name in GROUPS else [CASES[name]]
    return [Case(seed + 17 * i, **s) for i, s in enumerate(specs)]


def _halo(mode, s):
    """Whether the TMA-fed kernel takes halo tiles for this instance."""
    ch = s["c"] if mode == "forward" else s["k"]
    return (mode != "wgrad" and s["ksize"] == 3 and s["stride"] == 1 and (s["h"] * s["w"]) % 128 == 0
            and 128 + 2 * s["w"] + 2 <= 256 and ch % 16 == 0 and ch <= 64)


def _tma_ok(mode, s):
    pad = s["ksize"] // 2
    geom = s["stride"] == 1 and ((s["ksize"] == 1 and pad == 0) or (s["ksize"] == 3 and pad == 1))
    ch = s["c"] if mode in ("forward", "wgrad") else s["k"]
    ok = geom and ch % 8 == 0 and (64 % ch == 0 if ch <= 64 else ch % 64 == 0)
    if mode == "wgrad":
        c = s["c"]
        ok = geom and (c <= 64 and 64 % c == 0 or c % 128 == 0 and c <= 512) and s["k"] <= 128
        halo = pad * s["w"] + pad
        ok = ok and 64 + 2 * halo <= 256
    return ok


def _params(mode):
    out = []
    for name in list(CASES) + list(GROUPS):
        specs = GROUPS[name] if name in GROUPS else [CASES[name]]
        impls = ["gathered"]
        if all(_tma_ok(mode, s) or _halo(mode, s) for s in specs):
            impls.append("tma")
            if any(_halo(mode, s) for s in specs) and all(_tma_ok(mode, s) for s in specs):
                impls.append("tma_tap")  # the same launch with one box per tap
        out += [(name, impl) for impl in impls]
    return out


# ------------------------------------------------------------------ forward
@pytest.mark.parametrize("name,impl", _params("forward"))
def test_conv_forward(name, impl):
    import torch
    from paper_2103_08802_gb300 import pnn
    cases = _cases(name, seed=1)
    insts, outs = [], []
    for i, cs in enumerate(cases):
        d = cs.dev()
        M = cs.g["batch"] * cs.P * cs.Q
        rng = np.random.default_rng(100 + i)
        res = rng.standard_normal((cs.g["batch"], cs.P, cs.Q, cs.g["k"])).astype(np.float32)
        # three epilogues in turn: bf16 y; fp32 y + fp32 residual; bf16 y +
        # bf16 residual (the residual stream's two storage precisions)
        kind = (i + len(name)) % 3
        ybf = kind != 1
        d["y_mean"] = torch.full((cs.g["k"],), float("nan"), device="cuda")
        d["y_rstd"] = torch.full((cs.g["k"],), float("nan"), device="cuda")
        if kind == 2:
            res = _bf16_round_f32(res).astype(np.float32)
        d["y"] = torch.full((M, cs.g["k"]), float("nan"), device="cuda",
                            dtype=torch.bfloat16 if ybf else torch.float32)
        if kind:
            d["res"] = _t(res, torch.float32 if kind == 1 else torch.bfloat16)
        outs.append((cs, ybf, res if kind else None))
        insts.append(d)
    pnn.conv_run("forward", insts, impl=impl)
    torch.cuda.synchronize()
    for (cs, ybf, res), d in zip(outs, insts):
        n = cs.g["ksize"] ** 2 * cs.g["c"]
        a, w = _nchw(cs.a), cs.w_kcrs()
        exact = O.conv2d(a, w, cs.g["stride"], cs.pad)
        mag = O.conv2d(np.abs(a), np.abs(w), cs.g["stride"], cs.pad)
        got = _nchw(d["y"].float().cpu().numpy().reshape(cs.g["batch"], cs.P, cs.Q, cs.g["k"]))
        absb = 2 * n * U * mag
        if res is not None:
            r = _nchw(res)
            exact = exact + r
            absb = absb + U * np.abs(r)
        if ybf:
            _check(f"{name}/{impl} y(bf16){'+res' if res is not None else ''}", got, exact, absb, 2.0 ** -8 + U,
                   4e-3, 8e-3)
        else:
            _check(f"{name}/{impl} y(fp32)+res", got, exact, absb, U, 1e-5)
        # batch statistics of the stored y (what the next BN normalises with)
        y = got
        mean = y.mean(axis=(0, 2, 3))
        var = ((y - mean.reshape(1, -1, 1, 1)) ** 2).mean(axis=(0, 2, 3))
        rstd = 1.0 / np.sqrt(var + O.BN_EPS)
        gm, gr = d["y_mean"].cpu().numpy().astype(np.float64), d["y_rstd"].cpu().numpy().astype(np.float64)
        scale = np.sqrt((y ** 2).mean(axis=(0, 2, 3)))  # |mean| <= rms: the mean's natural scale
        assert np.all(np.abs(gm - mean) <= 1e-5 * scale + 1e-30), (np.abs(gm - mean) / scale).max()
        assert np.all(np.abs(gr - rstd) <= 1e-4 * rstd), (np.abs(gr - rstd) / rstd).max()


# ------------------------------------------------------------------ data gradient
@pytest.mark.parametrize("name,impl", _params("dgrad"))
def test_conv_data_gradient(name, impl):
    import torch
    from paper_2103_08802_gb300 import pnn
    cases = _cases(name, seed=2)
    insts, meta = [], []
    for i, cs in enumerate(cases):
        d = cs.dev()
        M = cs.g["batch"] * cs.g["h"] * cs.g["w"]
        d["dy"] = _t(cs.dy, torch.float32)
        acc = i == 1  # the second instance of a group accumulates into dx
        rng = np.random.default_rng(200 + i)
        dx0 = rng.standard_normal((M, cs.g["c"])).astype(np.float32) if acc else None
        d["dx"] = _t(dx0, torch.float32) if acc else torch.full((M, cs.g["c"]), float("nan"), device="cuda")
        d["accumulate"] = int(acc)
        bn = cs.scale is not None and not acc
        stats = None
        if bn:
            # the BN whose input is x: its forward statistics (of x) and the
            # scale/shift already in d; the sums of g = dx * relu'(BN x)
            xf = cs.x.astype(np.float64).reshape(-1, cs.g["c"])
            mean = xf.mean(0).astype(np.float32)
            rstd = (1.0 / np.sqrt(xf.var(0) + O.BN_EPS)).astype(np.float32)
            d["bn_mean"], d["bn_rstd"] = _t(mean, torch.float32), _t(rstd, torch.float32)
            d["dgamma"] = torch.full((cs.g["c"],), float("nan"), device="cuda")
            d["dbeta"] = torch.full((cs.g["c"],), float("nan"), device="cuda")
            stats = (mean, rstd)
        else:
            d.pop("x", None)
            d.pop("bn_scale", None)
            d.pop("bn_shift", None)
        insts.append(d)
        meta.append((cs, dx0, stats))
    pnn.conv_run("dgrad", insts, impl=impl)
    torch.cuda.synchronize()
    for (cs, dx0, stats), d in zip(meta, insts):
        n = cs.g["ksize"] ** 2 * cs.g["k"]
        a, w = _nchw(cs.a), cs.w_kcrs()
        dyq = _nchw(cs.dyq)
        exact, _ = O.conv2d_backward(a, w, cs.g["stride"], cs.pad, dyq)
        mag, _ = O.conv2d_backward(np.abs(a), np.abs(w), cs.g["stride"], cs.pad, np.abs(dyq))
        got = _nchw(d["dx"].cpu().numpy().reshape(cs.g["batch"], cs.g["h"], cs.g["w"], cs.g["c"]))
        absb = 2 * n * U * mag
        if dx0 is not None:
            base = _nchw(dx0.reshape(cs.g["batch"], cs.g["h"], cs.g["w"], cs.g["c"]))
            exact = exact + base
            absb = absb + U * np.abs(base)
        _check(f"{name}/{impl} dx{' (accumulate)' if dx0 is not None else ''}", got, exact, absb, U, 1e-5)
        if stats is not None:
            mean, rstd = stats
            z = (cs.scale.astype(np.float64) * cs.x.astype(np.float64) + cs.shift.astype(np.float64)).astype(np.float32)
            mask = _nchw(z > 0) if cs.relu else 1.0
            xhat = _nchw((cs.x.astype(np.float64) - mean) * rstd)
            g = exact * mask
            db, dg = g.sum(axis=(0, 2, 3)), (g * xhat).sum(axis=(0, 2, 3))
            gotb, gotg = d["dbeta"].cpu().numpy(), d["dgamma"].cpu().numpy()
            rows = g.shape[0] * g.shape[2] * g.shape[3]
            # each term carries the dx error above (norm-relative <= 1e-5) and
            # fp32 rounding of the product; the sums add ~rows terms
            sb = np.abs(g).sum(axis=(0, 2, 3))
            sg = np.abs(g * xhat).sum(axis=(0, 2, 3))
            tol_b = (2 * rows * U + 1e-5) * sb
            tol_g = (2 * rows * U + 1e-5) * sg
            print(f"{name}/{impl} BN sums: dbeta max err/bound {(np.abs(gotb - db) / tol_b).max():.3f}, "
                  f"dgamma {(np.abs(gotg - dg) / tol_g).max():.3f}")
            assert np.all(np.abs(gotb - db) <= tol_b)
            assert np.all(np.abs(gotg - dg) <= tol_g)


# ------------------------------------------------------------------ weight gradient
@pytest.mark.parametrize("name,impl", _params("wgrad"))
def test_conv_weight_gradient(name, impl):
    import torch
    from paper_2103_08802_gb300 import pnn
    cases = _cases(name, seed=3)
    insts = []
    for cs in cases:
        d = cs.dev()
        d["dy"] = _t(cs.dy, torch.float32)
        d["dw"] = torch.full((cs.g["k"] * cs.g["ksize"] ** 2 * cs.g["c"],), float("nan"), device="cuda")
        insts.append(d)
    pnn.conv_run("wgrad", insts, impl=impl)
    torch.cuda.synchronize()
    for cs, d in zip(cases, insts):
        n = cs.g["batch"] * cs.P * cs.Q
        a, w = _nchw(cs.a), cs.w_kcrs()
        dyq = _nchw(cs.dyq)
        _, exact = O.conv2d_backward(a, w, cs.g["stride"], cs.pad, dyq, need_dx=False)
        _, mag = O.conv2d_backward(np.abs(a), w, cs.g["stride"], cs.pad, np.abs(dyq), need_dx=False)
        k, r, c = cs.g["k"], cs.g["ksize"], cs.g["c"]
        got = d["dw"].cpu().numpy().astype(np.float64).reshape(k, r, r, c).transpose(0, 3, 1, 2)
        _check(f"{name}/{impl} dw", got, exact, 2 * n * U * mag, U, 1e-5)


def test_tma_kernels_ran():
    """The TMA-fed variants are exercised above for every mode."""
    assert any(i == "tma" for _, i in _params("forward"))
    assert any(i == "tma" for _, i in _params("dgrad"))
    assert any(i == "tma" for _, i in _params("wgrad"))
