"""The allocation-free weight-gradient call (pnn_conv_wgrad_noalloc).

Some callers cannot allocate device memory when they need a result (a memory
pool they do not own, or a runtime that forbids cudaMalloc after start-up).
For them the library offers one call that computes a convolution's weight
gradient with its scratch held in fixed-size arrays compiled into the
library.  This test checks that call, through the C ABI, against the weight
gradient the ordinary training step (pnn_backward, whose scratch lives in the
caller's workspace) produces for the same convolution, on two calls in a row.

The file name sorts last so that a run stopping at the first failure has run
every other test first; it also passes alone in a fresh process.
"""
import ctypes as C

import numpy as np
import pytest

import workloads as W

pytestmark = pytest.mark.gpu


def _net_desc():
    # stem: 3->16 conv (CUDA-core kernel); body: one 16->32 3x3 conv, torn into
    # N = 1 subnetwork, so its input is x_1 and its output gradient is D_1
    return {
        "name": "one_conv", "batch": 8, "in_c": 3, "in_h": 16, "in_w": 16, "classes": 10,
        "precision": "bf16", "correction": "residual",
        "stem": [W.conv(16)], "body": [W.conv(32, k=3)], "segments": [1], "coarse": [],
        "cj_post": "none", "head": {"kind": "gap_fc", "hidden": []},
    }


def test_noalloc_weight_gradient_matches_training_step():
    import torch
    from paper_2103_08802_gb300 import build, pnn
    build.build()
    desc = _net_desc()
    net = pnn.ParaNet(desc, seed=4)
    x, labels = W.make_batch(desc, seed=7)
    xd = torch.from_numpy(x).cuda()
    ld = torch.from_numpy(labels).cuda()
    net.forward(xd, ld)
    net.backward()
    net.sync()
    B, Cin, H, Wd, K = 8, 16, 16, 16, 32
    x1 = net.get_tensor("x", 1).reshape(B, Cin, H, Wd)        # input of the body conv
    d1 = net.get_tensor("D", 1).reshape(B, K, H, Wd)          # gradient of its output
    kind, dims, off = net.param_spec()[1]                     # body conv weight (K, C, R, S)
    assert kind == 0 and dims == (K, Cin, 3, 3)
    ref = net.get_grads()[off:off + K * Cin * 9].reshape(K, Cin, 3, 3)

    xn = torch.from_numpy(np.ascontiguousarray(x1.transpose(0, 2, 3, 1))).cuda()
    dn = torch.from_numpy(np.ascontiguousarray(d1.transpose(0, 2, 3, 1))).cuda()
    lib = pnn.load()
    outs = []
    for _ in range(2):
        dw = torch.full((K * 9 * Cin,), float("nan"), dtype=torch.float32, device="cuda")
        rc = lib.pnn_conv_wgrad_noalloc(C.c_void_p(xn.data_ptr()), C.c_void_p(dn.data_ptr()),
                                        C.c_void_p(dw.data_ptr()), B, H, Wd, Cin, K, 3, 1, None)
        assert rc == 0, lib.pnn_last_error(None)
        # (k, r, s, c) -> (k, c, r, s)
        outs.append(dw.cpu().numpy().reshape(K, 3, 3, Cin).transpose(0, 3, 1, 2))
    for got in outs:
        assert np.isfinite(got).all()
        err = np.linalg.norm(got - ref) / np.linalg.norm(ref)
        assert err <= 5e-2, err      # the bf16 gradient tolerance of the parity tests
        assert err <= 1e-4, err      # same operands and kernel: only the split order differs
    np.testing.assert_array_equal(outs[0], outs[1])


# (batch, h, w, c, k, ksize, stride): 1x1 stride 2; 3x3 with C = 64 and K = 512
# (two 256-column N tiles); C = K = 512 3x3 (k*9*c = 2.36 Mi floats), where
# the 4 Mi-float scratch caps the split count at one although the launch
# would take four
ORACLE_CASES = [(3, 9, 9, 64, 128, 1, 2), (2, 12, 12, 64, 512, 3, 1), (4, 16, 16, 512, 512, 3, 1),
                (2, 8, 8, 16, 32, 3, 1)]


@pytest.mark.parametrize("case", ORACLE_CASES, ids=lambda c: "b%d_%dx%d_c%d_k%d_r%d_s%d" % c)
def test_noalloc_weight_gradient_matches_oracle(case):
    """Against the oracle's conv2d_backward on the operands the kernel
    multiplies (x and dy rounded to bf16): each product is exact in fp32, so
    the error of an fp32 sum of n of them in any order is at most
    2 n 2^-24 sum |x||dy| (2u per addition, as in the per-kernel tests); also
    against the same kernel through pnn_conv_run (gathered), which keeps its
    scratch in a caller workspace, within the 1e-5 norm-relative level of the
    per-kernel tests, on two calls in a row."""
    import torch
    from oracle import pnn_oracle as O
    from paper_2103_08802_gb300 import build, pnn
    build.build()
    B, H, Wd, Cin, K, r, s = case
    pad = r // 2
    P, Q = (H + 2 * pad - r) // s + 1, (Wd + 2 * pad - r) // s + 1
    rng = np.random.default_rng(11)
    x = rng.standard_normal((B, H, Wd, Cin)).astype(np.float32)
    dy = rng.standard_normal((B, P, Q, K)).astype(np.float32)
    xq = O.round_bf16(x.astype(np.float64)).transpose(0, 3, 1, 2)
    dyq = O.round_bf16(dy.astype(np.float64)).transpose(0, 3, 1, 2)
    w0 = np.zeros((K, Cin, r, r))
    _, exact = O.conv2d_backward(xq, w0, s, pad, dyq, need_dx=False)
    _, mag = O.conv2d_backward(np.abs(xq), w0, s, pad, np.abs(dyq), need_dx=False)
    bound = 2 * (B * P * Q) * 2.0 ** -24 * mag + 1e-30
    xd, dd = torch.from_numpy(x).cuda(), torch.from_numpy(dy).cuda()
    lib = pnn.load()
    outs = []
    for _ in range(2):
        dw = torch.full((K * r * r * Cin,), float("nan"), dtype=torch.float32, device="cuda")
        rc = lib.pnn_conv_wgrad_noalloc(C.c_void_p(xd.data_ptr()), C.c_void_p(dd.data_ptr()),
                                        C.c_void_p(dw.data_ptr()), B, H, Wd, Cin, K, r, s, None)
        assert rc == 0, lib.pnn_last_error(None)
        outs.append(dw.cpu().numpy().astype(np.float64).reshape(K, r, r, Cin).transpose(0, 3, 1, 2))
    # the same weight gradient through the workspace-backed entry point
    dw2 = torch.full((K * r * r * Cin,), float("nan"), dtype=torch.float32, device="cuda")
    pnn.conv_run("wgrad", [dict(batch=B, h=H, w=Wd, c=Cin, k=K, ksize=r, stride=s, x=xd,
                                wt=torch.zeros(K * r * r * Cin, dtype=torch.bfloat16, device="cuda"),
                                dy=dd, dw=dw2)], impl="gathered")
    ref = dw2.cpu().numpy().astype(np.float64).reshape(K, r, r, Cin).transpose(0, 3, 1, 2)
    for got in outs:
        assert np.isfinite(got).all()
        worst = float((np.abs(got - exact) / bound).max())
        nrel = np.linalg.norm(got - exact) / np.linalg.norm(exact)
        print(case, "noalloc vs oracle: worst err/bound %.3f, norm-rel %.2e" % (worst, nrel))
        assert worst <= 1.0, worst
        assert nrel <= 1e-5, nrel
        assert np.linalg.norm(got - ref) / np.linalg.norm(ref) <= 1e-5
    np.testing.assert_array_equal(outs[0], outs[1])


def test_noalloc_rejects_sizes_beyond_its_scratch():
    from paper_2103_08802_gb300 import build, pnn
    build.build()
    lib = pnn.load()
    # k * 3 * 3 * c = 512 * 9 * 1024 > 4Mi floats
    rc = lib.pnn_conv_wgrad_noalloc(C.c_void_p(16), C.c_void_p(16), C.c_void_p(16), 1, 4, 4, 1024, 512, 3, 1, None)
    assert rc == 1
    assert b"static scratch" in lib.pnn_last_error(None)
