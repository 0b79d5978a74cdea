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


def test_noalloc_rejects_sizes_beyond_its_scratch():
    from paper_2103_08802_gb300 import build, pnn
    build.build()
    lib = pnn.load()
    # k * 3 * 3 * c = 512 * 9 * 1024 > 4Mi floats
    rc = lib.pnn_conv_wgrad_noalloc(C.c_void_p(16), C.c_void_p(16), C.c_void_p(16), 1, 4, 4, 1024, 512, 3, 1, None)
    assert rc == 1
    assert b"static scratch" in lib.pnn_last_error(None)
