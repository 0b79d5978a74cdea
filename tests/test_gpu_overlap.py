"""Coarse/fine overlap (opts.overlap): the last subnetwork's backward needs
only D_N (Algorithm 2), so it runs on a second stream beside the coarse
chain's backward, and the chain's term of dL/dx_N is added after both.  (The
correction's sums then keep launches of their own; the sequential schedule
they are compared with is planned the same way, fuse_correction=False.)  The
step computes the same quantities as the sequential schedule: everything but
dL/dx_N is accumulated in the same order and agrees bit for bit; dL/dx_N
sums the same two terms in the other order, so only the gradients of C^N
(which read it) may differ, by fp32 rounding."""
import numpy as np
import pytest

import workloads as W
from parity import compare, inputs, norm_rel, run_gpu, run_oracle

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2103_08802_gb300 import build
    build.build()


def test_overlap_tiny_fp32_matches_oracle():
    desc = W.config(0)
    onet, theta, x, labels = inputs(desc)
    g = run_gpu(desc, theta, x, labels, overlap=32)
    o = run_oracle(desc, theta, x, labels)
    report, fails = compare(desc, g, o)
    assert not fails, fails


@pytest.mark.parametrize("name", ["cfg4_reduced", "cfg2_reduced", "paper_n6"])
def test_overlap_matches_sequential(name):
    if name == "cfg4_reduced":
        desc = W.parareal_resnet1001(n_seg=8, batch=256, classes=200, hw=64, per_stage=3,
                                     segments=[2, 1, 1, 1, 1, 1, 1, 1])
    elif name == "cfg2_reduced":
        desc = W.parareal_resnet1001(n_seg=4, batch=128, classes=10, per_stage=2, segments=[2, 1, 2, 1])
    else:
        desc = W.paper_parareal_resnet(6, batch=128, per_stage=2)
    onet, theta, x, labels = inputs(desc)
    a = run_gpu(desc, theta, x, labels, fuse_correction=False)
    b = run_gpu(desc, theta, x, labels, overlap=32)
    for k in a:
        if k in ("net", "onet", "grad", "theta_new", "momentum"):
            continue
        np.testing.assert_array_equal(np.asarray(a[k]), np.asarray(b[k]), err_msg=k)
    # parameter gradients: bit-identical except C^N's
    N = len(desc["segments"])
    off = 0
    for name_, j, sp in onet.blocks:
        n = sum(int(np.prod(s)) for _, s in sp)
        if name_ == "pre" and j == N - 1:
            lo, hi = off, off + n
        off += n
    ga, gb = a["grad"], b["grad"]
    mask = np.ones(ga.size, bool)
    mask[lo:hi] = False
    np.testing.assert_array_equal(ga[mask], gb[mask])
    assert norm_rel(gb[lo:hi], ga[lo:hi]) <= 1e-5
