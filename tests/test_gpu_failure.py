"""Failure detection on the GPU without a fault.

Every device wait of the library's kernels is bounded: when a wait runs
out, the kernel records a status word, releases what it holds and returns,
and the host reports PNN_ETIMEOUT.  pnn_selftest_wait_timeout makes one such
wait run out on purpose (an mbarrier phase that can never complete, waited
on with the kernels' bounded wait and a short limit).  The test checks the
reported status and the elapsed time, and then that the same CUDA context
still trains: a strict-tolerance step of the tiny network against the oracle.
"""
import time

import numpy as np
import pytest

import workloads as W
from parity import TOL, compare, inputs, run_gpu, run_oracle

pytestmark = pytest.mark.gpu

PNN_ETIMEOUT = 5


def test_expired_device_wait_is_reported_and_the_context_stays_usable():
    from paper_2103_08802_gb300 import build, pnn
    build.build()
    lib = pnn.load()
    t0 = time.perf_counter()
    rc = lib.pnn_selftest_wait_timeout(100_000_000, None)   # 0.1 s limit
    dt = time.perf_counter() - t0
    assert rc == PNN_ETIMEOUT, lib.pnn_last_error(None)
    assert b"gave up" in lib.pnn_last_error(None)
    assert 0.09 <= dt < 10.0, dt
    # the context is intact: a full training step still matches the oracle at fp32 check-mode bounds
    desc = W.config(0)
    onet, theta, x, labels = inputs(desc)
    g = run_gpu(desc, theta, x, labels)
    o = run_oracle(desc, theta, x, labels)
    report, fails = compare(desc, g, o)
    assert not fails, fails
    assert np.isfinite(g["loss"])
