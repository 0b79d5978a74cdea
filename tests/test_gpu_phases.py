"""Per-phase timing of graph-replayed training steps (pnn_time_phases): the
phases of Tables gradvgg and grad, measured without the launch gaps of an
eager step.  The timed steps are ordinary training steps."""
import numpy as np
import pytest

import workloads as W
from parity import inputs

pytestmark = pytest.mark.gpu


def test_phase_timing_runs_whole_steps():
    import torch
    from paper_2103_08802_gb300 import build, pnn
    build.build()
    d = W.config(0)
    onet, theta, x, labels = inputs(d)
    xd, ld = torch.from_numpy(x).cuda(), torch.from_numpy(labels).cuda()
    a, b = pnn.ParaNet(d), pnn.ParaNet(d)
    a.set_params(theta)
    b.set_params(theta)
    for _ in range(4):
        a.train_step(xd, ld)
    a.sync()
    ms = b.time_phases(xd, ld, 3)
    # an untimed first step and three steps through the phase graphs leave
    # the same parameters and momentum as four steps of the whole-step graph
    np.testing.assert_array_equal(a.get_params(), b.get_params())
    np.testing.assert_array_equal(a.get_momentum(), b.get_momentum())
    assert all(v > 0 for v in ms.values()), ms
    parts = sum(v for k, v in ms.items() if k != "total")
    assert abs(parts - ms["total"]) <= 1e-3 * ms["total"]
    with pytest.raises(pnn.PnnError):
        b.time_phases(xd, ld, 0)
