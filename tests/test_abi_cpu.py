"""Host-side checks of the C-ABI library (no GPU needed): it loads, exports
every function include/pnn.h declares, plans the five workloads with the
parameter table of the oracle (eq:barf order and shapes) and rejects bad
descriptions with PNN_EINVAL."""
import copy
import ctypes as C
import os
import re

import numpy as np
import pytest

import workloads as W
from oracle import pnn_oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def pnn():
    from paper_2103_08802_gb300 import build, pnn as P
    build.build()
    P.load()
    return P


def declared_functions():
    src = open(os.path.join(ROOT, "include", "pnn.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(pnn_[a-z_0-9]+)\s*\(", src)))


def test_library_exports_every_declared_symbol(pnn):
    lib = C.CDLL(pnn.LIB_PATH)
    names = declared_functions()
    assert len(names) >= 20
    for n in names:
        assert hasattr(lib, n), n


PAPER_NETS = {
    "paper_resnet_n3": lambda: W.paper_parareal_resnet(3),
    "paper_resnet_n18": lambda: W.paper_parareal_resnet(18),
    "paper_resnet_n24_delta": lambda: W.paper_parareal_resnet(24, correction="delta"),
    "paper_vgg16_4": lambda: W.parareal_vgg16(coarse="paper"),
}


@pytest.mark.parametrize("idx", list(range(5)) + list(PAPER_NETS))
def test_plan_matches_oracle_parameter_table(pnn, idx):
    d = W.config(idx) if isinstance(idx, int) else PAPER_NETS[idx]()
    net = pnn.ParaNet(d, bind=False)
    spec = net.param_spec()
    ospec = O.ParaNet(d).spec
    assert len(spec) == len(ospec)
    off = 0
    for (kind, dims, o), (okind, shape) in zip(spec, ospec):
        assert kind == okind
        assert tuple(dims[:len(shape)]) == tuple(shape) and all(x == 1 for x in dims[len(shape):])
        assert o == off
        off += int(np.prod(shape))
    assert net.num_params == off
    assert net.workspace_bytes > 0


@pytest.mark.parametrize("mode", ["residual", "delta"])
def test_plan_delta_and_n1(pnn, mode):
    d = W.config(2)
    d["correction"] = mode
    net = pnn.ParaNet(d, bind=False)
    assert net.num_params == O.ParaNet(d).num_params()
    d1 = copy.deepcopy(d)
    d1["segments"] = [333]
    d1["coarse"] = []
    assert pnn.ParaNet(d1, bind=False).num_params == O.ParaNet(d1).num_params() == 10_327_706


def test_bad_descriptions_are_rejected(pnn):
    base = W.config(0)
    bad = []
    d = copy.deepcopy(base); d["segments"] = [1, 2]; bad.append(d)            # does not sum to body
    d = copy.deepcopy(base); d["batch"] = 0; bad.append(d)
    d = copy.deepcopy(base); d["coarse"] = [[W.conv_bn_relu(32)]]; bad.append(d)  # F^1 output is not X_2
    d = copy.deepcopy(base); d["body"][0] = W.basic(16) | {"cout": 0}; bad.append(d)
    d = copy.deepcopy(base); d["stem"] = [W.conv(16, k=5)]; bad.append(d)
    for d in bad:
        with pytest.raises(pnn.PnnError) as e:
            pnn.ParaNet(d, bind=False)
        assert e.value.status == 1


def test_calls_without_workspace_fail_cleanly(pnn):
    net = pnn.ParaNet(W.config(0), bind=False)
    lib = net.lib
    assert lib.pnn_backward(net.h) == 7          # PNN_ENOTBOUND
    assert lib.pnn_sgd_step(net.h, 0.1) == 7
    assert lib.pnn_backward(None) == 1            # null handle
    assert lib.pnn_status_string(5) == b"device wait timed out"


def test_wait_selftest_rejects_bad_limits(pnn):
    lib = pnn.load()
    assert lib.pnn_selftest_wait_timeout(0, None) == 1          # PNN_EINVAL, before any CUDA call
    assert lib.pnn_selftest_wait_timeout(-5, None) == 1
    assert b"limit_ns" in lib.pnn_last_error(None)


@pytest.mark.parametrize("idx", range(5))
def test_running_stats_layout_and_inference_plan(pnn, idx):
    """The library's running-statistics block has the oracle's layout size
    (2 C floats per BN layer), and an inference plan of the same network --
    forward only, activation buffers handed on by liveness -- needs a fraction
    of the training workspace."""
    import ctypes as C
    d = W.config(idx)
    train = pnn.ParaNet(d, bind=False)
    infer = pnn.ParaNet(d, bind=False, inference=True)
    n = C.c_size_t()
    assert train.lib.pnn_running_stats_size(train.h, C.byref(n)) == 0
    assert n.value == O.RunningStats(O.ParaNet(d).spec).flat().size
    assert infer.lib.pnn_running_stats_size(infer.h, C.byref(n)) == 0
    assert n.value == O.RunningStats(O.ParaNet(d).spec).flat().size
    assert infer.num_params == train.num_params
    assert infer.workspace_bytes < train.workspace_bytes / 2


def test_overlap_option_plans_the_last_subnetwork_apart(pnn):
    """opts.overlap moves the last subnetwork's backward out of the grouped
    launches (more backward launches) in the residual form with N > 1, and
    leaves the delta form and N = 1 as they are.  It also keeps the
    correction's sums as launches of their own (r_j, rt_{j+1} and ytilde:
    (N-1) + (N-2) + 1 of them) instead of folding them into conv epilogues."""
    import ctypes as C

    def counts(d, **kw):
        net = pnn.ParaNet(d, bind=False, **kw)
        c = (C.c_int32 * 3)()
        assert net.lib.pnn_launch_counts(net.h, c) == 0
        return list(c)

    d = W.config(2)
    N = len(d["segments"])
    seq, ov = counts(d), counts(d, overlap=32)
    assert ov[0] == seq[0] + (N - 1) + (N - 2) + 1 and ov[1] > seq[1] and ov[2] == seq[2]
    dd = W.config(2)
    dd["correction"] = "delta"
    assert counts(dd, overlap=32) == counts(dd)
    d1 = W.config(0)
    d1["segments"] = [4]
    d1["coarse"] = []
    assert counts(d1, overlap=32) == counts(d1)


def test_single_conv_call_checks_its_arguments(pnn):
    """pnn_conv_workspace_bytes / pnn_conv_run validate geometry and the kernel
    choice on the host (no device memory is touched): the TMA-fed kernels take
    stride 1 only, channel counts must be multiples of 8."""
    lib = pnn.load()
    fake = 256  # never dereferenced: the checks run before any device work

    def args(**kw):
        a = pnn.ConvArgs()
        g = dict(batch=2, h=8, w=8, c=16, k=32, ksize=3, stride=1)
        g.update(kw)
        for key, v in g.items():
            setattr(a, key, v)
        a.x = a.wt = a.y = a.dy = a.dx = a.dw = fake
        return (pnn.ConvArgs * 1)(a)

    nb = C.c_size_t()
    for mode in range(3):
        assert lib.pnn_conv_workspace_bytes(mode, 0, 1, args(), C.byref(nb)) == 0 and nb.value > 0
        assert lib.pnn_conv_workspace_bytes(mode, 1, 1, args(stride=2), C.byref(nb)) == 1   # TMA: stride 1 only
        assert lib.pnn_conv_workspace_bytes(mode, 2, 1, args(stride=2), C.byref(nb)) == 0
        assert lib.pnn_conv_workspace_bytes(mode, 0, 1, args(c=12), C.byref(nb)) == 1       # c % 8
        assert lib.pnn_conv_workspace_bytes(mode, 0, 1, args(ksize=5), C.byref(nb)) == 1
    # too small a workspace is refused before any launch
    assert lib.pnn_conv_run(0, 0, 1, args(), C.c_void_p(256), 256, None) == 2


def test_halo_tiles_kernel_choice(pnn):
    """The TMA-fed 3x3 forward / data gradient take halo tiles (one box per
    128-pixel tile) where 128 divides h*w, w <= 63 and the A source has 16 |
    channels <= 64, and two pipeline stages fit: impl 1 accepts such a
    source even when its channel count rules out one box per tap (48), impl
    3 (one box per tap) refuses it; the workspace holds a fourth tensor map
    per instance either way."""
    lib = pnn.load()
    fake = 256

    def args(**kw):
        a = pnn.ConvArgs()
        g = dict(batch=2, h=32, w=4, c=48, k=16, ksize=3, stride=1)
        g.update(kw)
        for key, v in g.items():
            setattr(a, key, v)
        a.x = a.wt = a.y = a.dy = a.dx = a.dw = fake
        return (pnn.ConvArgs * 1)(a)

    nb = C.c_size_t()
    # forward, A source c = 48: halo tiles only
    assert lib.pnn_conv_workspace_bytes(0, 1, 1, args(), C.byref(nb)) == 0
    assert lib.pnn_conv_workspace_bytes(0, 3, 1, args(), C.byref(nb)) == 1
    # 8x8 images: 128 does not divide h*w, no halo tiles, and 48 channels take no per-tap box
    assert lib.pnn_conv_workspace_bytes(0, 1, 1, args(h=8, w=8), C.byref(nb)) == 1
    # a 64-wide image needs a box of 128 + 2*64 + 2 > 256 rows
    assert lib.pnn_conv_workspace_bytes(0, 1, 1, args(h=8, w=64), C.byref(nb)) == 1
    # 16 channels: both layouts
    for impl in (1, 3):
        assert lib.pnn_conv_workspace_bytes(0, impl, 1, args(c=16), C.byref(nb)) == 0
    # data gradient: the A source is dy (k channels)
    assert lib.pnn_conv_workspace_bytes(1, 1, 1, args(c=16, k=48), C.byref(nb)) == 0
    assert lib.pnn_conv_workspace_bytes(1, 3, 1, args(c=16, k=48), C.byref(nb)) == 1


def test_roofline_group_has_algorithmic_work():
    """bench.py's roofline record takes the launch group with the most device
    time among those with algorithmic bytes or FLOPs: per-layer BN
    finalisations (no bytes counted, one trace shape for all layers) can sum
    to more time in an untorn network without being a roofline candidate."""
    import bench
    conv = {"kind": "conv_fwd_tc", "variant": 2, "shape": (16, 64, 1, 1, 32, 32), "instances": 8,
            "ms": 0.2, "flops": 4.3e9, "bytes": 3.5e8}
    fin = {"kind": "bn_finalize", "variant": 0, "shape": (0, 0, 0, 0, 0, 0), "instances": 8,
           "ms": 0.05, "flops": 0.0, "bytes": 0.0}
    trace = [dict(conv) for _ in range(3)] + [dict(fin) for _ in range(20)]
    r = bench.roofline_of({}, 1, trace)
    assert r["kernel"] == "k_conv_fwd_tma_w" and r["kind"] == "conv_fwd_tc", r
    assert r["launches_per_step"] == 3 and abs(r["ms_per_launch"] - 0.2) < 1e-12
    assert abs(r["achieved"] - 3.5e8 / 0.2e-3 / 1e9) < 1e-6 and r["bound"] == "hbm"
    groups = bench.launch_groups(trace, 1)
    assert [g["kernel"] for g in groups] == ["k_bn_fin", "k_conv_fwd_tma_w"]  # by time, bytes or not
    assert groups[0]["launches_per_step"] == 20 and groups[1]["gbs"] > 0
