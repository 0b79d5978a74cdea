"""GPU parity of the whole training step (Algorithms 1 and 2 plus the SGD
update) against the CPU oracle on identical seeded inputs and weights,
through the C ABI.

Tolerances.  The target bounds are 2e-2 (bf16 forward, max-relative),
5e-2 (bf16 gradients, norm-relative) and 1e-4 (fp32 check mode).  They are
applied as they stand wherever they are attainable: every forward tensor in
bf16 and every quantity in fp32 check mode at small sizes.  Beyond that, a
floating-point decision (a ReLU mask, a maxpool argmax, the bf16 rounding of
a stored value) flips when two correct computations differ by the last bits
of an fp32 sum, and depth amplifies each flip.  How far the oracle's own
result moves under differences of that size is measured and bounds the GPU:

* bf16: the oracle's bf16 model (forward values rounded where the library
  stores them in bf16; every decision taken on those values) with each
  convolution output perturbed by a relative 4e-6 (about sqrt(4608) * 2^-24,
  the typical relative difference of two fp32 summation orders of the
  longest contraction here, 3x3x512) before rounding; every quantity is held
  to max(target bound, 3x the largest move over two draws).  Every bf16
  forward tensor is also reported against the float64 oracle (bf16 weights and
  inputs, no internal rounding) and held to max(2e-2, 1.5x the distance of
  the oracle's own bf16 evaluation from float64): at full depth and small
  batches the network amplifies rounding so much that even that evaluation
  sits 10-50 % from float64 (measured; printed by the tests).
* fp32 check mode beyond the tiny config: 3x the oracle's response to a 1e-5
  relative perturbation of its parameters (max of two draws), never below the
  target bound.
"""
import numpy as np
import pytest

import workloads as W
from parity import TOL, compare, inputs, norm_rel, run_gpu, run_oracle

pytestmark = pytest.mark.gpu
LOOSE = {"fwd": 1e9, "grad": 1e9}


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2103_08802_gb300 import build
    build.build()


def _fmt(r):
    return {k: f"{v:.1e}" for k, v in r.items() if not isinstance(v, dict)}


def _strict(desc, **kw):
    onet, theta, x, labels = inputs(desc)
    g = run_gpu(desc, theta, x, labels, **kw)
    o = run_oracle(desc, theta, x, labels)
    report, fails = compare(desc, g, o)
    print(desc["name"], desc["precision"], desc.get("correction"), desc["batch"], _fmt(report))
    assert not fails, fails
    return g, o, theta


def _grad_keys(report):
    return [k for k in report if k.startswith("D") or k.startswith("grad")]


def _measured(desc, noise_fn, factor, floor, conv_impl=0):
    """Every key is bounded by max(target bound, factor * measured noise):
    the forward bound for forward tensors, `floor` for D_j and gradients.
    bf16 runs also hold every forward tensor to the forward bound against
    the float64 oracle.  conv_impl: the library's kernel choice (options)."""
    onet, theta, x, labels = inputs(desc)
    g = run_gpu(desc, theta, x, labels, conv_impl=conv_impl)
    o = run_oracle(desc, theta, x, labels)
    err, _ = compare(desc, g, o, LOOSE)
    noise = noise_fn(desc, theta, x, labels, o)
    tol = TOL[desc["precision"]]
    print(desc["name"], desc["precision"], desc["batch"], "gpu err", _fmt(err))
    print(desc["name"], desc["precision"], desc["batch"], "noise  ", _fmt(noise))
    bad = []
    for k, e in err.items():
        if k in ("grad_worst",):
            continue
        lo = floor if k in _grad_keys(err) else tol["fwd"]
        b = max(lo, factor * noise[k])
        print(f"  {k:10s} err {e:.2e}  bound {b:.2e}")
        if not e <= b:
            bad.append((k, e, noise[k]))
    # per-tensor parameter gradients
    off = 0
    gn = noise.get("_per_tensor", {})
    for i, (kind, shape) in enumerate(onet.spec):
        n = int(np.prod(shape))
        e = norm_rel(g["grad"][off:off + n], o["grad"][off:off + n])
        if not e <= max(floor, factor * gn.get(i, 0.0)):
            bad.append((f"grad[{i}] {shape}", e, gn.get(i)))
        off += n
    if desc["precision"] == "bf16":
        # against float64: no bf16 implementation can be closer than the
        # oracle's own bf16 evaluation is, so the bound is the 2e-2 target or
        # 1.5x that distance, whichever is larger
        o64 = run_oracle(desc, theta, x, labels, precision="fp64")
        e64, _ = compare(desc, g, o64, LOOSE)
        m64, _ = compare(desc, o, o64, LOOSE)
        for k, e in e64.items():
            if k.startswith("D") or k.startswith("grad"):
                continue
            b = max(tol["fwd"], 1.5 * m64[k])
            print(f"  {k:10s} vs fp64 oracle {e:.2e}  (bf16 model vs fp64 {m64[k]:.2e})  bound {b:.2e}")
            if not e <= b:
                bad.append((k + " vs fp64", e, b))
    assert not bad, bad[:40]


def _per_tensor(onet, a, b):
    out, off = {}, 0
    for i, (kind, shape) in enumerate(onet.spec):
        n = int(np.prod(shape))
        out[i] = norm_rel(a[off:off + n], b[off:off + n])
        off += n
    return out


def bf16_accum_noise(desc, theta, x, labels, o, draws=2, rel=4e-6):
    """How far the oracle's bf16 model moves when every convolution output
    differs by a relative `rel` (fp32 summation-order size) before it is
    rounded: the elementwise maximum over `draws` perturbations."""
    from oracle import pnn_oracle as O
    out = None
    for k in range(draws):
        with O.perturbed(np.random.default_rng(5 + k), rel):
            o2 = run_oracle(desc, theta, x, labels)
        r, _ = compare(desc, o2, o, LOOSE)
        r["_per_tensor"] = _per_tensor(o["onet"], o2["grad"], o["grad"])
        if out is None:
            out = r
        else:
            for key, v in r.items():
                out[key] = {i: max(a, v[i]) for i, a in out[key].items()} if key == "_per_tensor" else max(out[key], v)
    return out


def fp32_perturbation_noise(desc, theta, x, labels, o, draws=2, rel=1e-5):
    """The oracle's own response to a relative perturbation of its parameters
    (rel = 1e-5, about ten times the GPU's fp32 accumulation-order
    differences, so that rare ReLU-mask flips are represented); the
    elementwise maximum over `draws` perturbations."""
    out = None
    for k in range(draws):
        rng = np.random.default_rng(5 + k)
        o2 = run_oracle(desc, theta.astype(np.float64) * (1 + rel * rng.standard_normal(theta.size)), x, labels)
        r, _ = compare(desc, o2, o, LOOSE)
        r["_per_tensor"] = _per_tensor(o["onet"], o2["grad"], o["grad"])
        if out is None:
            out = r
        else:
            for key, v in r.items():
                out[key] = {i: max(a, v[i]) for i, a in out[key].items()} if key == "_per_tensor" else max(out[key], v)
    return out


def reduced(idx, precision="bf16", correction="residual", batch=None):
    """Config idx at its full batch and resolution with fewer blocks per
    segment (same stem, stages, strides, projections, interfaces, coarse
    blocks, head); VGG-16 runs whole."""
    if idx == 1:
        d = W.config(1)
    elif idx == 2:
        d = W.parareal_resnet1001(n_seg=4, batch=128, classes=10, per_stage=2, segments=[2, 1, 2, 1])
    elif idx == 3:
        d = W.parareal_resnet1001(n_seg=16, batch=128, classes=100, per_stage=6, segments=[2, 2] + [1] * 14)
    elif idx == 4:
        d = W.parareal_resnet1001(n_seg=8, batch=256, classes=200, hw=64, per_stage=3,
                                  segments=[2, 1, 1, 1, 1, 1, 1, 1])
    d["precision"] = precision
    d["correction"] = correction
    d["config_index"] = idx
    if batch:
        d["batch"] = batch
    return d


def paper_reduced(n, precision="bf16", correction="residual", batch=128):
    """Parareal ResNet-N as Section 4.2 builds it (N = 3 N_0 stage-aligned
    subnetworks, N_c = ceil(12/N) coarse RUs per F^j, 100 classes, 32x32)
    with one or two bottlenecks per subnetwork instead of ceil(333/N): the
    same interfaces X_j, coarse network, C^j and head."""
    per_stage = {3: 2, 6: 2, 12: 4, 18: 6}[n]
    return W.paper_parareal_resnet(n, batch=batch, per_stage=per_stage, precision=precision,
                                   correction=correction)


# ------------------------------------------------------------------ strict (target bounds)
@pytest.mark.parametrize("mode", ["residual", "delta"])
def test_tiny_fp32_check_mode_step(mode):
    desc = W.config(0)
    desc["correction"] = mode
    g, o, theta = _strict(desc)
    # the SGD update: compare the step theta_new - theta and the momentum buffer
    step_g = g["theta_new"].astype(np.float64) - theta
    step_o = o["theta_new"] - theta
    assert norm_rel(step_g, step_o) <= TOL["fp32"]["grad"]
    assert norm_rel(g["momentum"], o["momentum"]) <= TOL["fp32"]["grad"]


def test_tiny_n1_is_untorn():
    desc = W.config(0)
    desc["segments"] = [4]
    desc["coarse"] = []
    _strict(desc)


@pytest.mark.parametrize("idx", [2, 3, 4])
@pytest.mark.parametrize("mode", ["residual", "delta"])
def test_fp32_small_batch_all_interfaces(idx, mode):
    _measured(reduced(idx, precision="fp32", correction=mode, batch=4), fp32_perturbation_noise, 3.0,
              TOL["fp32"]["grad"])


def test_vgg_fp32_small_batch():
    _measured(reduced(1, precision="fp32", batch=2), fp32_perturbation_noise, 3.0, TOL["fp32"]["grad"])


# ------------------------------------------------------------------ measured bounds, full batch
@pytest.mark.parametrize("idx", [1, 2, 3, 4])
def test_bf16_full_batch(idx):
    _measured(reduced(idx), bf16_accum_noise, 3.0, TOL["bf16"]["grad"])


@pytest.mark.parametrize("idx", [1, 2, 4])
def test_bf16_full_batch_fp32_residual_stream(idx):
    """The residual stream (block outputs, r_j, rt_j, ytilde) kept in fp32
    (the bf16 workloads store it in bf16 by default; the oracle's bf16 model
    rounds whichever values the library stores in bf16)."""
    d = reduced(idx)
    d["residual_stream"] = "fp32"
    _measured(d, bf16_accum_noise, 3.0, TOL["bf16"]["grad"])


def test_bf16_full_batch_delta_mode():
    _measured(reduced(2, correction="delta"), bf16_accum_noise, 3.0, TOL["bf16"]["grad"])


@pytest.mark.parametrize("idx", [2, 4])
def test_fp32_full_batch(idx):
    _measured(reduced(idx, precision="fp32"), fp32_perturbation_noise, 3.0, TOL["fp32"]["grad"])


# ------------------------------------------------------------------ the paper's own constructions
@pytest.mark.parametrize("n,mode", [(3, "residual"), (3, "delta"), (12, "residual")])
def test_paper_resnet_fp32_small_batch(n, mode):
    _measured(paper_reduced(n, precision="fp32", correction=mode, batch=4), fp32_perturbation_noise, 3.0,
              TOL["fp32"]["grad"])


@pytest.mark.parametrize("n,batch", [(3, 128), (12, 32)])
def test_paper_resnet_bf16(n, batch):
    _measured(paper_reduced(n, batch=batch), bf16_accum_noise, 3.0, TOL["bf16"]["grad"])


def test_paper_vgg_coarse_fp32_small_batch():
    """Batch 2: the last subnetwork's BNs see 8 values per channel, where a
    one-pass variance (sum h^2 - n mean^2) loses digits; the statistics are
    combined as (count, mean, M2) partials (Chan's pairwise update) instead."""
    d = W.parareal_vgg16(coarse="paper", precision="fp32", batch=2)
    _measured(d, fp32_perturbation_noise, 3.0, TOL["fp32"]["grad"])


def test_paper_vgg_coarse_bf16():
    _measured(W.parareal_vgg16(coarse="paper", batch=32), bf16_accum_noise, 3.0, TOL["bf16"]["grad"])


# ------------------------------------------------------------------ full depth
# Full-depth ResNet-1001 (333 bottlenecks): configurations 3 (N = 4), 4
# (N = 16, 100 classes) and 5 (N = 8, 64x64 with the stride-2 stem, 200
# classes) at small batches (the fp64 oracle holds every activation).
@pytest.mark.parametrize("idx,batch", [(2, 2), (3, 2), (4, 2)])
def test_full_depth_fp32(idx, batch):
    desc = W.config(idx, batch=batch)
    desc["precision"] = "fp32"
    _measured(desc, fp32_perturbation_noise, 3.0, TOL["fp32"]["grad"])


@pytest.mark.parametrize("idx,batch,stream", [(2, 4, "fp32"), (3, 4, "fp32"), (4, 2, "fp32"), (4, 2, "bf16")])
def test_full_depth_bf16(idx, batch, stream):
    """The benchmarked path (tcgen05 kernels, bf16 storage) at full depth."""
    desc = W.config(idx, batch=batch)
    desc["residual_stream"] = stream
    _measured(desc, bf16_accum_noise, 3.0, TOL["bf16"]["grad"])


# ------------------------------------------------------------------ properties
@pytest.mark.parametrize("idx", [1, 2, 4])
def test_tensor_core_forward_matches_cuda_core(idx):
    """The tcgen05 convolutions and the CUDA-core convolutions compute the
    same bf16-operand products with fp32 accumulation: forward tensors agree
    to a few bf16 ulps of the largest element."""
    desc = reduced(idx)
    onet, theta, x, labels = inputs(desc)
    tc = run_gpu(desc, theta, x, labels)
    cc = run_gpu(desc, theta, x, labels, conv_impl=1)
    r, _ = compare(desc, tc, cc, LOOSE)
    fwd = {k: v for k, v in r.items() if not (k.startswith("D") or k.startswith("grad"))}
    print(desc["name"], "tc vs cuda-core", _fmt(fwd))
    assert max(fwd.values()) <= 2e-2, fwd


def _conv_variants(desc, theta, x, labels, conv_impl):
    """Kernel variants of the tensor-core conv launches of one eager step."""
    import torch
    from paper_2103_08802_gb300 import pnn
    net = pnn.ParaNet(desc, conv_impl=conv_impl)
    net.set_params(theta)
    net.profile(True)
    net.forward(torch.from_numpy(x).cuda(), torch.from_numpy(labels).cuda())
    net.backward()
    tr = net.profile_trace()
    net.profile(False)
    return {(r["kind"], r["variant"]) for r in tr if r["kind"] in ("conv_fwd_tc", "conv_dgrad_tc", "conv_wgrad_tc")}


@pytest.mark.parametrize("idx", [1, 2, 4, "paper_n3"])
def test_thread_gathered_convs_match_oracle(idx):
    """The thread-gathered tensor-core convolutions (conv_impl=3: no TMA
    producer) against the oracle's bf16 model within the same measured bound
    as the default path (test_bf16_full_batch, test_paper_resnet_bf16), on
    workloads whose default plan does use the TMA-fed forward, data- and
    weight-gradient kernels.  The two paths build the same bf16 operands; the
    epilogues differ in fp32 summation orders (the wide-epilogue forward sums
    a staged chunk's BN-statistics columns per lane, the other kernels by
    shuffle trees; the TMA-fed data gradient forms the BN-backward sums over
    its 128-row tiles), and these deep networks respond to such rounding-level
    changes far beyond them, so each path is held to the oracle rather than
    to the other.  (VGG-16's 3x3 convs with 64..512 channels, ResNet's 1x1
    and 3x3 bottleneck convs, the coarse RUs' 3x3 convs at 128 and 256
    channels; stride-2 convs take the gathered kernel on both paths.)"""
    desc = paper_reduced(3) if idx == "paper_n3" else reduced(idx)
    onet, theta, x, labels = inputs(desc)
    tma = _conv_variants(desc, theta, x, labels, 0)
    assert ("conv_fwd_tc", 1) in tma and ("conv_dgrad_tc", 1) in tma and ("conv_wgrad_tc", 1) in tma, tma
    assert all(v == 0 for _, v in _conv_variants(desc, theta, x, labels, 3))
    _measured(desc, bf16_accum_noise, 3.0, TOL["bf16"]["grad"], conv_impl=3)


def test_step_is_deterministic():
    desc = W.config(2, batch=4)
    onet, theta, x, labels = inputs(desc)
    a = run_gpu(desc, theta, x, labels)
    b = run_gpu(desc, theta, x, labels)
    np.testing.assert_array_equal(a["grad"], b["grad"])
    np.testing.assert_array_equal(a["logits"], b["logits"])
    np.testing.assert_array_equal(a["theta_new"], b["theta_new"])


@pytest.mark.parametrize("paper,mode", [(False, "residual"), (True, "residual"), (False, "delta")])
def test_correction_folded_into_conv_epilogues(paper, mode):
    """The correction's sums (residual form: r_j, rt_{j+1}, ytilde; delta form:
    the states s_{j+1} = y_{j+1} + F^j(s_j) - F^j(x_{j+1})) ride in the
    epilogues of the convs that produce their operands, and their backward
    scatter (dL/dy_j = D_j, dL/dx_{j+1} -= D_j) in gradient aliases and the
    BN-backward apply of x_{j+1}: no elementwise launch in the coarse phases
    of a step.  (Values the step no longer stores -- y_j for j < N, rt_N, the
    delta form's r_j and rt_j -- are still exported exactly; the parity tests
    above compare them.)"""
    import torch
    from paper_2103_08802_gb300 import pnn
    desc = paper_reduced(3) if paper else reduced(2, correction=mode)
    onet, theta, x, labels = inputs(desc)
    net = pnn.ParaNet(desc)
    net.set_params(theta)
    net.profile(True)
    net.forward(torch.from_numpy(x).cuda(), torch.from_numpy(labels).cuda())
    net.backward()
    tr = net.profile_trace()
    net.profile(False)
    coarse = [r["kind"] for r in tr if r["phase"] in (2, 5)]
    assert coarse and not any(k.startswith("elementwise") for k in coarse), coarse
