"""Workload descriptions and seeded input generators.

This module is shared by the tests and the benchmark.  It describes the five
parareal networks that are measured (as plain dictionaries) and draws their
seeded synthetic inputs.  It holds none of the method's arithmetic: it does not
evaluate a network, a correction or a gradient.  Both the CPU oracle and the
CUDA library receive the description and the arrays drawn here as inputs.

Description format (a dict):

  name, batch, in_c, in_h, in_w, classes
  precision    "fp32" (check mode) or "bf16"
  correction   "residual" (the paper's eq:correct) or "delta"
  stem         list of layers: the preprocessing operator C_delta = C^1
  body         list of layers: the block-repetitive part g_phi
  segments     list of N ints: body layers per fine subnetwork g^j (tearing)
  coarse       list of N-1 layer lists: the coarse blocks F^j : X_j -> X_{j+1}
  cj_post      "bn_relu" or "none": what follows the 1x1 conv of C^j, j > 1
  head         {"kind": "gap_fc" | "bn_relu_gap_fc" | "gap_mlp", "hidden": [...]}

Layer kinds:
  {"op": "conv", "cout", "k", "stride"}                 bare conv, pad k//2
  {"op": "conv_bn_relu", "cout", "k", "stride", "pool"} conv-BN-ReLU (+ 2x2/s2 maxpool if pool)
  {"op": "basic", "cout"}                               post-activation basic block
  {"op": "bottleneck", "cout", "mid", "stride"}         pre-activation bottleneck
  {"op": "coarse_ru", "cout", "stride"}                 coarse RU: two 3x3 convs + skip
"""
from __future__ import annotations

import copy
import numpy as np

__all__ = [
    "conv", "conv_bn_relu", "basic", "bottleneck", "coarse_ru",
    "tiny_resnet", "parareal_vgg16", "parareal_resnet1001", "paper_parareal_resnet",
    "config", "CONFIG_NAMES", "make_batch", "init_params", "bf16_round",
    "with_batch",
]


# ---------------------------------------------------------------- layers
def conv(cout, k=3, stride=1):
    return {"op": "conv", "cout": cout, "k": k, "stride": stride}


def conv_bn_relu(cout, k=3, stride=1, pool=0):
    return {"op": "conv_bn_relu", "cout": cout, "k": k, "stride": stride, "pool": pool}


def basic(cout):
    return {"op": "basic", "cout": cout}


def bottleneck(cout, mid, stride=1):
    return {"op": "bottleneck", "cout": cout, "mid": mid, "stride": stride}


def coarse_ru(cout, stride=1):
    return {"op": "coarse_ru", "cout": cout, "stride": stride}


# ---------------------------------------------------------------- configs
def tiny_resnet(batch=8, precision="fp32", correction="residual"):
    """Tiny parareal ResNet: stem conv3x3->16 (+BN+ReLU), N=2 subnetworks of
    2 basic blocks at 16 channels, one conv3x3+BN+ReLU coarse block."""
    return {
        "name": "tiny_resnet_n2", "batch": batch, "in_c": 3, "in_h": 32, "in_w": 32,
        "classes": 10, "precision": precision,
        "residual_stream": "bf16" if precision == "bf16" else "fp32", "correction": correction,
        "stem": [conv_bn_relu(16)],
        "body": [basic(16) for _ in range(4)],
        "segments": [2, 2],
        "coarse": [[conv_bn_relu(16)]],
        "cj_post": "bn_relu",
        "head": {"kind": "gap_fc", "hidden": []},
    }


def parareal_vgg16(batch=128, precision="bf16", correction="residual", classes=10, coarse="one_conv"):
    """Parareal VGG-16-4 at 32x32: the 13 conv layers with BN+ReLU and a 2x2
    maxpool closing each stage, torn after stages 2, 3, 4 and 5 (Section 4.1);
    3-FC head.  coarse="one_conv": one conv3x3+BN+ReLU+maxpool block per
    interface; coarse="paper": F^j of Section 4.1, two 3x3 convs (each with
    BN+ReLU, as the body's convs) and a 2x2/s2 maxpool, at the width of
    X_{j+1}."""
    body = [conv_bn_relu(64, pool=2),
            conv_bn_relu(128), conv_bn_relu(128, pool=2),
            conv_bn_relu(256), conv_bn_relu(256), conv_bn_relu(256, pool=2),
            conv_bn_relu(512), conv_bn_relu(512), conv_bn_relu(512, pool=2),
            conv_bn_relu(512), conv_bn_relu(512), conv_bn_relu(512, pool=2)]
    return {
        "name": "parareal_vgg16_n4", "batch": batch, "in_c": 3, "in_h": 32, "in_w": 32,
        "classes": classes, "precision": precision,
        "residual_stream": "bf16" if precision == "bf16" else "fp32", "correction": correction,
        "stem": [conv_bn_relu(64)],
        "body": body,
        "segments": [3, 3, 3, 3],
        "coarse": ([[conv_bn_relu(c, pool=2)] for c in (256, 512, 512)] if coarse == "one_conv" else
                   [[conv_bn_relu(c), conv_bn_relu(c, pool=2)] for c in (256, 512, 512)]),
        "cj_post": "bn_relu",
        "head": {"kind": "gap_mlp", "hidden": [4096, 4096]},
    }


def _resnet_stage(block_index, per_stage=111):
    return min(block_index // per_stage, 2)


def parareal_resnet1001(n_seg=4, batch=128, classes=10, hw=32, precision="bf16",
                        correction="residual", coarse_blocks=2, per_stage=111, segments=None):
    """Parareal pre-activation ResNet-1001 (Section 4.2): 333 bottleneck
    blocks in three stages (widths 64/128/256, bottleneck 16/32/64, stride 2
    at the first block of stages 2 and 3), torn into n_seg consecutive
    segments of ceil(333/n_seg) blocks (the last takes the remainder).  Each
    coarse block F^j is `coarse_blocks` pre-activation bottlenecks at the
    width of X_{j+1}; the first one is strided and projected when the shape
    changes.  hw=64 adds a stride-2 conv to the stem.

    per_stage < 111 gives the same family with fewer blocks per stage (a
    depth-reduced variant with the same stages, strides, projections and
    interface kinds); `segments` then overrides the tearing."""
    nb = 3 * per_stage
    body = []
    for b in range(nb):
        s = _resnet_stage(b, per_stage)
        first = b in (per_stage, 2 * per_stage)
        body.append(bottleneck(64 << s, 16 << s, 2 if first else 1))
    if segments is None:
        per = -(-nb // n_seg)
        segments = [per] * (n_seg - 1) + [nb - per * (n_seg - 1)]
    assert len(segments) == n_seg and sum(segments) == nb and min(segments) > 0
    # shape of X_j: output of the last block of segment j
    ends = [int(e) for e in np.cumsum(segments) - 1]
    shapes = [(64 << _resnet_stage(e, per_stage), 32 >> _resnet_stage(e, per_stage)) for e in ends]
    coarse = []
    for j in range(n_seg - 1):
        (c0, h0), (c1, h1) = shapes[j], shapes[j + 1]
        assert h0 in (h1, 2 * h1)
        blocks = [bottleneck(c1, c1 // 4, h0 // h1)]
        blocks += [bottleneck(c1, c1 // 4, 1) for _ in range(coarse_blocks - 1)]
        coarse.append(blocks)
    stem = [conv(16)] if hw == 32 else [conv_bn_relu(16), conv(16, stride=2)]
    assert hw in (32, 64)
    return {
        "name": f"parareal_resnet{9 * per_stage + 2}_n{n_seg}", "batch": batch, "in_c": 3,
        "in_h": hw, "in_w": hw, "classes": classes, "precision": precision,
        "residual_stream": "bf16" if precision == "bf16" else "fp32",
        "correction": correction,
        "stem": stem, "body": body, "segments": segments, "coarse": coarse,
        "cj_post": "none",
        "head": {"kind": "bn_relu_gap_fc", "hidden": []},
    }


def paper_parareal_resnet(n, batch=128, classes=100, hw=32, precision="bf16", correction="residual",
                          per_stage=111, n_c=None):
    """Parareal ResNet-N built from ResNet-1001 as Section 4.2 does.

    N = 3 N_0 subnetworks, N_0 per stage, so that X_j is 64x32x32 for
    j <= N_0, 128x16x16 for j <= 2 N_0 and 256x8x8 after.  Every g^j holds
    ceil(333/N) = ceil(111/N_0) pre-activation bottlenecks (the body thus has
    N ceil(333/N) >= 333 of them; the first block of stages 2 and 3 is the
    strided one).  Each F^j : X_j -> X_{j+1} is N_c = ceil(12/N) coarse RUs
    at the width of X_{j+1}, the first strided (and projected) when X_j and
    X_{j+1} differ in shape.  n = 1 is the untorn ResNet-1001 (Parareal
    ResNet-1).  per_stage < 111 gives the same construction with fewer
    bottlenecks per stage (ceil(per_stage/N_0) per subnetwork)."""
    if n == 1:
        d = parareal_resnet1001(n_seg=1, batch=batch, classes=classes, hw=hw, precision=precision,
                                correction=correction, per_stage=per_stage, segments=[3 * per_stage])
        d["name"] = "paper_parareal_resnet_n1"
        return d
    assert n % 3 == 0, "Parareal ResNet-N is defined for N = 3 N_0"
    n0 = n // 3
    seg = -(-per_stage // n0)
    n_c = -(-12 // n) if n_c is None else n_c
    body = []
    for s in range(3):
        for b in range(n0 * seg):
            body.append(bottleneck(64 << s, 16 << s, 2 if (s > 0 and b == 0) else 1))
    coarse = []
    for j in range(1, n):
        s0, s1 = (j - 1) // n0, j // n0   # stages of X_j and X_{j+1}
        c1 = 64 << s1
        coarse.append([coarse_ru(c1, 2 if s1 > s0 else 1)] + [coarse_ru(c1) for _ in range(n_c - 1)])
    assert hw in (32, 64)
    stem = [conv(16)] if hw == 32 else [conv_bn_relu(16), conv(16, stride=2)]
    return {
        "name": f"paper_parareal_resnet_n{n}", "batch": batch, "in_c": 3, "in_h": hw, "in_w": hw,
        "classes": classes, "precision": precision,
        "residual_stream": "bf16" if precision == "bf16" else "fp32", "correction": correction,
        "stem": stem, "body": body, "segments": [seg] * n, "coarse": coarse,
        "cj_post": "none",
        "head": {"kind": "bn_relu_gap_fc", "hidden": []},
    }


CONFIG_NAMES = [
    "tiny_resnet_n2_b8_fp32",
    "parareal_vgg16_n4_b128_bf16",
    "parareal_resnet1001_n4_b128_bf16",
    "parareal_resnet1001_n16_b128_c100_bf16",
    "parareal_resnet1001_n8_b256_64px_c200_bf16",
]


def config(index, batch=None, segments=None):
    """The five measured workloads, by index 0..4.  `segments` re-tears the
    ResNet-1001 workloads (2..4) with the same number of subnetworks."""
    if segments is not None and index not in (2, 3, 4):
        raise ValueError("only the ResNet-1001 workloads take another tearing")
    if index == 0:
        d = tiny_resnet()
    elif index == 1:
        d = parareal_vgg16()
    elif index == 2:
        d = parareal_resnet1001(n_seg=4, batch=128, classes=10, segments=segments)
    elif index == 3:
        d = parareal_resnet1001(n_seg=16, batch=128, classes=100, segments=segments)
    elif index == 4:
        d = parareal_resnet1001(n_seg=8, batch=256, classes=200, hw=64, segments=segments)
    else:
        raise ValueError(index)
    d["config_index"] = index
    if batch is not None:
        d["batch"] = batch
    return d


def with_batch(desc, batch):
    d = copy.deepcopy(desc)
    d["batch"] = batch
    return d


# ---------------------------------------------------------------- inputs
def bf16_round(a):
    """Round float32 values to the nearest bfloat16 (ties to even), returned
    as float32 (every bf16 value is exactly representable)."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    r = ((u + 0x7FFF + lsb) >> 16) << 16
    out = r.astype(np.uint32).view(np.float32)
    nan = np.isnan(a)
    if nan.any():
        out = out.copy()
        out[nan] = np.nan
    return out.reshape(a.shape)


def make_batch(desc, seed=None):
    """x ~ N(0,1) float32 in NCHW and labels uniform in [0, classes), int32.
    Seed defaults to 1000 + config index.  In bf16 workloads x is rounded to
    bf16 so that both sides start from the same representable input."""
    if seed is None:
        seed = 1000 + int(desc.get("config_index", 0))
    rng = np.random.default_rng(seed)
    shape = (desc["batch"], desc["in_c"], desc["in_h"], desc["in_w"])
    x = rng.standard_normal(shape, dtype=np.float64).astype(np.float32)
    labels = rng.integers(0, desc["classes"], size=desc["batch"], dtype=np.int64).astype(np.int32)
    if desc["precision"] == "bf16":
        x = bf16_round(x)
    return x, labels


# parameter kinds (shared vocabulary of the flat parameter vector)
KIND_CONV_W, KIND_BN_G, KIND_BN_B, KIND_FC_W, KIND_FC_B = 0, 1, 2, 3, 4


def init_params(spec, seed=0, bf16=False):
    """He-normal initialisation (std sqrt(2/fan_in)) of conv and FC weights,
    BN gamma = 1, beta = 0, FC bias = 0, drawn in `spec` order.

    spec: list of (kind, shape) with shape the PyTorch layout of the tensor
    ((K,C,R,S) for a conv, (out,in) for an FC).  Returns one flat float32
    vector.  With bf16=True every value is rounded to bf16."""
    rng = np.random.default_rng(seed)
    parts = []
    for kind, shape in spec:
        n = int(np.prod(shape))
        if kind in (KIND_CONV_W, KIND_FC_W):
            fan_in = int(np.prod(shape[1:]))
            v = rng.standard_normal(n) * np.sqrt(2.0 / fan_in)
        elif kind == KIND_BN_G:
            v = np.ones(n)
        else:
            v = np.zeros(n)
        parts.append(v.astype(np.float32))
    theta = np.concatenate(parts) if parts else np.zeros(0, np.float32)
    if bf16:
        theta = bf16_round(theta)
    return theta
