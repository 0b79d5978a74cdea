"""Cost-balanced tearing (Section 4.2, the remark after Table grad), host only:
the library's exact min-max cut against an exhaustive search, and its per-layer
FLOPs against the count written out from the layer shapes."""
import numpy as np
import pytest

import workloads as W
from oracle import pnn_oracle as O
from oracle import tearing as T


@pytest.fixture(scope="module")
def pnn():
    from paper_2103_08802_gb300 import build, pnn as P
    build.build()
    return P


def _check_cut(costs, seg, n_seg):
    assert len(seg) == n_seg and all(s >= 1 for s in seg) and sum(seg) == len(costs)
    b = np.cumsum([0] + seg)
    return max(sum(costs[b[i]:b[i + 1]]) for i in range(n_seg))


@pytest.mark.parametrize("seed", range(40))
def test_partition_is_optimal(pnn, seed):
    r = np.random.default_rng(seed)
    n = int(r.integers(1, 11))
    n_seg = int(r.integers(1, n + 1))
    # integer costs (with repeats and zeros): every sum is exact in both codes
    costs = [int(v) for v in r.integers(0, 20, size=n)]
    seg = pnn.partition(costs, n_seg)
    assert _check_cut(costs, seg, n_seg) == T.best_cut(costs, n_seg)


def test_partition_special_cases(pnn):
    assert pnn.partition([3.0] * 7, 1) == [7]
    assert pnn.partition([1.0, 5.0, 2.0], 3) == [1, 1, 1]
    # equal costs: the optimum is ceil(10/4) = 3 layers; each segment takes as
    # many as that allows, the last what is left
    assert pnn.partition([1.0] * 10, 4) == [3, 3, 3, 1]
    # one dominant layer sits alone
    seg = pnn.partition([1, 1, 1, 100, 1, 1, 1], 3)
    b = np.cumsum([0] + seg)
    assert any(b[i + 1] - b[i] == 1 and b[i] == 3 for i in range(3)), seg
    for bad in ([], [1.0, -1.0], [1.0, float("nan")]):
        with pytest.raises(pnn.PnnError):
            pnn.partition(bad, 1)
    with pytest.raises(pnn.PnnError):
        pnn.partition([1.0, 2.0], 3)
    with pytest.raises(pnn.PnnError):
        pnn.partition([1.0, 2.0], 0)


NETS = {
    "resnet1001_reduced": lambda: W.parareal_resnet1001(n_seg=4, per_stage=3, segments=[3, 2, 2, 2]),
    "resnet1001_64px": lambda: W.parareal_resnet1001(n_seg=4, batch=8, hw=64, per_stage=2, segments=[2, 2, 1, 1]),
    "vgg16": lambda: W.parareal_vgg16(batch=16),
    "tiny": lambda: W.tiny_resnet(),
    "paper_resnet_n3": lambda: W.paper_parareal_resnet(3, batch=8, per_stage=2),
}


@pytest.mark.parametrize("name", list(NETS))
def test_block_flops_match_layer_shapes(pnn, name):
    d = NETS[name]()
    got = pnn.block_costs(d, "flops")
    want = T.body_training_flops(d, O.ParaNet(d).X[0])
    assert got == [float(v) for v in want]


def test_block_bytes_are_positive_and_follow_activation_size(pnn):
    """HBM bytes of a stage-1 bottleneck (64 x 32 x 32 activations) exceed a
    stage-3 one's (256 x 8 x 8, four times fewer values) at equal FLOPs."""
    d = W.parareal_resnet1001(n_seg=1, per_stage=3, segments=[9])
    b = pnn.block_costs(d, "bytes")
    f = pnn.block_costs(d, "flops")
    assert all(v > 0 for v in b)
    assert f[1] == f[7] and b[1] > 1.5 * b[7]


def test_balanced_segments_of_resnet1001(pnn):
    """ResNet-1001 bottlenecks all cost the same FLOPs except the projected
    first units of each stage, so the FLOP-balanced cut of the N = 8 network is
    within a unit of the uniform one; by bytes the stage-1 units weigh ~3.5x
    the stage-3 ones and the byte-balanced cut gives early subnetworks fewer."""
    d = W.config(4)
    fl = pnn.balanced_segments(d, 8, "flops")
    by = pnn.balanced_segments(d, 8, "bytes")
    assert sum(fl) == sum(by) == 333
    assert max(fl) - min(fl) <= 1
    assert by[0] < by[-1] / 2


# ------------------------------------------------------------ pins of the oracle's own tearing helpers
def test_oracle_best_cut_textbook_cases():
    """The classic "split an array into m parts minimising the largest sum"
    examples, worked by hand."""
    assert T.best_cut([7, 2, 5, 10, 8], 2) == 18      # 7+2+5 | 10+8
    assert T.best_cut([1, 2, 3, 4, 5], 2) == 9        # 1+2+3 | 4+5
    assert T.best_cut([1, 4, 4], 3) == 4
    assert T.best_cut([5, 5, 5, 5], 1) == 20
    assert T.best_cut([3, 1, 4, 1, 5, 9, 2, 6], 8) == 9


def test_oracle_layer_flops_closed_form():
    """A non-strided ResNet-1001 bottleneck on a 32x32 map with 64 channels and
    width 16 takes 1024 * (64*16 + 9*16*16 + 16*64) multiply-adds per image in
    the forward pass (the same at every stage: 4x the pixels, 1/4 the channels
    squared), and three times that in training; the whole body of 333 units
    with its stem comes to about 8.95 GFLOP of training convolutions per 32x32
    image."""
    per_unit = 1024 * (64 * 16 + 9 * 16 * 16 + 16 * 64)
    d = W.parareal_resnet1001(n_seg=1, batch=2, segments=[333])
    f = T.body_training_flops(d, (16, 32, 32))
    assert f[5] == f[150] == f[300] == 6 * per_unit * 2
    stem = 3 * 2 * T.layer_forward_macs(d["stem"][0], (3, 32, 32))[0]
    assert abs((sum(f) / 2 + stem) / 8.95e9 - 1) < 1e-3


def test_partition_rejects_oversized_problems(pnn):
    with pytest.raises(pnn.PnnError):
        pnn.partition([1.0] * 40000, 3)
