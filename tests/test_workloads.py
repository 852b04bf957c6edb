"""The synthetic workload recipes (no GPU): the ResNet-50 sweep's shape table
and the exactness of its zero padding, checked through the oracle."""
import numpy as np
import pytest

import oracle as orc
from paper_2010_14298_gb300 import workloads as wl


def test_resnet50_sweep_shapes():
    """53 convolutions (16 bottlenecks of three, four projection shortcuts,
    the stem) and the fc; stride 2 on the 3 x 3 conv of the first block of
    stages 2-4; 4.09 GMACs per 224 x 224 image (the architecture's count)."""
    sh = wl.resnet50_shapes()
    assert len(sh) == 54 and sh[-1].name == "fc"
    assert sum(s.name.endswith("downsample") for s in sh) == 4
    assert sum(s.k == 3 for s in sh) == 16 and sh[0].k == 7
    assert [s.name for s in sh if s.stride == 2] == [
        "conv1", "layer2.0.conv2", "layer2.0.downsample", "layer3.0.conv2",
        "layer3.0.downsample", "layer4.0.conv2", "layer4.0.downsample"]
    # spatial sizes: 112 after the stem, 56 / 28 / 14 / 7 through the stages
    assert sh[0].hout == 112
    outs = {s.name.split(".")[0]: s.hout for s in sh if s.name.endswith("conv3")}
    assert outs == {"layer1": 56, "layer2": 28, "layer3": 14, "layer4": 7}
    macs = sum(s.rows(1) * s.cout * s.D for s in sh)
    assert abs(macs - 4.089e9) / 4.089e9 < 1e-3
    # the contractions' operands: multiples of 16 after padding
    assert all(s.D_pad % 16 == 0 and s.C_pad % 16 == 0 for s in sh)
    assert (sh[0].D, sh[0].D_pad) == (147, 160) and (sh[-1].cout, sh[-1].C_pad) == (1000, 1008)


def test_resnet50_sweep_layers_are_padded_with_zeros():
    L = wl.config(4, batch=1)
    assert len(L) == 54
    stem, fc = L[0], L[-1]
    assert stem.X.shape == (112 * 112, 160) and not stem.X[:, 147:].any()
    assert not stem.W[:, 147:].any()
    assert fc.dH.shape == (1, 1008) and not fc.dH[:, 1000:].any() and not fc.W[1000:].any()


def test_zero_padding_of_the_reduction_columns_is_exact():
    """The stem's D = 147 -> 160: zero columns of X and W lie inside the
    per-tensor ranges of X~ and W~ (both ranges straddle 0), so the codes of
    the real columns, and grad_X and grad_W on them, equal the unpadded
    layer's exactly (oracle, same seed)."""
    g = wl.rng(77)
    n, c, d, dp = 40, 16, 147, 160
    dH = wl.random_grad(g, n, c)
    X = g.uniform(-1, 1, (n, d)).astype(np.float32)
    W = (0.1 * g.standard_normal((c, d))).astype(np.float32)
    Xp = np.concatenate([X, np.zeros((n, dp - d), np.float32)], axis=1)
    Wp = np.concatenate([W, np.zeros((c, dp - d), np.float32)], axis=1)
    a = orc.linear_backward(dH, X, W, orc.BHQ, 5, 16, 3)
    b = orc.linear_backward(dH, Xp, Wp, orc.BHQ, 5, 16, 3)
    assert np.array_equal(a["grad_x"], b["grad_x"][:, :d])
    assert np.array_equal(a["grad_w"], b["grad_w"][:, :d])
