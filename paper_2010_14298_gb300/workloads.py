"""Seeded synthetic inputs shaped like the paper's workloads.

This module holds no arithmetic of the method: it only draws the layer
tensors (output gradient dH, layer input X, weight W) that both the CUDA
library and the CPU oracle consume.  Draws use numpy's counter-based Philox
bit generator keyed by the data seed, so a (config, seed, size) triple gives
the same arrays on any machine.

The paper trains on CIFAR10, ImageNet and IWSLT14 (Sec. 5), which are not
available here.  The gradients below stand in for them: rows (samples) with
sparse, heavy-tailed per-sample magnitudes, the structure Sec. 4.1 attributes
to cross-entropy gradients of a well-fit network (most rows near zero, a few
outliers).  Conv layers are lowered to a linear layer on im2col rows
(Sec. 2.1), padding zeros included.
"""
from __future__ import annotations

import dataclasses
from typing import List, Optional, Tuple

import numpy as np

PTQ, PSQ, BHQ = 0, 1, 2
KIND_NAMES = {PTQ: "ptq", PSQ: "psq", BHQ: "bhq"}


def rng(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.Philox(key=seed))


def to_bf16_values(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bf16 (ties to even), kept in fp32.

    Used for workloads whose source tensors are bf16: the GPU receives the
    bf16 tensor, the oracle its exact fp32 widening.
    """
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    lsb = (u >> 16) & 1
    r = (u + 0x7FFF + lsb) & 0xFFFF0000
    return r.astype(np.uint32).view(np.float32)


def im2col_nhwc(x: np.ndarray, kh: int, kw: int, stride: int,
                pad: int) -> np.ndarray:
    """im2col of an NHWC tensor: rows (n, oh, ow), columns (kh, kw, cin)."""
    n, h, w, c = x.shape
    xp = np.pad(x, ((0, 0), (pad, pad), (pad, pad), (0, 0)))
    oh = (h + 2 * pad - kh) // stride + 1
    ow = (w + 2 * pad - kw) // stride + 1
    cols = np.empty((n, oh, ow, kh, kw, c), dtype=x.dtype)
    for i in range(kh):
        for j in range(kw):
            cols[:, :, :, i, j, :] = xp[:, i:i + stride * oh:stride,
                                        j:j + stride * ow:stride, :]
    return cols.reshape(n * oh * ow, kh * kw * c)


@dataclasses.dataclass
class Layer:
    """One layer backward problem: dH (N x C), X (N x D), W (C x D)."""
    name: str
    dH: np.ndarray
    X: np.ndarray
    W: np.ndarray
    dtype: str  # "f32" or "bf16": the source tensor type handed to the GPU
    runs: List[Tuple[int, int, int]]  # (kind, bits, block) for Q_b2
    x_nhwc: Optional[np.ndarray] = None  # conv layers: the NHWC input X is the im2col of

    @property
    def N(self) -> int:
        return self.dH.shape[0]

    @property
    def C(self) -> int:
        return self.dH.shape[1]

    @property
    def D(self) -> int:
        return self.X.shape[1]


def _lognormal_rows(g: np.random.Generator, n: int, sigma: float) -> np.ndarray:
    return np.exp(sigma * g.standard_normal(n)).astype(np.float32)


CONFIG_NAMES = [
    "linear-128x256",
    "resnet18-conv3x3-b128-32x32-64ch",
    "resnet50-layer3-conv3x3-b256-14x14-256ch",
    "transformer-ffn-8192tok-1024x4096-bf16",
    "resnet50-sweep-b256-224x224",
]


@dataclasses.dataclass(frozen=True)
class ConvShape:
    """One layer of the ResNet-50 sweep lowered to im2col: a k x k conv of
    cin -> cout channels on an h x h input (stride, padding); the final fc is
    a 1 x 1 conv on a 1 x 1 map."""
    name: str
    cin: int
    cout: int
    k: int
    stride: int
    pad: int
    h: int

    @property
    def hout(self) -> int:
        return (self.h + 2 * self.pad - self.k) // self.stride + 1

    def rows(self, batch: int) -> int:
        return batch * self.hout * self.hout

    @property
    def D(self) -> int:  # im2col columns (kh, kw, cin)
        return self.k * self.k * self.cin

    @property
    def D_pad(self) -> int:  # to a multiple of 16 for the contractions
        return (self.D + 15) // 16 * 16

    @property
    def C_pad(self) -> int:
        return (self.cout + 15) // 16 * 16


def resnet50_shapes() -> List[ConvShape]:
    """The 53 convolutions of ResNet-50 v1.5 (stride 2 on the 3 x 3 conv of the
    first bottleneck of a stage; four projection shortcuts) and the fc, at a
    224 x 224 input, in forward order."""
    out = [ConvShape("conv1", 3, 64, 7, 2, 3, 224)]
    cin, h = 64, 56  # after the 3 x 3 / 2 max pool
    for stage, (blocks, width) in enumerate(((3, 64), (4, 128), (6, 256), (3, 512)), start=1):
        cout = 4 * width
        for b in range(blocks):
            s = 2 if (b == 0 and stage > 1) else 1
            pre = f"layer{stage}.{b}"
            out.append(ConvShape(pre + ".conv1", cin, width, 1, 1, 0, h))
            out.append(ConvShape(pre + ".conv2", width, width, 3, s, 1, h))
            h2 = (h + 2 - 3) // s + 1
            out.append(ConvShape(pre + ".conv3", width, cout, 1, 1, 0, h2))
            if b == 0:
                out.append(ConvShape(pre + ".downsample", cin, cout, 1, s, 0, h))
            cin, h = cout, h2
    out.append(ConvShape("fc", 2048, 1000, 1, 1, 0, 1))
    return out


def resnet50_layer(shape: ConvShape, batch: int, seed: int) -> "Layer":
    """One layer of the ResNet-50 sweep: input U[-1, 1] at the layer's NHWC
    input shape, lowered to im2col; dH rows N(0, 1) scaled per sample by
    lognormal(0, 2); W Kaiming normal N(0, 2/D).  D and C are padded to
    multiples of 16 with zero columns (the stem's D = 147 -> 160, the fc's
    C = 1000 -> 1008): the padded columns of X and W are zero and so are the
    padded columns of dH; the outputs of the real columns are those of the
    unpadded layer."""
    g = rng(seed)
    x = g.uniform(-1, 1, (batch, shape.h, shape.h, shape.cin)).astype(np.float32)
    X = im2col_nhwc(x, shape.k, shape.k, shape.stride, shape.pad)
    n = X.shape[0]
    if shape.D_pad != shape.D:
        X = np.concatenate([X, np.zeros((n, shape.D_pad - shape.D), np.float32)], axis=1)
    dH = (g.standard_normal((n, shape.cout), dtype=np.float32)
          * _lognormal_rows(g, n, 2.0)[:, None])
    W = (np.sqrt(2.0 / shape.D) * g.standard_normal((shape.cout, shape.D))).astype(np.float32)
    if shape.C_pad != shape.cout:
        dH = np.concatenate([dH, np.zeros((n, shape.C_pad - shape.cout), np.float32)], axis=1)
        W = np.concatenate([W, np.zeros((shape.C_pad - shape.cout, shape.D), np.float32)], axis=0)
    if shape.D_pad != shape.D:
        W = np.concatenate([W, np.zeros((W.shape[0], shape.D_pad - shape.D), np.float32)], axis=1)
    return Layer(f"{CONFIG_NAMES[4]}:{shape.name}", np.ascontiguousarray(dH),
                 np.ascontiguousarray(X), np.ascontiguousarray(W), "f32", [(BHQ, 5, 16)])


def config(index: int, batch: Optional[int] = None, rows: Optional[int] = None,
           seed: Optional[int] = None) -> List[Layer]:
    """Layers of workload `index` (0-based).

    `batch` shrinks the image batch of the conv workloads and `rows` the
    token / sample count of the others, keeping every other shape and the
    value distributions, so the same recipe yields oracle-sized cases.
    """
    g = rng(1234 + index if seed is None else seed)
    if index == 0:
        n = rows or 128
        dH = (g.standard_normal((n, 256)).astype(np.float32)
              * _lognormal_rows(g, n, 2.0)[:, None])
        X = g.uniform(-1, 1, (n, 256)).astype(np.float32)
        W = (0.02 * g.standard_normal((256, 256))).astype(np.float32)
        return [Layer(CONFIG_NAMES[0], dH, X, W, "f32",
                      [(PTQ, 8, 0), (PSQ, 8, 0), (BHQ, 5, 16)])]
    if index == 1:
        b = batch or 128
        x = g.uniform(-1, 1, (b, 32, 32, 64)).astype(np.float32)
        X = im2col_nhwc(x, 3, 3, 1, 1)
        n = X.shape[0]
        dH = g.standard_normal((n, 64)).astype(np.float32)
        big = g.random(n) < 0.01
        dH[big] *= 100.0
        W = (np.sqrt(2.0 / 576) * g.standard_normal((64, 576))).astype(np.float32)
        runs = [(k, b_, 16 if k == BHQ else 0) for k in (PTQ, PSQ, BHQ)
                for b_ in (4, 5, 8)]
        return [Layer(CONFIG_NAMES[1], dH, X, W, "f32", runs, x)]
    if index == 2:
        b = batch or 256
        x = g.uniform(-1, 1, (b, 14, 14, 256)).astype(np.float32)
        X = im2col_nhwc(x, 3, 3, 1, 1)
        n = X.shape[0]
        dH = (g.standard_normal((n, 256)).astype(np.float32)
              * _lognormal_rows(g, n, 2.5)[:, None])
        W = (np.sqrt(2.0 / 2304) * g.standard_normal((256, 2304))).astype(np.float32)
        return [Layer(CONFIG_NAMES[2], dH, X, W, "f32",
                      [(BHQ, 5, nb) for nb in (8, 16, 32, 64)], x)]
    if index == 3:
        n = rows or 8192
        out = []
        for name, c, d in (("ffn-up", 4096, 1024), ("ffn-down", 1024, 4096)):
            z = g.standard_normal((n, c)).astype(np.float32)
            chi = g.chisquare(3, (n, c)).astype(np.float32)
            t3 = z / np.sqrt(chi / 3.0)
            dH = to_bf16_values(t3 * _lognormal_rows(g, n, 1.5)[:, None])
            X = to_bf16_values(g.standard_normal((n, d)).astype(np.float32))
            W = to_bf16_values((0.02 * g.standard_normal((c, d))).astype(np.float32))
            out.append(Layer(f"{CONFIG_NAMES[3]}:{name}", dH, X, W, "bf16",
                             [(PTQ, 8, 0), (PSQ, 5, 0), (BHQ, 5, 16)]))
        return out
    if index == 4:
        # full size is 40+ GB of fp32 inputs: the bench draws it on the device
        # from the same shape table; here, small batches for the oracle
        b = batch or 1
        base = 1234 + index if seed is None else seed
        return [resnet50_layer(sh, b, base + i) for i, sh in enumerate(resnet50_shapes())]
    raise ValueError(f"no workload {index}")


def random_grad(g: np.random.Generator, n: int, c: int, sigma: float = 2.0,
                outlier_frac: float = 0.0) -> np.ndarray:
    """Generic per-sample-scaled gradient for edge-case tests."""
    dH = (g.standard_normal((n, c)).astype(np.float32)
          * _lognormal_rows(g, n, sigma)[:, None])
    if outlier_frac > 0:
        dH[g.random(n) < outlier_frac] *= 100.0
    return dH
