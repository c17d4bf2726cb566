"""Seeded synthetic inputs shaped like the Q-CNN paper's workloads.

This module is shared by the tests, the smoke check and the benchmark, and it
is the only code that both the CUDA path and the float64 oracle see.  It draws
random numbers and describes layer shapes; it computes nothing of the method
(no look-up table, no response, no reconstruction).

The paper's inputs (ILSVRC-12 images, trained AlexNet / CaffeNet / CNN-S /
VGG-16 weights and their sub-codebooks, Sec. 4.2) are not available, so every
tensor here is drawn from a seeded numpy PCG64 generator, which gives the same
stream on x86 and Arm hosts:

  seed 0 -> layer inputs        seed 1 -> sub-codebooks D[m][k][j]
  seed 2 -> sub-codeword codes  seed 3 -> biases
Each layer of a network salts its streams with its index, and a test can salt
them further, so every array is independent and reproducible.

Layouts match the C library and the oracle:
  fc   : x [N, Cs] fp32, D [M, K, Csp] fp32, codes [M, Ct] uint8, bias [Ct] fp32
  conv : x [N, Cs, H, W] fp32, D [M, K, Csp] fp32, codes [Ct, kh*kw, M] uint8
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional, Sequence, Union

import numpy as np

SEED_X, SEED_D, SEED_CODES, SEED_BIAS = 0, 1, 2, 3


def rng(seed: int, *salt: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([seed, *salt])))


def normal(shape, std: float, seed: int, *salt: int) -> np.ndarray:
    """float32 samples of N(0, std^2) (std is a standard deviation)."""
    a = rng(seed, *salt).standard_normal(size=shape, dtype=np.float32)
    if std != 1.0:
        a *= np.float32(std)
    return a


def relu_normal(shape, seed: int, *salt: int) -> np.ndarray:
    """float32 samples of max(0, z), z ~ N(0, 1) -- a post-ReLU activation."""
    a = rng(seed, *salt).standard_normal(size=shape, dtype=np.float32)
    np.maximum(a, 0, out=a)
    return a


def uniform_codes(shape, K: int, seed: int, *salt: int) -> np.ndarray:
    """uint8 sub-codeword indices, uniform over [0, K)."""
    return rng(seed, *salt).integers(0, K, size=shape, dtype=np.uint8)


def sample_indices(n: int, k: int, seed: int, *salt: int) -> np.ndarray:
    """k indices drawn from range(n): distinct when k <= n, with repeats
    otherwise (the initial-centroid draw of a k-means run)."""
    return rng(seed, *salt).choice(n, size=k, replace=k > n).astype(np.int64)


def small_integers(shape, lo: int, hi: int, seed: int, *salt: int) -> np.ndarray:
    """float32 holding integers uniform in [lo, hi] -- every sum of a few
    thousand products of such values is exact in fp32 and in fp64."""
    return rng(seed, *salt).integers(lo, hi + 1, size=shape).astype(np.float32)


# --------------------------------------------------------------------------
# Layer descriptions
# --------------------------------------------------------------------------
@dataclass
class Conv:
    Cs: int
    Ct: int
    kh: int
    kw: int
    stride: int
    pad: int
    Csp: int
    K: int
    relu: bool = True
    cb_std: Optional[float] = None  # None -> He scale sqrt(2 / (kh*kw*Cs))
    bias_std: float = 0.1
    kind: str = field(default="conv", init=False)

    @property
    def M(self) -> int:
        return self.Cs // self.Csp

    def out_hw(self, H: int, W: int):
        return ((H + 2 * self.pad - self.kh) // self.stride + 1,
                (W + 2 * self.pad - self.kw) // self.stride + 1)


@dataclass
class FC:
    Cs: int
    Ct: int
    Csp: int
    K: int
    relu: bool = True
    cb_std: Optional[float] = None  # None -> He scale sqrt(2 / Cs)
    bias_std: float = 0.1
    kind: str = field(default="fc", init=False)

    @property
    def M(self) -> int:
        return self.Cs // self.Csp


@dataclass
class Pool:
    k: int
    s: int
    kind: str = field(default="maxpool", init=False)

    def out_hw(self, H: int, W: int):
        return (H - self.k) // self.s + 1, (W - self.k) // self.s + 1


Layer = Union[Conv, FC, Pool]


def layer_params(L: Layer, index: int, *salt: int) -> dict:
    """Draw D, codes and bias for one layer (empty dict for a pool)."""
    if isinstance(L, Pool):
        return {}
    if isinstance(L, Conv):
        std = L.cb_std if L.cb_std is not None else float(np.sqrt(2.0 / (L.kh * L.kw * L.Cs)))
        codes_shape = (L.Ct, L.kh * L.kw, L.M)
    else:
        std = L.cb_std if L.cb_std is not None else float(np.sqrt(2.0 / L.Cs))
        codes_shape = (L.M, L.Ct)
    return {
        "D": normal((L.M, L.K, L.Csp), std, SEED_D, index, *salt),
        "codes": uniform_codes(codes_shape, L.K, SEED_CODES, index, *salt),
        "bias": normal((L.Ct,), L.bias_std, SEED_BIAS, index, *salt),
    }


def oracle_layer_dict(L: Layer, params: dict) -> dict:
    """The dict form that ``oracle.net_forward`` takes (plain data, no maths)."""
    if isinstance(L, Pool):
        return {"kind": "maxpool", "k": L.k, "s": L.s}
    d = {"kind": L.kind, "D": params["D"], "codes": params["codes"],
         "bias": params.get("bias"), "relu": L.relu}
    if isinstance(L, Conv):
        d.update(kh=L.kh, kw=L.kw, stride=L.stride, pad=L.pad)
    return d


# --------------------------------------------------------------------------
# The five workloads (shapes from the paper's networks, Sec. 4.2, Tables 3-8)
# --------------------------------------------------------------------------
@dataclass
class Workload:
    name: str
    layers: List[Layer]
    in_shape: Sequence[int]        # per-image shape: (Cs,) or (C, H, W)
    x_dist: str                    # "normal" or "relu_normal"
    batches: Sequence[int]
    description: str = ""

    def input(self, N: int, *salt: int) -> np.ndarray:
        shape = (N, *self.in_shape)
        if self.x_dist == "normal":
            return normal(shape, 1.0, SEED_X, *salt)
        return relu_normal(shape, SEED_X, *salt)

    def params(self, *salt: int) -> List[dict]:
        return [layer_params(L, i, *salt) for i, L in enumerate(self.layers)]

    def shapes(self):
        """Per-layer (input shape, output shape) for one image."""
        out = []
        s = tuple(self.in_shape)
        for L in self.layers:
            if isinstance(L, FC):
                o = (L.Ct,)
            elif isinstance(L, Conv):
                o = (L.Ct, *L.out_hw(s[1], s[2]))
            else:
                o = (s[0], *L.out_hw(s[1], s[2]))
            out.append((s, o))
            s = o
        return out


def fc_layer() -> Workload:
    """Single PQ FC layer: 512 -> 256, C's = 4 (M = 128), K = 16, batch 8."""
    return Workload("fc_512x256_b8",
                    [FC(512, 256, 4, 16, relu=False, cb_std=0.5, bias_std=0.1)],
                    (512,), "normal", (8,),
                    "x ~ N(0,1); D ~ N(0, 0.5^2); codes U[0,16); bias ~ N(0, 0.1^2)")


def conv_layer() -> Workload:
    """Single PQ 3x3 conv: 64 x 56 x 56 -> 64, C's = 4 (M = 16), K = 128."""
    return Workload("conv3x3_64x56x56_b1",
                    [Conv(64, 64, 3, 3, 1, 1, 4, 128, relu=False, cb_std=0.05)],
                    (64, 56, 56), "relu_normal", (1,),
                    "x ~ ReLU(N(0,1)); D ~ N(0, 0.05^2); codes U[0,128); bias ~ N(0, 0.1^2)")


def vgg_stack() -> Workload:
    """VGG-16-shaped conv stack (conv3/conv4/conv5 blocks of VGG-16): five
    3x3 s1 p1 layers, C's = 8, K = 128, ReLU after each, 2x2/2 max-pool where
    the spatial size halves."""
    c = dict(Csp=8, K=128, relu=True, cb_std=0.05)
    layers: List[Layer] = [
        Conv(256, 256, 3, 3, 1, 1, **c),
        Conv(256, 256, 3, 3, 1, 1, **c),
        Pool(2, 2),
        Conv(256, 512, 3, 3, 1, 1, **c),
        Pool(2, 2),
        Conv(512, 512, 3, 3, 1, 1, **c),
        Conv(512, 512, 3, 3, 1, 1, **c),
    ]
    return Workload("vgg16_conv_stack", layers, (256, 56, 56), "relu_normal", (1, 32),
                    "x ~ ReLU(N(0,1)); D ~ N(0, 0.05^2); codes U[0,128); bias ~ N(0, 0.1^2)")


def alexnet_fc() -> Workload:
    """AlexNet fc6 / fc7 / fc8 shapes, C's = 4, K = 32 (ReLU after fc6, fc7)."""
    c = dict(Csp=4, K=32, cb_std=0.01)
    layers: List[Layer] = [FC(9216, 4096, relu=True, **c), FC(4096, 4096, relu=True, **c),
                           FC(4096, 1000, relu=False, **c)]
    return Workload("alexnet_fc678", layers, (9216,), "relu_normal", (1, 64, 256),
                    "x ~ ReLU(N(0,1)); D ~ N(0, 0.01^2); codes U[0,32); bias ~ N(0, 0.1^2)")


def alexnet() -> Workload:
    """Ungrouped (CaffeNet-style) AlexNet: conv1 11x11/4 (C's=3, K=128),
    conv2 5x5 p2, conv3-5 3x3 p1 (C's=4, K=128), 3x3/2 max-pool after conv1,
    conv2, conv5, then fc6-8 (C's=4, K=32); ReLU after every layer but fc8."""
    k = dict(K=128, relu=True)
    f = dict(Csp=4, K=32)
    layers: List[Layer] = [
        Conv(3, 96, 11, 11, 4, 0, Csp=3, **k),
        Pool(3, 2),
        Conv(96, 256, 5, 5, 1, 2, Csp=4, **k),
        Pool(3, 2),
        Conv(256, 384, 3, 3, 1, 1, Csp=4, **k),
        Conv(384, 384, 3, 3, 1, 1, Csp=4, **k),
        Conv(384, 256, 3, 3, 1, 1, Csp=4, **k),
        Pool(3, 2),
        FC(9216, 4096, relu=True, **f),
        FC(4096, 4096, relu=True, **f),
        FC(4096, 1000, relu=False, **f),
    ]
    return Workload("alexnet_qcnn", layers, (3, 227, 227), "normal", (1, 128),
                    "x ~ N(0,1) images; D ~ N(0, 2/fan_in) (He scale); "
                    "codes uniform; bias ~ N(0, 0.1^2)")


WORKLOADS = {w.name: w for w in (fc_layer(), conv_layer(), vgg_stack(), alexnet_fc(), alexnet())}
