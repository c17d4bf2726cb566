"""Algorithmic work and storage of Q-CNN layers (Sec. 3.4, Table 1).

Table 1 counts, per image,
  conv  CNN  : d_t^2 C_t d_k^2 C_s                    multiply-adds
        Q-CNN: d_s^2 C_s K + d_t^2 C_t d_k^2 M        (table build + look-ups)
  FC    CNN  : C_s C_t
        Q-CNN: C_s K + C_t M
  bytes conv : 4 d_k^2 C_s C_t  vs  4 C_s K + d_k^2 M C_t log2(K) / 8
        FC   : 4 C_s C_t        vs  4 C_s K + M C_t log2(K) / 8
The paper counts one multiply-add as one FLOP.  Here the square sizes are
generalised to H x W input maps, Ho x Wo output maps and kh x kw kernels, and
M = C_s / C'_s is kept as a real number, which is how the paper's tables treat
settings such as C'_s = 3 on a 4096-wide layer (Table 7).

The same counts give the benchmark's algorithmic work per image:
  lut_entries  = H W M K   (each entry costs C'_s multiply-adds)
  lookups      = Ho Wo C_t kh kw M  (one fp32 load + one add each)
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from typing import Iterable, List, Optional, Tuple


@dataclass(frozen=True)
class LayerCost:
    dense_macs: float    # Table 1, CNN FLOPs (multiply-adds)
    lut_macs: float      # Table 1, first Q-CNN term
    lookups: float       # Table 1, second Q-CNN term
    lut_entries: float   # lut_macs / C'_s
    dense_bytes: float   # Table 1, CNN bytes
    q_bytes: float       # Table 1, Q-CNN bytes

    @property
    def q_macs(self) -> float:
        return self.lut_macs + self.lookups

    def __add__(self, o: "LayerCost") -> "LayerCost":
        return LayerCost(*(a + b for a, b in zip(self.astuple(), o.astuple())))

    def scale(self, f: float) -> "LayerCost":
        return LayerCost(*(a * f for a in self.astuple()))

    def astuple(self):
        return (self.dense_macs, self.lut_macs, self.lookups, self.lut_entries,
                self.dense_bytes, self.q_bytes)


ZERO = LayerCost(0, 0, 0, 0, 0, 0)


def conv_cost(Cs: int, Ct: int, H: int, W: int, kh: int, kw: int, Ho: int, Wo: int,
              Csp: float, K: int, groups: int = 1) -> LayerCost:
    """Table 1, convolutional row; a grouped layer is ``groups`` independent
    layers of Cs/groups inputs and Ct/groups outputs."""
    cs, ct = Cs / groups, Ct / groups
    M = cs / Csp
    dense = Ho * Wo * ct * kh * kw * cs
    lut = H * W * cs * K
    look = Ho * Wo * ct * kh * kw * M
    db = 4 * kh * kw * cs * ct
    qb = 4 * cs * K + kh * kw * M * ct * math.log2(K) / 8
    return LayerCost(dense, lut, look, lut / Csp, db, qb).scale(groups)


def fc_cost(Cs: int, Ct: int, Csp: float, K: int) -> LayerCost:
    """Table 1, fully-connected row."""
    M = Cs / Csp
    return LayerCost(Cs * Ct, Cs * K, Ct * M, Cs * K / Csp, 4 * Cs * Ct,
                     4 * Cs * K + M * Ct * math.log2(K) / 8)


def speedup(costs: Iterable[LayerCost]) -> float:
    tot = sum(costs, ZERO)
    return tot.dense_macs / tot.q_macs


def compression(costs: Iterable[LayerCost]) -> float:
    tot = sum(costs, ZERO)
    return tot.dense_bytes / tot.q_bytes


# ---------------------------------------------------------------------------
# Grouped AlexNet as used in the paper's experiments (Krizhevsky et al. 2012):
# conv2, conv4, conv5 have two groups.  Returns per-layer costs.
# ---------------------------------------------------------------------------
def alexnet_grouped(conv_csp: float, conv_k: int, fc_settings: List[Tuple[float, int]],
                    conv1_csp: float = 3, conv1_k: Optional[int] = None,
                    quantize_fc: bool = True) -> List[LayerCost]:
    """Per-layer costs of grouped AlexNet.  conv1 has only three input
    channels, so its sub-space is the whole RGB vector (C'_s = 3) with the
    same K as the other conv layers unless ``conv1_k`` is given."""
    k1 = conv_k if conv1_k is None else conv1_k
    layers = [
        conv_cost(3, 96, 227, 227, 11, 11, 55, 55, conv1_csp, k1),
        conv_cost(96, 256, 27, 27, 5, 5, 27, 27, conv_csp, conv_k, groups=2),
        conv_cost(256, 384, 13, 13, 3, 3, 13, 13, conv_csp, conv_k),
        conv_cost(384, 384, 13, 13, 3, 3, 13, 13, conv_csp, conv_k, groups=2),
        conv_cost(384, 256, 13, 13, 3, 3, 13, 13, conv_csp, conv_k, groups=2),
    ]
    if quantize_fc:
        dims = [(9216, 4096), (4096, 4096), (4096, 1000)]
        for (cs, ct), (csp, k) in zip(dims, fc_settings):
            layers.append(fc_cost(cs, ct, csp, k))
    return layers


def vgg16_conv(csp: float, k: int, conv1_csp: float = 3) -> List[LayerCost]:
    """The 13 conv layers of VGG-16 (3x3, pad 1) at 224 x 224 input."""
    spec = [(3, 64, 224), (64, 64, 224), (64, 128, 112), (128, 128, 112),
            (128, 256, 56), (256, 256, 56), (256, 256, 56),
            (256, 512, 28), (512, 512, 28), (512, 512, 28),
            (512, 512, 14), (512, 512, 14), (512, 512, 14)]
    out = []
    for i, (cs, ct, d) in enumerate(spec):
        out.append(conv_cost(cs, ct, d, d, 3, 3, d, d, conv1_csp if i == 0 else csp, k))
    return out
