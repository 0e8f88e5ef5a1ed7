"""Seeded synthetic workloads for pattern- and connectivity-pruned 3x3 conv.

This module only draws inputs: pattern sets, per-kernel pattern choices,
connectivity masks, pruned weights, biases, activations, and the layer lists of
the five benchmark workloads.  It holds none of the method's arithmetic (no
packing, reordering or convolution), so both the CUDA path and the CPU oracle
can take their inputs from it.

Readings of unstated details (all seeded with numpy's PCG64 ``default_rng``):
  * the 8 fixed patterns: the 8 neighbours of the centre tap in ring order
    0,1,2,5,8,7,6,3; pattern s = centre + ring[s], ring[s+1], ring[s+2];
  * a seed-chosen set of P patterns: the 56 neighbour triples in lexicographic
    order, P of them drawn without replacement, kept in ascending order;
  * "keeps a random X% of kernels": exactly round(X * Co * Ci) kernels, the
    first ones of a random permutation of the (o, i) grid;
  * per-kernel pattern: uniform over the set, drawn for every kernel;
  * draw order per layer: pattern ids, mask, dense weights, bias; the input
    activation is drawn last.  Pruned taps are then set to zero.
"""
from __future__ import annotations

import itertools
from dataclasses import dataclass, field
from typing import List, Optional

import numpy as np

CENTRE = 4
RING = (0, 1, 2, 5, 8, 7, 6, 3)
NEIGHBOURS = (0, 1, 2, 3, 5, 6, 7, 8)


def ring8_patterns() -> np.ndarray:
    """The fixed set of 8 patterns: centre plus 3 consecutive ring neighbours."""
    out = []
    for s in range(8):
        taps = sorted({CENTRE, RING[s], RING[(s + 1) % 8], RING[(s + 2) % 8]})
        out.append(taps)
    return np.array(out, dtype=np.uint8)


def all_centre_patterns() -> np.ndarray:
    """All 56 patterns made of the centre plus 3 of the 8 neighbours, lexicographic."""
    return np.array([sorted(c + (CENTRE,)) for c in itertools.combinations(NEIGHBOURS, 3)], dtype=np.uint8)


def seeded_patterns(rng: np.random.Generator, P: int) -> np.ndarray:
    allp = all_centre_patterns()
    idx = np.sort(rng.choice(len(allp), size=P, replace=False))
    return allp[idx].copy()


@dataclass
class PrunedLayer:
    """A pattern- and connectivity-pruned 3x3 layer as a user would hand it over."""

    w: np.ndarray  # [Co][Ci][9] float32, zero outside the kept taps
    mask: np.ndarray  # [Co][Ci] uint8
    pattern_ids: np.ndarray  # [Co][Ci] uint8 (the drawn pattern of every kernel)
    taps: np.ndarray  # [P][4] uint8
    bias: Optional[np.ndarray]  # [Co] float32 or None

    @property
    def Co(self) -> int:
        return self.w.shape[0]

    @property
    def Ci(self) -> int:
        return self.w.shape[1]

    @property
    def nk(self) -> int:
        return int(self.mask.sum())


@dataclass
class DenseLayer:
    """An unpruned 3x3 layer (all 9 taps of all kernels)."""

    w: np.ndarray  # [Co][Ci][9] float32
    bias: Optional[np.ndarray]

    @property
    def Co(self) -> int:
        return self.w.shape[0]

    @property
    def Ci(self) -> int:
        return self.w.shape[1]


def _nonzero_normal(rng: np.random.Generator, std: float, shape) -> np.ndarray:
    """float32 normal draws with exact zeros redrawn (a zero would hide a kept tap)."""
    w = (rng.standard_normal(shape) * std).astype(np.float32)
    bad = w == 0
    while bad.any():
        w[bad] = (rng.standard_normal(int(bad.sum())) * std).astype(np.float32)
        bad = w == 0
    return w


def make_pruned_layer(rng: np.random.Generator, Co: int, Ci: int, taps: np.ndarray, keep: float, w_std: float,
                      bias_std: Optional[float]) -> PrunedLayer:
    P = taps.shape[0]
    pattern_ids = rng.integers(0, P, size=(Co, Ci)).astype(np.uint8)
    nk = int(np.floor(keep * Co * Ci + 0.5))
    order = rng.permutation(Co * Ci)
    mask = np.zeros(Co * Ci, np.uint8)
    mask[order[:nk]] = 1
    mask = mask.reshape(Co, Ci)
    w = _nonzero_normal(rng, w_std, (Co, Ci, 9))
    keep_tap = np.zeros((Co, Ci, 9), bool)
    for p in range(P):
        sel = (pattern_ids == p) & (mask == 1)
        for t in taps[p]:
            keep_tap[:, :, t] |= sel
    w = np.where(keep_tap, w, np.float32(0)).astype(np.float32)
    bias = None if bias_std is None else (rng.standard_normal(Co) * bias_std).astype(np.float32)
    return PrunedLayer(w, mask, pattern_ids, taps.astype(np.uint8), bias)


def make_dense_layer(rng: np.random.Generator, Co: int, Ci: int, w_std: float, bias_std: Optional[float]) -> DenseLayer:
    w = _nonzero_normal(rng, w_std, (Co, Ci, 9))
    bias = None if bias_std is None else (rng.standard_normal(Co) * bias_std).astype(np.float32)
    return DenseLayer(w, bias)


def he_std(Ci: int) -> float:
    return float(np.sqrt(2.0 / (9.0 * Ci)))


# ----------------------------------------------------------------------------
# Network descriptions.  An op is one conv (pruned or dense) with its fused
# epilogue: optional residual add of an earlier activation, ReLU, 2x2 max pool.
# Activation 0 is the network input; op k writes activation k + 1.
# ----------------------------------------------------------------------------


@dataclass
class Op:
    layer: object  # PrunedLayer or DenseLayer
    relu: bool = False
    pool: bool = False
    skip_from: int = -1  # index of the activation added before the ReLU, -1 = none


@dataclass
class Net:
    name: str
    x: np.ndarray  # [N][C][H][W] float32 input
    ops: List[Op] = field(default_factory=list)

    def surviving_flops(self) -> int:
        """2 * (pattern taps of kept kernels, or 9 taps for dense layers) * pixels, per op, summed."""
        N, _, H, W = self.x.shape
        total = 0
        for op in self.ops:
            L = op.layer
            taps = 4 * L.nk if isinstance(L, PrunedLayer) else 9 * L.Co * L.Ci
            total += 2 * N * H * W * taps
            if op.pool:
                H //= 2
                W //= 2
        return total


def cfg0_single(seed: int = 0) -> Net:
    """1x16x32x32, 16->16, 8 fixed patterns, keep 0.5, w~N(0,0.1), b~N(0,0.01), x~U(-1,1)."""
    rng = np.random.default_rng(seed)
    L = make_pruned_layer(rng, 16, 16, ring8_patterns(), 0.5, 0.1, 0.01)
    x = rng.uniform(-1, 1, size=(1, 16, 32, 32)).astype(np.float32)
    return Net("single_layer_16x32x32", x, [Op(L)])


VGG16 = [64, 64, "P", 128, 128, "P", 256, 256, 256, "P", 512, 512, 512, "P", 512, 512, 512]


def cfg1_vgg16(seed: int = 0) -> Net:
    """VGG-16 conv trunk at 3x224x224: 13 pruned convs (bias+ReLU), 4 fused pools; conv1 keeps all kernels."""
    rng = np.random.default_rng(seed)
    taps = ring8_patterns()
    ops: List[Op] = []
    ci = 3
    for item in VGG16:
        if item == "P":
            ops[-1].pool = True
            continue
        co = int(item)
        keep = 1.0 if not ops else 0.3
        L = make_pruned_layer(rng, co, ci, taps, keep, 2.25 * he_std(ci), 0.01)
        ops.append(Op(L, relu=True))
        ci = co
    x = rng.uniform(0, 1, size=(1, 3, 224, 224)).astype(np.float32)
    return Net("vgg16_trunk_224", x, ops)


def cfg2_style(seed: int = 0) -> Net:
    """Style-transfer residual trunk: 5 blocks of two 128->128 pruned convs at 128x128, keep 0.25, no bias."""
    rng = np.random.default_rng(seed)
    taps = ring8_patterns()
    ops: List[Op] = []
    for b in range(5):
        La = make_pruned_layer(rng, 128, 128, taps, 0.25, 0.05, None)
        Lb = make_pruned_layer(rng, 128, 128, taps, 0.25, 0.05, None)
        block_in = len(ops)  # activation index feeding this block
        ops.append(Op(La, relu=True))
        ops.append(Op(Lb, relu=False, skip_from=block_in))
    x = rng.uniform(-1, 1, size=(1, 128, 128, 128)).astype(np.float32)
    return Net("style_residual_128x128", x, ops)


def cfg3_vdsr(seed: int = 0, H: int = 720, W: int = 1280) -> Net:
    """VDSR-shaped stack on 1x1x720x1280: dense 1->64, 18 pruned 64->64 (keep 0.4), dense 64->1, + input."""
    rng = np.random.default_rng(seed)
    taps = ring8_patterns()
    ops: List[Op] = [Op(make_dense_layer(rng, 64, 1, he_std(1), 0.01), relu=True)]
    for _ in range(18):
        ops.append(Op(make_pruned_layer(rng, 64, 64, taps, 0.4, he_std(64), 0.01), relu=True))
    ops.append(Op(make_dense_layer(rng, 1, 64, he_std(64), 0.01), relu=False, skip_from=0))
    x = rng.uniform(0, 1, size=(1, 1, H, W)).astype(np.float32)
    return Net("vdsr_720x1280", x, ops)


SWEEP_C = (64, 128, 256, 512)
SWEEP_P = (4, 8, 12)
SWEEP_KEEP = (0.2, 0.35, 0.5, 1.0)


def cfg4_point(C: int, P: int, keep: float, seed: int = 0, N: int = 8, H: int = 56, W: int = 56) -> Net:
    """One point of the sweep: batch 8, 56x56, C->C, P seed-chosen patterns, bias, no activation."""
    rng = np.random.default_rng(seed)
    taps = seeded_patterns(rng, P)
    L = make_pruned_layer(rng, C, C, taps, keep, 0.05, 0.01)
    x = rng.uniform(-1, 1, size=(N, C, H, W)).astype(np.float32)
    return Net(f"sweep_C{C}_P{P}_keep{keep}", x, [Op(L)])


def cfg4_points():
    return [(C, P, k) for C in SWEEP_C for P in SWEEP_P for k in SWEEP_KEEP]


def small_random_layer(rng: np.random.Generator, Co: int, Ci: int, P: int = 8, keep: float = 0.5,
                       ring: bool = True, w_std: float = 0.1, bias: bool = True) -> PrunedLayer:
    taps = ring8_patterns()[:P] if ring else seeded_patterns(rng, P)
    return make_pruned_layer(rng, Co, Ci, taps, keep, w_std, 0.01 if bias else None)


def integer_layer(rng: np.random.Generator, Co: int, Ci: int, taps: np.ndarray, keep: float) -> PrunedLayer:
    """A pruned layer with small nonzero integer weights in [-4, 4] and integer bias in [-8, 8]:
    with integer inputs every partial sum is an exactly representable integer in fp32."""
    L = make_pruned_layer(rng, Co, Ci, taps, keep, 1.0, 1.0)
    vals = rng.integers(1, 5, size=L.w.shape) * rng.choice([-1, 1], size=L.w.shape)
    L.w = np.where(L.w != 0, vals, 0).astype(np.float32)
    L.bias = rng.integers(-8, 9, size=Co).astype(np.float32)
    return L
