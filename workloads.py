"""Seeded synthetic weight sets shaped like the paper's models.

This module holds only input generation (shapes, initialisers, seeds) and none
of the regularizer's arithmetic; both the oracle and the CUDA path are fed from
it.  The paper trains on ImageNet-1K and FineWeb-Edu from timm / TorchVision /
OLMo checkpoints (Sec. 4, App. D, App. F); none of those are available, so
these seeded random weight sets with the models' matrix shapes and the stated
initialisation recipes stand in for them.

Shapes (conv kernels use the (C_out, C_in*k*k) view of App. D.1):

* ``cfg1``          8 independent 256 x 256, N(0, 1/256).
* ``resnet18``      21 matrices: stem 64x147; layer1 4 x 64x576; layer2 128x576,
                    3 x 128x1152, 128x64 (1x1 downsample); layer3 256x1152,
                    3 x 256x2304, 256x128; layer4 512x2304, 3 x 512x4608, 512x256;
                    fc 1000x512.  Kaiming normal: std sqrt(2/fan_out) for convs
                    (fan_out = C_out*k*k), sqrt(2/fan_in) for the fc.
* ``vit_b16``       12 blocks x {qkv 2304x768, proj 768x768, fc1 3072x768,
                    fc2 768x3072}: truncated normal std 0.02 cut at +-2 std,
                    plus a rank-32 spike 0.5 * U32 V32^T (orthonormal U, V from
                    QR of Gaussian matrices).
* ``vit_l16``       24 blocks x {3072x1024, 1024x1024, 4096x1024, 1024x4096},
                    same recipe.
* ``decoder_560m``  24 layers x {q 1280x1280, k 320x1280, v 320x1280,
                    o 1280x1280, gate 3456x1280, up 3456x1280, down 1280x3456},
                    N(0, 0.02^2) (GQA, 20 query / 5 key-value heads of dim 64).
* ``decoder_560m_mha``  the same with k, v 1280x1280 (multi-head attention).
* ``vit_ladder_<name>``  the ViT scaling ladder of the paper's ViT configuration
                    table (appendix "Scaling Up with Vision Transformers"):
                    embed dim d and depth of vit_ti 192x12, vit_256 256x12,
                    vit_s 384x12, vit_512 512x12, vit_b 768x12, vit_b24 768x24,
                    vit_960_24 960x24, vit_l 1024x24, vit_1152_28 1152x28,
                    vit_h 1280x32; MLP ratio 4; blocks as for ``vit_b16``.

Matrix i of weight set number c (the order of ``WEIGHT_SETS``) is drawn in
fp64 from ``numpy.random.default_rng(1000 * c + i)`` and rounded to fp32.
"""

from __future__ import annotations

import numpy as np


def _resnet18():
    out = []
    out.append(((64, 147), ("kaiming_fan_out", 64 * 49)))
    for _ in range(4):
        out.append(((64, 576), ("kaiming_fan_out", 64 * 9)))
    out.append(((128, 576), ("kaiming_fan_out", 128 * 9)))
    for _ in range(3):
        out.append(((128, 1152), ("kaiming_fan_out", 128 * 9)))
    out.append(((128, 64), ("kaiming_fan_out", 128)))
    out.append(((256, 1152), ("kaiming_fan_out", 256 * 9)))
    for _ in range(3):
        out.append(((256, 2304), ("kaiming_fan_out", 256 * 9)))
    out.append(((256, 128), ("kaiming_fan_out", 256)))
    out.append(((512, 2304), ("kaiming_fan_out", 512 * 9)))
    for _ in range(3):
        out.append(((512, 4608), ("kaiming_fan_out", 512 * 9)))
    out.append(((512, 256), ("kaiming_fan_out", 512)))
    out.append(((1000, 512), ("kaiming_fan_in", 512)))
    return out


def _vit(blocks, d, hidden):
    spec = ("trunc_normal_spike", 0.02)
    out = []
    for _ in range(blocks):
        out += [((3 * d, d), spec), ((d, d), spec), ((hidden, d), spec), ((d, hidden), spec)]
    return out


def _decoder(layers, d, kv, ffn):
    spec = ("normal", 0.02)
    out = []
    for _ in range(layers):
        out += [((d, d), spec), ((kv, d), spec), ((kv, d), spec), ((d, d), spec),
                ((ffn, d), spec), ((ffn, d), spec), ((d, ffn), spec)]
    return out


WEIGHT_SETS = {
    "cfg1": [((256, 256), ("normal", 1.0 / 16.0))] * 8,
    "resnet18": _resnet18(),
    "vit_b16": _vit(12, 768, 3072),
    "vit_l16": _vit(24, 1024, 4096),
    "decoder_560m": _decoder(24, 1280, 320, 3456),
    "decoder_560m_mha": _decoder(24, 1280, 1280, 3456),
}

# ViT scaling ladder (appended: the seeds of the sets above are unchanged).
VIT_LADDER = [("vit_ti", 192, 12), ("vit_256", 256, 12), ("vit_s", 384, 12), ("vit_512", 512, 12),
              ("vit_b", 768, 12), ("vit_b24", 768, 24), ("vit_960_24", 960, 24), ("vit_l", 1024, 24),
              ("vit_1152_28", 1152, 28), ("vit_h", 1280, 32)]
for _name, _d, _depth in VIT_LADDER:
    WEIGHT_SETS["vit_ladder_" + _name] = _vit(_depth, _d, 4 * _d)

SET_INDEX = {name: i for i, name in enumerate(WEIGHT_SETS)}


def shapes(name: str):
    """[(m, n), ...] of a weight set."""
    return [s for s, _ in WEIGHT_SETS[name]]


def _draw(rng, shape, spec):
    kind = spec[0]
    m, n = shape
    if kind == "normal":
        return rng.normal(0.0, spec[1], size=shape)
    if kind == "kaiming_fan_out" or kind == "kaiming_fan_in":
        return rng.normal(0.0, np.sqrt(2.0 / spec[1]), size=shape)
    if kind == "trunc_normal_spike":
        std = spec[1]
        W = rng.normal(0.0, std, size=shape)
        bad = np.abs(W) > 2.0 * std
        while bad.any():
            W[bad] = rng.normal(0.0, std, size=int(bad.sum()))
            bad = np.abs(W) > 2.0 * std
        r = min(32, m, n)
        U, _ = np.linalg.qr(rng.normal(size=(m, r)))
        V, _ = np.linalg.qr(rng.normal(size=(n, r)))
        return W + 0.5 * (U @ V.T)
    raise ValueError(kind)


def generate_one(name: str, i: int) -> np.ndarray:
    """Matrix i of weight set ``name`` as a C-contiguous fp32 array."""
    shape, spec = WEIGHT_SETS[name][i]
    rng = np.random.default_rng(1000 * SET_INDEX[name] + i)
    return np.ascontiguousarray(_draw(rng, shape, spec).astype(np.float32))


def generate(name: str, indices=None):
    """All (or the selected) matrices of a weight set, fp32."""
    idx = range(len(WEIGHT_SETS[name])) if indices is None else indices
    return [generate_one(name, i) for i in idx]


def random_matrix(shape, seed: int, std: float = 1.0) -> np.ndarray:
    """A plain N(0, std^2) fp32 test matrix from ``default_rng(seed)``."""
    rng = np.random.default_rng(seed)
    return np.ascontiguousarray(rng.normal(0.0, std, size=shape).astype(np.float32))
