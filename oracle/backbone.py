"""fp64 oracle of the ResNet-18-style quaternion backbone (TEST INFRASTRUCTURE ONLY:
used by tests/ and by the CPU legs of bench.py, never by the product path).

The layer list and the seeded parameters come from the input-generator module; every
layer is computed by the oracle's quaternion convolution (Eq. 5, IQBN inference
epilogue of Eq. 11-12) or its component-wise max pooling (QSPPF rule, Sec. III-D).
"""
from __future__ import annotations

import numpy as np

from . import ACT_NONE, bf16_bits_to_f64, maxpool2d, qconv2d


def layer_forward(layer, params, x, residual=None):
    """One backbone layer on float64 input x [N, H, W, C]."""
    if layer.kind == "maxpool":
        return maxpool2d(x, k=layer.k, stride=layer.stride, pad=layer.pad)
    s = layer.spec
    w = [bf16_bits_to_f64(params[k]) for k in ("wr", "wi", "wj", "wk")]
    return qconv2d(x, *w, stride=s.stride, pad=s.pad, bias=None, scale=params["scale"],
                   shift=params["shift"], residual=residual, act=s.act)


def forward(layers, params, x_bits, keep=False):
    """Whole backbone on bf16 input bits; returns the last output (and every output when
    keep=True).  Intermediate values stay in float64 (no rounding between layers)."""
    outs = []
    x0 = bf16_bits_to_f64(x_bits)
    for i, L in enumerate(layers):
        x = x0 if L.src == -1 else outs[L.src]
        res = outs[L.res] if (L.kind == "conv" and L.res is not None) else None
        outs.append(layer_forward(L, params[i], x, res))
    return (outs[-1], outs) if keep else outs[-1]
