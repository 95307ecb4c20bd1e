"""Seeded synthetic inputs for the quaternion convolution layers.

This module is shared by the CUDA path's tests and benchmark and by the oracle
checks.  It holds only random-number draws, the bfloat16 round-to-nearest-even
quantisation of those draws, and the layer shapes -- none of the quaternion
convolution arithmetic.  Both sides consume the identical values it returns.

Recipe (the paper's data sets are not available; these stand in for them):
  * activations ~ N(0, 1) (the backbone input ~ U(-1, 1) on 4 components),
  * each letter tensor W_r, W_i, W_j, W_k ~ N(0, 1 / (C_in * kh * kw)), C_in in
    real channels, so every real output has variance close to 1,
  * bias ~ N(0, 0.1^2) (fp32 layer only), IQBN scale ~ U(0.5, 1.5),
    IQBN shift ~ N(0, 0.1^2),
  * numpy PCG64 generators seeded with (config, layer, 0) for the activations
    (images drawn in batch order, so a smaller batch is a prefix of the full one)
    and (config, layer, 1) for the parameters, drawn in the order
    W_r, W_i, W_j, W_k, bias, scale, shift; a residual input uses (config, layer, 7),
    the output gradient of the backward pass ~ N(0, 1) uses (config, layer, 9).
Shapes follow the paper's workloads: CIFAR 32x32, ImageNet ResNet stages at
56/28/14/7, and a 640-px detector neck at stride 8/16.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace

import numpy as np

ACT_NONE, ACT_RELU, ACT_SILU = 0, 1, 2


def to_bf16_bits(a) -> np.ndarray:
    """Round float32 values to bfloat16 (nearest, ties to even); returns uint16 bits."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)
    rounding = ((u >> 16) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + rounding) >> 16).astype(np.uint16)


@dataclass(frozen=True)
class LayerSpec:
    name: str
    N: int
    H: int
    W: int
    Cin: int
    Cout: int
    kh: int
    kw: int
    stride: int
    pad: int
    act: int = ACT_RELU
    bias: bool = False
    iqbn: bool = True
    residual: bool = False
    dtype: str = "bf16"          # "bf16" or "f32"
    seed: tuple = (0, 0)
    x_dist: str = "normal"       # "normal" or "uniform"

    @property
    def Ho(self) -> int:
        return (self.H + 2 * self.pad - self.kh) // self.stride + 1

    @property
    def Wo(self) -> int:
        return (self.W + 2 * self.pad - self.kw) // self.stride + 1

    @property
    def flops(self) -> float:
        """Real-equivalent FLOPs: 2 * N * Ho * Wo * C_out * C_in * kh * kw."""
        return 2.0 * self.N * self.Ho * self.Wo * self.Cout * self.Cin * self.kh * self.kw

    @property
    def elem_bytes(self) -> int:
        return 2 if self.dtype == "bf16" else 4

    @property
    def algorithmic_bytes(self) -> float:
        """x read once (only the sampled pixels for a 1x1 strided layer), compact
        weights, three fp32 per-channel vectors, y written (+ residual read)."""
        e = self.elem_bytes
        if self.kh == 1 and self.kw == 1 and self.pad == 0:
            xb = self.N * self.Ho * self.Wo * self.Cin * e
        else:
            xb = self.N * self.H * self.W * self.Cin * e
        wb = self.Cout * self.Cin * self.kh * self.kw * e / 4
        pb = 3 * self.Cout * 4
        yb = self.N * self.Ho * self.Wo * self.Cout * e
        rb = yb if self.residual else 0
        return xb + wb + pb + yb + rb


LAYERS = {
    # fp32 single layer, bias, no IQBN
    "c0": LayerSpec("c0", 2, 8, 8, 16, 16, 3, 3, 1, 1, act=ACT_NONE, bias=True, iqbn=False,
                    dtype="f32", seed=(0, 0)),
    # CIFAR-shaped layer
    "c1": LayerSpec("c1", 128, 32, 32, 64, 64, 3, 3, 1, 1, seed=(1, 0)),
    # ImageNet ResNet stage layers
    "c2a": LayerSpec("c2a", 64, 56, 56, 256, 256, 3, 3, 1, 1, seed=(2, 0)),
    "c2b": LayerSpec("c2b", 64, 56, 56, 256, 512, 3, 3, 2, 1, seed=(2, 1)),
    # detection neck (640-px input at stride 8 and 16)
    "c3a": LayerSpec("c3a", 16, 80, 80, 512, 1024, 1, 1, 1, 0, seed=(3, 0)),
    "c3b": LayerSpec("c3b", 16, 40, 40, 1024, 1024, 3, 3, 1, 1, seed=(3, 1)),
}

# Workload groups: the small fp32 check layer, the CIFAR-shaped layer, the two
# ImageNet ResNet-stage layers, the two detection-neck layers.
CONFIGS = {
    "small": ["c0"],
    "cifar": ["c1"],
    "imagenet_stage": ["c2a", "c2b"],
    "detection_neck": ["c3a", "c3b"],
}


def layer_inputs(spec: LayerSpec, n_images: int | None = None) -> dict:
    """Draw the inputs of one layer.  bf16 tensors are returned as uint16 bit
    patterns, fp32 tensors as float32; per-channel vectors are float32 or None.

    ``n_images`` limits the batch that is drawn; the result is a prefix of the
    full batch and the parameters are unchanged."""
    N = spec.N if n_images is None else n_images
    Qin, Qout = spec.Cin // 4, spec.Cout // 4
    xrng = np.random.default_rng(spec.seed + (0,))
    xshape = (N, spec.H, spec.W, spec.Cin)
    if spec.x_dist == "uniform":
        x = xrng.uniform(-1.0, 1.0, size=xshape).astype(np.float32)
    else:
        x = xrng.standard_normal(xshape, dtype=np.float32)
    rng = np.random.default_rng(spec.seed + (1,))
    wstd = 1.0 / np.sqrt(spec.Cin * spec.kh * spec.kw)
    wshape = (Qout, spec.kh, spec.kw, Qin)
    w = [(rng.standard_normal(wshape, dtype=np.float32) * np.float32(wstd)) for _ in range(4)]
    bias = (rng.standard_normal(spec.Cout, dtype=np.float32) * np.float32(0.1)
            if spec.bias else None)
    if spec.iqbn:
        scale = rng.uniform(0.5, 1.5, size=spec.Cout).astype(np.float32)
        shift = (rng.standard_normal(spec.Cout, dtype=np.float32) * np.float32(0.1))
    else:
        scale = shift = None
    out = {"spec": spec, "bias": bias, "scale": scale, "shift": shift}
    if spec.dtype == "bf16":
        out["x"] = to_bf16_bits(x)
        out["wr"], out["wi"], out["wj"], out["wk"] = (to_bf16_bits(t) for t in w)
    else:
        out["x"] = x
        out["wr"], out["wi"], out["wj"], out["wk"] = w
    if spec.residual:
        rr = np.random.default_rng(spec.seed + (7,))
        r = rr.standard_normal((N, spec.Ho, spec.Wo, spec.Cout), dtype=np.float32)
        out["residual"] = to_bf16_bits(r) if spec.dtype == "bf16" else r
    else:
        out["residual"] = None
    return out


def grad_output(spec: LayerSpec, n_images: int | None = None) -> np.ndarray:
    """The output gradient dy [N, Ho, Wo, C_out] for the backward pass of one layer, as
    bf16 bits (a prefix of the full batch for a smaller ``n_images``)."""
    N = spec.N if n_images is None else n_images
    rng = np.random.default_rng(spec.seed + (9,))
    dy = rng.standard_normal((N, spec.Ho, spec.Wo, spec.Cout), dtype=np.float32)
    return to_bf16_bits(dy)


def small_layer(name: str, N: int, H: int, W: int, Cin: int, Cout: int, k: int, stride: int,
                pad: int, *, kw: int | None = None, act=ACT_RELU, bias=False, iqbn=True,
                residual=False, dtype="bf16", seed=(100, 0)) -> LayerSpec:
    """A LayerSpec for tests (same value recipe as the configured layers)."""
    return LayerSpec(name, N, H, W, Cin, Cout, k, k if kw is None else kw, stride, pad,
                     act=act, bias=bias, iqbn=iqbn, residual=residual, dtype=dtype, seed=seed)


# ---------------------------------------------------------------------------
# ResNet-18-style quaternion backbone, 224x224x4 input
# ---------------------------------------------------------------------------

@dataclass(frozen=True)
class BackboneLayer:
    kind: str                 # "conv" or "maxpool"
    spec: LayerSpec | None = None
    src: int = -1             # index of the layer whose output feeds this one (-1: image)
    res: int | None = None    # index of the layer whose output is added before act
    k: int = 0
    stride: int = 0
    pad: int = 0


def backbone_layers(N: int = 256, H: int = 224, seed: int = 4, act: int = ACT_RELU) -> list:
    """Layer list of the ResNet-18-style backbone: 7x7/2 stem, 3x3/2 max pool applied
    per real channel, 4 stages x 2 basic blocks at 64/128/256/512 real channels with
    1x1/2 shortcut convolutions; every convolution is a quaternion convolution with
    fused IQBN; the activation `act` (ReLU by default, SiLU for the detector-style
    variant) everywhere except on the shortcut, and on the second convolution of a block
    after the block input (or shortcut) is added."""
    layers = []
    idx = [0]
    block_act = act

    def conv(src, Hin, Cin, Cout, k, s, p, act=block_act, res=None):
        spec = LayerSpec("bb%d" % idx[0], N, Hin, Hin, Cin, Cout, k, k, s, p, act=act,
                         residual=False, seed=(seed, idx[0]),
                         x_dist="uniform" if src == -1 else "normal")
        layers.append(BackboneLayer("conv", spec, src=src, res=res))
        idx[0] += 1
        return len(layers) - 1, spec.Ho

    cur, Hc = conv(-1, H, 4, 64, 7, 2, 3)
    layers.append(BackboneLayer("maxpool", None, src=cur, k=3, stride=2, pad=1))
    idx[0] += 1
    cur, Hc = len(layers) - 1, (Hc + 2 - 3) // 2 + 1
    C = 64
    for width in (64, 128, 256, 512):
        for b in range(2):
            s = 2 if (b == 0 and width != 64) else 1
            inp, Hin = cur, Hc
            a, Ha = conv(inp, Hin, C, width, 3, s, 1)
            if s != 1 or C != width:
                sc, _ = conv(inp, Hin, C, width, 1, s, 0, act=ACT_NONE)
            else:
                sc = inp
            cur, Hc = conv(a, Ha, width, width, 3, 1, 1, res=sc)
            C = width
    return layers


def backbone_input(N: int = 256, H: int = 224, seed: int = 4, n_images: int | None = None):
    """Backbone image batch, 4 quaternion components per pixel ~ U(-1, 1), bf16 bits."""
    rng = np.random.default_rng((seed, 1000))
    x = rng.uniform(-1.0, 1.0, size=(N, H, H, 4)).astype(np.float32)
    if n_images is not None:
        x = x[:n_images]
    return to_bf16_bits(x)


def backbone_rgb(N: int = 256, H: int = 224, seed: int = 4, n_images: int | None = None):
    """Backbone RGB image batch for the Eq. 4 input mapping, fp32 [N][H][H][3] ~ U(0, 1)."""
    rng = np.random.default_rng((seed, 1001))
    rgb = rng.uniform(0.0, 1.0, size=(N, H, H, 3)).astype(np.float32)
    return rgb if n_images is None else rgb[:n_images]


def backbone_params(layer: BackboneLayer) -> dict:
    """Weights and IQBN vectors of one backbone convolution (no activations drawn)."""
    spec = layer.spec
    rng = np.random.default_rng(spec.seed + (1,))
    Qin, Qout = spec.Cin // 4, spec.Cout // 4
    wstd = 1.0 / np.sqrt(spec.Cin * spec.kh * spec.kw)
    wshape = (Qout, spec.kh, spec.kw, Qin)
    w = [to_bf16_bits(rng.standard_normal(wshape, dtype=np.float32) * np.float32(wstd))
         for _ in range(4)]
    scale = rng.uniform(0.5, 1.5, size=spec.Cout).astype(np.float32)
    shift = rng.standard_normal(spec.Cout, dtype=np.float32) * np.float32(0.1)
    return {"wr": w[0], "wi": w[1], "wj": w[2], "wk": w[3], "bias": None, "scale": scale,
            "shift": shift}
