"""The seeded generators: bf16 rounding agrees with torch's round-to-nearest-even
conversion, draws are deterministic, and a smaller batch is a prefix of the full one."""
import numpy as np
import torch

from paper_2509_05512_gb300 import inputs


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    a = np.concatenate([rng.standard_normal(100000).astype(np.float32),
                        np.array([0.0, -0.0, 1.0, 1.00390625, 1.01171875, 3.0e38, -1e-38],
                                 dtype=np.float32)])
    ours = inputs.to_bf16_bits(a)
    ref = torch.from_numpy(a).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(ours, ref)


def test_layer_inputs_deterministic_and_prefix():
    spec = inputs.small_layer("t", 4, 5, 6, 16, 32, 3, 1, 1, bias=True)
    a = inputs.layer_inputs(spec)
    b = inputs.layer_inputs(spec)
    c = inputs.layer_inputs(spec, n_images=2)
    for k in ("x", "wr", "wi", "wj", "wk", "bias", "scale", "shift"):
        np.testing.assert_array_equal(a[k], b[k])
    np.testing.assert_array_equal(a["x"][:2], c["x"])
    np.testing.assert_array_equal(a["wk"], c["wk"])
    assert a["x"].shape == (4, 5, 6, 16) and a["wr"].shape == (8, 3, 3, 4)


def test_config_shapes_and_flops():
    L = inputs.LAYERS
    assert (L["c2b"].Ho, L["c2b"].Wo) == (28, 28)
    assert abs(L["c1"].flops - 9.66e9) / 9.66e9 < 1e-3
    assert abs(L["c3b"].flops - 483.2e9) / 483.2e9 < 1e-3
    layers = inputs.backbone_layers()
    convs = [l for l in layers if l.kind == "conv"]
    assert len(convs) == 20
    assert sum(l.kind == "maxpool" for l in layers) == 1
    total = sum(l.spec.flops for l in convs)
    assert 9.0e11 < total < 1.0e12


def test_backbone_activation_variant():
    relu = inputs.backbone_layers(N=2, act=inputs.ACT_RELU)
    silu = inputs.backbone_layers(N=2, act=inputs.ACT_SILU)
    for a, b in zip(relu, silu):
        if a.kind != "conv":
            continue
        # shortcuts keep no activation; every other convolution switches
        if a.spec.act == inputs.ACT_NONE:
            assert b.spec.act == inputs.ACT_NONE and a.spec.kh == 1
        else:
            assert a.spec.act == inputs.ACT_RELU and b.spec.act == inputs.ACT_SILU
        assert a.spec.seed == b.spec.seed  # same weights


def test_grad_output_seeded_and_prefix():
    spec = inputs.small_layer("g", 4, 6, 5, 16, 32, 3, 2, 1, seed=(7, 3))
    a = inputs.grad_output(spec)
    assert a.shape == (4, spec.Ho, spec.Wo, 32) and a.dtype.name == "uint16"
    np.testing.assert_array_equal(a, inputs.grad_output(spec))      # same seed, same bits
    np.testing.assert_array_equal(a[:2], inputs.grad_output(spec, n_images=2))
    other = inputs.grad_output(inputs.small_layer("g", 4, 6, 5, 16, 32, 3, 2, 1, seed=(7, 4)))
    assert (a != other).any()


def test_round_bf16_of_the_checks():
    # the tests' fp64 -> bf16 rounding (nearest, ties to even) agrees with the input
    # quantiser on float32 values and rounds float64 values once, directly
    from tests._util import round_bf16
    rng = np.random.default_rng(1)
    a = np.concatenate([rng.standard_normal(100000).astype(np.float32) * 3,
                        np.array([0.0, 1.0, 1e-30, -7.5], dtype=np.float32)])
    want = (inputs.to_bf16_bits(a).astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    np.testing.assert_array_equal(round_bf16(a.astype(np.float64)), want)
    ulp = 2.0 ** -7
    assert round_bf16(1 + ulp / 2) == 1.0                        # tie -> even (down)
    assert round_bf16(1 + 3 * ulp / 2) == 1 + 2 * ulp            # tie -> even (up)
    assert round_bf16(1 + ulp / 2 + 2.0 ** -40) == 1 + ulp       # just above the tie
    assert round_bf16(-(1 + ulp / 2 + 2.0 ** -40)) == -(1 + ulp)
    assert round_bf16(255.9) == 256.0 and round_bf16(2.0 ** -130) == 2.0 ** -130


def test_bf16_reference_straddled_midpoint():
    # the other neighbour is accepted only for an exact value within 2^-16 of a midpoint
    from tests._util import bf16_reference
    ulp = 2.0 ** -5                      # bf16 spacing in [4, 8)
    mid = 4.0 + ulp / 2                  # between 4 and 4 + ulp
    ref = np.array([mid * (1 + 2.0 ** -30), mid * (1 + 2.0 ** -10), 5.0])
    got = np.array([4.0, 4.0, 5.0 + ulp])
    want = np.array([4.0, 4.0 + ulp, 5.0])
    np.testing.assert_array_equal(bf16_reference(got, ref), want)
