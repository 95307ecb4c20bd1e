"""GPU parity of the Poincare RGB -> quaternion mapping (Eq. 4) against the fp64 oracle
(`oracle.poincare`), through the C ABI entry point quan_poincare_fwd, and the mapping
feeding the 4-channel stem convolution."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2509_05512_gb300 import build, inputs, quan
from tests._util import BF16_HALF_ULP, assert_bf16_close, out_f64, to_dev, to_dev_f32

pytestmark = pytest.mark.gpu

# bf16 round-to-nearest-even (7 explicit mantissa bits): |rounded - exact| is at most half
# an ulp, <= 2^-8 |exact| for normal values; the fp32 evaluation before the rounding adds a
# few fp32 ulps
BF16_REL = BF16_HALF_ULP * 1.001
ABS_SLACK = 1e-6


@pytest.fixture(scope="module", autouse=True)
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build_library()
    yield quan.load()


def gpu_map(rgb_np, offset=0):
    """Map on the GPU; `offset` bf16 elements of misalignment for the output."""
    rgb = torch.from_numpy(np.ascontiguousarray(rgb_np, dtype=np.float32)).cuda()
    n = rgb.numel() // 3
    buf = torch.full((4 * n + offset + 8,), float("nan"), dtype=torch.bfloat16, device="cuda")
    out = buf[offset:offset + 4 * n].view(rgb_np.shape[:-1] + (4,))
    quan.poincare(rgb, out=out)
    torch.cuda.synchronize()
    assert torch.isnan(buf[offset + 4 * n:].float()).all()  # nothing written past the end
    return out_f64(out)


def check_elementwise(got, ref):
    err = np.abs(got - ref)
    bound = BF16_REL * np.abs(ref) + ABS_SLACK
    assert (err <= bound).all(), "max excess %.3e" % (err - bound).max()


@pytest.mark.parametrize("offset", [0, 1])
def test_poincare_matches_oracle(offset):
    rng = np.random.default_rng(40)
    rgb = rng.uniform(-1.0, 1.0, size=(2, 37, 29, 3))  # odd pixel count
    rgb32 = rgb.astype(np.float32)
    got = gpu_map(rgb32, offset)
    check_elementwise(got, oracle.poincare(rgb32.astype(np.float64)))


def test_poincare_unit_norm_and_special_values():
    rgb = np.array([[0, 0, 0], [1, 0, 0], [0, 1, 0], [0, 0, 1], [0.5, -0.5, 2.0],
                    [-3.0, 4.0, 0.0]], dtype=np.float32)
    got = gpu_map(rgb)
    np.testing.assert_array_equal(got[:4], [[1, 0, 0, 0], [0, 1, 0, 0], [0, 0, 1, 0],
                                            [0, 0, 0, 1]])
    check_elementwise(got, oracle.poincare(rgb.astype(np.float64)))
    np.testing.assert_allclose(np.linalg.norm(got, axis=-1), 1.0, atol=2 * BF16_HALF_ULP)


def test_poincare_image_batch_full_size():
    # the backbone's input size: N = 256 images of 224 x 224
    rng = np.random.default_rng(41)
    rgb = rng.uniform(0.0, 1.0, size=(256, 224, 224, 3)).astype(np.float32)
    got = gpu_map(rgb)
    idx = rng.integers(0, rgb.size // 3, size=4096)
    flat_rgb, flat_got = rgb.reshape(-1, 3), got.reshape(-1, 4)
    check_elementwise(flat_got[idx], oracle.poincare(flat_rgb[idx].astype(np.float64)))
    assert np.isfinite(flat_got).all()


def test_poincare_zero_pixels_is_a_no_op():
    quan.quan_poincare_fwd(None, 0, None)


def test_poincare_feeds_the_stem():
    # RGB -> Eq. 4 -> 7x7/2 stem on the GPU, against the oracle stem on the GPU's mapping
    rng = np.random.default_rng(42)
    rgb = rng.uniform(0.0, 1.0, size=(2, 32, 32, 3)).astype(np.float32)
    q = quan.poincare(torch.from_numpy(rgb).cuda())
    spec = inputs.small_layer("stem_rgb", 2, 32, 32, 4, 64, 7, 2, 3, seed=(406, 0))
    d = inputs.layer_inputs(spec)
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    sc, sh = to_dev_f32(d["scale"]), to_dev_f32(d["shift"])
    y = quan.qconv2d(q, *w, stride=2, pad=3, scale=sc, shift=sh, act=quan.QUAN_ACT_RELU)
    torch.cuda.synchronize()
    assert quan.quan_last_kernel() == "qconv_pairs_kernel"
    f64 = oracle.bf16_bits_to_f64
    ref = oracle.qconv2d(out_f64(q), *(f64(d[k]) for k in ("wr", "wi", "wj", "wk")), stride=2,
                         pad=3, scale=d["scale"], shift=d["shift"], act=oracle.ACT_RELU)
    assert_bf16_close(out_f64(y), ref, "poincare-stem")
