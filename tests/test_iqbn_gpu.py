"""GPU parity of training-mode IQBN (Eq. 11-12) against the fp64 oracle, through the C ABI
entry points quan_iqbn_batch_stats and quan_iqbn_train_fwd: the 16-byte vector path and the
scalar path, large channel offsets, in-place normalisation and the activations, and an
ImageNet-stage activation tensor in full."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2509_05512_gb300 import build, inputs, quan
from tests._util import BF16_HALF_ULP, out_f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build_library()
    yield quan.load()


def _bf16(rng, shape, scale=1.0, offset=0.0):
    bits = inputs.to_bf16_bits(rng.standard_normal(shape).astype(np.float32) * scale + offset)
    return bits, oracle.bf16_bits_to_f64(bits)


def _dev(bits, offset=0):
    """bf16 bits on the device, `offset` elements past a 16-byte boundary."""
    flat = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16).reshape(-1))
    buf = torch.empty(flat.numel() + 8, dtype=torch.int16)
    buf[offset:offset + flat.numel()] = flat
    return buf.cuda().view(torch.bfloat16)[offset:offset + flat.numel()].view(bits.shape)


def check_stats(x_dev, x64):
    mean, var = quan.iqbn_batch_stats(x_dev)
    torch.cuda.synchronize()
    rm, rv = oracle.iqbn_batch_stats(x64)
    sd = np.sqrt(rv)
    # fp32 sums of shifted values: errors far below the bf16 input resolution
    mean_err = np.abs(out_f64(mean) - rm) - 1e-5 * (sd + np.abs(rm))
    assert (mean_err <= 0).all(), "mean: max excess %.3e" % mean_err.max()
    var_err = np.abs(out_f64(var) - rv) - (1e-4 * rv + 1e-12)
    assert (var_err <= 0).all(), "var: max excess %.3e" % var_err.max()
    return mean, var


STAT_CASES = [
    # name, shape (N, H, W, C), pointer offset: vector path (C % 8 == 0, aligned) or scalar
    ("vec_c64", (4, 9, 7, 64), 0),
    ("vec_c256", (2, 5, 11, 256), 0),
    ("vec_c2048", (1, 3, 5, 2048), 0),
    ("scalar_c4", (2, 13, 17, 4), 0),
    ("scalar_c12", (3, 6, 5, 12), 0),
    ("scalar_misaligned", (2, 7, 5, 64), 1),
    ("one_pixel", (1, 1, 1, 64), 0),
]


@pytest.mark.parametrize("case", STAT_CASES, ids=[c[0] for c in STAT_CASES])
def test_batch_stats(case):
    name, shape, off = case
    rng = np.random.default_rng(800 + len(name))
    scale = np.linspace(0.2, 3.0, shape[-1])
    bits, x64 = _bf16(rng, shape, scale=scale, offset=np.linspace(-2, 2, shape[-1]))
    check_stats(_dev(bits, off), x64)


def test_batch_stats_repeat_bit_identical():
    # partial sums are added in a fixed order: the same input gives the same bits
    rng = np.random.default_rng(811)
    bits, _ = _bf16(rng, (16, 20, 20, 128))
    x = _dev(bits)
    m1, v1 = quan.iqbn_batch_stats(x)
    m2, v2 = quan.iqbn_batch_stats(x)
    torch.cuda.synchronize()
    assert torch.equal(m1, m2) and torch.equal(v1, v2)


def test_batch_stats_large_mean():
    # channels centred at 64 with unit spread: the per-channel shift keeps the variance
    rng = np.random.default_rng(810)
    bits, x64 = _bf16(rng, (8, 16, 16, 64), scale=1.0, offset=64.0)
    check_stats(_dev(bits), x64)


def check_train(x_dev, x64, gamma, beta, eps, act, inplace=False):
    g = None if gamma is None else torch.from_numpy(gamma.astype(np.float32)).cuda()
    b = None if beta is None else torch.from_numpy(beta.astype(np.float32)).cuda()
    out = x_dev if inplace else None
    y, _, _ = quan.iqbn_train(x_dev, g, b, eps=eps, act=act, out=out)
    torch.cuda.synchronize()
    C = x64.shape[-1]
    ref = oracle.iqbn_train(x64, np.ones(C) if gamma is None else gamma,
                            np.zeros(C) if beta is None else beta, eps=eps, act=act)
    got = out_f64(y)
    err = np.abs(got - ref)
    # one bf16 rounding of the output, plus the fp32 statistics' error on x_hat
    bound = BF16_HALF_ULP * 1.001 * np.abs(ref) + 1e-4 * (np.abs(ref).max() + 1.0)
    assert (err <= bound).all(), "max excess %.3e" % (err - bound).max()


@pytest.mark.parametrize("act", [quan.QUAN_ACT_NONE, quan.QUAN_ACT_RELU, quan.QUAN_ACT_SILU])
@pytest.mark.parametrize("C", [64, 12])
def test_train_forward(act, C):
    rng = np.random.default_rng(820 + C + act)
    bits, x64 = _bf16(rng, (3, 7, 9, C), scale=np.linspace(0.5, 2.0, C), offset=1.0)
    gamma = rng.uniform(0.5, 1.5, C)
    beta = rng.standard_normal(C) * 0.1
    check_train(_dev(bits), x64, gamma, beta, 1e-5, act)


def test_train_forward_in_place_and_defaults():
    rng = np.random.default_rng(830)
    bits, x64 = _bf16(rng, (2, 8, 8, 128), scale=2.0, offset=-1.0)
    check_train(_dev(bits), x64, None, None, 1e-3, quan.QUAN_ACT_RELU, inplace=True)


def test_batch_stats_rejects_small_workspace():
    x = torch.zeros((4, 64), dtype=torch.bfloat16, device="cuda")
    ws = torch.empty(quan.quan_iqbn_batch_stats_workspace_size(64) - 4, dtype=torch.uint8,
                     device="cuda")
    with pytest.raises(quan.QuanError) as ei:
        quan.iqbn_batch_stats(x, workspace=ws)
    assert ei.value.status == quan.QUAN_ERR_INVALID_ARG


def test_imagenet_stage_activation_full():
    # 64 images of 56 x 56 with 256 real channels (the ImageNet-stage layer's output)
    rng = np.random.default_rng(840)
    bits, x64 = _bf16(rng, (64, 56, 56, 256), scale=1.0, offset=0.5)
    x = _dev(bits)
    mean, var = check_stats(x, x64)
    gamma, beta = rng.uniform(0.5, 1.5, 256), rng.standard_normal(256) * 0.1
    y = torch.empty_like(x)
    quan.quan_iqbn_train_fwd(x, x.numel() // 256, 256, mean, var,
                             torch.from_numpy(gamma.astype(np.float32)).cuda(),
                             torch.from_numpy(beta.astype(np.float32)).cuda(), 1e-5,
                             quan.QUAN_ACT_RELU, y)
    torch.cuda.synchronize()
    idx = rng.integers(0, x64.size // 256, size=2048)
    xs = x64.reshape(-1, 256)
    rm, rv = oracle.iqbn_batch_stats(x64)
    ref = np.maximum((xs[idx] - rm) / np.sqrt(rv + 1e-5) * gamma + beta, 0.0)
    got = out_f64(y).reshape(-1, 256)[idx]
    bound = BF16_HALF_ULP * 1.001 * np.abs(ref) + 1e-4 * (np.abs(ref).max() + 1.0)
    assert (np.abs(got - ref) <= bound).all()
