"""GPU parity of the separable QUAN convolution (Eq. 7) against the fp64 oracle
(`oracle.qconv2d_separable`), through the C ABI entry point quan_qconv2d_sep_fwd: small
layers spanning several tiles with ragged tails, every (kappa, bnq) tile, the CUDA-core
path, and the CIFAR- and ImageNet-shaped layers in full."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2509_05512_gb300 import build, inputs, quan
from tests._util import assert_bf16_close, host_f64, out_f64, to_dev, to_dev_f32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build_library()
    yield quan.load()
    quan.quan_set_path(quan.QUAN_PATH_AUTO)
    quan.quan_set_tc_tiles(0, 0, 0, 0)


@pytest.fixture(autouse=True)
def _reset():
    yield
    quan.quan_set_path(quan.QUAN_PATH_AUTO)
    quan.quan_set_tc_tiles(0, 0, 0, 0)


def run_sep(d, path=quan.QUAN_PATH_AUTO):
    spec = d["spec"]
    x = to_dev(d["x"], "bf16")
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    bias, scale, shift = (to_dev_f32(d[k]) for k in ("bias", "scale", "shift"))
    n_out = spec.N * spec.Ho * spec.Wo * spec.Cout
    pad = 4096
    buf = torch.full((n_out + 2 * pad,), float("nan"), dtype=torch.bfloat16, device="cuda")
    out = buf[pad:pad + n_out].view(spec.N, spec.Ho, spec.Wo, spec.Cout)
    quan.quan_set_path(path)
    quan.qconv2d(x, *w, stride=spec.stride, pad=spec.pad, bias=bias, scale=scale, shift=shift,
                 act=spec.act, out=out, separable=True)
    torch.cuda.synchronize()
    # guard bands on both sides of the output stay untouched
    assert torch.isnan(buf[:pad].float()).all() and torch.isnan(buf[pad + n_out:].float()).all()
    st, bits = quan.quan_device_status()
    assert st == quan.QUAN_OK, bits
    return out_f64(out), quan.quan_last_path()


def oracle_sep(d):
    f = lambda k: host_f64(d[k], "bf16")
    spec = d["spec"]
    return oracle.qconv2d_separable(f("x"), f("wr"), f("wi"), f("wj"), f("wk"),
                                    stride=spec.stride, pad=spec.pad, bias=d["bias"],
                                    scale=d["scale"], shift=d["shift"], act=spec.act)


def check_sep(spec, path=quan.QUAN_PATH_AUTO, expect_path=None):
    d = inputs.layer_inputs(spec)
    got, used = run_sep(d, path)
    if expect_path is not None:
        assert used == expect_path
    assert_bf16_close(got, oracle_sep(d), spec.name + "-sep")
    return d, got


SEP_CASES = [
    # name, N, H, W, Cin, Cout, k, stride, pad, extra
    ("ragged", 3, 13, 11, 64, 64, 3, 1, 1, {}),
    ("stride2", 2, 15, 17, 64, 128, 3, 2, 1, {}),
    ("pointwise", 2, 12, 10, 128, 256, 1, 1, 0, {}),
    ("wide_q", 1, 9, 9, 256, 256, 3, 1, 1, {}),
    ("pad2_5x5", 1, 11, 12, 64, 64, 5, 1, 2, {}),
    ("bias_silu", 2, 9, 8, 64, 128, 3, 1, 1, {"bias": True, "act": quan.QUAN_ACT_SILU}),
    ("no_iqbn", 2, 9, 8, 64, 64, 3, 1, 1, {"iqbn": False, "act": quan.QUAN_ACT_NONE}),
    ("tiny_image", 1, 1, 1, 64, 64, 3, 1, 1, {}),
]


@pytest.mark.parametrize("case", SEP_CASES, ids=[c[0] for c in SEP_CASES])
def test_separable_tc_layers(case):
    name, N, H, W, Cin, Cout, k, s, p, extra = case
    spec = inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(500, len(name)), **extra)
    check_sep(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    kernel = quan.quan_last_kernel()
    if Cin == Cout == 64 and k * k <= 9:
        # 16 -> 16 quaternion channels: the vertical-tap (3x3 stride 1, one box per input
        # row) or the weight-stationary kernel, with the separable block weight expanded
        # on chip
        assert kernel.startswith(("qconv_vs_kernel<", "qconv_ws_kernel<")), kernel
        assert kernel.endswith(",sep>"), kernel
    else:
        assert kernel.startswith("qconv_tc_kernel<sep,"), kernel


@pytest.mark.parametrize("kappa,bnq", [(k, b) for k in (16, 32, 64) for b in (16, 32, 64)])
def test_separable_tile_variants(kappa, bnq):
    spec = inputs.small_layer("sep_tiles", 2, 11, 13, 256, 256, 3, 1, 1,
                              seed=(501, kappa + bnq))
    quan.quan_set_tc_tiles(kappa, bnq, 0, 0)
    check_sep(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    assert quan.quan_last_kernel() == "qconv_tc_kernel<sep,kappa=%d,bnq=%d>" % (kappa, bnq)


def test_separable_few_ctas_many_tiles():
    # 3 CTAs: every stage ring and both accumulator buffers wrap many times
    spec = inputs.small_layer("sep_few", 4, 24, 24, 128, 128, 3, 1, 1, seed=(502, 0))
    quan.quan_set_tc_tiles(0, 0, 3, 0)
    check_sep(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)


@pytest.mark.parametrize("case", [
    ("simt_qin12", 2, 7, 9, 48, 64, 3, 1, 1),     # Cin/4 = 12: CUDA cores only
    ("simt_stem", 1, 16, 16, 4, 64, 7, 2, 3),     # the stem's shape has no separable TC form
], ids=lambda c: c[0])
def test_separable_simt_shapes(case):
    name, N, H, W, Cin, Cout, k, s, p = case
    spec = inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(503, len(name)))
    check_sep(spec, expect_path=quan.QUAN_PATH_SIMT)
    assert quan.quan_last_kernel() == "qconv_simt_kernel<bf16,sep>"


@pytest.mark.parametrize("path", [quan.QUAN_PATH_TC, quan.QUAN_PATH_SIMT])
def test_separable_cifar_layer_full(path):
    check_sep(inputs.LAYERS["c1"], path=path, expect_path=path)


def test_separable_imagenet_layer_full():
    check_sep(inputs.LAYERS["c2a"], path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)


def test_separable_differs_from_full_form():
    # the cross-component terms the separable form drops are not small: the two forms
    # disagree on the same inputs, so a path that ran the full form would fail here
    spec = inputs.small_layer("sep_vs_full", 1, 8, 8, 64, 64, 3, 1, 1, seed=(504, 0),
                              act=quan.QUAN_ACT_NONE, iqbn=False)
    d = inputs.layer_inputs(spec)
    got, _ = run_sep(d, quan.QUAN_PATH_TC)
    f = lambda k: host_f64(d[k], "bf16")
    full = oracle.qconv2d(f("x"), f("wr"), f("wi"), f("wj"), f("wk"), stride=1, pad=1)
    rel = np.linalg.norm(got - full) / np.linalg.norm(full)
    assert rel > 0.5


def test_separable_rejects_mode_override():
    spec = inputs.small_layer("sep_mode", 1, 8, 8, 64, 64, 3, 1, 1, seed=(505, 0))
    d = inputs.layer_inputs(spec)
    quan.quan_set_tc_tiles(0, 0, 0, 2)
    with pytest.raises(quan.QuanError) as ei:
        run_sep(d, quan.QUAN_PATH_TC)
    assert ei.value.status == quan.QUAN_ERR_UNSUPPORTED
