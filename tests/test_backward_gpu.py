"""GPU parity of the backward pass against the fp64 oracle, through the C ABI entry points
quan_qconv2d_bwd_data / quan_qconv2d_bwd_weight (full Hamilton form, gradients of Eq. 5
before its epilogue) and quan_qconv2d_sep_bwd_data / quan_qconv2d_sep_bwd_weight (the
separable form, Eq. 8-10): the tensor-core input gradient (stride 1) and the CUDA-core
kernels over ragged, strided and padded shapes, and the CIFAR layer in full."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2509_05512_gb300 import build, inputs, quan
from tests._util import assert_bf16_close, assert_f32_close, host_f64, out_f64, to_dev

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


def layer(spec):
    d = inputs.layer_inputs(spec)
    d["dy"] = inputs.grad_output(spec)
    return d


def gpu_bwd_data(d, separable=False, path=quan.QUAN_PATH_AUTO, letters_only=False):
    """letters_only: a workspace for the transformed letters alone (a strided layer then
    runs on CUDA cores); else the larger one of quan_qconv2d_bwd_data_workspace_size_ex."""
    spec = d["spec"]
    dy = to_dev(d["dy"], "bf16")
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    if letters_only:
        nb = quan.quan_qconv2d_bwd_data_workspace_size(spec.Cin, spec.Cout, spec.kh, spec.kw)
    else:
        nb = quan.quan_qconv2d_bwd_data_workspace_size_ex(spec.N, spec.H, spec.W, spec.Cin,
                                                          spec.Cout, spec.kh, spec.kw,
                                                          spec.stride, spec.pad)
    ws = torch.empty(nb, dtype=torch.uint8, device="cuda")
    n = spec.N * spec.H * spec.W * spec.Cin
    pad = 4096
    buf = torch.full((n + 2 * pad,), float("nan"), dtype=torch.bfloat16, device="cuda")
    dx = buf[pad:pad + n].view(spec.N, spec.H, spec.W, spec.Cin)
    quan.quan_set_path(path)
    quan.qconv2d_backward_data(dy, *w, H=spec.H, W=spec.W, stride=spec.stride, pad=spec.pad,
                               separable=separable, workspace=ws, out=dx)
    torch.cuda.synchronize()
    assert torch.isnan(buf[:pad].float()).all() and torch.isnan(buf[pad + n:].float()).all()
    st, bits = quan.quan_device_status()
    assert st == quan.QUAN_OK, bits
    return out_f64(dx), quan.quan_last_path(), quan.quan_last_kernel()


def gpu_bwd_weight(d, separable=False, path=quan.QUAN_PATH_AUTO):
    spec = d["spec"]
    quan.quan_set_path(path)
    x, dy = to_dev(d["x"], "bf16"), to_dev(d["dy"], "bf16")
    # the outputs start as garbage: the call zeroes them itself
    out = tuple(torch.full((spec.Cout // 4, spec.kh, spec.kw, spec.Cin // 4), 7.0,
                           dtype=torch.float32, device="cuda") for _ in range(4))
    quan.qconv2d_backward_weight(x, dy, kh=spec.kh, kw=spec.kw, stride=spec.stride,
                                 pad=spec.pad, separable=separable, out=out)
    torch.cuda.synchronize()
    return [out_f64(t) for t in out], quan.quan_last_kernel()


def oracle_bwd_data(d, separable=False):
    spec = d["spec"]
    f = lambda k: host_f64(d[k], "bf16")
    fn = oracle.qconv2d_sep_bwd_data if separable else oracle.qconv2d_bwd_data
    return fn(f("dy"), f("wr"), f("wi"), f("wj"), f("wk"), H=spec.H, W=spec.W,
              stride=spec.stride, pad=spec.pad)


def oracle_bwd_weight(d, separable=False):
    spec = d["spec"]
    fn = oracle.qconv2d_sep_bwd_weight if separable else oracle.qconv2d_bwd_weight
    return fn(host_f64(d["x"], "bf16"), host_f64(d["dy"], "bf16"), kh=spec.kh, kw=spec.kw,
              stride=spec.stride, pad=spec.pad)


def tc_weight_shape(spec):
    return (spec.stride in (1, 2) and spec.Cin % 64 == 0 and spec.Cout % 64 == 0 and
            (spec.Cout <= 256 or spec.Cout % 256 == 0))


def check_weight(d, separable=False, path=quan.QUAN_PATH_AUTO):
    got, kernel = gpu_bwd_weight(d, separable, path)
    spec = d["spec"]
    if path != quan.QUAN_PATH_SIMT and tc_weight_shape(spec):
        assert kernel.startswith("qconv_dw_kernel<"), kernel
        assert kernel.endswith(",sep>") == separable, kernel
    else:
        assert kernel == ("bwd_weight_simt_kernel<sep>" if separable
                          else "bwd_weight_simt_kernel"), kernel
    ref = oracle_bwd_weight(d, separable)
    for L in range(4):
        assert_f32_close(got[L], ref[L], "%s dW[%d] (%s)" % (spec.name, L, kernel))
    return got


TC_CASES = [
    # name, N, H, W, Cin, Cout, k, stride, pad: stride 1, square filter, pad < k
    ("ws_16to16", 2, 13, 11, 64, 64, 3, 1, 1),       # weight-stationary kernel
    ("wide_out", 2, 12, 10, 64, 128, 3, 1, 1),       # dx has 16, dy 32 quaternion channels
    ("wide_in", 1, 9, 13, 256, 64, 3, 1, 1),
    ("pointwise", 2, 10, 9, 128, 256, 1, 1, 0),
    ("pad0", 2, 11, 12, 64, 128, 3, 1, 0),           # transposed padding 2
    ("k5_pad2", 1, 12, 11, 64, 64, 5, 1, 2),
    ("k5_pad1", 1, 12, 11, 128, 64, 5, 1, 1),        # transposed padding 3
    # strided: dy spread out with zeros in the workspace, then the stride-1 convolution
    ("s2_odd", 2, 15, 17, 64, 128, 3, 2, 1),
    ("s2_16to16", 1, 16, 16, 64, 64, 3, 2, 1),       # weight-stationary kernel
    ("s2_shortcut", 2, 14, 14, 64, 128, 1, 2, 0),
    ("s2_imagenet", 1, 56, 56, 256, 512, 3, 2, 1),
    ("s2_5x5", 1, 13, 12, 64, 64, 5, 2, 2),
]


@pytest.mark.parametrize("case", TC_CASES, ids=[c[0] for c in TC_CASES])
def test_bwd_data_tensor_cores(case):
    name, N, H, W, Cin, Cout, k, s, p = case
    d = layer(inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(600, len(name))))
    got, path, kernel = gpu_bwd_data(d, path=quan.QUAN_PATH_TC)
    assert path == quan.QUAN_PATH_TC, kernel
    assert kernel.startswith("qconv_"), kernel
    assert_bf16_close(got, oracle_bwd_data(d), name + " dx")


SIMT_CASES = [
    ("stride2", 2, 15, 17, 64, 128, 3, 2, 1),
    ("stride2_even", 1, 16, 16, 64, 64, 3, 2, 1),
    ("shortcut_1x1_s2", 2, 14, 14, 64, 128, 1, 2, 0),
    ("stem", 1, 20, 18, 4, 64, 7, 2, 3),
    ("qin12", 2, 7, 9, 48, 64, 3, 1, 1),
    ("pad_gt_k", 1, 6, 7, 64, 64, 1, 1, 1),          # pad >= k: no transposed padding
    ("stride3_k5", 1, 17, 16, 16, 32, 5, 3, 2),
]


@pytest.mark.parametrize("case", SIMT_CASES, ids=[c[0] for c in SIMT_CASES])
def test_bwd_data_cuda_cores(case):
    name, N, H, W, Cin, Cout, k, s, p = case
    d = layer(inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(601, len(name))))
    got, path, kernel = gpu_bwd_data(d, letters_only=True)
    assert path == quan.QUAN_PATH_SIMT and kernel == "bwd_data_simt_kernel"
    assert_bf16_close(got, oracle_bwd_data(d), name + " dx")


def test_bwd_data_rectangular_filter():
    d = layer(inputs.small_layer("k3x1", 2, 9, 8, 64, 64, 3, 1, 1, kw=1, seed=(602, 0)))
    got, path, _ = gpu_bwd_data(d)
    assert path == quan.QUAN_PATH_SIMT
    assert_bf16_close(got, oracle_bwd_data(d), "k3x1 dx")


def test_bwd_data_paths_agree():
    # the same stride-1 layer on both paths
    d = layer(inputs.small_layer("both", 2, 11, 9, 64, 128, 3, 1, 1, seed=(603, 0)))
    tc, p1, _ = gpu_bwd_data(d, path=quan.QUAN_PATH_TC)
    simt, p2, _ = gpu_bwd_data(d, path=quan.QUAN_PATH_SIMT)
    assert (p1, p2) == (quan.QUAN_PATH_TC, quan.QUAN_PATH_SIMT)
    ref = oracle_bwd_data(d)
    assert_bf16_close(tc, ref, "tc")
    assert_bf16_close(simt, ref, "simt")


def test_bwd_data_tc_strided_needs_the_larger_workspace():
    d = layer(inputs.small_layer("tc_s2", 1, 9, 9, 64, 64, 3, 2, 1, seed=(604, 0)))
    with pytest.raises(quan.QuanError) as ei:
        gpu_bwd_data(d, path=quan.QUAN_PATH_TC, letters_only=True)
    assert ei.value.status == quan.QUAN_ERR_UNSUPPORTED
    got, path, _ = gpu_bwd_data(d, path=quan.QUAN_PATH_TC)
    assert path == quan.QUAN_PATH_TC
    assert_bf16_close(got, oracle_bwd_data(d), "tc_s2 dx")


def test_bwd_data_workspace_reuse():
    # one workspace for two layers with different weights: every call rewrites it
    ws = torch.empty(quan.quan_qconv2d_bwd_data_workspace_size(64, 128, 3, 3),
                     dtype=torch.uint8, device="cuda")
    for seed in (605, 606):
        d = layer(inputs.small_layer("reuse", 1, 10, 10, 64, 128, 3, 1, 1, seed=(seed, 0)))
        spec = d["spec"]
        dx = quan.qconv2d_backward_data(to_dev(d["dy"], "bf16"),
                                        *(to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")),
                                        H=spec.H, W=spec.W, stride=1, pad=1, workspace=ws)
        torch.cuda.synchronize()
        assert quan.quan_last_path() == quan.QUAN_PATH_TC
        assert_bf16_close(out_f64(dx), oracle_bwd_data(d), "reuse dx")


WEIGHT_CASES = [
    ("w3x3", 2, 13, 11, 64, 64, 3, 1, 1),
    ("w_stride2", 2, 15, 17, 64, 128, 3, 2, 1),
    ("w_pointwise", 2, 10, 9, 128, 256, 1, 1, 0),
    ("w_stem", 1, 20, 18, 4, 64, 7, 2, 3),
    ("w_qin12", 2, 7, 9, 48, 64, 3, 1, 1),
    ("w_tiny", 1, 1, 1, 8, 8, 3, 1, 1),
]


@pytest.mark.parametrize("case", WEIGHT_CASES, ids=[c[0] for c in WEIGHT_CASES])
def test_bwd_weight(case):
    name, N, H, W, Cin, Cout, k, s, p = case
    check_weight(layer(inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p,
                                          seed=(607, len(name)))))


TC_WEIGHT_CASES = [
    # name, N, H, W, Cin, Cout, k, stride, pad: the tensor-core weight gradient
    ("dw_odd_units", 2, 13, 11, 64, 64, 3, 1, 1),    # 9 taps: the last unit pair repeats
    ("dw_cout128", 2, 12, 10, 64, 128, 3, 1, 1),
    ("dw_cin256", 1, 9, 13, 256, 64, 3, 1, 1),       # 8 unit pairs per CTA, 3 pair groups
    ("dw_c192", 1, 7, 9, 192, 192, 3, 1, 1),
    ("dw_pointwise", 2, 10, 9, 128, 256, 1, 1, 0),
    ("dw_pad0", 2, 11, 12, 64, 128, 3, 1, 0),
    ("dw_k5", 1, 12, 11, 64, 64, 5, 1, 2),
    ("dw_cout512", 1, 6, 7, 64, 512, 3, 1, 1),       # two output-channel groups
    ("dw_tiny", 1, 1, 1, 64, 64, 3, 1, 1),
    ("dw_wide_row", 1, 3, 200, 64, 64, 3, 1, 1),     # 200 columns: one row per block
    # stride 2: the x boxes traverse every second input pixel
    ("dw_s2", 2, 15, 17, 64, 128, 3, 2, 1),
    ("dw_s2_even", 1, 16, 16, 128, 64, 3, 2, 1),
    ("dw_s2_shortcut", 2, 14, 14, 64, 128, 1, 2, 0),
    ("dw_s2_imagenet", 1, 56, 56, 256, 512, 3, 2, 1),  # one image of the stride-2 layer
    ("dw_s2_5x5", 1, 13, 12, 64, 64, 5, 2, 2),
]


@pytest.mark.parametrize("case", TC_WEIGHT_CASES, ids=[c[0] for c in TC_WEIGHT_CASES])
def test_bwd_weight_tensor_cores(case):
    name, N, H, W, Cin, Cout, k, s, p = case
    d = layer(inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(610, len(name))))
    check_weight(d, path=quan.QUAN_PATH_TC)


def test_bwd_weight_paths_agree():
    d = layer(inputs.small_layer("dw_both", 2, 9, 10, 64, 128, 3, 1, 1, seed=(611, 0)))
    tc = check_weight(d, path=quan.QUAN_PATH_TC)
    simt = check_weight(d, path=quan.QUAN_PATH_SIMT)
    for L in range(4):
        assert_f32_close(tc[L], simt[L], "tc vs simt dW[%d]" % L)


SEP_CASES = [
    ("sep_3x3", 2, 13, 11, 64, 64, 3, 1, 1),
    ("sep_wide", 2, 9, 10, 128, 256, 3, 1, 1),
    ("sep_pad0_5x5", 1, 12, 11, 64, 128, 5, 1, 0),
    ("sep_stride2", 2, 15, 17, 64, 128, 3, 2, 1),
    ("sep_pointwise", 1, 10, 9, 128, 64, 1, 1, 0),
    ("sep_qin3", 1, 8, 9, 12, 16, 3, 1, 1),
]


@pytest.mark.parametrize("case", SEP_CASES, ids=[c[0] for c in SEP_CASES])
def test_separable_backward(case):
    name, N, H, W, Cin, Cout, k, s, p = case
    d = layer(inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(608, len(name))))
    got, path, kernel = gpu_bwd_data(d, separable=True)
    if Cin % 64 == 0 and Cout % 64 == 0:
        assert kernel.startswith("qconv_tc_kernel<sep_t,"), kernel
    else:
        assert kernel == "bwd_data_simt_kernel<sep>", kernel
    assert_bf16_close(got, oracle_bwd_data(d, True), name + " sep dx")
    check_weight(d, separable=True)


@pytest.mark.parametrize("case", [("sepw_3x3", 2, 12, 10, 64, 128, 3, 1, 1),
                                  ("sepw_c256", 1, 9, 7, 256, 64, 3, 1, 1)],
                         ids=lambda c: c[0])
def test_separable_weight_gradient_paths(case):
    # the tensor-core kernel with Eq. 7's fold against the oracle and the CUDA-core kernel
    name, N, H, W, Cin, Cout, k, s, p = case
    d = layer(inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(612, len(name))))
    tc = check_weight(d, separable=True, path=quan.QUAN_PATH_TC)
    simt = check_weight(d, separable=True, path=quan.QUAN_PATH_SIMT)
    for L in range(4):
        assert_f32_close(tc[L], simt[L], "sep tc vs simt dW[%d]" % L)


def test_separable_input_gradient_paths_agree():
    d = layer(inputs.small_layer("sep_both", 2, 11, 9, 64, 128, 3, 1, 1, seed=(613, 0)))
    tc, p1, k1 = gpu_bwd_data(d, separable=True, path=quan.QUAN_PATH_TC)
    simt, p2, _ = gpu_bwd_data(d, separable=True, path=quan.QUAN_PATH_SIMT)
    assert (p1, p2) == (quan.QUAN_PATH_TC, quan.QUAN_PATH_SIMT), k1
    ref = oracle_bwd_data(d, True)
    assert_bf16_close(tc, ref, "sep tc")
    assert_bf16_close(simt, ref, "sep simt")


def test_separable_backward_differs_from_full_form():
    d = layer(inputs.small_layer("sep_vs_full", 1, 8, 8, 64, 64, 3, 1, 1, seed=(609, 0)))
    got, _, _ = gpu_bwd_data(d, separable=True)
    full = oracle_bwd_data(d)
    assert np.linalg.norm(got - full) / np.linalg.norm(full) > 0.5


def test_cifar_layer_backward_full():
    # the 32x32, 64 -> 64 channel 3x3 layer, batch 128, both gradients in full
    d = layer(inputs.LAYERS["c1"])
    got, path, _ = gpu_bwd_data(d)
    assert path == quan.QUAN_PATH_TC
    assert_bf16_close(got, oracle_bwd_data(d), "c1 dx")
    check_weight(d)
