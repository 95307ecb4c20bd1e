"""GPU parity of the fused convolution + 1x1 shortcut call (quan_qconv2d_fwd_shortcut), the
downsampling block's 3x3/2 convolution and its 1x1/2 shortcut of the same input (Sec.
III-D): both outputs against the fp64 oracle, each layer on its own (Eq. 5/6 with its
epilogue); bit-identity with separate calls on the same pair-kernel tiles; shapes without a
fused form (two calls); guard bands; failure injection."""
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2509_05512_gb300 import build, inputs, quan
from tests._util import assert_bf16_close, host_f64, out_f64, to_dev, to_dev_f32

pytestmark = pytest.mark.gpu

LETTERS = ("wr", "wi", "wj", "wk")


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
    quan.quan_set_fault_injection(False)
    quan.quan_set_wait_limit_ns(0)


def make(name, N, H, W, Cin, Cout, Cout_sc, k, stride, pad, seed, conv_kw=None, sc_kw=None):
    conv = inputs.small_layer(name, N, H, W, Cin, Cout, k, stride, pad, seed=(600, seed),
                              **(conv_kw or {}))
    sc = inputs.small_layer(name + "_sc", N, H, W, Cin, Cout_sc, 1, stride, 0,
                            seed=(601, seed), **(sc_kw or {}))
    return conv, sc, inputs.layer_inputs(conv), inputs.layer_inputs(sc)


def dev(conv, sc, dc, ds):
    x = to_dev(dc["x"], "bf16")  # the shortcut reads the convolution's input
    w = [to_dev(dc[k], "bf16") for k in LETTERS]
    sw = [to_dev(ds[k], "bf16") for k in LETTERS]
    vec = [to_dev_f32(dc[k]) for k in ("bias", "scale", "shift")]
    svec = [to_dev_f32(ds[k]) for k in ("bias", "scale", "shift")]
    return x, w, sw, vec, svec


def guarded(n):
    pad = 4096
    buf = torch.full((n + 2 * pad,), float("nan"), dtype=torch.bfloat16, device="cuda")
    return buf, buf[pad:pad + n], pad


def run_fused(conv, sc, dc, ds):
    x, w, sw, (b, s, h), (sb, ss, sh) = dev(conv, sc, dc, ds)
    n1, n2 = conv.N * conv.Ho * conv.Wo * conv.Cout, sc.N * sc.Ho * sc.Wo * sc.Cout
    buf1, o1, p1 = guarded(n1)
    buf2, o2, p2 = guarded(n2)
    out = o1.view(conv.N, conv.Ho, conv.Wo, conv.Cout)
    out_sc = o2.view(sc.N, sc.Ho, sc.Wo, sc.Cout)
    quan.qconv2d_shortcut(x, w, sw, stride=conv.stride, pad=conv.pad, bias=b, scale=s, shift=h,
                          act=conv.act, sc_bias=sb, sc_scale=ss, sc_shift=sh, sc_act=sc.act,
                          out=out, out_sc=out_sc)
    torch.cuda.synchronize()
    for buf, p, n in ((buf1, p1, n1), (buf2, p2, n2)):  # guard bands untouched
        assert torch.isnan(buf[:p].float()).all() and torch.isnan(buf[p + n:].float()).all()
    st, bits = quan.quan_device_status()
    assert st == quan.QUAN_OK, bits
    return out, out_sc, quan.quan_last_kernel()


def oracle_pair(conv, sc, dc, ds):
    x = host_f64(dc["x"], "bf16")
    y = oracle.qconv2d(x, *(host_f64(dc[k], "bf16") for k in LETTERS), stride=conv.stride,
                       pad=conv.pad, bias=dc["bias"], scale=dc["scale"], shift=dc["shift"],
                       act=conv.act)
    y_sc = oracle.qconv2d(x, *(host_f64(ds[k], "bf16") for k in LETTERS), stride=sc.stride,
                          pad=0, bias=ds["bias"], scale=ds["scale"], shift=ds["shift"],
                          act=sc.act)
    return y, y_sc


SILU, NONE = quan.QUAN_ACT_SILU, quan.QUAN_ACT_NONE
CASES = [
    # name, N, H, W, Cin, Cout, Cout_sc, k, stride, pad, conv extras, shortcut extras, kernel
    ("block2", 2, 28, 28, 128, 256, 256, 3, 2, 1, {}, {"act": NONE},
     "qconv_tc_kernel<pair,kappa=32,bnq=64,shortcut>"),
    ("block3", 1, 14, 14, 256, 512, 512, 3, 2, 1, {}, {"act": NONE},
     "qconv_tc_kernel<pair,kappa=32,bnq=64,shortcut>"),
    ("ragged_bias_silu", 3, 15, 13, 64, 128, 128, 3, 2, 1, {"bias": True, "act": SILU},
     {"bias": True}, "qconv_tc_kernel<pair,kappa=16,bnq=32,shortcut>"),
    ("more_sc_tiles", 2, 16, 16, 128, 256, 512, 3, 2, 1, {}, {"iqbn": False, "act": NONE},
     "qconv_tc_kernel<pair,kappa=32,bnq=64,shortcut>"),
    ("stride1", 2, 10, 12, 64, 128, 128, 3, 1, 1, {}, {}, "qconv_tc_kernel<pair,kappa=16,bnq=32,shortcut>"),
    ("pad2_5x5", 1, 13, 11, 64, 128, 128, 5, 2, 2, {}, {"act": NONE},
     "qconv_tc_kernel<pair,kappa=16,bnq=32,shortcut>"),
    ("one_tile", 1, 4, 4, 64, 128, 128, 3, 2, 1, {}, {}, "qconv_tc_kernel<pair,kappa=16,bnq=32,shortcut>"),
]


@pytest.mark.parametrize("case", CASES, ids=[c[0] for c in CASES])
def test_fused_shortcut_layers(case):
    name, N, H, W, Cin, Cout, Cout_sc, k, s, p, ck, sk, kernel = case
    conv, sc, dc, ds = make(name, N, H, W, Cin, Cout, Cout_sc, k, s, p, len(name), ck, sk)
    assert (conv.Ho, conv.Wo) == (sc.Ho, sc.Wo)
    out, out_sc, kern = run_fused(conv, sc, dc, ds)
    assert kern == kernel
    y, y_sc = oracle_pair(conv, sc, dc, ds)
    assert_bf16_close(out_f64(out), y, name)
    assert_bf16_close(out_f64(out_sc), y_sc, name + "_sc")


def test_fused_shortcut_bit_identical_to_separate_calls():
    # the same pair-kernel tiles, K blocks and epilogue arithmetic: the fused launch
    # reproduces the two separate launches bit for bit
    conv, sc, dc, ds = make("sep_calls", 2, 28, 28, 128, 256, 256, 3, 2, 1, 7, {},
                            {"act": NONE})
    quan.quan_set_tc_tiles(32, 64, 0, 2)
    out, out_sc, kern = run_fused(conv, sc, dc, ds)
    assert kern == "qconv_tc_kernel<pair,kappa=32,bnq=64,shortcut>"
    x, w, sw, (b, s, h), (sb, ss, sh) = dev(conv, sc, dc, ds)
    ref = quan.qconv2d(x, *w, stride=2, pad=1, bias=b, scale=s, shift=h, act=conv.act)
    assert quan.quan_last_kernel() == "qconv_tc_kernel<pair,kappa=32,bnq=64>"
    ref_sc = quan.qconv2d(x, *sw, stride=2, pad=0, bias=sb, scale=ss, shift=sh, act=sc.act)
    assert quan.quan_last_kernel() == "qconv_tc_kernel<pair,kappa=32,bnq=64>"
    torch.cuda.synchronize()
    assert torch.equal(out, ref)
    assert torch.equal(out_sc, ref_sc)


def test_shortcut_without_fused_form_runs_two_calls():
    # 32 quaternion output channels per tile and a 16-channel shortcut: no fused tiling, so
    # the call runs the two layers separately (the shortcut last, on its own kernel)
    conv, sc, dc, ds = make("two_calls", 2, 16, 16, 64, 128, 64, 3, 2, 1, 8)
    out, out_sc, kern = run_fused(conv, sc, dc, ds)
    assert "shortcut" not in kern
    y, y_sc = oracle_pair(conv, sc, dc, ds)
    assert_bf16_close(out_f64(out), y, "two_calls")
    assert_bf16_close(out_f64(out_sc), y_sc, "two_calls_sc")


def test_fused_shortcut_on_cuda_cores():
    conv, sc, dc, ds = make("simt_sc", 1, 9, 7, 64, 128, 128, 3, 2, 1, 9)
    quan.quan_set_path(quan.QUAN_PATH_SIMT)
    out, out_sc, kern = run_fused(conv, sc, dc, ds)
    assert kern == "qconv_simt_kernel<bf16>"
    y, y_sc = oracle_pair(conv, sc, dc, ds)
    assert_bf16_close(out_f64(out), y, "simt_sc")
    assert_bf16_close(out_f64(out_sc), y_sc, "simt_sc_sc")


def test_fused_shortcut_bounded_wait_timeout():
    # failure injection on the fused launch: every wait ends with a timeout status, the
    # context stays usable, and the next call is right
    conv, sc, dc, ds = make("inject_sc", 2, 16, 16, 128, 256, 256, 3, 2, 1, 10)
    x, w, sw, (b, s, h), (sb, ss, sh) = dev(conv, sc, dc, ds)
    quan.quan_set_wait_limit_ns(5_000_000)
    quan.quan_set_fault_injection(True)
    quan.qconv2d_shortcut(x, w, sw, stride=2, pad=1, bias=b, scale=s, shift=h, act=conv.act,
                          sc_bias=sb, sc_scale=ss, sc_shift=sh, sc_act=sc.act)
    st, bits = quan.quan_device_status()
    assert st == quan.QUAN_ERR_DEVICE_TIMEOUT and bits != 0
    assert quan.quan_last_kernel() == "qconv_tc_kernel<pair,kappa=32,bnq=64,shortcut>"
    quan.quan_set_fault_injection(False)
    quan.quan_set_wait_limit_ns(0)
    out, out_sc, _ = run_fused(conv, sc, dc, ds)
    y, y_sc = oracle_pair(conv, sc, dc, ds)
    assert_bf16_close(out_f64(out), y, "inject_sc")
    assert_bf16_close(out_f64(out_sc), y_sc, "inject_sc_sc")
