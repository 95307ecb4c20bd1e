"""The stem convolution with its 3x3/2 max pooling in one kernel (quan_qconv2d_maxpool_fwd):
bit for bit the two separate calls (max commutes with the monotone bf16 rounding), within
the bf16 tolerance of the oracle's convolution followed by the oracle's pooling, and
through the backbone."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2509_05512_gb300 import build, inputs, quan
from paper_2509_05512_gb300.backbone import BackboneRunner
from tests._util import assert_bf16_close, host_f64, out_f64, to_dev, to_dev_f32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    build.build_library()
    yield quan.load()


def run_both(spec, act, negate_scale=None, max_ctas=0):
    d = inputs.layer_inputs(spec)
    if negate_scale is not None:
        d["scale"] = np.where(negate_scale, -d["scale"], d["scale"]).astype(np.float32)
    x = to_dev(d["x"], "bf16")
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    sc, sh = to_dev_f32(d["scale"]), to_dev_f32(d["shift"])
    N, H, W = spec.N, spec.H, spec.W
    conv = quan.qconv2d(x, *w, stride=spec.stride, pad=spec.pad, scale=sc, shift=sh, act=act)
    ref_gpu = quan.maxpool2d(conv, k=3, stride=2, pad=1)
    # one kernel writes the pooled tensor: no workspace
    assert quan.quan_qconv2d_maxpool_workspace_size(N, H, W, spec.Cout, spec.kh, spec.kw,
                                                    spec.stride, spec.pad) == 0
    out = torch.full_like(ref_gpu, float("nan"))
    quan.quan_set_tc_tiles(0, 0, max_ctas, 0)
    try:
        quan.quan_qconv2d_maxpool_fwd(x, *w, None, sc, sh, N, H, W, spec.Cin, spec.Cout,
                                      spec.kh, spec.kw, spec.stride, spec.pad, act, None, 0,
                                      out)
        torch.cuda.synchronize()
    finally:
        quan.quan_set_tc_tiles(0, 0, 0, 0)
    assert quan.quan_last_kernel() == "qconv_stem_pool_kernel"
    assert quan.quan_device_status()[0] == quan.QUAN_OK
    return d, out, ref_gpu


STEM_CASES = [
    # name, N, H, W: the 7x7/2 pad-3 stem, 4 -> 64 real channels
    ("even_wo", 2, 32, 32),
    ("odd_wo", 2, 30, 30),       # Wo = Ho = 15: the last pooled column and row are partial
    ("wide", 1, 20, 224),        # a full 112-pixel output row
    ("tall", 1, 41, 16),
]


@pytest.mark.parametrize("act", [quan.QUAN_ACT_RELU, quan.QUAN_ACT_SILU])
@pytest.mark.parametrize("case", STEM_CASES, ids=[c[0] for c in STEM_CASES])
def test_fused_equals_separate_calls_and_oracle(case, act):
    name, N, H, W = case
    spec = inputs.small_layer("stem_" + name, N, H, W, 4, 64, 7, 2, 3, seed=(900, len(name)),
                              act=act)
    d, out, ref_gpu = run_both(spec, act)
    assert torch.equal(out, ref_gpu)
    f = lambda k: host_f64(d[k], "bf16")
    y = oracle.qconv2d(f("x"), f("wr"), f("wi"), f("wj"), f("wk"), stride=2, pad=3,
                       scale=d["scale"], shift=d["shift"], act=act)
    assert_bf16_close(out_f64(out), oracle.maxpool2d(y, k=3, stride=2, pad=1), name)


@pytest.mark.parametrize("act", [quan.QUAN_ACT_RELU, quan.QUAN_ACT_NONE, quan.QUAN_ACT_SILU])
def test_fused_negative_scales_and_bands_across_images(act):
    # channels with a negative IQBN scale (the pooling is then a min of the accumulators,
    # taken on negated weights); a 3-CTA grid, so that each CTA's band of pooled rows
    # crosses image boundaries and starts inside an image (its priming tile)
    spec = inputs.small_layer("stem_neg", 3, 38, 36, 4, 64, 7, 2, 3, seed=(902, act), act=act)
    neg = (np.arange(64) % 3) == 1
    d, out, ref_gpu = run_both(spec, act, negate_scale=neg, max_ctas=3)
    assert torch.equal(out, ref_gpu)
    f = lambda k: host_f64(d[k], "bf16")
    y = oracle.qconv2d(f("x"), f("wr"), f("wi"), f("wj"), f("wk"), stride=2, pad=3,
                       scale=d["scale"], shift=d["shift"], act=act)
    assert_bf16_close(out_f64(out), oracle.maxpool2d(y, k=3, stride=2, pad=1), "stem_neg")


def test_fused_rejects_other_shapes():
    spec = inputs.small_layer("not_stem", 1, 16, 16, 64, 64, 3, 1, 1, seed=(901, 0))
    d = inputs.layer_inputs(spec)
    x = to_dev(d["x"], "bf16")
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    out = torch.empty((1, 8, 8, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(quan.QuanError) as ei:
        quan.quan_qconv2d_maxpool_fwd(x, *w, None, None, None, 1, 16, 16, 64, 64, 3, 3, 1, 1,
                                      quan.QUAN_ACT_RELU, None, 0, out)
    assert ei.value.status == quan.QUAN_ERR_UNSUPPORTED


def test_backbone_fused_stem_is_bit_identical():
    x_bits = inputs.backbone_input(n_images=2)
    stream = torch.cuda.current_stream().cuda_stream
    outs = []
    for fuse in (False, True):
        runner = BackboneRunner(torch, quan, inputs, N=2, x_bits=x_bits, fuse_stem_pool=fuse)
        assert runner.fused == fuse
        runner.step(stream)
        torch.cuda.synchronize()
        assert quan.quan_device_status()[0] == quan.QUAN_OK
        outs.append((runner.outs[1].clone(), runner.output.clone()))
    assert torch.equal(outs[0][0], outs[1][0])  # the pooled stem output
    assert torch.equal(outs[0][1], outs[1][1])  # the backbone output


def test_fused_call_first_in_a_fresh_process():
    # the fused entry point sets up everything it needs on its own (nothing else has
    # been called in the process before it)
    import os
    import subprocess
    import sys
    code = (
        "import torch\n"
        "from paper_2509_05512_gb300 import inputs, quan\n"
        "from paper_2509_05512_gb300.backbone import BackboneRunner\n"
        "r = BackboneRunner(torch, quan, inputs, N=2, fuse_stem_pool=True)\n"
        "r.run_layer(0, torch.cuda.current_stream().cuda_stream)\n"
        "torch.cuda.synchronize()\n"
        "assert quan.quan_last_kernel() == 'qconv_stem_pool_kernel'\n"
        "assert quan.quan_device_status()[0] == quan.QUAN_OK\n")
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    res = subprocess.run([sys.executable, "-c", code], cwd=root, capture_output=True, text=True,
                         timeout=300)
    assert res.returncode == 0, res.stderr[-2000:]


def test_fused_bounded_wait_timeout_and_recovery():
    # the failure-injection path: the first issuer waits on a barrier nothing arrives on;
    # the timeout is reported and the next call on the same context is correct
    spec = inputs.small_layer("stem_inject", 2, 32, 32, 4, 64, 7, 2, 3, seed=(903, 0))
    quan.quan_set_wait_limit_ns(5_000_000)
    quan.quan_set_fault_injection(True)
    try:
        d = inputs.layer_inputs(spec)
        x = to_dev(d["x"], "bf16")
        w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
        out = torch.empty((2, 8, 8, 64), dtype=torch.bfloat16, device="cuda")
        quan.quan_qconv2d_maxpool_fwd(x, *w, None, None, None, 2, 32, 32, 4, 64, 7, 7, 2, 3,
                                      quan.QUAN_ACT_RELU, None, 0, out)
        st, bits = quan.quan_device_status()
        assert st == quan.QUAN_ERR_DEVICE_TIMEOUT and bits != 0
    finally:
        quan.quan_set_fault_injection(False)
        quan.quan_set_wait_limit_ns(0)
    d, out, ref_gpu = run_both(spec, quan.QUAN_ACT_RELU)
    assert torch.equal(out, ref_gpu)


# ------------------------------------------------------------------ RGB input (Eq. 4 fused)

def run_rgb(N, H, W, act, seed, max_ctas=0):
    """The RGB stem-pool call and, for comparison, quan_poincare_fwd followed by the
    quaternion-input call, on the same fp32 pixels and weights."""
    spec = inputs.small_layer("stem_rgb", N, H, W, 4, 64, 7, 2, 3, seed=(904, seed), act=act)
    d = inputs.layer_inputs(spec)
    rgb_np = np.random.default_rng(905 + seed).uniform(0.0, 1.0, size=(N, H, W, 3))
    rgb_np = rgb_np.astype(np.float32)
    rgb = torch.from_numpy(rgb_np).cuda()
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    sc, sh = to_dev_f32(d["scale"]), to_dev_f32(d["shift"])
    Ho, Wo = (H - 1) // 2 + 1, (W - 1) // 2 + 1
    out = torch.full((N, (Ho - 1) // 2 + 1, (Wo - 1) // 2 + 1, 64), float("nan"),
                     dtype=torch.bfloat16, device="cuda")
    quan.quan_set_tc_tiles(0, 0, max_ctas, 0)
    try:
        quan.quan_qconv2d_maxpool_rgb_fwd(rgb, *w, None, sc, sh, N, H, W, 64, 7, 7, 2, 3, act,
                                          out)
        torch.cuda.synchronize()
        assert quan.quan_last_kernel() == "qconv_stem_pool_kernel<rgb>"
        mapped = quan.poincare(rgb)
        ref = torch.full_like(out, float("nan"))
        quan.quan_qconv2d_maxpool_fwd(mapped, *w, None, sc, sh, N, H, W, 4, 64, 7, 7, 2, 3, act,
                                      None, 0, ref)
        torch.cuda.synchronize()
    finally:
        quan.quan_set_tc_tiles(0, 0, 0, 0)
    assert quan.quan_device_status()[0] == quan.QUAN_OK
    return d, rgb_np, out, ref


RGB_CASES = [
    # name, N, H, W, act, max_ctas
    ("square", 2, 32, 32, quan.QUAN_ACT_RELU, 0),
    ("odd_h", 2, 35, 64, quan.QUAN_ACT_SILU, 0),      # Ho = 18, Hp = 9; 64 wide
    ("wide", 1, 12, 224, quan.QUAN_ACT_RELU, 0),      # a full 112-pixel output row
    ("bands", 3, 40, 32, quan.QUAN_ACT_NONE, 3),      # bands across images
]


@pytest.mark.parametrize("case", RGB_CASES, ids=[c[0] for c in RGB_CASES])
def test_rgb_stem_pool_equals_mapping_then_stem_and_oracle(case):
    name, N, H, W, act, max_ctas = case
    d, rgb_np, out, ref = run_rgb(N, H, W, act, len(name), max_ctas)
    assert torch.equal(out, ref)
    # the oracle: Eq. 4 on the same fp32 pixels, rounded to bf16 as the kernel's loader
    # stores them, then the stem convolution and the pooling in fp64
    q = oracle.poincare(rgb_np.astype(np.float64))
    q_bits = inputs.to_bf16_bits(q.astype(np.float32))
    f = lambda k: host_f64(d[k], "bf16")
    y = oracle.qconv2d(host_f64(q_bits, "bf16"), f("wr"), f("wi"), f("wj"), f("wk"), stride=2,
                       pad=3, scale=d["scale"], shift=d["shift"], act=act)
    assert_bf16_close(out_f64(out), oracle.maxpool2d(y, k=3, stride=2, pad=1), name)


def test_rgb_stem_pool_rejects_width_not_multiple_of_32():
    spec = inputs.small_layer("stem_rgb_w", 1, 16, 30, 4, 64, 7, 2, 3, seed=(906, 0))
    d = inputs.layer_inputs(spec)
    rgb = torch.zeros((1, 16, 30, 3), dtype=torch.float32, device="cuda")
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    out = torch.empty((1, 4, 8, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(quan.QuanError) as ei:
        quan.quan_qconv2d_maxpool_rgb_fwd(rgb, *w, None, None, None, 1, 16, 30, 64, 7, 7, 2, 3,
                                          quan.QUAN_ACT_RELU, out)
    assert ei.value.status == quan.QUAN_ERR_UNSUPPORTED
