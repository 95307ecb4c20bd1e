"""GPU parity: libquan (through the C ABI) against the fp64 oracle on identical seeded
inputs.  Small layers are compared element by element over several tiles with a
ragged tail; the full-size layers of the five configurations are compared on sampled
output pixels (first/last pixels, tile boundaries, random picks) plus quaternion
identities that hold at any size."""
import dataclasses

import numpy as np
import pytest

torch = pytest.importorskip("torch")

import oracle
from paper_2509_05512_gb300 import build, inputs, quan
from tests._util import (assert_bf16_close, assert_f32_close, host_f64, out_f64, to_dev,
                         to_dev_f32)

pytestmark = pytest.mark.gpu

NEEDS_GPU = not torch.cuda.is_available()


@pytest.fixture(scope="module", autouse=True)
def lib():
    if NEEDS_GPU:
        pytest.skip("no CUDA device")
    build.build_library()
    lib = quan.load()
    yield lib
    quan.quan_set_path(quan.QUAN_PATH_AUTO)
    quan.quan_set_tc_tiles(0, 0, 0, 0)


@pytest.fixture(autouse=True)
def _reset_paths():
    yield
    quan.quan_set_path(quan.QUAN_PATH_AUTO)
    quan.quan_set_tc_tiles(0, 0, 0, 0)
    quan.quan_set_fault_injection(False)
    quan.quan_set_wait_limit_ns(0)
    quan.quan_set_tc_halo(True)
    quan.quan_set_tc_issuers(0)
    quan.quan_set_tc_band_rows(0)


def run_gpu(d, path=quan.QUAN_PATH_AUTO, guard=True):
    """Upload a generated layer, run it through the C ABI, return float64 output."""
    spec = d["spec"]
    dt = spec.dtype
    x = to_dev(d["x"], dt)
    w = [to_dev(d[k], dt) for k in ("wr", "wi", "wj", "wk")]
    bias, scale, shift = (to_dev_f32(d[k]) for k in ("bias", "scale", "shift"))
    res = to_dev(d["residual"], dt) if d["residual"] is not None else None
    tdt = torch.bfloat16 if dt == "bf16" else torch.float32
    n_out = spec.N * spec.Ho * spec.Wo * spec.Cout
    pad = 4096
    buf = torch.full((n_out + 2 * pad,), float("nan"), dtype=tdt, device="cuda")
    out = buf[pad:pad + n_out].view(spec.N, spec.Ho, spec.Wo, spec.Cout)
    quan.quan_set_path(path)
    quan.qconv2d(x, *w, stride=spec.stride, pad=spec.pad, bias=bias, scale=scale, shift=shift,
                 act=spec.act, residual=res, out=out)
    torch.cuda.synchronize()
    if guard:  # guard bands on both sides of the output stay untouched
        assert torch.isnan(buf[:pad].float()).all() and torch.isnan(buf[pad + n_out:].float()).all()
    st, bits = quan.quan_device_status()
    assert st == quan.QUAN_OK, bits
    return out_f64(out), quan.quan_last_path()


def oracle_full(d):
    spec = d["spec"]
    dt = spec.dtype
    return oracle.qconv2d(host_f64(d["x"], dt), *(host_f64(d[k], dt) for k in ("wr", "wi", "wj", "wk")),
                          stride=spec.stride, pad=spec.pad, bias=d["bias"], scale=d["scale"],
                          shift=d["shift"], residual=host_f64(d["residual"], dt), act=spec.act)


def check(spec, path=quan.QUAN_PATH_AUTO, expect_path=None, **kw):
    d = inputs.layer_inputs(spec)
    got, used = run_gpu(d, path)
    if expect_path is not None:
        assert used == expect_path
    ref = oracle_full(d)
    if spec.dtype == "bf16":
        return assert_bf16_close(got, ref, spec.name)
    return assert_f32_close(got, ref, spec.name)


# ------------------------------------------------------------------ configs 0 and 1 in full

def test_config0_fp32_full():
    check(inputs.LAYERS["c0"], expect_path=quan.QUAN_PATH_SIMT)


@pytest.mark.parametrize("path", [quan.QUAN_PATH_TC, quan.QUAN_PATH_SIMT])
def test_config1_full(path):
    check(inputs.LAYERS["c1"], path=path, expect_path=path)


@pytest.mark.parametrize("mode", [1, 2, 3, 7])
def test_config1_full_every_mode(mode):
    quan.quan_set_tc_tiles(0, 0, 0, mode)
    check(inputs.LAYERS["c1"], path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)


WS_CASES = [
    ("ws_ragged", 3, 13, 11, 64, 64, 3, 1, 1, {}),
    ("ws_stride2", 2, 15, 17, 64, 64, 3, 2, 1, {"residual": True}),
    ("ws_1x1", 2, 9, 7, 64, 64, 1, 1, 0, {"bias": True, "act": quan.QUAN_ACT_SILU}),
    ("ws_5x1", 1, 9, 8, 64, 64, 5, 1, 2, {"kw": 1}),
    # row-block halo staging: partial last block (R = 5), 112-row tiles, 1x1, valid conv
    ("ws_halo_24", 2, 24, 24, 64, 64, 3, 1, 1, {"residual": True}),
    ("ws_halo_56", 1, 56, 56, 64, 64, 3, 1, 1, {}),
    ("ws_halo_1x1", 2, 16, 16, 64, 64, 1, 1, 0, {"act": quan.QUAN_ACT_NONE}),
    ("ws_halo_valid", 2, 18, 18, 64, 64, 3, 1, 0, {"bias": True}),
    ("ws_halo_1x3", 1, 12, 16, 64, 64, 1, 1, 0, {"kw": 3}),
]


@pytest.mark.parametrize("issuers", [0, 2, 3])
@pytest.mark.parametrize("halo", [1, 0])
@pytest.mark.parametrize("case", WS_CASES, ids=[c[0] for c in WS_CASES])
def test_tc_weight_stationary_layers(case, halo, issuers):
    name, N, H, W, Cin, Cout, k, s, p, extra = case
    spec = inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(205, len(name)), **extra)
    quan.quan_set_tc_tiles(0, 0, 0, 3)
    quan.quan_set_tc_halo(bool(halo))
    quan.quan_set_tc_issuers(issuers)
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    kernel = quan.quan_last_kernel()
    assert kernel.startswith("qconv_ws_kernel<")
    if issuers:
        assert kernel.endswith("issuers=%d>" % issuers)


@pytest.mark.parametrize("issuers", [2, 3])
@pytest.mark.parametrize("halo", [1, 0])
def test_tc_weight_stationary_few_ctas(halo, issuers):
    # 96 tiles on 3 CTAs: the accumulator buffers and every issuer's stages wrap many
    # times
    spec = inputs.small_layer("ws_few", 12, 32, 32, 64, 64, 3, 1, 1, residual=True,
                              seed=(209, halo))
    quan.quan_set_tc_tiles(0, 0, 3, 3)
    quan.quan_set_tc_halo(bool(halo))
    quan.quan_set_tc_issuers(issuers)
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)


@pytest.mark.parametrize("issuers", [2, 3])
@pytest.mark.parametrize("halo", [1, 0])
def test_config1_weight_stationary_staging(halo, issuers):
    quan.quan_set_tc_tiles(0, 0, 0, 3)
    quan.quan_set_tc_halo(bool(halo))
    quan.quan_set_tc_issuers(issuers)
    check(inputs.LAYERS["c1"], path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)


# vertical-tap kernel (3x3 stride 1, 16 -> 16 quaternion channels): one box per input row
# (P = Wo + 2 lanes per image) or three (P = Wo, Wo dividing 128), bands of 1 to 4 output
# rows, image groups with a ragged last group, padding 0 and 2, the epilogue's options
VS_CASES = [
    # name, N, H, W, pad, extra
    ("vs_56", 3, 56, 56, 1, {"residual": True}),              # 1 box, E = 2, ragged groups
    ("vs_32", 5, 32, 32, 1, {}),                               # 3 boxes, E = 4
    ("vs_13x11", 3, 13, 11, 1, {"bias": True, "act": quan.QUAN_ACT_SILU}),  # 1 box, E = 9
    ("vs_16", 9, 16, 16, 1, {"residual": True}),               # 3 boxes, E = 8
    ("vs_valid", 2, 18, 18, 0, {"iqbn": False, "act": quan.QUAN_ACT_NONE}),  # Wo = 16
    ("vs_pad2", 3, 10, 6, 2, {}),                              # Wo = 8: 3 boxes, E = 16
    ("vs_wide", 2, 5, 126, 1, {}),                             # P = 128, one image
    ("vs_tiny", 2, 1, 1, 1, {}),                               # Wo = 1: E = 128
    ("vs_24", 2, 24, 24, 1, {"residual": True}),               # 1 box, E = 4
]


@pytest.mark.parametrize("rows", [0, 1, 2, 3, 4])
@pytest.mark.parametrize("case", VS_CASES, ids=[c[0] for c in VS_CASES])
def test_tc_vertical_tap_layers(case, rows):
    name, N, H, W, p, extra = case
    spec = inputs.small_layer(name, N, H, W, 64, 64, 3, 1, p, seed=(206, len(name)), **extra)
    quan.quan_set_tc_tiles(0, 0, 0, 7)
    quan.quan_set_tc_band_rows(rows)
    try:
        check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    finally:
        quan.quan_set_tc_band_rows(0)
    kernel = quan.quan_last_kernel()
    assert kernel.startswith("qconv_vs_kernel<"), kernel
    if rows:
        assert ",rows=%d" % rows in kernel, kernel


@pytest.mark.parametrize("rows", [1, 4])
def test_tc_vertical_tap_few_ctas(rows):
    # 2 CTAs: the stage ring and both band buffers wrap many times
    spec = inputs.small_layer("vs_few", 7, 32, 32, 64, 64, 3, 1, 1, residual=True,
                              seed=(207, rows))
    quan.quan_set_tc_tiles(0, 0, 2, 7)
    quan.quan_set_tc_band_rows(rows)
    try:
        check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    finally:
        quan.quan_set_tc_band_rows(0)


@pytest.mark.parametrize("case", [("vs_auto_56", 2, 56, 56, True), ("vs_auto_32", 2, 32, 32, False),
                                  ("vs_auto_13x11", 2, 13, 11, True)], ids=lambda c: c[0])
def test_tc_vertical_tap_default_choice(case):
    # mode 0 takes the vertical-tap kernel where one box per input row serves, the
    # weight-stationary kernel where the row needs three boxes
    name, N, H, W, vs = case
    spec = inputs.small_layer(name, N, H, W, 64, 64, 3, 1, 1, seed=(210, len(name)))
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    kernel = quan.quan_last_kernel()
    assert kernel.startswith("qconv_vs_kernel<boxes=1" if vs else "qconv_ws_kernel<"), kernel


def test_tc_vertical_tap_mode_rejects_other_shapes():
    spec = inputs.small_layer("vs_reject", 1, 9, 9, 64, 64, 3, 2, 1, seed=(208, 0))
    quan.quan_set_tc_tiles(0, 0, 0, 7)
    with pytest.raises(quan.QuanError):
        run_gpu(inputs.layer_inputs(spec), quan.QUAN_PATH_TC, guard=False)


# split K (quan_qconv2d_fwd_ex): the (tile, K block) iterations cut evenly over a grid that
# the tile count does not divide, tiles shared by two CTAs finished through the workspace
SPLITK_CASES = [
    # name, N, H, W, Cin, Cout, k, stride, pad, extra, grid, (kappa, bnq, mode)
    ("sk_pair_res", 4, 12, 12, 128, 256, 3, 1, 1, {"residual": True}, 3, (0, 0, 0)),  # 5 tiles
    ("sk_quad", 4, 12, 12, 128, 256, 3, 1, 1, {}, 4, (0, 0, 1)),
    ("sk_two_ntiles", 3, 11, 13, 128, 256, 3, 1, 1, {"bias": True, "act": quan.QUAN_ACT_SILU},
     5, (32, 32, 2)),                                        # 8 tiles (2 channel blocks)
    ("sk_kappa16", 4, 10, 12, 64, 128, 3, 1, 1, {}, 3, (16, 32, 2)),  # 4 tiles
    ("sk_stride2", 5, 15, 17, 128, 256, 3, 2, 1, {}, 2, (0, 0, 0)),   # 3 tiles
    ("sk_5x5", 2, 11, 12, 64, 256, 5, 1, 2, {"residual": True}, 2, (0, 0, 0)),  # 3 tiles
]


def run_split(d, ws, grid, tiles):
    kappa, bnq, mode = tiles
    quan.quan_set_tc_tiles(kappa, bnq, grid, mode)
    spec = d["spec"]
    x = to_dev(d["x"], "bf16")
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    bias, scale, shift = (to_dev_f32(d[k]) for k in ("bias", "scale", "shift"))
    res = to_dev(d["residual"], "bf16") if d["residual"] is not None else None
    quan.quan_set_path(quan.QUAN_PATH_TC)
    y = quan.qconv2d(x, *w, stride=spec.stride, pad=spec.pad, bias=bias, scale=scale,
                     shift=shift, act=spec.act, residual=res, workspace=ws)
    torch.cuda.synchronize()
    assert quan.quan_device_status()[0] == quan.QUAN_OK
    return y, quan.quan_last_kernel()


@pytest.mark.parametrize("case", SPLITK_CASES, ids=[c[0] for c in SPLITK_CASES])
def test_tc_split_k_layers(case):
    name, N, H, W, Cin, Cout, k, st, p, extra, grid, tiles = case
    spec = inputs.small_layer(name, N, H, W, Cin, Cout, k, st, p, seed=(211, len(name)), **extra)
    d = inputs.layer_inputs(spec)
    ws = quan.fwd_workspace()
    y1, kernel = run_split(d, ws, grid, tiles)
    assert kernel.endswith(",splitk>"), kernel
    ref = oracle_full(d)
    assert_bf16_close(out_f64(y1), ref, name)
    # a second call on the same workspace: the same result (the split is deterministic), and
    # every flag is clear again afterwards
    y2, _ = run_split(d, ws, grid, tiles)
    assert torch.equal(y1, y2)
    flags = ws.view(torch.uint8)[grid * 512 * (tiles[1] or 64) * 4:]
    assert int(flags[:grid * 4].count_nonzero()) == 0
    # no workspace: the unsplit kernel, within rounding of the split one
    y0, kernel0 = run_split(d, None, grid, tiles)
    assert not kernel0.endswith(",splitk>")
    assert_bf16_close(out_f64(y0), ref, name + "-unsplit")


def test_tc_split_k_full_size_stage4():
    # the backbone's 7x7 512 -> 512 residual layer on the full grid (196 tiles on the SMs)
    spec = inputs.small_layer("sk_stage4", 256, 7, 7, 512, 512, 3, 1, 1, residual=True,
                              seed=(212, 0))
    d = inputs.layer_inputs(spec)
    ws = quan.fwd_workspace()
    y1, kernel = run_split(d, ws, 0, (0, 0, 0))
    assert kernel.endswith(",splitk>"), kernel
    y0, kernel0 = run_split(d, None, 0, (0, 0, 0))
    a, b = out_f64(y1), out_f64(y0)
    rel = float(np.linalg.norm(a - b) / np.linalg.norm(b))
    assert rel < 2e-3, rel
    # images 0, N/2, N-1 against the oracle
    for n in (0, 128, 255):
        dn = dict(d)
        dn["x"] = d["x"][n:n + 1]
        dn["residual"] = d["residual"][n:n + 1]
        dn["spec"] = dataclasses.replace(spec, N=1)
        assert_bf16_close(a[n:n + 1], oracle_full(dn), "sk_stage4 image %d" % n)


# ------------------------------------------------------------------ tensor-core small layers

SMALL_TC = [
    # name, N, H, W, Cin, Cout, k, stride, pad, extra
    ("ragged", 3, 13, 11, 64, 64, 3, 1, 1, {}),
    ("stride2", 2, 15, 17, 64, 128, 3, 2, 1, {}),
    ("pointwise", 2, 12, 10, 128, 256, 1, 1, 0, {}),
    ("pointwise_s2", 2, 14, 14, 64, 128, 1, 2, 0, {"act": quan.QUAN_ACT_NONE}),
    ("tiny_image", 1, 1, 1, 64, 64, 3, 1, 1, {}),
    ("stem_like_7x7", 1, 20, 18, 64, 64, 7, 2, 3, {}),
    ("wide_q", 1, 9, 9, 256, 256, 3, 1, 1, {}),
    ("qin48", 2, 7, 9, 192, 64, 3, 1, 1, {}),
    ("bias_silu", 2, 9, 8, 64, 128, 3, 1, 1, {"bias": True, "act": quan.QUAN_ACT_SILU}),
    ("no_iqbn", 2, 9, 8, 64, 64, 3, 1, 1, {"iqbn": False, "act": quan.QUAN_ACT_NONE}),
    ("residual", 2, 10, 9, 128, 128, 3, 1, 1, {"residual": True}),
    ("pad2_5x5", 1, 11, 12, 64, 64, 5, 1, 2, {}),
]


@pytest.mark.parametrize("case", SMALL_TC, ids=[c[0] for c in SMALL_TC])
def test_tc_small_layers(case):
    name, N, H, W, Cin, Cout, k, s, p, extra = case
    spec = inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(200, len(name)), **extra)
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)


# every (kappa, bnq, mode)
TILE_CASES = [(k, b, m) for m in (1, 2) for k in (16, 32, 64) for b in (16, 32, 64)]


@pytest.mark.parametrize("kappa,bnq,mode", TILE_CASES)
def test_tc_tile_variants(kappa, bnq, mode):
    spec = inputs.small_layer("tiles", 2, 11, 13, 256, 256, 3, 1, 1, seed=(201, kappa + bnq))
    quan.quan_set_tc_tiles(kappa, bnq, 0, mode)
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    assert quan.quan_last_kernel() == "qconv_tc_kernel<%s,kappa=%d,bnq=%d>" % (
        "quad" if mode == 1 else "pair", kappa, bnq)


@pytest.mark.parametrize("mode", [1, 2])
def test_tc_pair_mode_layers(mode):
    # stride-2, ragged tail, residual and both modes on the same layer
    spec = inputs.small_layer("pairs", 3, 15, 13, 128, 256, 3, 2, 1, residual=True,
                              seed=(204, mode))
    quan.quan_set_tc_tiles(0, 0, 0, mode)
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)


def test_tc_few_ctas_many_tiles():
    # a small persistent grid walks many tiles per CTA (accumulator double buffering,
    # ring wrap-around many times)
    spec = inputs.small_layer("few_ctas", 4, 16, 16, 64, 128, 3, 1, 1, seed=(202, 0))
    quan.quan_set_tc_tiles(0, 16, 3, 0)
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)


# ------------------------------------------------------------------ pixel-pair gather (Cin = 4)

GATHER_CASES = [
    # name, N, H, W, Cin, Cout, k, stride, pad, extra
    ("stem_7x7", 2, 32, 32, 4, 64, 7, 2, 3, {}),             # 512 pixels, 4 whole tiles
    ("stem_ragged", 2, 22, 22, 4, 64, 7, 2, 3, {}),          # 242 pixels, ragged tail
    ("stem_rect_res", 3, 19, 30, 4, 64, 7, 2, 3,             # odd H, residual, SiLU
     {"residual": True, "act": quan.QUAN_ACT_SILU}),
    ("even_pad_5x5", 2, 18, 16, 4, 64, 5, 2, 2, {"bias": True}),  # 15 units + 1 zero unit
    ("k3_pad1", 2, 20, 14, 4, 64, 3, 2, 1, {"iqbn": False, "act": quan.QUAN_ACT_NONE}),
    ("k4x2_valid", 1, 17, 12, 4, 64, 4, 2, 0, {"kw": 2}),     # one pair per filter row
    ("tiny", 1, 2, 2, 4, 64, 7, 2, 3, {}),                   # a single output pixel
    ("wide_rows", 1, 6, 300, 4, 64, 7, 2, 3, {}),            # Wo = 150: two tiles per row
    ("odd_kw", 2, 12, 20, 4, 64, 3, 2, 2, {"kw": 5}),        # 3x5, pad 2: zero pair slot
]


@pytest.mark.parametrize("case", GATHER_CASES, ids=[c[0] for c in GATHER_CASES])
def test_tc_pixel_pair_gather_layers(case):
    name, N, H, W, Cin, Cout, k, s, p, extra = case
    spec = inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(206, len(name)), **extra)
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    assert quan.quan_last_kernel() == "qconv_pairs_kernel"


def test_tc_pixel_pair_gather_few_ctas():
    # 32 tiles on 3 CTAs: every CTA wraps the stage ring and both accumulators many times
    spec = inputs.small_layer("gather_few", 4, 64, 64, 4, 64, 7, 2, 3, seed=(207, 0))
    quan.quan_set_tc_tiles(0, 0, 3, 4)
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)


def test_tc_pixel_pair_gather_mode_rejects_other_shapes():
    spec = inputs.small_layer("not_stem", 1, 8, 8, 64, 64, 3, 1, 1, seed=(208, 0))
    d = inputs.layer_inputs(spec)
    quan.quan_set_tc_tiles(0, 0, 0, 4)
    with pytest.raises(quan.QuanError) as ei:
        run_gpu(d, path=quan.QUAN_PATH_TC)
    assert ei.value.status == quan.QUAN_ERR_UNSUPPORTED


# ------------------------------------------------------------------ pointwise (1x1) kernel

PW_CASES = [
    # name, N, H, W, Cin, Cout, k, stride, pad, extra
    ("pw_s1_ragged", 3, 9, 13, 64, 128, 1, 1, 0, {}),        # 351 pixels: a ragged tile
    ("pw_s1_tiny", 1, 3, 5, 128, 256, 1, 1, 0, {}),          # 15 pixels, less than a tile
    ("pw_s1_cin512", 2, 16, 17, 512, 256, 1, 1, 0,           # 8 K chunks through 3 stages
     {"bias": True, "act": quan.QUAN_ACT_SILU}),
    ("pw_s1_cout512", 1, 20, 20, 256, 512, 1, 1, 0,          # 4 channel blocks
     {"iqbn": False, "act": quan.QUAN_ACT_NONE}),
    ("pw_s2_shortcut", 3, 28, 28, 64, 128, 1, 2, 0,          # 18 output rows per tile
     {"act": quan.QUAN_ACT_NONE}),
    ("pw_s2_wide", 2, 14, 14, 256, 512, 1, 2, 0, {"act": quan.QUAN_ACT_NONE}),  # Wo = 7
    ("pw_s2_odd_out", 1, 30, 22, 128, 256, 1, 2, 0, {}),     # Ho = 15, Wo = 11: one short tile
]


@pytest.mark.parametrize("case", PW_CASES, ids=[c[0] for c in PW_CASES])
def test_tc_pointwise_layers(case):
    name, N, H, W, Cin, Cout, k, s, p, extra = case
    spec = inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(209, len(name)), **extra)
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    assert quan.quan_last_kernel() == "qconv_pw_kernel<s%d>" % s


@pytest.mark.parametrize("max_ctas", [2, 5])
def test_tc_pointwise_few_ctas(max_ctas):
    # 2 channel blocks on a grid of 2 (5 rounds down to 4): every CTA walks many pixel
    # tiles, wrapping the stage ring and both accumulators many times
    spec = inputs.small_layer("pw_few", 4, 32, 32, 128, 256, 1, 1, 0, seed=(210, max_ctas))
    quan.quan_set_tc_tiles(0, 0, max_ctas, 5)
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    assert quan.quan_last_kernel() == "qconv_pw_kernel<s1>"


def test_tc_pointwise_matches_pair_kernel():
    # the same stride-2 shortcut on the pointwise and the pair kernel: both within the
    # oracle's tolerance, and close to each other
    spec = inputs.small_layer("pw_vs_pair", 2, 28, 28, 128, 256, 1, 2, 0, seed=(211, 0),
                              act=quan.QUAN_ACT_NONE)
    d = inputs.layer_inputs(spec)
    ref = oracle_full(d)
    outs = []
    for mode, kern in ((5, "qconv_pw_kernel<s2>"), (2, None)):
        quan.quan_set_tc_tiles(0, 0, 0, mode)
        got, used = run_gpu(d, path=quan.QUAN_PATH_TC)
        assert used == quan.QUAN_PATH_TC
        if kern:
            assert quan.quan_last_kernel() == kern
        assert_bf16_close(got, ref, "mode %d" % mode)
        outs.append(got)
    assert_bf16_close(outs[0], outs[1], "pointwise vs pair")


def test_tc_pointwise_mode_rejects_other_shapes():
    for args in ((1, 8, 8, 64, 128, 3, 1, 1), (1, 8, 8, 64, 64, 1, 1, 0),
                 (1, 9, 8, 64, 128, 1, 2, 0)):   # 3x3; Cout 64; odd H at stride 2
        spec = inputs.small_layer("not_pw", *args, seed=(212, 0))
        d = inputs.layer_inputs(spec)
        quan.quan_set_tc_tiles(0, 0, 0, 5)
        with pytest.raises(quan.QuanError) as ei:
            run_gpu(d, path=quan.QUAN_PATH_TC)
        assert ei.value.status == quan.QUAN_ERR_UNSUPPORTED


# ------------------------------------------------------------------ CTA-pair kernel (Cout 128)

HALO, HALO2, PER_TAP = "qconv_cg2_kernel<halo>", "qconv_cg2_kernel<halo2>", "qconv_cg2_kernel"
CG2_CASES = [
    # name, N, H, W, Cin, Cout, k, stride, pad, extra, kernel
    # halo staging (stride 1, 3x3): 8 rows of 15 per tile, the image's second tile 6 rows
    ("cg2_s1_res", 2, 14, 13, 128, 128, 3, 1, 1, {"residual": True}, HALO),
    ("cg2_one_tile", 1, 8, 8, 128, 128, 3, 1, 1,                         # one tile: the odd
     {"bias": True, "act": quan.QUAN_ACT_SILU}, HALO),                   # CTA has none
    ("cg2_no_iqbn", 2, 12, 12, 64, 128, 3, 1, 1,                         # one 64-channel chunk
     {"iqbn": False, "act": quan.QUAN_ACT_NONE}, HALO),
    ("cg2h_wide", 1, 6, 90, 128, 128, 3, 1, 1, {}, HALO),    # 92-pixel pitch: one row per tile
    ("cg2h_pad0", 2, 10, 12, 128, 128, 3, 1, 0, {}, HALO),   # box from column 0
    ("cg2h_pad2", 1, 9, 7, 64, 128, 3, 1, 2, {"residual": True}, HALO),  # box from column -2
    ("cg2h_deep", 3, 28, 28, 128, 128, 3, 1, 1, {"residual": True}, HALO),  # the stage-2 shape
    # stride-2 halo staging (four parity boxes per stage): odd input sizes, one tile of
    # 8 rows of 10 per image
    ("cg2h2_odd", 3, 15, 17, 64, 128, 3, 2, 1, {}, HALO2),
    ("cg2h2_stage2", 3, 56, 56, 64, 128, 3, 2, 1, {"residual": True}, HALO2),  # 7 tiles of 4 rows
    ("cg2h2_ragged", 2, 20, 58, 64, 128, 3, 2, 1,                # 29 columns, 10 rows: the
     {"bias": True, "act": quan.QUAN_ACT_SILU}, HALO2),          # third tile has 2 of 4 rows
    ("cg2h2_pad0", 2, 13, 13, 64, 128, 3, 2, 0, {}, HALO2),      # boxes from column 0 and 1
    ("cg2h2_pad2", 1, 11, 11, 64, 128, 3, 2, 2, {"residual": True}, HALO2),  # from -2 and -1
    ("cg2h2_one_col", 2, 9, 2, 64, 128, 3, 2, 1, {}, HALO2),     # Wo = 1: 64 rows per tile
    # per-tap staging: other filters, rows too wide for two halo stages, or a block weight
    # that leaves room for one stride-2 stage only
    ("cg2_s2_wide_k", 3, 15, 17, 128, 128, 3, 2, 1, {}, PER_TAP),        # 216 pixels
    ("cg2_5x1", 2, 11, 9, 128, 128, 5, 1, 2, {"kw": 1}, PER_TAP),        # 5 taps x 128
    ("cg2_too_wide", 1, 3, 100, 128, 128, 3, 1, 1, {}, PER_TAP),         # 102-pixel pitch
    ("cg2_s2_too_wide", 1, 5, 120, 64, 128, 3, 2, 1, {}, PER_TAP),       # 61-pixel pitch
]


@pytest.mark.parametrize("case", CG2_CASES, ids=[c[0] for c in CG2_CASES])
def test_tc_cta_pair_layers(case):
    name, N, H, W, Cin, Cout, k, s, p, extra, kernel = case
    spec = inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(213, len(name)), **extra)
    quan.quan_set_tc_tiles(0, 0, 0, 6)
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    assert quan.quan_last_kernel() == kernel


@pytest.mark.parametrize("max_ctas", [4, 6])
def test_tc_cta_pair_few_pairs(max_ctas):
    # 2 or 3 pairs walk many pair tiles: every stage ring and all four accumulators wrap
    spec = inputs.small_layer("cg2_few", 4, 20, 20, 128, 128, 3, 1, 1, residual=True,
                              seed=(214, max_ctas))
    quan.quan_set_tc_tiles(0, 0, max_ctas, 6)
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    assert quan.quan_last_kernel() == HALO


@pytest.mark.parametrize("max_ctas", [4, 6])
def test_tc_cta_pair_per_tap_few_pairs(max_ctas):
    # the per-tap staging's ring (12 stages) wraps many times
    spec = inputs.small_layer("cg2_few_s2", 4, 30, 30, 128, 128, 3, 2, 1, seed=(217, max_ctas))
    quan.quan_set_tc_tiles(0, 0, max_ctas, 6)
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    assert quan.quan_last_kernel() == PER_TAP


@pytest.mark.parametrize("max_ctas", [2, 6])
def test_tc_cta_pair_stride2_few_pairs(max_ctas):
    # one or three pairs: the two-stage ring of parity boxes and the four accumulators wrap
    # many times (6 images of 2 tiles of 8 rows)
    spec = inputs.small_layer("cg2h2_few", 6, 30, 30, 64, 128, 3, 2, 1, residual=True,
                              seed=(218, max_ctas))
    quan.quan_set_tc_tiles(0, 0, max_ctas, 6)
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    assert quan.quan_last_kernel() == HALO2


def test_tc_cta_pair_stride2_default_choice():
    # the backbone's first stage-2 convolution (3x3 / 2, 64 -> 128) takes the CTA-pair
    # kernel with parity boxes by default
    spec = inputs.small_layer("cg2h2_default", 2, 56, 56, 64, 128, 3, 2, 1, seed=(219, 0))
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)
    assert quan.quan_last_kernel() == HALO2


def test_tc_cta_pair_matches_pair_kernel():
    # the stage-2 shape of the backbone on the CTA-pair kernel (the default choice for it)
    # and on the pair kernel: both within the oracle's tolerance and close to each other
    spec = inputs.small_layer("cg2_vs_pair", 2, 28, 28, 128, 128, 3, 1, 1, seed=(215, 0))
    d = inputs.layer_inputs(spec)
    ref = oracle_full(d)
    outs = []
    for mode, kern in ((0, HALO), (2, "qconv_tc_kernel<pair,kappa=32,bnq=32>")):
        quan.quan_set_tc_tiles(0, 0, 0, mode)
        got, used = run_gpu(d, path=quan.QUAN_PATH_TC)
        assert used == quan.QUAN_PATH_TC
        assert quan.quan_last_kernel() == kern
        assert_bf16_close(got, ref, "mode %d" % mode)
        outs.append(got)
    assert_bf16_close(outs[0], outs[1], "pair of CTAs vs pair kernel")


def test_tc_cta_pair_mode_rejects_other_shapes():
    for args in ((1, 8, 8, 64, 64, 3, 1, 1), (1, 8, 8, 192, 128, 3, 1, 1)):  # Cout 64; K > 1152
        spec = inputs.small_layer("not_cg2", *args, seed=(216, 0))
        d = inputs.layer_inputs(spec)
        quan.quan_set_tc_tiles(0, 0, 0, 6)
        with pytest.raises(quan.QuanError) as ei:
            run_gpu(d, path=quan.QUAN_PATH_TC)
        assert ei.value.status == quan.QUAN_ERR_UNSUPPORTED


def test_tc_nonsquare_kernel():
    spec = inputs.small_layer("k3x1", 2, 9, 10, 64, 64, 3, 1, 1, kw=1, seed=(203, 0))
    # pad 1 on both sides with kw = 1 widens the output; valid for the oracle too
    check(spec, path=quan.QUAN_PATH_TC, expect_path=quan.QUAN_PATH_TC)


# ------------------------------------------------------------------ CUDA-core path

SMALL_SIMT = [
    ("q3", 2, 7, 6, 12, 8, 3, 1, 1, {}),
    ("stem", 2, 23, 21, 4, 64, 7, 2, 3, {}),
    ("q1_to_q1", 1, 5, 5, 4, 4, 3, 1, 1, {"act": quan.QUAN_ACT_SILU, "bias": True}),
    ("residual", 1, 6, 6, 8, 8, 3, 1, 1, {"residual": True}),
]


@pytest.mark.parametrize("case", SMALL_SIMT, ids=[c[0] for c in SMALL_SIMT])
def test_simt_small_layers(case):
    name, N, H, W, Cin, Cout, k, s, p, extra = case
    spec = inputs.small_layer(name, N, H, W, Cin, Cout, k, s, p, seed=(300, len(name)), **extra)
    check(spec, expect_path=quan.QUAN_PATH_SIMT)


def test_simt_fp32_shapes():
    spec = inputs.small_layer("f32", 2, 9, 7, 8, 12, 3, 2, 1, dtype="f32", bias=True,
                              act=quan.QUAN_ACT_RELU, seed=(301, 0))
    check(spec, expect_path=quan.QUAN_PATH_SIMT)


def test_misaligned_pointer_demotes_to_simt():
    spec = inputs.small_layer("mis", 1, 6, 6, 64, 64, 3, 1, 1, seed=(302, 0))
    d = inputs.layer_inputs(spec)
    x = to_dev(d["x"], "bf16")
    xs = torch.empty(x.numel() + 8, dtype=torch.bfloat16, device="cuda")
    xs[1:1 + x.numel()] = x.flatten()
    xm = xs[1:1 + x.numel()].view_as(x)          # 2-byte aligned only
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    sc, sh = to_dev_f32(d["scale"]), to_dev_f32(d["shift"])
    with pytest.raises(quan.QuanError) as ei:
        quan.quan_set_path(quan.QUAN_PATH_TC)
        quan.qconv2d(xm, *w, stride=1, pad=1, scale=sc, shift=sh, act=spec.act)
    assert ei.value.status == quan.QUAN_ERR_UNSUPPORTED
    quan.quan_set_path(quan.QUAN_PATH_AUTO)
    y = quan.qconv2d(xm, *w, stride=1, pad=1, scale=sc, shift=sh, act=spec.act)
    torch.cuda.synchronize()
    assert quan.quan_last_path() == quan.QUAN_PATH_SIMT
    assert_bf16_close(out_f64(y), oracle_full(d), "misaligned")


def test_misaligned_channel_vector_demotes_to_simt():
    # the tensor-core epilogues read the per-channel vectors 16 bytes at a time
    spec = inputs.small_layer("mis_vec", 1, 6, 6, 64, 64, 3, 1, 1, seed=(302, 1))
    d = inputs.layer_inputs(spec)
    x = to_dev(d["x"], "bf16")
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    sc, sh = to_dev_f32(d["scale"]), to_dev_f32(d["shift"])
    buf = torch.empty(sc.numel() + 4, dtype=torch.float32, device="cuda")
    buf[1:1 + sc.numel()] = sc
    scm = buf[1:1 + sc.numel()]                   # 4-byte aligned only
    with pytest.raises(quan.QuanError) as ei:
        quan.quan_set_path(quan.QUAN_PATH_TC)
        quan.qconv2d(x, *w, stride=1, pad=1, scale=scm, shift=sh, act=spec.act)
    assert ei.value.status == quan.QUAN_ERR_UNSUPPORTED
    quan.quan_set_path(quan.QUAN_PATH_AUTO)
    y = quan.qconv2d(x, *w, stride=1, pad=1, scale=scm, shift=sh, act=spec.act)
    torch.cuda.synchronize()
    assert quan.quan_last_path() == quan.QUAN_PATH_SIMT
    assert_bf16_close(out_f64(y), oracle_full(d), "misaligned-vector")


# ------------------------------------------------------------------ full-size layers, sampled

def sample_points(spec, n_random, seed):
    rng = np.random.default_rng(seed)
    M = spec.N * spec.Ho * spec.Wo
    idx = set([0, 1, M - 1, M - 2, 127, 128, 129, (M // 128) * 128 - 1])
    idx.update(int(i) for i in rng.integers(0, M, n_random))
    idx = sorted(i for i in idx if 0 <= i < M)
    hw = spec.Ho * spec.Wo
    return [(i // hw, (i % hw) // spec.Wo, i % spec.Wo) for i in idx]


@pytest.mark.parametrize("name", ["c2a", "c2b", "c3a", "c3b"])
def test_full_size_layer_whole_images(name):
    # the full launch, compared with the oracle element by element on images 0, N/2, N - 1
    spec = inputs.LAYERS[name]
    d = inputs.layer_inputs(spec)
    got, used = run_gpu(d, guard=True)
    assert used == quan.QUAN_PATH_TC
    images = [0, spec.N // 2, spec.N - 1]
    w = [host_f64(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    ref = oracle.qconv2d(host_f64(d["x"][images], "bf16"), *w, stride=spec.stride,
                         pad=spec.pad, bias=d["bias"], scale=d["scale"], shift=d["shift"],
                         act=spec.act)
    for k, n in enumerate(images):
        assert_bf16_close(got[n], ref[k], "%s image %d" % (name, n))


@pytest.mark.parametrize("name", ["c1", "c2a", "c2b", "c3a", "c3b"])
def test_full_size_layer_sampled(name):
    spec = inputs.LAYERS[name]
    d = inputs.layer_inputs(spec)
    got, used = run_gpu(d, guard=True)
    assert used == quan.QUAN_PATH_TC
    pts = sample_points(spec, 384, 7)
    images = sorted(set(p[0] for p in pts))
    remap = {n: i for i, n in enumerate(images)}
    xs = host_f64(d["x"][images], "bf16")
    w = [host_f64(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    ref = oracle.qconv2d_points(xs, *w, [(remap[n], h, ww) for n, h, ww in pts],
                                stride=spec.stride, pad=spec.pad, bias=d["bias"],
                                scale=d["scale"], shift=d["shift"], act=spec.act)
    g = np.stack([got[n, h, ww] for n, h, ww in pts])
    assert_bf16_close(g, ref, name)
    # whole-output sanity: finite, ReLU non-negative, not all zero
    assert np.isfinite(got).all() and (got >= 0).all() and (got > 0).mean() > 0.2


def _left_mul_unit(wl, unit):
    """Letters of u (x) W for a basis unit u (exact in bf16: a signed permutation)."""
    wr, wi, wj, wk = wl
    if unit == "i":
        return [-wi, wr, -wk, wj]
    if unit == "j":
        return [-wj, wk, wr, -wi]
    return [-wk, -wj, wi, wr]


def _left_mul_out(y, unit, Q):
    r, i, j, k = (y[..., m * Q:(m + 1) * Q] for m in range(4))
    if unit == "i":
        parts = [-i, r, -k, j]
    elif unit == "j":
        parts = [-j, k, r, -i]
    else:
        parts = [-k, -j, i, r]
    return np.concatenate(parts, axis=-1)


@pytest.mark.parametrize("name,unit", [("c2a", "i"), ("c3a", "j"), ("c2b", "k")])
def test_full_size_left_multiplication_identity(name, unit):
    # u (x) (W (x) X) = (u (x) W) (x) X for a constant quaternion u (associativity of
    # Eq. 3, lifted to the convolution by linearity); with u a basis unit both sides
    # are exact signed permutations, so the check covers the whole output.
    # The signed permutations used here: i (x) (a + bi + cj + dk) = -b + ai - dj + ck, etc.
    spec = inputs.LAYERS[name]
    d = inputs.layer_inputs(spec)
    dd = dict(d)
    dd["scale"] = dd["shift"] = None
    base_spec = dataclasses.replace(spec, iqbn=False, act=quan.QUAN_ACT_NONE)
    dd["spec"] = base_spec
    y, _ = run_gpu(dd)
    wl = [d[k] for k in ("wr", "wi", "wj", "wk")]
    # negate bf16 by flipping the sign bit (exact)
    neg = lambda b: (b ^ np.uint16(0x8000)).astype(np.uint16)
    mapping = {"i": [("wi", 1), ("wr", 0), ("wk", 1), ("wj", 0)],
               "j": [("wj", 1), ("wk", 0), ("wr", 0), ("wi", 1)],
               "k": [("wk", 1), ("wj", 1), ("wi", 0), ("wr", 0)]}[unit]
    d2 = dict(dd)
    for L, (src, negate) in zip(("wr", "wi", "wj", "wk"), mapping):
        d2[L] = neg(d[src]) if negate else d[src]
    y2, _ = run_gpu(d2)
    lhs = _left_mul_out(y, unit, spec.Cout // 4)
    rel = np.linalg.norm(y2 - lhs) / np.linalg.norm(lhs)
    assert rel < 1e-3, rel


# ------------------------------------------------------------------ pooling

@pytest.mark.parametrize("shape", [(2, 9, 8, 64, 3, 2, 1), (1, 7, 7, 12, 3, 2, 1),
                                   (2, 112, 112, 64, 3, 2, 1)])
def test_maxpool(shape):
    N, H, W, C, k, s, p = shape
    rng = np.random.default_rng(sum(shape))
    bits = inputs.to_bf16_bits(rng.standard_normal((N, H, W, C)).astype(np.float32))
    x = to_dev(bits, "bf16")
    y = quan.maxpool2d(x, k=k, stride=s, pad=p)
    torch.cuda.synchronize()
    ref = oracle.maxpool2d(host_f64(bits, "bf16"), k=k, stride=s, pad=p)
    np.testing.assert_array_equal(out_f64(y), ref)


# ------------------------------------------------------------------ failure detection

@pytest.mark.parametrize("mode,issuers", [(2, 0), (3, 2), (3, 3), (4, 0), (5, 0), (6, 0),
                                          (6, 1), (6, 2), (7, 0)])
def test_bounded_wait_timeout_every_kernel(mode, issuers):
    # the failure-injection path of the pair-mode, weight-stationary (two and three
    # issuers), gather, pointwise and CTA-pair kernels (the CTA-pair kernel ignores the
    # issuer count, which selects its staging here: halo, stride-2 halo, per tap)
    if mode == 4:
        spec = inputs.small_layer("inject_m", 2, 32, 32, 4, 64, 7, 2, 3, seed=(401, mode))
    elif mode == 5:
        spec = inputs.small_layer("inject_m", 2, 16, 16, 64, 128, 1, 1, 0, seed=(401, mode))
    elif mode == 6:
        spec = inputs.small_layer("inject_m", 2, 16, 16, 128 if issuers == 2 else 64, 128, 3,
                                  1 if issuers == 0 else 2, 1, seed=(401, mode))
        issuers = 0
    else:
        spec = inputs.small_layer("inject_m", 1, 16, 16, 64, 64, 3, 1, 1, seed=(401, mode))
    d = inputs.layer_inputs(spec)
    x = to_dev(d["x"], "bf16")
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    quan.quan_set_path(quan.QUAN_PATH_TC)
    quan.quan_set_tc_tiles(0, 16 if mode == 2 else 0, 0, mode)
    quan.quan_set_tc_issuers(issuers)
    quan.quan_set_wait_limit_ns(5_000_000)
    quan.quan_set_fault_injection(True)
    quan.qconv2d(x, *w, stride=spec.stride, pad=spec.pad, act=spec.act)
    st, bits = quan.quan_device_status()
    assert st == quan.QUAN_ERR_DEVICE_TIMEOUT and bits != 0
    quan.quan_set_fault_injection(False)
    quan.quan_set_wait_limit_ns(0)
    y = quan.qconv2d(x, *w, stride=spec.stride, pad=spec.pad, act=spec.act)
    torch.cuda.synchronize()
    assert quan.quan_device_status()[0] == quan.QUAN_OK
    d2 = dict(d); d2["scale"] = d2["shift"] = None
    assert_bf16_close(out_f64(y), oracle_full(d2), "after-timeout-%d" % mode)


def test_bounded_wait_timeout_split_k():
    # failure injection on a split launch: the waits end with a timeout status, the
    # context stays usable, and after zeroing the workspace again the split call is right
    spec = inputs.small_layer("inject_sk", 4, 12, 12, 128, 256, 3, 1, 1, seed=(402, 0))
    d = inputs.layer_inputs(spec)
    x = to_dev(d["x"], "bf16")
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    ws = quan.fwd_workspace()
    quan.quan_set_path(quan.QUAN_PATH_TC)
    quan.quan_set_tc_tiles(0, 0, 3, 0)
    quan.quan_set_wait_limit_ns(5_000_000)
    quan.quan_set_fault_injection(True)
    quan.qconv2d(x, *w, stride=1, pad=1, act=spec.act, workspace=ws)
    st, bits = quan.quan_device_status()
    assert st == quan.QUAN_ERR_DEVICE_TIMEOUT and bits != 0
    quan.quan_set_fault_injection(False)
    quan.quan_set_wait_limit_ns(0)
    ws.zero_()
    y = quan.qconv2d(x, *w, stride=1, pad=1, act=spec.act, workspace=ws)
    torch.cuda.synchronize()
    assert quan.quan_device_status()[0] == quan.QUAN_OK
    assert quan.quan_last_kernel().endswith(",splitk>")
    d2 = dict(d); d2["scale"] = d2["shift"] = None
    assert_bf16_close(out_f64(y), oracle_full(d2), "after-timeout-splitk")


def test_bounded_wait_timeout_reports_status_and_context_survives():
    spec = inputs.small_layer("inject", 1, 16, 16, 64, 64, 3, 1, 1, seed=(400, 0))
    d = inputs.layer_inputs(spec)
    x = to_dev(d["x"], "bf16")
    w = [to_dev(d[k], "bf16") for k in ("wr", "wi", "wj", "wk")]
    sc, sh = to_dev_f32(d["scale"]), to_dev_f32(d["shift"])
    quan.quan_set_path(quan.QUAN_PATH_TC)
    quan.quan_set_wait_limit_ns(5_000_000)          # 5 ms
    quan.quan_set_fault_injection(True)
    quan.qconv2d(x, *w, stride=1, pad=1, scale=sc, shift=sh, act=spec.act)
    st, bits = quan.quan_device_status()
    assert st == quan.QUAN_ERR_DEVICE_TIMEOUT and bits != 0
    quan.quan_set_fault_injection(False)
    quan.quan_set_wait_limit_ns(0)
    st, bits = quan.quan_device_status()            # cleared
    assert st == quan.QUAN_OK
    y = quan.qconv2d(x, *w, stride=1, pad=1, scale=sc, shift=sh, act=spec.act)
    torch.cuda.synchronize()
    assert_bf16_close(out_f64(y), oracle_full(d), "after-timeout")
