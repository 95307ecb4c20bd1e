"""Host-side checks of the C ABI that need no GPU: the library builds, loads and
exports every function include/quan.h declares, and argument errors are rejected on
the host before anything is launched."""
import ctypes

import pytest

from paper_2509_05512_gb300 import build, quan


@pytest.fixture(scope="module")
def lib():
    build.build_library()
    return quan.load()


def test_exports_every_header_function(lib):
    names = quan.header_functions()
    assert "quan_qconv2d_fwd" in names and "quan_maxpool2d_fwd" in names
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing, missing


def test_status_strings_and_version(lib):
    assert quan.quan_status_string(quan.QUAN_OK) == "QUAN_OK"
    assert quan.quan_status_string(quan.QUAN_ERR_DEVICE_TIMEOUT) == "QUAN_ERR_DEVICE_TIMEOUT"
    assert quan.quan_status_string(99) == "QUAN_ERR_UNKNOWN"
    assert quan.quan_version() >= 100


FAKE = 0x10000  # never dereferenced: every case below fails validation first


def _call(lib, **kw):
    a = dict(x=FAKE, wr=FAKE + 0x1000, wi=FAKE + 0x2000, wj=FAKE + 0x3000, wk=FAKE + 0x4000,
             bias=None, scale=None, shift=None, N=1, H=8, W=8, Cin=64, Cout=64, kh=3, kw=3,
             stride=1, pad=1, act=1, out=0x7000000, stream=None)
    a.update(kw)
    return lib.quan_qconv2d_fwd(a["x"], a["wr"], a["wi"], a["wj"], a["wk"], a["bias"], a["scale"],
                                a["shift"], a["N"], a["H"], a["W"], a["Cin"], a["Cout"], a["kh"],
                                a["kw"], a["stride"], a["pad"], a["act"], a["out"], a["stream"])


@pytest.mark.parametrize("bad", [
    dict(x=None), dict(wk=None), dict(out=None),
    dict(Cin=6), dict(Cout=10), dict(N=0), dict(H=-1), dict(stride=0), dict(pad=-1),
    dict(kh=0), dict(act=7), dict(kh=11, pad=1),
    dict(scale=0x9000000),            # scale without shift
    dict(shift=0x9000000),            # shift without scale
    dict(out=FAKE),                   # out overlaps x
])
def test_invalid_arguments(lib, bad):
    assert _call(lib, **bad) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_last_error_message()


def test_maxpool_and_setters_validate(lib):
    assert lib.quan_maxpool2d_fwd(None, 1, 4, 4, 8, 3, 2, 1, FAKE, None) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_maxpool2d_fwd(FAKE, 1, 4, 4, 8, 3, 2, 2, FAKE * 64, None) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_set_path(5) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_set_tc_tiles(24, 0, 0, 0) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_set_tc_tiles(0, 0, 0, 8) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_set_tc_tiles(0, 0, 0, 7) == quan.QUAN_OK
    assert lib.quan_set_tc_tiles(0, 0, 0, 6) == quan.QUAN_OK
    assert lib.quan_set_tc_tiles(0, 0, 0, 4) == quan.QUAN_OK
    assert lib.quan_set_tc_tiles(0, 0, 0, 0) == quan.QUAN_OK
    assert lib.quan_poincare_fwd(None, 4, FAKE, None) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_poincare_fwd(FAKE, -1, FAKE * 64, None) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_poincare_fwd(FAKE + 1, 4, FAKE * 64, None) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_poincare_fwd(FAKE, 4, FAKE + 8, None) == quan.QUAN_ERR_INVALID_ARG  # overlap
    assert lib.quan_poincare_fwd(None, 0, None, None) == quan.QUAN_OK
    assert lib.quan_set_tc_issuers(1) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_set_tc_issuers(4) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_set_tc_issuers(2) == quan.QUAN_OK
    assert lib.quan_set_tc_issuers(0) == quan.QUAN_OK
    assert lib.quan_set_tc_band_rows(-1) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_set_tc_band_rows(5) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_set_tc_band_rows(3) == quan.QUAN_OK
    assert lib.quan_set_tc_band_rows(0) == quan.QUAN_OK
    assert lib.quan_set_path(0) == quan.QUAN_OK
    assert lib.quan_set_wait_limit_ns(0) == quan.QUAN_OK
    # quan_qconv2d_fwd_ex: the workspace arguments are checked before anything else
    conv = [FAKE] * 8 + [1, 8, 8, 64, 64, 3, 3, 1, 1, 1]
    assert lib.quan_qconv2d_fwd_ex(*conv, None, None, 64, FAKE * 64, None) == \
        quan.QUAN_ERR_INVALID_ARG  # workspace NULL with bytes > 0
    assert lib.quan_qconv2d_fwd_ex(*conv, None, FAKE + 16, 4096, FAKE * 64, None) == \
        quan.QUAN_ERR_INVALID_ARG  # not 256-byte aligned


def test_f32_entry_point_validates(lib):
    f = lib.quan_qconv2d_fwd_f32
    assert f(None, FAKE, FAKE, FAKE, FAKE, None, None, None, 1, 4, 4, 4, 4, 3, 3, 1, 1, 0,
             FAKE * 16, None) == quan.QUAN_ERR_INVALID_ARG
    r = lib.quan_qconv2d_fwd_res
    assert r(FAKE, FAKE, FAKE, FAKE, FAKE, None, None, None, 1, 4, 4, 4, 4, 3, 3, 1, 1, 0,
             None, FAKE * 16, None) == quan.QUAN_ERR_INVALID_ARG


def test_no_python_fallback_when_library_missing(monkeypatch, tmp_path):
    # The binding must fail loudly, never compute elsewhere, if libquan.so is absent.
    monkeypatch.setattr(quan, "LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(quan, "_lib", None)
    with pytest.raises(RuntimeError, match="not built"):
        quan.load()


def _bwd_data(lib, sep=False, **kw):
    a = dict(dy=FAKE, wr=FAKE + 0x1000, wi=FAKE + 0x2000, wj=FAKE + 0x3000, wk=FAKE + 0x4000,
             N=1, H=8, W=8, Cin=64, Cout=128, kh=3, kw=3, stride=1, pad=1,
             ws=0x8000000, ws_bytes=36864, dx=0x7000000)
    a.update(kw)
    f = lib.quan_qconv2d_sep_bwd_data if sep else lib.quan_qconv2d_bwd_data
    return f(a["dy"], a["wr"], a["wi"], a["wj"], a["wk"], a["N"], a["H"], a["W"], a["Cin"],
             a["Cout"], a["kh"], a["kw"], a["stride"], a["pad"], a["ws"], a["ws_bytes"], a["dx"],
             None)


def _bwd_weight(lib, sep=False, **kw):
    a = dict(x=FAKE, dy=FAKE * 16, N=1, H=8, W=8, Cin=64, Cout=128, kh=3, kw=3, stride=1,
             pad=1, dwr=0x7000000, dwi=0x7100000, dwj=0x7200000, dwk=0x7300000)
    a.update(kw)
    f = lib.quan_qconv2d_sep_bwd_weight if sep else lib.quan_qconv2d_bwd_weight
    return f(a["x"], a["dy"], a["N"], a["H"], a["W"], a["Cin"], a["Cout"], a["kh"], a["kw"],
             a["stride"], a["pad"], a["dwr"], a["dwi"], a["dwj"], a["dwk"], None)


def test_backward_workspace_size(lib):
    # four transformed letters of (Cin/4) * kh * kw * (Cout/4) bf16 values
    assert lib.quan_qconv2d_bwd_data_workspace_size(64, 128, 3, 3) == 4 * 16 * 9 * 32 * 2
    assert lib.quan_qconv2d_bwd_data_workspace_size(4, 64, 7, 7) == 4 * 1 * 49 * 16 * 2
    assert lib.quan_qconv2d_bwd_data_workspace_size(6, 64, 3, 3) == 0
    assert lib.quan_qconv2d_bwd_data_workspace_size(64, 64, 0, 3) == 0
    # strided: the letters (rounded to 256 bytes) and dy spread out to H + 2 pad - kh + 1 rows
    lt = lib.quan_qconv2d_bwd_data_workspace_size(64, 128, 3, 3)
    assert lib.quan_qconv2d_bwd_data_workspace_size_ex(2, 8, 8, 64, 128, 3, 3, 1, 1) == lt
    assert lib.quan_qconv2d_bwd_data_workspace_size_ex(2, 8, 8, 64, 128, 3, 3, 2, 1) == \
        (lt + 255) // 256 * 256 + 2 * 8 * 8 * 128 * 2
    assert lib.quan_qconv2d_bwd_data_workspace_size_ex(2, 8, 8, 64, 128, 3, 3, 0, 1) == 0


@pytest.mark.parametrize("sep", [False, True])
@pytest.mark.parametrize("bad", [
    dict(dy=None), dict(wj=None), dict(dx=None), dict(Cin=6), dict(stride=0), dict(kh=11),
    dict(ws=None), dict(ws_bytes=36863),   # workspace missing or one byte short
    dict(dx=FAKE),                         # dx overlaps dy
    dict(ws=FAKE + 0x2000),                # workspace overlaps a weight tensor
    dict(ws=0x7000000 + 64),               # workspace overlaps dx
])
def test_backward_data_invalid_arguments(lib, sep, bad):
    assert _bwd_data(lib, sep, **bad) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_last_error_message()


@pytest.mark.parametrize("sep", [False, True])
@pytest.mark.parametrize("bad", [
    dict(x=None), dict(dwk=None), dict(Cout=10), dict(pad=-1),
    dict(dwi=0x7000000 + 4),               # two weight gradients overlap
    dict(dwr=FAKE),                        # a weight gradient overlaps x
    dict(dwj=0x7200002),                   # misaligned fp32 output
])
def test_backward_weight_invalid_arguments(lib, sep, bad):
    assert _bwd_weight(lib, sep, **bad) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_last_error_message()


def test_backward_weight_tensor_core_shapes(lib):
    # the tensor-core weight gradient takes stride 1 or 2, Cin and Cout multiples of 64:
    # forcing it on another shape fails on the host
    assert lib.quan_set_path(quan.QUAN_PATH_TC) == quan.QUAN_OK
    try:
        assert _bwd_weight(lib, stride=3) == quan.QUAN_ERR_UNSUPPORTED
        assert _bwd_weight(lib, Cin=48) == quan.QUAN_ERR_UNSUPPORTED
        assert _bwd_weight(lib, Cout=320) == quan.QUAN_ERR_UNSUPPORTED
        assert _bwd_weight(lib, x=FAKE + 8) == quan.QUAN_ERR_UNSUPPORTED  # misaligned for TMA
    finally:
        assert lib.quan_set_path(quan.QUAN_PATH_AUTO) == quan.QUAN_OK


def test_iqbn_entry_points_validate(lib):
    st, tr = lib.quan_iqbn_batch_stats, lib.quan_iqbn_train_fwd
    bad = quan.QUAN_ERR_INVALID_ARG
    ws, wsb = 0x8000000, lib.quan_iqbn_batch_stats_workspace_size(64)
    assert wsb == 1024 * 2 * 64 * 4 and lib.quan_iqbn_batch_stats_workspace_size(0) == 0
    args = lambda **k: [k.get("x", FAKE), k.get("npix", 16), k.get("C", 64), k.get("ws", ws),
                        k.get("wsb", wsb), k.get("mean", 0x7000000), k.get("var", 0x7100000),
                        None]
    assert st(*args(x=None)) == bad
    assert st(*args(npix=0)) == bad
    assert st(*args(C=0)) == bad
    assert st(*args(ws=None)) == bad
    assert st(*args(wsb=wsb - 1)) == bad
    assert st(*args(var=0x7000000 + 8)) == bad          # mean overlaps var
    assert st(*args(mean=FAKE + 64)) == bad             # mean overlaps x
    assert st(*args(mean=0x7000002)) == bad             # misaligned mean
    assert st(*args(ws=0x7100000 - 64)) == bad          # workspace overlaps var
    assert st(*args(C=260, wsb=lib.quan_iqbn_batch_stats_workspace_size(260))) == \
        quan.QUAN_ERR_UNSUPPORTED
    v = (FAKE, 16, 64, 0x7000000, 0x7100000, None, None)
    assert tr(*v, ctypes.c_float(1e-5), 7, 0x7200000, None) == bad      # unknown activation
    assert tr(*v, ctypes.c_float(-1.0), 0, 0x7200000, None) == bad      # negative eps
    assert tr(*v, ctypes.c_float(float("nan")), 0, 0x7200000, None) == bad
    assert tr(*v, ctypes.c_float(1e-5), 0, FAKE + 2, None) == bad       # partial overlap
    assert tr(*v, ctypes.c_float(1e-5), 0, 0x7000000, None) == bad      # out overlaps mean
    assert tr(FAKE, 16, 260, 0x7000000, 0x7100000, None, None, ctypes.c_float(1e-5), 0,
              0x7200000, None) == quan.QUAN_ERR_UNSUPPORTED


def test_fused_stem_pool_validates(lib):
    f = lib.quan_qconv2d_maxpool_fwd
    # one kernel writes the pooled tensor: no workspace for any shape
    assert lib.quan_qconv2d_maxpool_workspace_size(2, 32, 32, 64, 7, 7, 2, 3) == 0
    args = lambda out, x=FAKE: (x, FAKE + 0x1000, FAKE + 0x2000, FAKE + 0x3000,
                                FAKE + 0x4000, None, None, None, 2, 32, 32, 4, 64, 7, 7, 2, 3,
                                1, None, 0, out, None)
    bad = quan.QUAN_ERR_INVALID_ARG
    assert f(*args(None)) == bad                           # no output
    assert f(*args(FAKE + 0x10)) == bad                    # output overlaps the input
    assert f(*args(0x9000000, x=None)) == bad              # no input


def _call_sc(lib, **kw):
    # quan_qconv2d_fwd_shortcut: the downsampling block's 3x3/2 convolution and its 1x1/2
    # shortcut of the same input
    a = dict(x=FAKE, w=FAKE + 0x1000, bias=None, scale=None, shift=None, N=1, H=8, W=8,
             Cin=64, Cout=128, kh=3, kw=3, stride=2, pad=1, act=1, sw=FAKE + 0x100000,
             sbias=None, sscale=None, sshift=None, Cout_sc=128, sact=0, out=0x7000000,
             out_sc=0x8000000, stream=None)
    a.update(kw)
    at = lambda base, k: None if base is None else base + k
    return lib.quan_qconv2d_fwd_shortcut(
        a["x"], a["w"], at(a["w"], 0x10000), at(a["w"], 0x20000), at(a["w"], 0x30000),
        a["bias"], a["scale"], a["shift"], a["N"], a["H"], a["W"], a["Cin"], a["Cout"],
        a["kh"], a["kw"], a["stride"], a["pad"], a["act"], a["sw"], at(a["sw"], 0x10000),
        at(a["sw"], 0x20000), at(a["sw"], 0x30000), a["sbias"], a["sscale"], a["sshift"],
        a["Cout_sc"], a["sact"], a["out"], a["out_sc"], a["stream"])


@pytest.mark.parametrize("bad", [
    dict(x=None), dict(sw=None), dict(out_sc=None),
    dict(Cout_sc=10),                 # not a multiple of 4
    dict(sact=7),
    dict(sscale=0x9000000),           # shortcut scale without shift
    dict(pad=0),                      # 3x3/2 without padding: 3x3 output, the 1x1/2 one 4x4
    dict(out_sc=0x7000000 + 64),      # out_sc overlaps out
    dict(out_sc=FAKE),                # out_sc overlaps x
])
def test_fused_shortcut_invalid_arguments(lib, bad):
    assert _call_sc(lib, **bad) == quan.QUAN_ERR_INVALID_ARG
    assert lib.quan_last_error_message()
