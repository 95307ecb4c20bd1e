"""ctypes binding of libquan (include/quan.h).  Argument marshalling only: every
arithmetic step runs in the library's CUDA kernels.  Tensor arguments may be torch
tensors (their device pointer is passed), integer device addresses, or None.

The library must have been built (``paper_2509_05512_gb300.build.build_library()``);
there is no fallback implementation, and a missing library raises immediately.
"""
from __future__ import annotations

import ctypes
import os
import re
import threading

PKG_DIR = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(PKG_DIR, "libquan.so")
HEADER = os.path.join(os.path.dirname(PKG_DIR), "include", "quan.h")

QUAN_OK, QUAN_ERR_INVALID_ARG, QUAN_ERR_UNSUPPORTED, QUAN_ERR_CUDA, QUAN_ERR_DEVICE_TIMEOUT = range(5)
QUAN_ACT_NONE, QUAN_ACT_RELU, QUAN_ACT_SILU = 0, 1, 2
QUAN_PATH_AUTO, QUAN_PATH_TC, QUAN_PATH_SIMT = 0, 1, 2

_lock = threading.Lock()
_lib = None

_vp = ctypes.c_void_p
_i = ctypes.c_int
_conv_args = [_vp] * 8 + [_i] * 10


class QuanError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__("%s: %s" % (_status_name(status), message))
        self.status = status


def _status_name(st: int) -> str:
    names = ["QUAN_OK", "QUAN_ERR_INVALID_ARG", "QUAN_ERR_UNSUPPORTED", "QUAN_ERR_CUDA",
             "QUAN_ERR_DEVICE_TIMEOUT"]
    return names[st] if 0 <= st < len(names) else "QUAN_ERR_%d" % st


def header_functions() -> list:
    """Names of the functions include/quan.h declares."""
    with open(HEADER) as f:
        text = f.read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(quan_[a-z0-9_]+)\s*\(", text)))


def load():
    """Load libquan.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(LIB_PATH):
            raise RuntimeError("libquan.so is not built; run "
                               "paper_2509_05512_gb300.build.build_library() first")
        lib = ctypes.CDLL(LIB_PATH)
        lib.quan_qconv2d_fwd.argtypes = _conv_args + [_vp, _vp]
        lib.quan_qconv2d_fwd_f32.argtypes = _conv_args + [_vp, _vp]
        lib.quan_qconv2d_fwd_res.argtypes = _conv_args + [_vp, _vp, _vp]
        lib.quan_qconv2d_fwd_ex.argtypes = _conv_args + [_vp, _vp, ctypes.c_size_t, _vp, _vp]
        lib.quan_qconv2d_fwd_shortcut.argtypes = (_conv_args + [_vp] * 7 + [_i, _i] +
                                                  [_vp, _vp, _vp])
        lib.quan_qconv2d_fwd_workspace_size.argtypes = []
        lib.quan_qconv2d_fwd_workspace_size.restype = ctypes.c_size_t
        lib.quan_qconv2d_sep_fwd.argtypes = _conv_args + [_vp, _vp]
        lib.quan_maxpool2d_fwd.argtypes = [_vp] + [_i] * 7 + [_vp, _vp]
        lib.quan_poincare_fwd.argtypes = [_vp, ctypes.c_longlong, _vp, _vp]
        _bwd_data_args = [_vp] * 5 + [_i] * 9 + [_vp, ctypes.c_size_t, _vp, _vp]
        lib.quan_qconv2d_bwd_data.argtypes = _bwd_data_args
        lib.quan_qconv2d_sep_bwd_data.argtypes = _bwd_data_args
        lib.quan_qconv2d_maxpool_fwd.argtypes = _conv_args + [_vp, ctypes.c_size_t, _vp, _vp]
        lib.quan_qconv2d_maxpool_rgb_fwd.argtypes = [_vp] * 8 + [_i] * 9 + [_vp, _vp]
        lib.quan_qconv2d_maxpool_workspace_size.argtypes = [_i] * 8
        lib.quan_qconv2d_maxpool_workspace_size.restype = ctypes.c_size_t
        lib.quan_iqbn_batch_stats.argtypes = [_vp, ctypes.c_longlong, _i, _vp, ctypes.c_size_t,
                                              _vp, _vp, _vp]
        lib.quan_iqbn_batch_stats_workspace_size.argtypes = [_i]
        lib.quan_iqbn_batch_stats_workspace_size.restype = ctypes.c_size_t
        lib.quan_iqbn_train_fwd.argtypes = ([_vp, ctypes.c_longlong, _i] + [_vp] * 4 +
                                            [ctypes.c_float, _i, _vp, _vp])
        lib.quan_qconv2d_bwd_data_static.argtypes = [_vp] * 5 + [_i] * 9 + [_vp, _vp]
        lib.quan_qconv2d_bwd_data_workspace_size.argtypes = [_i] * 4
        lib.quan_qconv2d_bwd_data_workspace_size.restype = ctypes.c_size_t
        lib.quan_qconv2d_bwd_data_workspace_size_ex.argtypes = [_i] * 9
        lib.quan_qconv2d_bwd_data_workspace_size_ex.restype = ctypes.c_size_t
        _bwd_weight_args = [_vp] * 2 + [_i] * 9 + [_vp] * 5
        lib.quan_qconv2d_bwd_weight.argtypes = _bwd_weight_args
        lib.quan_qconv2d_sep_bwd_weight.argtypes = _bwd_weight_args
        lib.quan_set_path.argtypes = [_i]
        lib.quan_last_path.argtypes = []
        lib.quan_last_kernel.argtypes = []
        lib.quan_last_kernel.restype = ctypes.c_char_p
        lib.quan_set_tc_tiles.argtypes = [_i, _i, _i, _i]
        lib.quan_set_wait_limit_ns.argtypes = [ctypes.c_ulonglong]
        lib.quan_set_tc_halo.argtypes = [_i]
        lib.quan_set_tc_issuers.argtypes = [_i]
        lib.quan_set_tc_band_rows.argtypes = [_i]
        lib.quan_device_status.argtypes = [_vp, ctypes.POINTER(ctypes.c_uint)]
        lib.quan_set_fault_injection.argtypes = [_i]
        lib.quan_status_string.argtypes = [_i]
        lib.quan_status_string.restype = ctypes.c_char_p
        lib.quan_last_error_message.argtypes = []
        lib.quan_last_error_message.restype = ctypes.c_char_p
        lib.quan_version.argtypes = []
        for name in ("quan_qconv2d_fwd", "quan_qconv2d_fwd_f32", "quan_qconv2d_fwd_res",
                     "quan_qconv2d_fwd_ex", "quan_qconv2d_fwd_shortcut",
                     "quan_qconv2d_sep_fwd", "quan_poincare_fwd", "quan_qconv2d_bwd_data",
                     "quan_qconv2d_sep_bwd_data", "quan_qconv2d_bwd_weight",
                     "quan_qconv2d_bwd_data_static", "quan_iqbn_batch_stats",
                     "quan_qconv2d_maxpool_fwd", "quan_qconv2d_maxpool_rgb_fwd",
                     "quan_iqbn_train_fwd",
                     "quan_qconv2d_sep_bwd_weight",
                     "quan_maxpool2d_fwd", "quan_set_path", "quan_set_tc_tiles",
                     "quan_set_wait_limit_ns", "quan_device_status", "quan_set_fault_injection",
                     "quan_set_tc_halo", "quan_set_tc_issuers", "quan_set_tc_band_rows"):
            getattr(lib, name).restype = _i
        lib.quan_last_path.restype = _i
        lib.quan_version.restype = _i
        _lib = lib
        return lib


def _ptr(t):
    if t is None:
        return None
    if isinstance(t, int):
        return t
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(st: int):
    if st != QUAN_OK:
        msg = load().quan_last_error_message().decode(errors="replace")
        raise QuanError(st, msg)


def quan_qconv2d_fwd(x, wr, wi, wj, wk, bias, iqbn_scale, iqbn_shift, N, H, W, Cin, Cout, kh, kw,
                     stride, pad, act, out, stream=None) -> None:
    _check(load().quan_qconv2d_fwd(_ptr(x), _ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk), _ptr(bias),
                                   _ptr(iqbn_scale), _ptr(iqbn_shift), N, H, W, Cin, Cout, kh, kw,
                                   stride, pad, act, _ptr(out), _stream(stream)))


def quan_qconv2d_fwd_f32(x, wr, wi, wj, wk, bias, iqbn_scale, iqbn_shift, N, H, W, Cin, Cout, kh,
                         kw, stride, pad, act, out, stream=None) -> None:
    _check(load().quan_qconv2d_fwd_f32(_ptr(x), _ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk),
                                       _ptr(bias), _ptr(iqbn_scale), _ptr(iqbn_shift), N, H, W,
                                       Cin, Cout, kh, kw, stride, pad, act, _ptr(out),
                                       _stream(stream)))


def quan_qconv2d_fwd_res(x, wr, wi, wj, wk, bias, iqbn_scale, iqbn_shift, N, H, W, Cin, Cout, kh,
                         kw, stride, pad, act, residual, out, stream=None) -> None:
    _check(load().quan_qconv2d_fwd_res(_ptr(x), _ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk),
                                       _ptr(bias), _ptr(iqbn_scale), _ptr(iqbn_shift), N, H, W,
                                       Cin, Cout, kh, kw, stride, pad, act, _ptr(residual),
                                       _ptr(out), _stream(stream)))


def quan_qconv2d_fwd_ex(x, wr, wi, wj, wk, bias, iqbn_scale, iqbn_shift, N, H, W, Cin, Cout, kh,
                        kw, stride, pad, act, residual, workspace, workspace_bytes, out,
                        stream=None) -> None:
    _check(load().quan_qconv2d_fwd_ex(_ptr(x), _ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk),
                                      _ptr(bias), _ptr(iqbn_scale), _ptr(iqbn_shift), N, H, W,
                                      Cin, Cout, kh, kw, stride, pad, act, _ptr(residual),
                                      _ptr(workspace), workspace_bytes, _ptr(out),
                                      _stream(stream)))


def quan_qconv2d_fwd_shortcut(x, wr, wi, wj, wk, bias, iqbn_scale, iqbn_shift, N, H, W, Cin,
                              Cout, kh, kw, stride, pad, act, sc_wr, sc_wi, sc_wj, sc_wk,
                              sc_bias, sc_iqbn_scale, sc_iqbn_shift, Cout_sc, sc_act, out,
                              out_sc, stream=None) -> None:
    _check(load().quan_qconv2d_fwd_shortcut(
        _ptr(x), _ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk), _ptr(bias), _ptr(iqbn_scale),
        _ptr(iqbn_shift), N, H, W, Cin, Cout, kh, kw, stride, pad, act, _ptr(sc_wr),
        _ptr(sc_wi), _ptr(sc_wj), _ptr(sc_wk), _ptr(sc_bias), _ptr(sc_iqbn_scale),
        _ptr(sc_iqbn_shift), Cout_sc, sc_act, _ptr(out), _ptr(out_sc), _stream(stream)))


def qconv2d_shortcut(x, w, sc_w, *, stride=2, pad=1, bias=None, scale=None, shift=None,
                     act=QUAN_ACT_NONE, sc_bias=None, sc_scale=None, sc_shift=None,
                     sc_act=QUAN_ACT_NONE, out=None, out_sc=None, stream=None):
    """A convolution (letters w = (wr, wi, wj, wk)) and the 1x1 shortcut of the same input
    (letters sc_w, same stride, no padding) in one call: returns (out, out_sc), allocated
    like qconv2d's when not given (bf16 CUDA tensors)."""
    import torch
    N, H, W, Cin = x.shape
    Qout, kh, kw, _ = w[0].shape
    Cout, Cout_sc = 4 * Qout, 4 * sc_w[0].shape[0]
    Ho, Wo = out_size(H, kh, stride, pad), out_size(W, kw, stride, pad)
    if out is None:
        out = torch.empty((N, Ho, Wo, Cout), dtype=x.dtype, device=x.device)
    if out_sc is None:
        out_sc = torch.empty((N, Ho, Wo, Cout_sc), dtype=x.dtype, device=x.device)
    quan_qconv2d_fwd_shortcut(x, *w, bias, scale, shift, N, H, W, Cin, Cout, kh, kw, stride, pad,
                              act, *sc_w, sc_bias, sc_scale, sc_shift, Cout_sc, sc_act, out,
                              out_sc, stream)
    return out, out_sc


def quan_qconv2d_fwd_workspace_size() -> int:
    return int(load().quan_qconv2d_fwd_workspace_size())


def fwd_workspace(device=None):
    """A zero-filled workspace (uint8 CUDA tensor) for quan_qconv2d_fwd_ex."""
    import torch
    return torch.zeros(quan_qconv2d_fwd_workspace_size(), dtype=torch.uint8,
                       device=device or "cuda")


def quan_maxpool2d_fwd(x, N, H, W, C, k, stride, pad, out, stream=None) -> None:
    _check(load().quan_maxpool2d_fwd(_ptr(x), N, H, W, C, k, stride, pad, _ptr(out),
                                     _stream(stream)))


def quan_set_path(path: int) -> None:
    _check(load().quan_set_path(path))


def quan_last_path() -> int:
    return load().quan_last_path()


def quan_last_kernel() -> str:
    return load().quan_last_kernel().decode()


def quan_set_tc_tiles(kappa: int = 0, bnq: int = 0, max_ctas: int = 0, mode: int = 0) -> None:
    _check(load().quan_set_tc_tiles(kappa, bnq, max_ctas, mode))


def quan_set_tc_halo(enable: bool) -> None:
    _check(load().quan_set_tc_halo(1 if enable else 0))


def quan_set_tc_issuers(issuers: int = 0) -> None:
    _check(load().quan_set_tc_issuers(issuers))


def quan_set_tc_band_rows(rows: int = 0) -> None:
    _check(load().quan_set_tc_band_rows(rows))


def quan_set_wait_limit_ns(ns: int) -> None:
    _check(load().quan_set_wait_limit_ns(ns))


def quan_set_fault_injection(enable: bool) -> None:
    _check(load().quan_set_fault_injection(1 if enable else 0))


def quan_device_status(stream=None) -> tuple:
    """Returns (status, bits); does not raise on QUAN_ERR_DEVICE_TIMEOUT."""
    bits = ctypes.c_uint(0)
    st = load().quan_device_status(_stream(stream), ctypes.byref(bits))
    if st not in (QUAN_OK, QUAN_ERR_DEVICE_TIMEOUT):
        _check(st)
    return st, bits.value


def quan_status_string(status: int) -> str:
    return load().quan_status_string(status).decode()


def quan_version() -> int:
    return load().quan_version()


def quan_qconv2d_sep_fwd(x, wr, wi, wj, wk, bias, iqbn_scale, iqbn_shift, N, H, W, Cin, Cout, kh,
                         kw, stride, pad, act, out, stream=None) -> None:
    _check(load().quan_qconv2d_sep_fwd(_ptr(x), _ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk),
                                       _ptr(bias), _ptr(iqbn_scale), _ptr(iqbn_shift), N, H, W,
                                       Cin, Cout, kh, kw, stride, pad, act, _ptr(out),
                                       _stream(stream)))


# ------------------------------------------------------------------ tensor helpers

def out_size(n: int, k: int, stride: int, pad: int) -> int:
    return (n + 2 * pad - k) // stride + 1


def qconv2d(x, wr, wi, wj, wk, *, stride=1, pad=0, bias=None, scale=None, shift=None,
            act=QUAN_ACT_NONE, residual=None, out=None, stream=None, separable=False,
            workspace=None):
    """Allocate the output (torch, same dtype/device as x) and run the convolution.
    x: [N, H, W, Cin] (bf16 or fp32, CUDA); w*: [Cout/4, kh, kw, Cin/4].  separable=True
    runs the separable form of Eq. 7 (bf16 only, no residual).  workspace (a zero-filled
    uint8 CUDA tensor, see fwd_workspace) runs the bf16 full form through
    quan_qconv2d_fwd_ex."""
    import torch
    N, H, W, Cin = x.shape
    Qout, kh, kw, _ = wr.shape
    Cout = 4 * Qout
    Ho, Wo = out_size(H, kh, stride, pad), out_size(W, kw, stride, pad)
    if out is None:
        out = torch.empty((N, Ho, Wo, Cout), dtype=x.dtype, device=x.device)
    if separable:
        if x.dtype != torch.bfloat16 or residual is not None:
            raise ValueError("the separable form takes bf16 tensors and no residual")
        quan_qconv2d_sep_fwd(x, wr, wi, wj, wk, bias, scale, shift, N, H, W, Cin, Cout, kh, kw,
                             stride, pad, act, out, stream)
    elif x.dtype == torch.float32:
        if residual is not None:
            raise ValueError("the fp32 entry point has no residual input")
        quan_qconv2d_fwd_f32(x, wr, wi, wj, wk, bias, scale, shift, N, H, W, Cin, Cout, kh, kw,
                             stride, pad, act, out, stream)
    elif workspace is not None:
        quan_qconv2d_fwd_ex(x, wr, wi, wj, wk, bias, scale, shift, N, H, W, Cin, Cout, kh, kw,
                            stride, pad, act, residual, workspace,
                            workspace.numel() * workspace.element_size(), out, stream)
    elif residual is not None:
        quan_qconv2d_fwd_res(x, wr, wi, wj, wk, bias, scale, shift, N, H, W, Cin, Cout, kh, kw,
                             stride, pad, act, residual, out, stream)
    else:
        quan_qconv2d_fwd(x, wr, wi, wj, wk, bias, scale, shift, N, H, W, Cin, Cout, kh, kw,
                         stride, pad, act, out, stream)
    return out


def quan_poincare_fwd(rgb, npix, out, stream=None) -> None:
    _check(load().quan_poincare_fwd(_ptr(rgb), npix, _ptr(out), _stream(stream)))


def poincare(rgb, *, out=None, stream=None):
    """Eq. 4 on the GPU: fp32 rgb [..., 3] (CUDA) -> bf16 quaternion pixels [..., 4]."""
    import torch
    if rgb.dtype != torch.float32 or rgb.shape[-1] != 3:
        raise ValueError("rgb must be float32 with a last dimension of 3")
    if out is None:
        out = torch.empty(rgb.shape[:-1] + (4,), dtype=torch.bfloat16, device=rgb.device)
    quan_poincare_fwd(rgb, rgb.numel() // 3, out, stream)
    return out


def quan_qconv2d_bwd_data_workspace_size(Cin, Cout, kh, kw) -> int:
    return load().quan_qconv2d_bwd_data_workspace_size(Cin, Cout, kh, kw)


def quan_qconv2d_bwd_data_workspace_size_ex(N, H, W, Cin, Cout, kh, kw, stride, pad) -> int:
    return load().quan_qconv2d_bwd_data_workspace_size_ex(N, H, W, Cin, Cout, kh, kw, stride,
                                                          pad)


def quan_qconv2d_bwd_data(dy, wr, wi, wj, wk, N, H, W, Cin, Cout, kh, kw, stride, pad, workspace,
                          workspace_bytes, dx, stream=None) -> None:
    _check(load().quan_qconv2d_bwd_data(_ptr(dy), _ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk), N, H,
                                        W, Cin, Cout, kh, kw, stride, pad, _ptr(workspace),
                                        workspace_bytes, _ptr(dx), _stream(stream)))


def quan_qconv2d_bwd_data_static(dy, wr, wi, wj, wk, N, H, W, Cin, Cout, kh, kw, stride, pad,
                                 dx, stream=None) -> None:
    _check(load().quan_qconv2d_bwd_data_static(_ptr(dy), _ptr(wr), _ptr(wi), _ptr(wj),
                                               _ptr(wk), N, H, W, Cin, Cout, kh, kw, stride,
                                               pad, _ptr(dx), _stream(stream)))


def quan_qconv2d_sep_bwd_data(dy, wr, wi, wj, wk, N, H, W, Cin, Cout, kh, kw, stride, pad,
                              workspace, workspace_bytes, dx, stream=None) -> None:
    _check(load().quan_qconv2d_sep_bwd_data(_ptr(dy), _ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk), N,
                                            H, W, Cin, Cout, kh, kw, stride, pad,
                                            _ptr(workspace), workspace_bytes, _ptr(dx),
                                            _stream(stream)))


def quan_qconv2d_bwd_weight(x, dy, N, H, W, Cin, Cout, kh, kw, stride, pad, dwr, dwi, dwj, dwk,
                            stream=None) -> None:
    _check(load().quan_qconv2d_bwd_weight(_ptr(x), _ptr(dy), N, H, W, Cin, Cout, kh, kw, stride,
                                          pad, _ptr(dwr), _ptr(dwi), _ptr(dwj), _ptr(dwk),
                                          _stream(stream)))


def quan_qconv2d_sep_bwd_weight(x, dy, N, H, W, Cin, Cout, kh, kw, stride, pad, dwr, dwi, dwj,
                                dwk, stream=None) -> None:
    _check(load().quan_qconv2d_sep_bwd_weight(_ptr(x), _ptr(dy), N, H, W, Cin, Cout, kh, kw,
                                              stride, pad, _ptr(dwr), _ptr(dwi), _ptr(dwj),
                                              _ptr(dwk), _stream(stream)))


def qconv2d_backward_data(dy, wr, wi, wj, wk, *, H, W, stride=1, pad=0, separable=False,
                          workspace=None, out=None, stream=None):
    """Input gradient of the pre-epilogue convolution: dy [N, Ho, Wo, Cout] (bf16, CUDA) ->
    dx [N, H, W, Cin] bf16.  `workspace` (a uint8 CUDA tensor) is allocated when not given,
    with quan_qconv2d_bwd_data_workspace_size_ex bytes (the tensor-core path of strided
    layers included)."""
    import torch
    N, Ho, Wo, Cout = dy.shape
    Qout, kh, kw, Qin = wr.shape
    Cin = 4 * Qin
    need = quan_qconv2d_bwd_data_workspace_size_ex(N, H, W, Cin, Cout, kh, kw, stride, pad)
    if workspace is None:
        workspace = torch.empty(need, dtype=torch.uint8, device=dy.device)
    if out is None:
        out = torch.empty((N, H, W, Cin), dtype=torch.bfloat16, device=dy.device)
    fn = quan_qconv2d_sep_bwd_data if separable else quan_qconv2d_bwd_data
    fn(dy, wr, wi, wj, wk, N, H, W, Cin, Cout, kh, kw, stride, pad, workspace,
       workspace.numel() * workspace.element_size(), out, stream)
    return out


def qconv2d_backward_weight(x, dy, *, kh, kw, stride=1, pad=0, separable=False, out=None,
                            stream=None):
    """Weight gradients of the pre-epilogue convolution: x [N, H, W, Cin], dy
    [N, Ho, Wo, Cout] (bf16, CUDA) -> (dW_r, dW_i, dW_j, dW_k), fp32 [Cout/4, kh, kw, Cin/4]."""
    import torch
    N, H, W, Cin = x.shape
    Cout = dy.shape[-1]
    if out is None:
        out = tuple(torch.empty((Cout // 4, kh, kw, Cin // 4), dtype=torch.float32,
                                device=x.device) for _ in range(4))
    fn = quan_qconv2d_sep_bwd_weight if separable else quan_qconv2d_bwd_weight
    fn(x, dy, N, H, W, Cin, Cout, kh, kw, stride, pad, *out, stream)
    return out


def quan_qconv2d_maxpool_workspace_size(N, H, W, Cout, kh, kw, stride, pad) -> int:
    return load().quan_qconv2d_maxpool_workspace_size(N, H, W, Cout, kh, kw, stride, pad)


def quan_qconv2d_maxpool_rgb_fwd(rgb, wr, wi, wj, wk, bias, iqbn_scale, iqbn_shift, N, H, W,
                                 Cout, kh, kw, stride, pad, act, out, stream=None) -> None:
    _check(load().quan_qconv2d_maxpool_rgb_fwd(_ptr(rgb), _ptr(wr), _ptr(wi), _ptr(wj),
                                               _ptr(wk), _ptr(bias), _ptr(iqbn_scale),
                                               _ptr(iqbn_shift), N, H, W, Cout, kh, kw, stride,
                                               pad, act, _ptr(out), _stream(stream)))


def quan_qconv2d_maxpool_fwd(x, wr, wi, wj, wk, bias, iqbn_scale, iqbn_shift, N, H, W, Cin,
                             Cout, kh, kw, stride, pad, act, workspace, workspace_bytes, out,
                             stream=None) -> None:
    _check(load().quan_qconv2d_maxpool_fwd(_ptr(x), _ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk),
                                           _ptr(bias), _ptr(iqbn_scale), _ptr(iqbn_shift), N,
                                           H, W, Cin, Cout, kh, kw, stride, pad, act,
                                           _ptr(workspace), workspace_bytes, _ptr(out),
                                           _stream(stream)))


def quan_iqbn_batch_stats_workspace_size(C) -> int:
    return load().quan_iqbn_batch_stats_workspace_size(C)


def quan_iqbn_batch_stats(x, npix, C, workspace, workspace_bytes, mean, var,
                          stream=None) -> None:
    _check(load().quan_iqbn_batch_stats(_ptr(x), npix, C, _ptr(workspace), workspace_bytes,
                                        _ptr(mean), _ptr(var), _stream(stream)))


def quan_iqbn_train_fwd(x, npix, C, mean, var, gamma, beta, eps, act, out, stream=None) -> None:
    _check(load().quan_iqbn_train_fwd(_ptr(x), npix, C, _ptr(mean), _ptr(var), _ptr(gamma),
                                      _ptr(beta), eps, act, _ptr(out), _stream(stream)))


def iqbn_batch_stats(x, *, workspace=None, stream=None):
    """Eq. 11 on the GPU: bf16 x [..., C] (CUDA) -> (mean, biased var), fp32 [C] each.
    `workspace` (a CUDA tensor of at least quan_iqbn_batch_stats_workspace_size(C) bytes)
    is allocated when not given."""
    import torch
    C = x.shape[-1]
    if workspace is None:
        workspace = torch.empty(quan_iqbn_batch_stats_workspace_size(C), dtype=torch.uint8,
                                device=x.device)
    mean = torch.empty(C, dtype=torch.float32, device=x.device)
    var = torch.empty(C, dtype=torch.float32, device=x.device)
    quan_iqbn_batch_stats(x, x.numel() // C, C, workspace,
                          workspace.numel() * workspace.element_size(), mean, var, stream)
    return mean, var


def iqbn_train(x, gamma=None, beta=None, *, eps=1e-5, act=QUAN_ACT_NONE, out=None,
               stream=None):
    """Training-mode IQBN (Eq. 11-12) with the batch's statistics, then the activation:
    bf16 x [..., C] -> bf16, same shape; returns (out, mean, var)."""
    import torch
    mean, var = iqbn_batch_stats(x, stream=stream)
    if out is None:
        out = torch.empty_like(x)
    C = x.shape[-1]
    quan_iqbn_train_fwd(x, x.numel() // C, C, mean, var, gamma, beta, eps, act, out, stream)
    return out, mean, var


def maxpool2d(x, *, k=3, stride=2, pad=1, out=None, stream=None):
    import torch
    N, H, W, C = x.shape
    Ho, Wo = out_size(H, k, stride, pad), out_size(W, k, stride, pad)
    if out is None:
        out = torch.empty((N, Ho, Wo, C), dtype=x.dtype, device=x.device)
    quan_maxpool2d_fwd(x, N, H, W, C, k, stride, pad, out, stream)
    return out
