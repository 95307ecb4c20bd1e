"""fp64 CPU oracle for the QUAN quaternion convolution forward pass.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
package.  The product path (the CUDA library and its Python binding) never
imports, links or runs it, and it shares no code with them.

The arithmetic lives in ``quan_oracle.c`` (plain C, double precision, one
OpenMP loop over independent output pixels).  This module compiles it with
gcc on first use and wraps it with ctypes; the wrappers only convert arrays.

Passages followed (Grant & Wang, arXiv 2509.05512):
  * Hamilton product ............ Eq. 3 (Sec. III-A)
  * Poincare RGB mapping ........ Eq. 4 (Sec. III-A)
  * quaternion convolution ...... Eq. 5 (Sec. III-B), weight on the left
  * block (Hamilton) matrix ..... Eq. 6 (Sec. III-B)
  * separable variant ........... Eq. 7 (Sec. III-B)
  * backward pass ............... the input and weight gradients of Eq. 5 (the
                                  pre-epilogue convolution), from the Jacobians of
                                  Eq. 3
  * separable backward .......... Eq. 8-10 (Sec. III-B): mixing matrix M of Eq. 9,
                                  then per-component convolution gradients
  * IQBN, inference form ........ Eq. 11-12 (Sec. III-C), folded to scale/shift
  * IQBN, training mode ......... Eq. 11 batch statistics (biased variance), Eq. 12
                                  normalisation and affine
  * component-wise pooling ...... QSPPF (Sec. III-D)
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "quan_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

ACT_NONE, ACT_RELU, ACT_SILU = 0, 1, 2

_dp = ctypes.POINTER(ctypes.c_double)
_ip = ctypes.POINTER(ctypes.c_int)


def build(force: bool = False) -> str:
    """Compile quan_oracle.c into a shared library (gcc, -O2, OpenMP)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            lib.oracle_qmul.argtypes = [_dp, _dp, _dp]
            lib.oracle_qmul.restype = None
            conv = [_dp] * 9 + [ctypes.c_int] * 10
            lib.oracle_qconv2d.argtypes = conv + [_dp]
            lib.oracle_qconv2d.restype = ctypes.c_int
            lib.oracle_qconv2d_points.argtypes = conv + [ctypes.c_int, _ip, _ip, _ip, _dp]
            lib.oracle_qconv2d_points.restype = ctypes.c_int
            lib.oracle_qconv2d_separable.argtypes = [_dp] * 8 + [ctypes.c_int] * 10 + [_dp]
            lib.oracle_qconv2d_separable.restype = ctypes.c_int
            lib.oracle_expand_block_weight.argtypes = [_dp] * 4 + [ctypes.c_int] * 4 + [_dp]
            lib.oracle_expand_block_weight.restype = ctypes.c_int
            lib.oracle_real_conv2d.argtypes = [_dp, _dp] + [ctypes.c_int] * 9 + [_dp]
            lib.oracle_real_conv2d.restype = ctypes.c_int
            lib.oracle_maxpool2d.argtypes = [_dp] + [ctypes.c_int] * 7 + [_dp]
            lib.oracle_maxpool2d.restype = ctypes.c_int
            lib.oracle_qconv2d_bwd_data.argtypes = [_dp] * 5 + [ctypes.c_int] * 9 + [_dp]
            lib.oracle_qconv2d_bwd_data.restype = ctypes.c_int
            lib.oracle_qconv2d_bwd_weight.argtypes = [_dp] * 2 + [ctypes.c_int] * 9 + [_dp] * 4
            lib.oracle_qconv2d_bwd_weight.restype = ctypes.c_int
            lib.oracle_qconv2d_sep_bwd_data.argtypes = [_dp] * 5 + [ctypes.c_int] * 9 + [_dp]
            lib.oracle_qconv2d_sep_bwd_data.restype = ctypes.c_int
            lib.oracle_qconv2d_sep_bwd_weight.argtypes = ([_dp] * 2 + [ctypes.c_int] * 9 +
                                                          [_dp] * 4)
            lib.oracle_qconv2d_sep_bwd_weight.restype = ctypes.c_int
            lib.oracle_iqbn_batch_stats.argtypes = [_dp, ctypes.c_longlong, ctypes.c_int, _dp,
                                                    _dp]
            lib.oracle_iqbn_batch_stats.restype = ctypes.c_int
            lib.oracle_iqbn_train.argtypes = [_dp, ctypes.c_longlong, ctypes.c_int, _dp, _dp,
                                              ctypes.c_double, ctypes.c_int, _dp]
            lib.oracle_iqbn_train.restype = ctypes.c_int
            lib.oracle_poincare.argtypes = [_dp, ctypes.c_longlong, _dp]
            lib.oracle_poincare.restype = None
            lib.oracle_num_threads.argtypes = []
            lib.oracle_num_threads.restype = ctypes.c_int
            _lib = lib
    return _lib


def _f64(a):
    if a is None:
        return None
    return np.ascontiguousarray(a, dtype=np.float64)


def _ptr(a):
    if a is None:
        return ctypes.cast(None, _dp)
    return a.ctypes.data_as(_dp)


def bf16_bits_to_f64(bits) -> np.ndarray:
    """Exact value of bfloat16 bit patterns (uint16) as float64."""
    b = np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def out_size(n: int, k: int, stride: int, pad: int) -> int:
    return (n + 2 * pad - k) // stride + 1


def num_threads() -> int:
    return _load().oracle_num_threads()


def qmul(p, q) -> np.ndarray:
    """Hamilton product p (x) q of two quaternions (r, i, j, k), Eq. 3."""
    p, q = _f64(p).reshape(4), _f64(q).reshape(4)
    out = np.zeros(4)
    _load().oracle_qmul(_ptr(p), _ptr(q), _ptr(out))
    return out


def qconv2d(x, wr, wi, wj, wk, *, stride=1, pad=0, bias=None, scale=None, shift=None,
            residual=None, act=ACT_NONE) -> np.ndarray:
    """Quaternion convolution forward with the fused epilogue, Eq. 5 + Eq. 11-12.

    x: [N, H, W, C_in] (component-major channels); w*: [C_out/4, kh, kw, C_in/4].
    Returns y: [N, Ho, Wo, C_out] in float64.
    """
    x, wr, wi, wj, wk = map(_f64, (x, wr, wi, wj, wk))
    bias, scale, shift, residual = map(_f64, (bias, scale, shift, residual))
    N, H, W, Cin = x.shape
    Qout, kh, kw, Qin = wr.shape
    Cout = 4 * Qout
    Ho, Wo = out_size(H, kh, stride, pad), out_size(W, kw, stride, pad)
    y = np.zeros((N, Ho, Wo, Cout))
    rc = _load().oracle_qconv2d(_ptr(x), _ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk), _ptr(bias),
                                _ptr(scale), _ptr(shift), _ptr(residual), N, H, W, Cin, Cout,
                                kh, kw, stride, pad, act, _ptr(y))
    if rc != 0:
        raise ValueError("oracle_qconv2d: invalid arguments")
    return y


def qconv2d_points(x, wr, wi, wj, wk, pts, *, stride=1, pad=0, bias=None, scale=None,
                   shift=None, residual=None, act=ACT_NONE) -> np.ndarray:
    """Same as :func:`qconv2d` but only at output pixels ``pts`` = [(n, ho, wo), ...].

    Returns [len(pts), C_out] float64.
    """
    x, wr, wi, wj, wk = map(_f64, (x, wr, wi, wj, wk))
    bias, scale, shift, residual = map(_f64, (bias, scale, shift, residual))
    N, H, W, Cin = x.shape
    Qout, kh, kw, Qin = wr.shape
    Cout = 4 * Qout
    pts = np.ascontiguousarray(np.asarray(pts, dtype=np.int32).reshape(-1, 3))
    pn, pho, pwo = (np.ascontiguousarray(pts[:, i]) for i in range(3))
    y = np.zeros((len(pts), Cout))
    rc = _load().oracle_qconv2d_points(
        _ptr(x), _ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk), _ptr(bias), _ptr(scale), _ptr(shift),
        _ptr(residual), N, H, W, Cin, Cout, kh, kw, stride, pad, act, len(pts),
        pn.ctypes.data_as(_ip), pho.ctypes.data_as(_ip), pwo.ctypes.data_as(_ip), _ptr(y))
    if rc != 0:
        raise ValueError("oracle_qconv2d_points: invalid arguments")
    return y


def qconv2d_separable(x, wr, wi, wj, wk, *, stride=1, pad=0, bias=None, scale=None,
                      shift=None, act=ACT_NONE) -> np.ndarray:
    """Separable QUAN convolution of Eq. 7 (diagonal terms with the printed signs)."""
    x, wr, wi, wj, wk = map(_f64, (x, wr, wi, wj, wk))
    bias, scale, shift = map(_f64, (bias, scale, shift))
    N, H, W, Cin = x.shape
    Qout, kh, kw, Qin = wr.shape
    Cout = 4 * Qout
    Ho, Wo = out_size(H, kh, stride, pad), out_size(W, kw, stride, pad)
    y = np.zeros((N, Ho, Wo, Cout))
    rc = _load().oracle_qconv2d_separable(_ptr(x), _ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk),
                                          _ptr(bias), _ptr(scale), _ptr(shift), N, H, W, Cin,
                                          Cout, kh, kw, stride, pad, act, _ptr(y))
    if rc != 0:
        raise ValueError("oracle_qconv2d_separable: invalid arguments")
    return y


def expand_block_weight(wr, wi, wj, wk) -> np.ndarray:
    """Real [C_out, kh, kw, C_in] weight built from the Hamilton matrix of Eq. 6."""
    wr, wi, wj, wk = map(_f64, (wr, wi, wj, wk))
    Qout, kh, kw, Qin = wr.shape
    wb = np.zeros((4 * Qout, kh, kw, 4 * Qin))
    rc = _load().oracle_expand_block_weight(_ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk), 4 * Qin,
                                            4 * Qout, kh, kw, _ptr(wb))
    if rc != 0:
        raise ValueError("oracle_expand_block_weight: invalid arguments")
    return wb


def real_conv2d(x, w, *, stride=1, pad=0) -> np.ndarray:
    """Plain real cross-correlation: x [N,H,W,Cin], w [Cout,kh,kw,Cin] -> [N,Ho,Wo,Cout]."""
    x, w = _f64(x), _f64(w)
    N, H, W, Cin = x.shape
    Cout, kh, kw, _ = w.shape
    Ho, Wo = out_size(H, kh, stride, pad), out_size(W, kw, stride, pad)
    y = np.zeros((N, Ho, Wo, Cout))
    rc = _load().oracle_real_conv2d(_ptr(x), _ptr(w), N, H, W, Cin, Cout, kh, kw, stride, pad,
                                    _ptr(y))
    if rc != 0:
        raise ValueError("oracle_real_conv2d: invalid arguments")
    return y


def maxpool2d(x, *, k=3, stride=2, pad=1) -> np.ndarray:
    """Per-real-channel max pooling (QSPPF pooling rule); x [N,H,W,C]."""
    x = _f64(x)
    N, H, W, C = x.shape
    Ho, Wo = out_size(H, k, stride, pad), out_size(W, k, stride, pad)
    y = np.zeros((N, Ho, Wo, C))
    rc = _load().oracle_maxpool2d(_ptr(x), N, H, W, C, k, stride, pad, _ptr(y))
    if rc != 0:
        raise ValueError("oracle_maxpool2d: invalid arguments")
    return y


def qconv2d_bwd_data(dy, wr, wi, wj, wk, *, H, W, stride=1, pad=0) -> np.ndarray:
    """Input gradient of the pre-epilogue convolution: dy [N, Ho, Wo, C_out] -> dx
    [N, H, W, C_in] (H, W: the forward input size)."""
    dy, wr, wi, wj, wk = map(_f64, (dy, wr, wi, wj, wk))
    N, Ho, Wo, Cout = dy.shape
    Qout, kh, kw, Qin = wr.shape
    Cin = 4 * Qin
    if (out_size(H, kh, stride, pad), out_size(W, kw, stride, pad)) != (Ho, Wo):
        raise ValueError("dy does not match the forward output size")
    dx = np.zeros((N, H, W, Cin))
    rc = _load().oracle_qconv2d_bwd_data(_ptr(dy), _ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk), N,
                                         H, W, Cin, Cout, kh, kw, stride, pad, _ptr(dx))
    if rc != 0:
        raise ValueError("oracle_qconv2d_bwd_data: invalid arguments")
    return dx


def qconv2d_bwd_weight(x, dy, *, kh, kw, stride=1, pad=0):
    """Weight gradients of the pre-epilogue convolution: (dW_r, dW_i, dW_j, dW_k), each
    [C_out/4, kh, kw, C_in/4]."""
    x, dy = map(_f64, (x, dy))
    N, H, W, Cin = x.shape
    Cout = dy.shape[-1]
    if dy.shape[:3] != (N, out_size(H, kh, stride, pad), out_size(W, kw, stride, pad)):
        raise ValueError("dy does not match the forward output size")
    shape = (Cout // 4, kh, kw, Cin // 4)
    dw = [np.zeros(shape) for _ in range(4)]
    rc = _load().oracle_qconv2d_bwd_weight(_ptr(x), _ptr(dy), N, H, W, Cin, Cout, kh, kw,
                                           stride, pad, *(_ptr(t) for t in dw))
    if rc != 0:
        raise ValueError("oracle_qconv2d_bwd_weight: invalid arguments")
    return tuple(dw)


def qconv2d_sep_bwd_data(dy, wr, wi, wj, wk, *, H, W, stride=1, pad=0) -> np.ndarray:
    """Input gradient of the separable convolution (Eq. 7) before its epilogue, by Eq. 8-9:
    dy [N, Ho, Wo, C_out] -> dx [N, H, W, C_in]."""
    dy, wr, wi, wj, wk = map(_f64, (dy, wr, wi, wj, wk))
    N, Ho, Wo, Cout = dy.shape
    Qout, kh, kw, Qin = wr.shape
    Cin = 4 * Qin
    if (out_size(H, kh, stride, pad), out_size(W, kw, stride, pad)) != (Ho, Wo):
        raise ValueError("dy does not match the forward output size")
    dx = np.zeros((N, H, W, Cin))
    rc = _load().oracle_qconv2d_sep_bwd_data(_ptr(dy), _ptr(wr), _ptr(wi), _ptr(wj), _ptr(wk),
                                             N, H, W, Cin, Cout, kh, kw, stride, pad, _ptr(dx))
    if rc != 0:
        raise ValueError("oracle_qconv2d_sep_bwd_data: invalid arguments")
    return dx


def qconv2d_sep_bwd_weight(x, dy, *, kh, kw, stride=1, pad=0):
    """Weight gradients of the separable convolution (Eq. 7) before its epilogue, by
    Eq. 9-10: (dW_r, dW_i, dW_j, dW_k), each [C_out/4, kh, kw, C_in/4]."""
    x, dy = map(_f64, (x, dy))
    N, H, W, Cin = x.shape
    Cout = dy.shape[-1]
    if dy.shape[:3] != (N, out_size(H, kh, stride, pad), out_size(W, kw, stride, pad)):
        raise ValueError("dy does not match the forward output size")
    shape = (Cout // 4, kh, kw, Cin // 4)
    dw = [np.zeros(shape) for _ in range(4)]
    rc = _load().oracle_qconv2d_sep_bwd_weight(_ptr(x), _ptr(dy), N, H, W, Cin, Cout, kh, kw,
                                               stride, pad, *(_ptr(t) for t in dw))
    if rc != 0:
        raise ValueError("oracle_qconv2d_sep_bwd_weight: invalid arguments")
    return tuple(dw)


def iqbn_batch_stats(x):
    """Batch statistics of Eq. 11 per real channel: x [..., C] -> (mean, biased var), each
    [C], over every leading index (N, H, W)."""
    x = _f64(x)
    C = x.shape[-1]
    npix = x.size // C
    mean, var = np.zeros(C), np.zeros(C)
    if _load().oracle_iqbn_batch_stats(_ptr(x), npix, C, _ptr(mean), _ptr(var)) != 0:
        raise ValueError("oracle_iqbn_batch_stats: invalid arguments")
    return mean, var


def iqbn_train(x, gamma, beta, *, eps=1e-5, act=ACT_NONE):
    """Training-mode IQBN (Eq. 11-12) with the batch's own statistics, then the split
    activation: x [..., C] -> same shape."""
    x, gamma, beta = map(_f64, (x, gamma, beta))
    C = x.shape[-1]
    y = np.zeros_like(x)
    if _load().oracle_iqbn_train(_ptr(x), x.size // C, C, _ptr(gamma), _ptr(beta), float(eps),
                                 act, _ptr(y)) != 0:
        raise ValueError("oracle_iqbn_train: invalid arguments")
    return y


def poincare(rgb) -> np.ndarray:
    """Poincare RGB -> quaternion mapping of Eq. 4; rgb [..., 3] -> [..., 4]."""
    rgb = _f64(rgb)
    shape = rgb.shape[:-1]
    npix = int(np.prod(shape)) if shape else 1
    q = np.zeros(shape + (4,))
    _load().oracle_poincare(_ptr(rgb), npix, _ptr(q))
    return q


def iqbn_fold(gamma, beta, mean, var, eps=1e-5):
    """Fold IQBN running statistics (Eq. 12) into the per-channel scale/shift pair."""
    gamma, beta, mean, var = map(_f64, (gamma, beta, mean, var))
    scale = gamma / np.sqrt(var + eps)
    return scale, beta - mean * scale
