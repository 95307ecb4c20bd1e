"""Pins for the fp64 oracle: each test checks it against something other than
itself -- values fixed by the paper's algebra (Eq. 2-3 basis table, a hand-computed
product), closed forms, invariants, special cases that reduce to a library routine
(torch.nn.functional.conv2d / max_pool2d in float64, numpy statistics), or
brute-force equality of two independent formulations (Eq. 5 vs Eq. 6)."""
import os

import numpy as np
import pytest
import torch

import oracle

UNITS = {"1": (1, 0, 0, 0), "i": (0, 1, 0, 0), "j": (0, 0, 1, 0), "k": (0, 0, 0, 1)}


def _unit(tok):
    sgn = -1.0 if tok.startswith("-") else 1.0
    return sgn * np.array(UNITS[tok.lstrip("-")], dtype=np.float64)


def _rows(path):
    with open(path) as f:
        return [ln.split() for ln in f if ln.strip() and not ln.startswith("#")]


# ----------------------------------------------------------------- Hamilton product

def test_qmul_basis_table(golden_dir):
    rows = _rows(os.path.join(golden_dir, "hamilton_basis.txt"))
    assert len(rows) == 16
    for left, right, res in rows:
        np.testing.assert_array_equal(oracle.qmul(_unit(left), _unit(right)), _unit(res))


def test_qmul_ijk_is_minus_one():
    # Eq. 2: ijk = -1 (evaluated left to right)
    ij = oracle.qmul(_unit("i"), _unit("j"))
    np.testing.assert_array_equal(oracle.qmul(ij, _unit("k")), _unit("-1"))


def test_qmul_worked_example(golden_dir):
    for row in _rows(os.path.join(golden_dir, "qmul_worked_example.txt")):
        v = np.array([float(t) for t in row])
        np.testing.assert_array_equal(oracle.qmul(v[0:4], v[4:8]), v[8:12])


def test_qmul_norm_multiplicative_and_associative():
    rng = np.random.default_rng(11)
    for _ in range(200):
        p, q, r = rng.standard_normal((3, 4))
        pq = oracle.qmul(p, q)
        assert abs(np.linalg.norm(pq) - np.linalg.norm(p) * np.linalg.norm(q)) <= 1e-12 * (
            1 + np.linalg.norm(pq))
        lhs = oracle.qmul(pq, r)
        rhs = oracle.qmul(p, oracle.qmul(q, r))
        np.testing.assert_allclose(lhs, rhs, rtol=0, atol=1e-12 * (1 + np.abs(lhs).max()))
        # conj(p q) = conj(q) conj(p)
        conj = np.array([1.0, -1.0, -1.0, -1.0])
        np.testing.assert_allclose(conj * pq, oracle.qmul(conj * q, conj * p), atol=1e-12)


def test_qmul_bilinear_matches_matrix_form():
    # p (x) q is linear in q; its 4x4 matrix, read off from basis images, must be the
    # left-multiplication (Hamilton) matrix of Eq. 6 with the letters of p.
    p = np.array([0.3, -1.2, 0.7, 2.5])
    cols = [oracle.qmul(p, _unit(u)) for u in ("1", "i", "j", "k")]
    mat = np.stack(cols, axis=1)
    r, i, j, k = p
    eq6 = np.array([[r, -i, -j, -k], [i, r, -k, j], [j, k, r, -i], [k, -j, i, r]])
    np.testing.assert_array_equal(mat, eq6)


# ----------------------------------------------------------------- convolution

def _rand_layer(rng, N, H, W, Cin, Cout, kh, kw):
    x = rng.standard_normal((N, H, W, Cin))
    w = [rng.standard_normal((Cout // 4, kh, kw, Cin // 4)) for _ in range(4)]
    return x, w


def _torch_conv(x_nhwc, w_ohwi, stride, pad):
    x = torch.from_numpy(np.ascontiguousarray(x_nhwc)).permute(0, 3, 1, 2)
    w = torch.from_numpy(np.ascontiguousarray(w_ohwi)).permute(0, 3, 1, 2)
    y = torch.nn.functional.conv2d(x, w, stride=stride, padding=pad)
    return y.permute(0, 2, 3, 1).numpy()


def test_qconv_1x1_basis_pixels():
    # single quaternion channel, 1x1: y(pixel) = w (x) x(pixel) (Eq. 5 special case);
    # with w = i and x = j everywhere the answer is k (basis table), never -k.
    x = np.zeros((1, 3, 2, 4)); x[..., 2] = 1.0            # x = j
    w = [np.zeros((1, 1, 1, 1)) for _ in range(4)]; w[1][:] = 1.0  # w = i
    y = oracle.qconv2d(x, *w)
    expect = np.zeros_like(y); expect[..., 3] = 1.0          # k
    np.testing.assert_array_equal(y, expect)
    # and with w = j, x = i: ji = -k
    x = np.zeros((1, 2, 2, 4)); x[..., 1] = 1.0
    w = [np.zeros((1, 1, 1, 1)) for _ in range(4)]; w[2][:] = 1.0
    y = oracle.qconv2d(x, *w)
    np.testing.assert_array_equal(y[..., 3], -np.ones((1, 2, 2)))
    np.testing.assert_array_equal(y[..., :3], np.zeros((1, 2, 2, 3)))


def test_qconv_1x1_norm_multiplicative():
    rng = np.random.default_rng(3)
    x, w = _rand_layer(rng, 2, 4, 5, 4, 4, 1, 1)
    y = oracle.qconv2d(x, *w)
    wn = np.sqrt(sum(t.reshape(()) ** 2 for t in w))
    np.testing.assert_allclose(np.linalg.norm(y, axis=-1), wn * np.linalg.norm(x, axis=-1),
                               rtol=1e-12)


@pytest.mark.parametrize("shape", [
    (2, 5, 6, 8, 12, 3, 3, 1, 1),
    (1, 7, 5, 4, 8, 3, 3, 2, 1),
    (2, 6, 6, 12, 4, 1, 1, 2, 0),
    (1, 9, 8, 8, 8, 7, 7, 2, 3),
    (1, 4, 4, 8, 8, 3, 2, 1, 0),
])
def test_direct_equals_eq6_block_conv_equals_torch(shape):
    N, H, W, Cin, Cout, kh, kw, s, p = shape
    rng = np.random.default_rng(sum(shape))
    x, w = _rand_layer(rng, N, H, W, Cin, Cout, kh, kw)
    direct = oracle.qconv2d(x, *w, stride=s, pad=p)
    wb = oracle.expand_block_weight(*w)
    block = oracle.real_conv2d(x, wb, stride=s, pad=p)
    ref = _torch_conv(x, wb, s, p)
    scale = np.abs(ref).max()
    np.testing.assert_allclose(block, ref, rtol=0, atol=1e-12 * scale)
    np.testing.assert_allclose(direct, block, rtol=0, atol=1e-12 * scale)


def _comp(a, m, Q):
    return a[..., m * Q:(m + 1) * Q]


@pytest.mark.parametrize("letter", [0, 1, 2, 3])
def test_single_letter_rows_of_eq5(letter):
    # With only one letter tensor non-zero, every output component is one real
    # convolution of one input component, with the sign and pairing printed in
    # Eq. 5 (rows y_r, y_i, y_j, y_k):
    #   W_r: ( +x_r, +x_i, +x_j, +x_k )     W_i: ( -x_i, +x_r, -x_k, +x_j )
    #   W_j: ( -x_j, +x_k, +x_r, -x_i )     W_k: ( -x_k, -x_j, +x_i, +x_r )
    table = {
        0: [(+1, 0), (+1, 1), (+1, 2), (+1, 3)],
        1: [(-1, 1), (+1, 0), (-1, 3), (+1, 2)],
        2: [(-1, 2), (+1, 3), (+1, 0), (-1, 1)],
        3: [(-1, 3), (-1, 2), (+1, 1), (+1, 0)],
    }[letter]
    rng = np.random.default_rng(40 + letter)
    N, H, W, Cin, Cout = 2, 6, 5, 8, 12
    x, w = _rand_layer(rng, N, H, W, Cin, Cout, 3, 3)
    for L in range(4):
        if L != letter:
            w[L] = np.zeros_like(w[L])
    y = oracle.qconv2d(x, *w, stride=1, pad=1)
    Qin, Qout = Cin // 4, Cout // 4
    for m, (sgn, src) in enumerate(table):
        ref = sgn * _torch_conv(_comp(x, src, Qin), w[letter], 1, 1)
        np.testing.assert_allclose(_comp(y, m, Qout), ref, rtol=0, atol=1e-12)


def test_points_match_full():
    rng = np.random.default_rng(5)
    x, w = _rand_layer(rng, 3, 7, 9, 8, 8, 3, 3)
    bias = rng.standard_normal(8); scale = rng.uniform(0.5, 1.5, 8); shift = rng.standard_normal(8)
    full = oracle.qconv2d(x, *w, stride=2, pad=1, bias=bias, scale=scale, shift=shift,
                          act=oracle.ACT_RELU)
    pts = [(0, 0, 0), (2, 3, 4), (1, 2, 0), (2, 0, 4)]
    got = oracle.qconv2d_points(x, *w, pts, stride=2, pad=1, bias=bias, scale=scale,
                                shift=shift, act=oracle.ACT_RELU)
    for i, (n, h, ww) in enumerate(pts):
        np.testing.assert_array_equal(got[i], full[n, h, ww])


def test_invalid_arguments_rejected():
    x = np.zeros((1, 4, 4, 6))
    w = [np.zeros((1, 3, 3, 1))] * 4   # C_in = 6 is not a multiple of 4 with Q_in = 1
    with pytest.raises(ValueError):
        oracle.qconv2d(x, *w)
    x = np.zeros((1, 2, 2, 4))
    w = [np.zeros((1, 5, 5, 1))] * 4   # kernel larger than the padded input
    with pytest.raises(ValueError):
        oracle.qconv2d(x, *w)


# ----------------------------------------------------------------- epilogue

def test_iqbn_epilogue_matches_eq11_normalisation():
    # Eq. 11-12: x_hat = (x - mu) / sqrt(var + eps); out = x_hat * gamma + beta,
    # statistics per real channel over (batch, H, W).  The oracle takes the folded
    # (scale, shift) pair and adds the bias before normalising.
    rng = np.random.default_rng(8)
    x, w = _rand_layer(rng, 3, 6, 6, 8, 8, 3, 3)
    bias = rng.standard_normal(8)
    gamma = rng.uniform(0.5, 1.5, 8); beta = rng.standard_normal(8)
    pre = oracle.qconv2d(x, *w, stride=1, pad=1, bias=bias)
    mu = pre.mean(axis=(0, 1, 2)); var = pre.var(axis=(0, 1, 2))
    eps = 1e-5
    ref = (pre - mu) / np.sqrt(var + eps) * gamma + beta
    scale, shift = oracle.iqbn_fold(gamma, beta, mu, var, eps)
    got = oracle.qconv2d(x, *w, stride=1, pad=1, bias=bias, scale=scale, shift=shift)
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-12 * np.abs(ref).max())
    # after normalisation each channel has mean beta and standard deviation ~gamma
    np.testing.assert_allclose(got.mean(axis=(0, 1, 2)), beta, atol=1e-10)
    np.testing.assert_allclose(got.std(axis=(0, 1, 2)), gamma * np.sqrt(var / (var + eps)),
                               rtol=1e-10)


def test_activations_and_residual():
    rng = np.random.default_rng(9)
    x, w = _rand_layer(rng, 2, 5, 5, 8, 8, 3, 3)
    res = rng.standard_normal((2, 5, 5, 8))
    z = oracle.qconv2d(x, *w, pad=1)
    relu = oracle.qconv2d(x, *w, pad=1, act=oracle.ACT_RELU)
    np.testing.assert_array_equal(relu, np.maximum(z, 0.0))
    silu = oracle.qconv2d(x, *w, pad=1, act=oracle.ACT_SILU)
    ref = torch.nn.functional.silu(torch.from_numpy(z)).numpy()
    np.testing.assert_allclose(silu, ref, rtol=1e-14, atol=1e-15)
    zr = oracle.qconv2d(x, *w, pad=1, residual=res, act=oracle.ACT_RELU)
    np.testing.assert_allclose(zr, np.maximum(z + res, 0.0), rtol=0, atol=1e-14)


# ----------------------------------------------------------------- pooling, mapping

@pytest.mark.parametrize("k,s,p", [(3, 2, 1), (2, 2, 0), (3, 1, 1)])
def test_maxpool_matches_torch(k, s, p):
    rng = np.random.default_rng(k * 10 + s)
    x = rng.standard_normal((2, 9, 8, 8))
    got = oracle.maxpool2d(x, k=k, stride=s, pad=p)
    t = torch.from_numpy(x).permute(0, 3, 1, 2)
    ref = torch.nn.functional.max_pool2d(t, k, s, p).permute(0, 2, 3, 1).numpy()
    np.testing.assert_array_equal(got, ref)


def test_poincare_unit_norm_and_special_values():
    rng = np.random.default_rng(12)
    rgb = rng.uniform(-2, 2, size=(50, 3))
    q = oracle.poincare(rgb)
    np.testing.assert_allclose(np.linalg.norm(q, axis=-1), 1.0, rtol=1e-14)
    np.testing.assert_array_equal(oracle.poincare(np.zeros(3)), [1.0, 0.0, 0.0, 0.0])
    np.testing.assert_array_equal(oracle.poincare(np.array([1.0, 0, 0])), [0.0, 1.0, 0.0, 0.0])
    np.testing.assert_array_equal(oracle.poincare(np.array([0, 0, 1.0])), [0.0, 0.0, 0.0, 1.0])


# ----------------------------------------------------------------- separable variant

def test_separable_eq7_against_eq9_mixing_matrix():
    # Eq. 7's sign table is the transpose of the backward mixing matrix M of Eq. 9.
    # With a single non-zero letter W_p every output component is +-(W_p conv x_p),
    # the sign being M[p][q].
    M = np.array([[1, 1, 1, 1], [-1, 1, -1, 1], [-1, 1, 1, -1], [-1, -1, 1, 1]], dtype=float)
    rng = np.random.default_rng(21)
    N, H, W, Cin, Cout = 1, 5, 6, 8, 8
    x, w = _rand_layer(rng, N, H, W, Cin, Cout, 3, 3)
    for p in range(4):
        wl = [t if L == p else np.zeros_like(t) for L, t in enumerate(w)]
        y = oracle.qconv2d_separable(x, *wl, pad=1)
        base = _torch_conv(_comp(x, p, Cin // 4), w[p], 1, 1)
        for q in range(4):
            np.testing.assert_allclose(_comp(y, q, Cout // 4), M[p, q] * base, atol=1e-12)


# ----------------------------------------------------------------- backward pass
# The convolution before its epilogue is linear in x and in each letter, so its gradients
# are the adjoints of the forward map: <dy, F(x, W)> = <dx(dy), x> = sum_L <dW_L(x, dy), W_L>
# exactly (up to fp64 rounding).  The forward oracle is pinned above.

BWD_CASES = [
    # N, H, W, Cin, Cout, kh, kw, stride, pad
    (2, 6, 7, 8, 12, 3, 3, 1, 1),
    (1, 9, 8, 4, 8, 3, 3, 2, 1),
    (2, 7, 7, 8, 4, 5, 3, 2, 2),
    (1, 5, 6, 12, 8, 1, 1, 1, 0),
    (1, 8, 9, 4, 4, 7, 7, 2, 3),
]


@pytest.mark.parametrize("case", BWD_CASES)
def test_backward_is_the_adjoint_of_the_forward(case):
    N, H, W, Cin, Cout, kh, kw, s, p = case
    rng = np.random.default_rng(sum(case))
    x, w = _rand_layer(rng, N, H, W, Cin, Cout, kh, kw)
    y = oracle.qconv2d(x, *w, stride=s, pad=p)
    dy = rng.standard_normal(y.shape)
    lhs = float(np.sum(dy * y))
    dx = oracle.qconv2d_bwd_data(dy, *w, H=H, W=W, stride=s, pad=p)
    dw = oracle.qconv2d_bwd_weight(x, dy, kh=kh, kw=kw, stride=s, pad=p)
    assert dx.shape == x.shape and all(g.shape == t.shape for g, t in zip(dw, w))
    np.testing.assert_allclose(float(np.sum(dx * x)), lhs, rtol=1e-11)
    np.testing.assert_allclose(sum(float(np.sum(g * t)) for g, t in zip(dw, w)), lhs,
                               rtol=1e-11)


def test_backward_finite_differences():
    # one perturbed entry at a time: the forward map is linear, so the difference quotient
    # is the gradient entry up to rounding
    rng = np.random.default_rng(31)
    N, H, W, Cin, Cout, kh, kw, s, p = 1, 5, 5, 8, 8, 3, 3, 2, 1
    x, w = _rand_layer(rng, N, H, W, Cin, Cout, kh, kw)
    y0 = oracle.qconv2d(x, *w, stride=s, pad=p)
    dy = rng.standard_normal(y0.shape)
    dx = oracle.qconv2d_bwd_data(dy, *w, H=H, W=W, stride=s, pad=p)
    dw = oracle.qconv2d_bwd_weight(x, dy, kh=kh, kw=kw, stride=s, pad=p)
    eps = 0.5
    for idx in [(0, 0, 0, 0), (0, 2, 3, 5), (0, 4, 4, 7), (0, 1, 2, 2)]:
        xp = x.copy()
        xp[idx] += eps
        fd = np.sum(dy * (oracle.qconv2d(xp, *w, stride=s, pad=p) - y0)) / eps
        np.testing.assert_allclose(fd, dx[idx], rtol=1e-10, atol=1e-12)
    for L in range(4):
        for idx in [(0, 0, 0, 0), (1, 2, 1, 1), (0, 1, 2, 1)]:
            wp = [t.copy() for t in w]
            wp[L][idx] += eps
            fd = np.sum(dy * (oracle.qconv2d(x, *wp, stride=s, pad=p) - y0)) / eps
            np.testing.assert_allclose(fd, dw[L][idx], rtol=1e-10, atol=1e-12)


def test_backward_single_pixel_is_conjugate_multiplication():
    # 1x1 kernel, one quaternion channel, one pixel: y = w (x) x, so the input gradient is
    # conj(w) (x) dy and the weight gradient is dy (x) conj(x) (quaternion algebra)
    rng = np.random.default_rng(32)
    wq, xq, g = rng.standard_normal(4), rng.standard_normal(4), rng.standard_normal(4)
    conj = lambda q: q * np.array([1.0, -1, -1, -1])
    w = [np.full((1, 1, 1, 1), wq[m]) for m in range(4)]
    dx = oracle.qconv2d_bwd_data(g.reshape(1, 1, 1, 4), *w, H=1, W=1)
    np.testing.assert_allclose(dx.reshape(4), oracle.qmul(conj(wq), g), rtol=1e-14, atol=1e-15)
    dw = oracle.qconv2d_bwd_weight(xq.reshape(1, 1, 1, 4), g.reshape(1, 1, 1, 4), kh=1, kw=1)
    np.testing.assert_allclose(np.array([t.item() for t in dw]), oracle.qmul(g, conj(xq)),
                               rtol=1e-14, atol=1e-15)


# ----------------------------------------------------------------- separable backward
# Eq. 8-10: the same adjoint identities against the separable forward (Eq. 7), and the
# per-component reduction to PyTorch's own convolution gradients with Eq. 9's M.

EQ9_M = np.array([[1, 1, 1, 1], [-1, 1, -1, 1], [-1, 1, 1, -1], [-1, -1, 1, 1]], dtype=float)


@pytest.mark.parametrize("case", BWD_CASES)
def test_separable_backward_is_the_adjoint_of_eq7(case):
    N, H, W, Cin, Cout, kh, kw, s, p = case
    rng = np.random.default_rng(100 + sum(case))
    x, w = _rand_layer(rng, N, H, W, Cin, Cout, kh, kw)
    y = oracle.qconv2d_separable(x, *w, stride=s, pad=p)
    dy = rng.standard_normal(y.shape)
    lhs = float(np.sum(dy * y))
    dx = oracle.qconv2d_sep_bwd_data(dy, *w, H=H, W=W, stride=s, pad=p)
    dw = oracle.qconv2d_sep_bwd_weight(x, dy, kh=kh, kw=kw, stride=s, pad=p)
    assert dx.shape == x.shape and all(g.shape == t.shape for g, t in zip(dw, w))
    np.testing.assert_allclose(float(np.sum(dx * x)), lhs, rtol=1e-11)
    np.testing.assert_allclose(sum(float(np.sum(g * t)) for g, t in zip(dw, w)), lhs,
                               rtol=1e-11)


@pytest.mark.parametrize("case", [(1, 7, 6, 8, 12, 3, 3, 1, 1), (2, 9, 8, 8, 4, 3, 3, 2, 1)])
def test_separable_backward_matches_torch_gradients(case):
    # component p: dx_p = conv2d_input(sum_m M[p][m] dy_m, W_p) and
    # dW_p = conv2d_weight(x_p, ..., sum_m M[p][m] dy_m), PyTorch fp64 on the CPU
    N, H, W, Cin, Cout, kh, kw, s, p = case
    rng = np.random.default_rng(200 + sum(case))
    x, w = _rand_layer(rng, N, H, W, Cin, Cout, kh, kw)
    Qin, Qout = Cin // 4, Cout // 4
    Ho, Wo = (H + 2 * p - kh) // s + 1, (W + 2 * p - kw) // s + 1
    dy = rng.standard_normal((N, Ho, Wo, Cout))
    dx = oracle.qconv2d_sep_bwd_data(dy, *w, H=H, W=W, stride=s, pad=p)
    dw = oracle.qconv2d_sep_bwd_weight(x, dy, kh=kh, kw=kw, stride=s, pad=p)
    nchw = lambda a: torch.from_numpy(np.ascontiguousarray(a)).permute(0, 3, 1, 2)
    for comp in range(4):
        g = sum(EQ9_M[comp, m] * _comp(dy, m, Qout) for m in range(4))
        wt = nchw(w[comp])  # [Qout][Qin][kh][kw]
        ref_dx = torch.nn.grad.conv2d_input((N, Qin, H, W), wt, nchw(g), stride=s, padding=p)
        np.testing.assert_allclose(_comp(dx, comp, Qin), ref_dx.permute(0, 2, 3, 1).numpy(),
                                   rtol=1e-12, atol=1e-12)
        ref_dw = torch.nn.grad.conv2d_weight(nchw(_comp(x, comp, Qin)), (Qout, Qin, kh, kw),
                                             nchw(g), stride=s, padding=p)
        np.testing.assert_allclose(dw[comp], ref_dw.permute(0, 2, 3, 1).numpy(), rtol=1e-12,
                                   atol=1e-12)



# ----------------------------------------------------------------- IQBN, training mode
# Eq. 11: per real channel, mu = E[x], sigma^2 = E[(x - mu)^2] over N, H, W; Eq. 12: the
# normalised value times gamma plus beta.

def test_iqbn_stats_hand_example():
    # channel 0: 1, 2, 3, 6 -> mu = 12 / 4 = 3, sigma^2 = (4 + 1 + 0 + 9) / 4 = 3.5;
    # channel 1: constant -2 -> mu = -2, sigma^2 = 0
    x = np.array([[1.0, -2.0], [2.0, -2.0], [3.0, -2.0], [6.0, -2.0]]).reshape(2, 1, 2, 2)
    mean, var = oracle.iqbn_batch_stats(x)
    np.testing.assert_array_equal(mean, [3.0, -2.0])
    np.testing.assert_array_equal(var, [3.5, 0.0])


def test_iqbn_stats_large_offset_is_exact():
    # 1e6 + (0, 1, 2, 3): mu = 1e6 + 1.5, sigma^2 = 1.25 exactly (two-pass definition; the
    # one-pass E[x^2] - mu^2 loses every digit here)
    x = (1e6 + np.arange(4.0)).reshape(4, 1)
    mean, var = oracle.iqbn_batch_stats(x)
    assert mean[0] == 1e6 + 1.5 and var[0] == 1.25


def test_iqbn_stats_affine_and_channel_independence():
    rng = np.random.default_rng(50)
    x = rng.standard_normal((3, 5, 4, 8))
    mean, var = oracle.iqbn_batch_stats(x)
    a = np.linspace(-2.0, 3.0, 8)
    b = np.linspace(5.0, -1.0, 8)
    m2, v2 = oracle.iqbn_batch_stats(a * x + b)
    np.testing.assert_allclose(m2, a * mean + b, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(v2, a * a * var, rtol=1e-12, atol=1e-14)
    y = x.copy()
    y[..., 3] *= 7.0
    m3, v3 = oracle.iqbn_batch_stats(y)
    keep = np.arange(8) != 3
    np.testing.assert_array_equal(m3[keep], mean[keep])
    np.testing.assert_array_equal(v3[keep], var[keep])


def test_iqbn_train_normalised_moments():
    # gamma = 1, beta = 0: every channel of the output has mean 0 and mean square
    # sigma^2 / (sigma^2 + eps); with gamma, beta the output is their affine image
    rng = np.random.default_rng(51)
    x = rng.standard_normal((2, 6, 5, 12)) * np.linspace(0.1, 4.0, 12) + np.linspace(-3, 3, 12)
    eps = 1e-3
    ones, zeros = np.ones(12), np.zeros(12)
    xh = oracle.iqbn_train(x, ones, zeros, eps=eps)
    _, var = oracle.iqbn_batch_stats(x)
    np.testing.assert_allclose(xh.reshape(-1, 12).mean(0), 0.0, atol=1e-12)
    np.testing.assert_allclose((xh ** 2).reshape(-1, 12).mean(0), var / (var + eps), rtol=1e-12)
    g, b = np.linspace(0.5, 1.5, 12), np.linspace(-0.2, 0.2, 12)
    np.testing.assert_allclose(oracle.iqbn_train(x, g, b, eps=eps), xh * g + b, rtol=1e-12,
                               atol=1e-12)


def test_iqbn_train_constant_channel_and_activations():
    # a constant channel normalises to 0, so the output is act(beta)
    x = np.full((4, 3), 2.5)
    g, b = np.array([1.3, 0.7, 2.0]), np.array([-0.5, 0.25, 1.0])
    np.testing.assert_array_equal(oracle.iqbn_train(x, g, b), np.broadcast_to(b, (4, 3)))
    np.testing.assert_array_equal(oracle.iqbn_train(x, g, b, act=oracle.ACT_RELU),
                                  np.broadcast_to([0.0, 0.25, 1.0], (4, 3)))
    silu = b / (1.0 + np.exp(-b))
    np.testing.assert_allclose(oracle.iqbn_train(x, g, b, act=oracle.ACT_SILU)[0], silu,
                               rtol=1e-15)
