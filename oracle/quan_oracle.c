/*
 * quan_oracle.c -- plain fp64 CPU oracle for the QUAN quaternion convolution
 * forward pass (Grant & Wang, "Quaternion Approximate Networks ...").
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call, link or
 * execute this file: it is used by tests/, by __graft_entry__.smoke() to check
 * the GPU result, and by the cpu_baseline / --impl reference legs of bench.py.
 * It shares no code, header, table or helper with the CUDA library.
 *
 * Everything is written as the plain definition, in double precision, with no
 * blocking, fusion or reordering.  The only parallelism is an OpenMP loop over
 * independent output pixels, which does not change any result.
 *
 * Tensor layouts (all row-major, C-contiguous):
 *   x   [N][H][W][C_in]            channel c = comp * Q_in + ci   (comp 0..3 = r,i,j,k)
 *   w_L [Q_out][kh][kw][Q_in]      one real tensor per letter L in {r,i,j,k}
 *   y   [N][Ho][Wo][C_out]         channel c = comp * Q_out + co
 * with Q = C / 4 and Ho = floor((H + 2 pad - kh) / stride) + 1.
 *
 * Readings of the paper used here (each is also recorded with the design notes):
 *   - "standard convolution" in Sec. III-B is a cross-correlation (no kernel
 *     flip) with zero padding;
 *   - the weight multiplies from the left, Y = W (x) X, as in the i-row of Eq. 5;
 *   - the epilogue is  act(scale * (acc + bias) + shift + residual), each piece
 *     optional, applied per real channel (IQBN inference form of Eq. 11-12);
 *   - activations are split (elementwise per real component).
 */
#include <math.h>
#include <stdlib.h>
#include <stddef.h>
#include <stdint.h>
#include <string.h>

#define ACT_NONE 0
#define ACT_RELU 1
#define ACT_SILU 2

/* Hamilton product p (x) q, Eq. 3 (Sec. III-A), written term by term. */
void oracle_qmul(const double p[4], const double q[4], double out[4]) {
    const double pr = p[0], pi = p[1], pj = p[2], pk = p[3];
    const double qr = q[0], qi = q[1], qj = q[2], qk = q[3];
    out[0] = pr * qr - pi * qi - pj * qj - pk * qk;
    out[1] = pr * qi + pi * qr + pj * qk - pk * qj;
    out[2] = pr * qj - pi * qk + pj * qr + pk * qi;
    out[3] = pr * qk + pi * qj - pj * qi + pk * qr;
}

static double apply_act(double z, int act) {
    if (act == ACT_RELU) return z > 0.0 ? z : 0.0;
    if (act == ACT_SILU) return z / (1.0 + exp(-z));
    return z;
}

typedef struct {
    const double *x, *wr, *wi, *wj, *wk, *bias, *scale, *shift, *residual;
    int N, H, W, Cin, Cout, kh, kw, stride, pad, act, Ho, Wo;
} qconv_args;

/* One output pixel (all C_out channels) of the quaternion convolution, Eq. 5:
 * for every output quaternion channel co, accumulate W[co, tap, ci] (x) X[pixel+tap, ci]
 * over taps and input quaternion channels with the Hamilton product of Eq. 3,
 * then apply the per-real-channel epilogue. */
static void qconv_pixel(const qconv_args *a, int n, int ho, int wo, double *yout) {
    const int Qin = a->Cin / 4, Qout = a->Cout / 4;
    for (int co = 0; co < Qout; ++co) {
        double acc[4] = {0.0, 0.0, 0.0, 0.0};
        for (int dh = 0; dh < a->kh; ++dh) {
            const int h = ho * a->stride - a->pad + dh;
            if (h < 0 || h >= a->H) continue;            /* zero padding */
            for (int dw = 0; dw < a->kw; ++dw) {
                const int w = wo * a->stride - a->pad + dw;
                if (w < 0 || w >= a->W) continue;        /* zero padding */
                const double *xp = a->x + (((size_t)n * a->H + h) * a->W + w) * a->Cin;
                for (int ci = 0; ci < Qin; ++ci) {
                    const size_t widx = (((size_t)co * a->kh + dh) * a->kw + dw) * Qin + ci;
                    const double wq[4] = {a->wr[widx], a->wi[widx], a->wj[widx], a->wk[widx]};
                    const double xq[4] = {xp[0 * Qin + ci], xp[1 * Qin + ci],
                                          xp[2 * Qin + ci], xp[3 * Qin + ci]};
                    double t[4];
                    oracle_qmul(wq, xq, t);
                    acc[0] += t[0]; acc[1] += t[1]; acc[2] += t[2]; acc[3] += t[3];
                }
            }
        }
        for (int m = 0; m < 4; ++m) {
            const int c = m * Qout + co;
            double z = acc[m];
            if (a->bias) z += a->bias[c];
            if (a->scale) z = a->scale[c] * z + a->shift[c];
            if (a->residual)
                z += a->residual[(((size_t)n * a->Ho + ho) * a->Wo + wo) * a->Cout + c];
            yout[c] = apply_act(z, a->act);
        }
    }
}

static int out_dim(int in, int k, int stride, int pad) {
    return (in + 2 * pad - k) / stride + 1;
}

static int check_args(const qconv_args *a) {
    if (a->N <= 0 || a->H <= 0 || a->W <= 0 || a->Cin <= 0 || a->Cout <= 0) return -1;
    if (a->Cin % 4 || a->Cout % 4) return -1;
    if (a->kh <= 0 || a->kw <= 0 || a->stride <= 0 || a->pad < 0) return -1;
    if (a->Ho <= 0 || a->Wo <= 0) return -1;
    if (a->scale && !a->shift) return -1;
    if (!a->x || !a->wr || !a->wi || !a->wj || !a->wk) return -1;
    return 0;
}

/* Full quaternion convolution forward (Eq. 5 + IQBN inference epilogue of Eq. 11-12).
 * bias, scale, shift: [C_out] or NULL; residual: [N][Ho][Wo][C_out] or NULL.
 * Returns 0 on success, -1 on invalid arguments. */
int oracle_qconv2d(const double *x, const double *wr, const double *wi, const double *wj,
                   const double *wk, const double *bias, const double *scale,
                   const double *shift, const double *residual, int N, int H, int W,
                   int Cin, int Cout, int kh, int kw, int stride, int pad, int act,
                   double *y) {
    qconv_args a = {x, wr, wi, wj, wk, bias, scale, shift, residual,
                    N, H, W, Cin, Cout, kh, kw, stride, pad, act, 0, 0};
    if (stride <= 0) return -1;
    a.Ho = out_dim(H, kh, stride, pad);
    a.Wo = out_dim(W, kw, stride, pad);
    if (check_args(&a)) return -1;
    const long long npix = (long long)N * a.Ho * a.Wo;
#pragma omp parallel for schedule(dynamic, 16)
    for (long long p = 0; p < npix; ++p) {
        const int n = (int)(p / ((long long)a.Ho * a.Wo));
        const int rem = (int)(p % ((long long)a.Ho * a.Wo));
        qconv_pixel(&a, n, rem / a.Wo, rem % a.Wo, y + (size_t)p * Cout);
    }
    return 0;
}

/* Same computation at a list of output pixels only (n[i], ho[i], wo[i]);
 * y is [npts][C_out].  Used to check full-size layers on sampled outputs. */
int oracle_qconv2d_points(const double *x, const double *wr, const double *wi,
                          const double *wj, const double *wk, const double *bias,
                          const double *scale, const double *shift, const double *residual,
                          int N, int H, int W, int Cin, int Cout, int kh, int kw, int stride,
                          int pad, int act, int npts, const int *pn, const int *pho,
                          const int *pwo, double *y) {
    qconv_args a = {x, wr, wi, wj, wk, bias, scale, shift, residual,
                    N, H, W, Cin, Cout, kh, kw, stride, pad, act, 0, 0};
    if (stride <= 0) return -1;
    a.Ho = out_dim(H, kh, stride, pad);
    a.Wo = out_dim(W, kw, stride, pad);
    if (check_args(&a)) return -1;
    for (int i = 0; i < npts; ++i)
        if (pn[i] < 0 || pn[i] >= N || pho[i] < 0 || pho[i] >= a.Ho || pwo[i] < 0 ||
            pwo[i] >= a.Wo)
            return -1;
#pragma omp parallel for schedule(dynamic, 4)
    for (int i = 0; i < npts; ++i) qconv_pixel(&a, pn[i], pho[i], pwo[i], y + (size_t)i * Cout);
    return 0;
}

/* Separable QUAN convolution of Eq. 7 (Sec. III-B): only the diagonal terms
 * W_p (x) x_p, combined with the printed sign table
 *   y_r = +r -i -j -k,  y_i = +r +i +j -k,  y_j = +r -i +j +k,  y_k = +r +i -j +k,
 * where "r" stands for W_r conv x_r, and so on.  Same epilogue as the full form. */
int oracle_qconv2d_separable(const double *x, const double *wr, const double *wi,
                             const double *wj, const double *wk, const double *bias,
                             const double *scale, const double *shift, int N, int H, int W,
                             int Cin, int Cout, int kh, int kw, int stride, int pad, int act,
                             double *y) {
    static const double sgn[4][4] = {
        {+1, -1, -1, -1},  /* y_r */
        {+1, +1, +1, -1},  /* y_i */
        {+1, -1, +1, +1},  /* y_j */
        {+1, +1, -1, +1},  /* y_k */
    };
    const double *wl[4] = {wr, wi, wj, wk};
    const int Ho = out_dim(H, kh, stride > 0 ? stride : 1, pad);
    const int Wo = out_dim(W, kw, stride > 0 ? stride : 1, pad);
    qconv_args a = {x, wr, wi, wj, wk, bias, scale, shift, NULL,
                    N, H, W, Cin, Cout, kh, kw, stride, pad, act, Ho, Wo};
    if (stride <= 0 || check_args(&a)) return -1;
    const int Qin = Cin / 4, Qout = Cout / 4;
    const long long npix = (long long)N * Ho * Wo;
#pragma omp parallel for schedule(dynamic, 16)
    for (long long p = 0; p < npix; ++p) {
        const int n = (int)(p / ((long long)Ho * Wo));
        const int rem = (int)(p % ((long long)Ho * Wo));
        const int ho = rem / Wo, wo = rem % Wo;
        for (int co = 0; co < Qout; ++co) {
            double conv[4] = {0, 0, 0, 0};   /* conv[p] = W_p conv x_p */
            for (int dh = 0; dh < kh; ++dh) {
                const int h = ho * stride - pad + dh;
                if (h < 0 || h >= H) continue;
                for (int dw = 0; dw < kw; ++dw) {
                    const int w = wo * stride - pad + dw;
                    if (w < 0 || w >= W) continue;
                    const double *xp = x + (((size_t)n * H + h) * W + w) * Cin;
                    for (int ci = 0; ci < Qin; ++ci) {
                        const size_t widx = (((size_t)co * kh + dh) * kw + dw) * Qin + ci;
                        for (int comp = 0; comp < 4; ++comp)
                            conv[comp] += wl[comp][widx] * xp[comp * Qin + ci];
                    }
                }
            }
            for (int m = 0; m < 4; ++m) {
                const int c = m * Qout + co;
                double z = 0.0;
                for (int comp = 0; comp < 4; ++comp) z += sgn[m][comp] * conv[comp];
                if (bias) z += bias[c];
                if (scale) z = scale[c] * z + shift[c];
                y[(size_t)p * Cout + c] = apply_act(z, act);
            }
        }
    }
    return 0;
}

/* The real block weight of Eq. 6 (Sec. III-B): for every tap, output component q
 * and input component p, the [Q_out x Q_in] block is the signed letter tensor at
 * row q, column p of
 *     [ w_r  -w_i  -w_j  -w_k ]
 *     [ w_i   w_r  -w_k   w_j ]
 *     [ w_j   w_k   w_r  -w_i ]
 *     [ w_k  -w_j   w_i   w_r ].
 * Output wb is [C_out][kh][kw][C_in] with component-major channels on both sides. */
int oracle_expand_block_weight(const double *wr, const double *wi, const double *wj,
                               const double *wk, int Cin, int Cout, int kh, int kw,
                               double *wb) {
    if (Cin <= 0 || Cout <= 0 || Cin % 4 || Cout % 4 || kh <= 0 || kw <= 0) return -1;
    const double *L[4] = {wr, wi, wj, wk};
    /* letter index and sign at (row q, column p) of the matrix above */
    static const int letter[4][4] = {{0, 1, 2, 3}, {1, 0, 3, 2}, {2, 3, 0, 1}, {3, 2, 1, 0}};
    static const double sign[4][4] = {
        {+1, -1, -1, -1}, {+1, +1, -1, +1}, {+1, +1, +1, -1}, {+1, -1, +1, +1}};
    const int Qin = Cin / 4, Qout = Cout / 4;
    for (int q = 0; q < 4; ++q)
        for (int co = 0; co < Qout; ++co)
            for (int dh = 0; dh < kh; ++dh)
                for (int dw = 0; dw < kw; ++dw)
                    for (int p = 0; p < 4; ++p)
                        for (int ci = 0; ci < Qin; ++ci) {
                            const size_t src = (((size_t)co * kh + dh) * kw + dw) * Qin + ci;
                            const size_t dst =
                                (((size_t)(q * Qout + co) * kh + dh) * kw + dw) * Cin +
                                p * Qin + ci;
                            wb[dst] = sign[q][p] * L[letter[q][p]][src];
                        }
    return 0;
}

/* Ordinary real cross-correlation, NHWC input, weight [C_out][kh][kw][C_in],
 * zero padding, no epilogue. */
int oracle_real_conv2d(const double *x, const double *w, int N, int H, int W, int Cin,
                       int Cout, int kh, int kw, int stride, int pad, double *y) {
    if (N <= 0 || H <= 0 || W <= 0 || Cin <= 0 || Cout <= 0 || stride <= 0 || pad < 0)
        return -1;
    const int Ho = out_dim(H, kh, stride, pad), Wo = out_dim(W, kw, stride, pad);
    if (Ho <= 0 || Wo <= 0) return -1;
    const long long npix = (long long)N * Ho * Wo;
#pragma omp parallel for schedule(dynamic, 16)
    for (long long p = 0; p < npix; ++p) {
        const int n = (int)(p / ((long long)Ho * Wo));
        const int rem = (int)(p % ((long long)Ho * Wo));
        const int ho = rem / Wo, wo = rem % Wo;
        for (int co = 0; co < Cout; ++co) {
            double acc = 0.0;
            for (int dh = 0; dh < kh; ++dh) {
                const int h = ho * stride - pad + dh;
                if (h < 0 || h >= H) continue;
                for (int dw = 0; dw < kw; ++dw) {
                    const int wq = wo * stride - pad + dw;
                    if (wq < 0 || wq >= W) continue;
                    for (int ci = 0; ci < Cin; ++ci)
                        acc += x[(((size_t)n * H + h) * W + wq) * Cin + ci] *
                               w[(((size_t)co * kh + dh) * kw + dw) * Cin + ci];
                }
            }
            y[(size_t)p * Cout + co] = acc;
        }
    }
    return 0;
}

/* Max pooling applied to each real channel independently (the component-wise
 * pooling rule of QSPPF, Sec. III-D); padded positions never win (-inf). */
int oracle_maxpool2d(const double *x, int N, int H, int W, int C, int k, int stride, int pad,
                     double *y) {
    if (N <= 0 || H <= 0 || W <= 0 || C <= 0 || k <= 0 || stride <= 0 || pad < 0) return -1;
    const int Ho = out_dim(H, k, stride, pad), Wo = out_dim(W, k, stride, pad);
    if (Ho <= 0 || Wo <= 0) return -1;
    const long long npix = (long long)N * Ho * Wo;
#pragma omp parallel for schedule(static)
    for (long long p = 0; p < npix; ++p) {
        const int n = (int)(p / ((long long)Ho * Wo));
        const int rem = (int)(p % ((long long)Ho * Wo));
        const int ho = rem / Wo, wo = rem % Wo;
        for (int c = 0; c < C; ++c) {
            double m = -INFINITY;
            for (int dh = 0; dh < k; ++dh) {
                const int h = ho * stride - pad + dh;
                if (h < 0 || h >= H) continue;
                for (int dw = 0; dw < k; ++dw) {
                    const int w = wo * stride - pad + dw;
                    if (w < 0 || w >= W) continue;
                    const double v = x[(((size_t)n * H + h) * W + w) * C + c];
                    if (v > m) m = v;
                }
            }
            y[(size_t)p * C + c] = m;
        }
    }
    return 0;
}

/* ---------------------------------------------------------------- backward pass
 * Gradients of the convolution of Eq. 5 before its epilogue, y = sum over taps and input
 * quaternion channels of W (x) X, given dy = dL/dy (same layout as y).  Both are written
 * from the Jacobians of the Hamilton product (Eq. 3) taken literally:
 *   d(W (x) X)_q / dX_p = (W (x) e_p)_q,    d(W (x) X)_q / dW_L = (e_L (x) X)_q,
 * e_m the quaternion basis element m, each evaluated with oracle_qmul. */
static const double BASIS[4][4] = {{1, 0, 0, 0}, {0, 1, 0, 0}, {0, 0, 1, 0}, {0, 0, 0, 1}};

/* dx [N][H][W][C_in]: every output pixel and tap that reads input pixel (h, w) adds
 * sum_q (W (x) e_p)_q dy_q to dx_p.  Returns 0, or -1 on invalid arguments. */
int oracle_qconv2d_bwd_data(const double *dy, const double *wr, const double *wi,
                            const double *wj, const double *wk, int N, int H, int W, int Cin,
                            int Cout, int kh, int kw, int stride, int pad, double *dx) {
    qconv_args a = {dy, wr, wi, wj, wk, NULL, NULL, NULL, NULL,
                    N, H, W, Cin, Cout, kh, kw, stride, pad, ACT_NONE, 0, 0};
    if (stride <= 0 || !dx) return -1;
    a.Ho = out_dim(H, kh, stride, pad);
    a.Wo = out_dim(W, kw, stride, pad);
    if (check_args(&a)) return -1;
    const int Qin = Cin / 4, Qout = Cout / 4;
    memset(dx, 0, sizeof(double) * (size_t)N * H * W * Cin);
#pragma omp parallel for schedule(dynamic, 1)
    for (int n = 0; n < N; ++n) {          /* one image per thread: no shared dx entry */
        for (int ho = 0; ho < a.Ho; ++ho)
            for (int wo = 0; wo < a.Wo; ++wo) {
                const double *g = dy + (((size_t)n * a.Ho + ho) * a.Wo + wo) * Cout;
                for (int dh = 0; dh < kh; ++dh) {
                    const int h = ho * stride - pad + dh;
                    if (h < 0 || h >= H) continue;
                    for (int dw = 0; dw < kw; ++dw) {
                        const int w = wo * stride - pad + dw;
                        if (w < 0 || w >= W) continue;
                        double *d = dx + (((size_t)n * H + h) * W + w) * Cin;
                        for (int co = 0; co < Qout; ++co)
                            for (int ci = 0; ci < Qin; ++ci) {
                                const size_t widx = (((size_t)co * kh + dh) * kw + dw) * Qin + ci;
                                const double wq[4] = {wr[widx], wi[widx], wj[widx], wk[widx]};
                                for (int p = 0; p < 4; ++p) {
                                    double col[4];
                                    oracle_qmul(wq, BASIS[p], col);
                                    for (int q = 0; q < 4; ++q)
                                        d[p * Qin + ci] += col[q] * g[q * Qout + co];
                                }
                            }
                    }
                }
            }
    }
    return 0;
}

/* dW_L [Q_out][kh][kw][Q_in] for L = r, i, j, k: the sum over output pixels of
 * sum_q (e_L (x) X)_q dy_q, X the input quaternion the tap reads.  Returns 0 or -1. */
int oracle_qconv2d_bwd_weight(const double *x, const double *dy, int N, int H, int W, int Cin,
                              int Cout, int kh, int kw, int stride, int pad, double *dwr,
                              double *dwi, double *dwj, double *dwk) {
    const double dummy = 0.0;
    qconv_args a = {x, &dummy, &dummy, &dummy, &dummy, NULL, NULL, NULL, NULL,
                    N, H, W, Cin, Cout, kh, kw, stride, pad, ACT_NONE, 0, 0};
    if (stride <= 0 || !dy || !dwr || !dwi || !dwj || !dwk) return -1;
    a.Ho = out_dim(H, kh, stride, pad);
    a.Wo = out_dim(W, kw, stride, pad);
    if (check_args(&a)) return -1;
    const int Qin = Cin / 4, Qout = Cout / 4;
    double *dwl[4] = {dwr, dwi, dwj, dwk};
#pragma omp parallel for schedule(dynamic, 1)
    for (int co = 0; co < Qout; ++co)       /* one output channel per thread */
        for (int dh = 0; dh < kh; ++dh)
            for (int dw = 0; dw < kw; ++dw)
                for (int ci = 0; ci < Qin; ++ci) {
                    double acc[4] = {0, 0, 0, 0};
                    for (int n = 0; n < N; ++n)
                        for (int ho = 0; ho < a.Ho; ++ho) {
                            const int h = ho * stride - pad + dh;
                            if (h < 0 || h >= H) continue;
                            for (int wo = 0; wo < a.Wo; ++wo) {
                                const int w = wo * stride - pad + dw;
                                if (w < 0 || w >= W) continue;
                                const double *xp = x + (((size_t)n * H + h) * W + w) * Cin;
                                const double *g =
                                    dy + (((size_t)n * a.Ho + ho) * a.Wo + wo) * Cout;
                                const double xq[4] = {xp[ci], xp[Qin + ci], xp[2 * Qin + ci],
                                                      xp[3 * Qin + ci]};
                                for (int L = 0; L < 4; ++L) {
                                    double t[4];
                                    oracle_qmul(BASIS[L], xq, t);
                                    for (int q = 0; q < 4; ++q) acc[L] += t[q] * g[q * Qout + co];
                                }
                            }
                        }
                    const size_t widx = (((size_t)co * kh + dh) * kw + dw) * Qin + ci;
                    for (int L = 0; L < 4; ++L) dwl[L][widx] = acc[L];
                }
    return 0;
}

/* ---------------------------------------------------------------- separable backward
 * Gradients of the separable convolution of Eq. 7 before its epilogue, by Eq. 8-10:
 * the output gradients are mixed by the matrix M of Eq. 9,
 *     [  1  1  1  1 ]
 *     [ -1  1 -1  1 ]
 *     [ -1  1  1 -1 ]
 *     [ -1 -1  1  1 ],
 * row p giving the weights of dy_r, dy_i, dy_j, dy_k for input component p, and each
 * component p then takes the plain convolution gradients with its own letter W_p:
 *     dx_p = sum_m M[p][m] (dy_m correlated back through W_p),
 *     dW_p = sum_m M[p][m] (dy_m correlated with x_p).
 * (Eq. 8 and 10 print the same letter q on the sum and inside it; this is the reading
 * that makes them the gradient of Eq. 7, whose sign table is M transposed.) */
static const double MIX_EQ9[4][4] = {
    {+1, +1, +1, +1},
    {-1, +1, -1, +1},
    {-1, +1, +1, -1},
    {-1, -1, +1, +1},
};

/* dx [N][H][W][C_in] of the separable form.  Returns 0, or -1 on invalid arguments. */
int oracle_qconv2d_sep_bwd_data(const double *dy, const double *wr, const double *wi,
                                const double *wj, const double *wk, int N, int H, int W,
                                int Cin, int Cout, int kh, int kw, int stride, int pad,
                                double *dx) {
    qconv_args a = {dy, wr, wi, wj, wk, NULL, NULL, NULL, NULL,
                    N, H, W, Cin, Cout, kh, kw, stride, pad, ACT_NONE, 0, 0};
    if (stride <= 0 || !dx) return -1;
    a.Ho = out_dim(H, kh, stride, pad);
    a.Wo = out_dim(W, kw, stride, pad);
    if (check_args(&a)) return -1;
    const int Qin = Cin / 4, Qout = Cout / 4;
    const double *wl[4] = {wr, wi, wj, wk};
    memset(dx, 0, sizeof(double) * (size_t)N * H * W * Cin);
#pragma omp parallel for schedule(dynamic, 1)
    for (int n = 0; n < N; ++n) {          /* one image per thread: no shared dx entry */
        for (int ho = 0; ho < a.Ho; ++ho)
            for (int wo = 0; wo < a.Wo; ++wo) {
                const double *g = dy + (((size_t)n * a.Ho + ho) * a.Wo + wo) * Cout;
                for (int dh = 0; dh < kh; ++dh) {
                    const int h = ho * stride - pad + dh;
                    if (h < 0 || h >= H) continue;
                    for (int dw = 0; dw < kw; ++dw) {
                        const int w = wo * stride - pad + dw;
                        if (w < 0 || w >= W) continue;
                        double *d = dx + (((size_t)n * H + h) * W + w) * Cin;
                        for (int co = 0; co < Qout; ++co)
                            for (int ci = 0; ci < Qin; ++ci) {
                                const size_t widx = (((size_t)co * kh + dh) * kw + dw) * Qin + ci;
                                for (int p = 0; p < 4; ++p)
                                    for (int m = 0; m < 4; ++m)
                                        d[p * Qin + ci] +=
                                            MIX_EQ9[p][m] * wl[p][widx] * g[m * Qout + co];
                            }
                    }
                }
            }
    }
    return 0;
}

/* dW_p [Q_out][kh][kw][Q_in] of the separable form.  Returns 0 or -1. */
int oracle_qconv2d_sep_bwd_weight(const double *x, const double *dy, int N, int H, int W,
                                  int Cin, int Cout, int kh, int kw, int stride, int pad,
                                  double *dwr, double *dwi, double *dwj, double *dwk) {
    const double dummy = 0.0;
    qconv_args a = {x, &dummy, &dummy, &dummy, &dummy, NULL, NULL, NULL, NULL,
                    N, H, W, Cin, Cout, kh, kw, stride, pad, ACT_NONE, 0, 0};
    if (stride <= 0 || !dy || !dwr || !dwi || !dwj || !dwk) return -1;
    a.Ho = out_dim(H, kh, stride, pad);
    a.Wo = out_dim(W, kw, stride, pad);
    if (check_args(&a)) return -1;
    const int Qin = Cin / 4, Qout = Cout / 4;
    double *dwl[4] = {dwr, dwi, dwj, dwk};
#pragma omp parallel for schedule(dynamic, 1)
    for (int co = 0; co < Qout; ++co)       /* one output channel per thread */
        for (int dh = 0; dh < kh; ++dh)
            for (int dw = 0; dw < kw; ++dw)
                for (int ci = 0; ci < Qin; ++ci) {
                    double acc[4] = {0, 0, 0, 0};
                    for (int n = 0; n < N; ++n)
                        for (int ho = 0; ho < a.Ho; ++ho) {
                            const int h = ho * stride - pad + dh;
                            if (h < 0 || h >= H) continue;
                            for (int wo = 0; wo < a.Wo; ++wo) {
                                const int w = wo * stride - pad + dw;
                                if (w < 0 || w >= W) continue;
                                const double *xp = x + (((size_t)n * H + h) * W + w) * Cin;
                                const double *g =
                                    dy + (((size_t)n * a.Ho + ho) * a.Wo + wo) * Cout;
                                for (int p = 0; p < 4; ++p)
                                    for (int m = 0; m < 4; ++m)
                                        acc[p] += MIX_EQ9[p][m] * g[m * Qout + co] *
                                                  xp[p * Qin + ci];
                            }
                        }
                    const size_t widx = (((size_t)co * kh + dh) * kw + dw) * Qin + ci;
                    for (int p = 0; p < 4; ++p) dwl[p][widx] = acc[p];
                }
    return 0;
}

/* ---------------------------------------------------------------- IQBN, training mode
 * Batch statistics of Eq. 11 (Sec. III-C), one real channel at a time: over the N H W
 * values of channel c (one component of one quaternion channel),
 *     mu_c = E[x_c],   sigma2_c = E[(x_c - mu_c)^2]      (two passes, biased variance).
 * x is [npix][C] (NHWC flattened).  Returns 0, or -1 on invalid arguments. */
int oracle_iqbn_batch_stats(const double *x, long long npix, int C, double *mean,
                            double *var) {
    if (!x || !mean || !var || npix < 1 || C < 1) return -1;
#pragma omp parallel for schedule(static)
    for (int c = 0; c < C; ++c) {
        double s = 0.0;
        for (long long p = 0; p < npix; ++p) s += x[(size_t)p * C + c];
        const double mu = s / (double)npix;
        double s2 = 0.0;
        for (long long p = 0; p < npix; ++p) {
            const double d = x[(size_t)p * C + c] - mu;
            s2 += d * d;
        }
        mean[c] = mu;
        var[c] = s2 / (double)npix;
    }
    return 0;
}

/* Training-mode IQBN output of Eq. 11-12: x_hat = (x - mu) / sqrt(sigma2 + eps) with the
 * batch statistics above, then x_hat * gamma + beta per real channel, then the split
 * activation.  Returns 0 or -1. */
int oracle_iqbn_train(const double *x, long long npix, int C, const double *gamma,
                      const double *beta, double eps, int act, double *y) {
    if (!x || !gamma || !beta || !y || npix < 1 || C < 1 || eps < 0.0) return -1;
    if (act < ACT_NONE || act > ACT_SILU) return -1;
    double *mean = (double *)malloc(sizeof(double) * (size_t)C);
    double *var = (double *)malloc(sizeof(double) * (size_t)C);
    if (!mean || !var) {
        free(mean);
        free(var);
        return -1;
    }
    oracle_iqbn_batch_stats(x, npix, C, mean, var);
#pragma omp parallel for schedule(static)
    for (long long p = 0; p < npix; ++p)
        for (int c = 0; c < C; ++c) {
            const double xh = (x[(size_t)p * C + c] - mean[c]) / sqrt(var[c] + eps);
            y[(size_t)p * C + c] = apply_act(xh * gamma[c] + beta[c], act);
        }
    free(mean);
    free(var);
    return 0;
}

/* Poincare mapping of Eq. 4 (Sec. III-A): rgb [npix][3] -> q [npix][4] as
 * (q_r, q_i, q_j, q_k) = ((1 - n^2), 2r, 2g, 2b) / (1 + n^2), n^2 = r^2 + g^2 + b^2. */
void oracle_poincare(const double *rgb, long long npix, double *q) {
    for (long long p = 0; p < npix; ++p) {
        const double r = rgb[3 * p], g = rgb[3 * p + 1], b = rgb[3 * p + 2];
        const double n2 = r * r + g * g + b * b;
        const double d = 1.0 + n2;
        q[4 * p + 0] = (1.0 - n2) / d;
        q[4 * p + 1] = 2.0 * r / d;
        q[4 * p + 2] = 2.0 * g / d;
        q[4 * p + 3] = 2.0 * b / d;
    }
}

int oracle_num_threads(void) {
#ifdef _OPENMP
    extern int omp_get_max_threads(void);
    return omp_get_max_threads();
#else
    return 1;
#endif
}
