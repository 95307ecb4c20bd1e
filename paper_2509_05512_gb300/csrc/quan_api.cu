// quan_api.cu -- the C ABI of libquan: argument validation, path selection, launch.
// See include/quan.h for the contract of every entry point.
#include <cuda_runtime.h>

#include <atomic>
#include <cstdarg>
#include <cstdint>
#include <cmath>
#include <cstdio>
#include <mutex>

#include "internal.h"
#include "quan.h"

namespace {

thread_local char t_errmsg[512] = "";
thread_local int t_last_path = 0;
thread_local const char* t_last_kernel = "";
std::atomic<int> g_path{QUAN_PATH_AUTO};
std::atomic<int> g_kappa{0}, g_bnq{0}, g_max_ctas{0}, g_mode{0}, g_ws_halo{1}, g_ws_issuers{0},
    g_vs_rows{0};
std::atomic<unsigned long long> g_wait_limit{2000000000ull};
std::atomic<int> g_inject{0};

constexpr int kMaxDevices = 64;
int g_num_sms[kMaxDevices] = {0};
int g_cc[kMaxDevices] = {0};
void* g_static_scratch[kMaxDevices] = {nullptr};  // quan_qconv2d_bwd_data_static, per device
std::mutex g_dev_mu;

quan_status_t fail(quan_status_t st, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(t_errmsg, sizeof(t_errmsg), fmt, ap);
    va_end(ap);
    return st;
}

quan_status_t cuda_fail(cudaError_t e, const char* what) {
    return fail(QUAN_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

// Number of SMs and compute capability (major*10+minor) of the current device.
bool device_info(int* num_sms, int* cc, cudaError_t* err) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        *err = e;
        return false;
    }
    if (dev >= 0 && dev < kMaxDevices) {
        std::lock_guard<std::mutex> lk(g_dev_mu);
        if (g_num_sms[dev] == 0) {
            int sms = 0, maj = 0, mnr = 0;
            if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) !=
                    cudaSuccess ||
                (e = cudaDeviceGetAttribute(&maj, cudaDevAttrComputeCapabilityMajor, dev)) !=
                    cudaSuccess ||
                (e = cudaDeviceGetAttribute(&mnr, cudaDevAttrComputeCapabilityMinor, dev)) !=
                    cudaSuccess) {
                *err = e;
                return false;
            }
            g_num_sms[dev] = sms;
            g_cc[dev] = maj * 10 + mnr;
        }
        *num_sms = g_num_sms[dev];
        *cc = g_cc[dev];
        return true;
    }
    *err = cudaErrorInvalidDevice;
    return false;
}

bool overlaps(const void* a, size_t na, const void* b, size_t nb) {
    if (!a || !b) return false;
    const uintptr_t a0 = reinterpret_cast<uintptr_t>(a), b0 = reinterpret_cast<uintptr_t>(b);
    return a0 < b0 + nb && b0 < a0 + na;
}

// Checks the sizes of one convolution and fills *s (epilogue-free, full form).
quan_status_t geometry(quan::ConvShape* s, int N, int H, int W, int Cin, int Cout, int kh,
                       int kw, int stride, int pad) {
    if (N < 1 || H < 1 || W < 1 || Cin < 1 || Cout < 1 || kh < 1 || kw < 1 || stride < 1 ||
        pad < 0)
        return fail(QUAN_ERR_INVALID_ARG,
                    "sizes must be positive (N=%d H=%d W=%d Cin=%d Cout=%d kh=%d kw=%d "
                    "stride=%d) and pad >= 0 (pad=%d)",
                    N, H, W, Cin, Cout, kh, kw, stride, pad);
    if (Cin % 4 || Cout % 4)
        return fail(QUAN_ERR_INVALID_ARG, "Cin=%d and Cout=%d must be multiples of 4", Cin, Cout);
    const long long Ho = (static_cast<long long>(H) + 2LL * pad - kh) / stride + 1;
    const long long Wo = (static_cast<long long>(W) + 2LL * pad - kw) / stride + 1;
    if (static_cast<long long>(H) + 2LL * pad < kh || static_cast<long long>(W) + 2LL * pad < kw ||
        Ho < 1 || Wo < 1)
        return fail(QUAN_ERR_INVALID_ARG, "filter %dx%d larger than the padded input %dx%d", kh,
                    kw, H + 2 * pad, W + 2 * pad);
    const long long xin = static_cast<long long>(N) * H * W * Cin;
    const long long yout = static_cast<long long>(N) * Ho * Wo * Cout;
    if (xin >= (1LL << 40) || yout >= (1LL << 40) || Ho > 0x7fffffff / Wo)
        return fail(QUAN_ERR_UNSUPPORTED, "tensor too large");
    s->N = N; s->H = H; s->W = W; s->Cin = Cin; s->Cout = Cout;
    s->kh = kh; s->kw = kw; s->stride = stride; s->pad = pad; s->act = QUAN_ACT_NONE;
    s->Ho = static_cast<int>(Ho); s->Wo = static_cast<int>(Wo);
    s->Qin = Cin / 4; s->Qout = Cout / 4;
    s->M = static_cast<long long>(N) * Ho * Wo;
    s->sep = 0;
    return QUAN_OK;
}

size_t x_bytes(const quan::ConvShape& s, size_t esize) {
    return static_cast<size_t>(s.N) * s.H * s.W * s.Cin * esize;
}
size_t y_bytes(const quan::ConvShape& s, size_t esize) {
    return static_cast<size_t>(s.M) * s.Cout * esize;
}
size_t w_bytes(const quan::ConvShape& s, size_t esize) {
    return static_cast<size_t>(s.Qout) * s.kh * s.kw * s.Qin * esize;
}

quan_status_t validate(quan::ConvShape* s, const void* x, const void* const w[4],
                       const float* bias, const float* scale, const float* shift, int N, int H,
                       int W, int Cin, int Cout, int kh, int kw, int stride, int pad, int act,
                       const void* residual, const void* out, size_t esize) {
    if (!x || !w[0] || !w[1] || !w[2] || !w[3] || !out)
        return fail(QUAN_ERR_INVALID_ARG, "null tensor pointer");
    quan_status_t st = geometry(s, N, H, W, Cin, Cout, kh, kw, stride, pad);
    if (st != QUAN_OK) return st;
    if ((scale == nullptr) != (shift == nullptr))
        return fail(QUAN_ERR_INVALID_ARG, "iqbn_scale and iqbn_shift must both be given or both NULL");
    if (act < QUAN_ACT_NONE || act > QUAN_ACT_SILU)
        return fail(QUAN_ERR_INVALID_ARG, "unknown activation %d", act);
    const size_t wbytes = w_bytes(*s, esize), xbytes = x_bytes(*s, esize);
    const size_t ybytes = y_bytes(*s, esize);
    if (overlaps(out, ybytes, x, xbytes) || overlaps(out, ybytes, w[0], wbytes) ||
        overlaps(out, ybytes, w[1], wbytes) || overlaps(out, ybytes, w[2], wbytes) ||
        overlaps(out, ybytes, w[3], wbytes) || overlaps(out, ybytes, residual, ybytes) ||
        overlaps(out, ybytes, bias, Cout * 4u) || overlaps(out, ybytes, scale, Cout * 4u) ||
        overlaps(out, ybytes, shift, Cout * 4u))
        return fail(QUAN_ERR_INVALID_ARG, "out overlaps an input");
    s->act = act;
    return QUAN_OK;
}

quan_status_t run_bf16(const void* x, const void* wr, const void* wi, const void* wj,
                       const void* wk, const float* bias, const float* scale, const float* shift,
                       int N, int H, int W, int Cin, int Cout, int kh, int kw, int stride, int pad,
                       int act, const void* residual, void* out, quan_stream_t stream,
                       bool separable = false, void* sk_ws = nullptr, size_t sk_ws_bytes = 0) {
    const void* w[4] = {wr, wi, wj, wk};
    quan::ConvShape s;
    quan_status_t st = validate(&s, x, w, bias, scale, shift, N, H, W, Cin, Cout, kh, kw,
                                stride, pad, act, residual, out, 2);
    if (st != QUAN_OK) return st;
    s.sep = separable ? 1 : 0;
    int num_sms = 0, cc = 0;
    cudaError_t e;
    if (!device_info(&num_sms, &cc, &e)) return cuda_fail(e, "device query");
    const int path = g_path.load();
    const quan::EpilogueArgs ep{bias, scale, shift, residual};
    const bool tc_ok = cc == 103 && quan::tc_supported(s, x, w, out, ep);
    bool use_tc;
    if (path == QUAN_PATH_TC) {
        if (!tc_ok)
            return fail(QUAN_ERR_UNSUPPORTED,
                        "tensor-core path needs sm_103, Cin/4 and Cout/4 multiples of 16 (or, "
                        "for the full form, Cin = 4, Cout = 64, stride 2, even W) and 16-byte "
                        "aligned tensors (device cc %d, Cin=%d, Cout=%d)",
                        cc, Cin, Cout);
        use_tc = true;
    } else if (path == QUAN_PATH_SIMT) {
        use_tc = false;
    } else {
        use_tc = tc_ok;
    }
    cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
    if (use_tc) {
        quan::TcOptions opt;
        opt.kappa = g_kappa.load();
        opt.bnq = g_bnq.load();
        opt.max_ctas = g_max_ctas.load();
        opt.mode = g_mode.load();
        opt.ws_halo = g_ws_halo.load();
        opt.ws_issuers = g_ws_issuers.load();
        opt.vs_rows = g_vs_rows.load();
        opt.sk_ws = sk_ws;
        opt.sk_ws_bytes = sk_ws_bytes;
        opt.wait_limit_ns = g_wait_limit.load();
        opt.inject_stall = g_inject.load();
        char err[256] = "";
        e = quan::launch_qconv_tc(s, x, w, ep, out, opt, num_sms, cs, err, sizeof(err));
        if (err[0] != '\0') return fail(QUAN_ERR_UNSUPPORTED, "%s", err);
        if (e != cudaSuccess) return cuda_fail(e, "qconv_tc launch");
        t_last_path = QUAN_PATH_TC;
        t_last_kernel = quan::last_tc_kernel();
    } else {
        e = quan::launch_qconv_simt_bf16(s, x, w, ep, out, cs);
        if (e != cudaSuccess) return cuda_fail(e, "qconv_simt launch");
        t_last_path = QUAN_PATH_SIMT;
        t_last_kernel = s.sep ? "qconv_simt_kernel<bf16,sep>" : "qconv_simt_kernel<bf16>";
    }
    return QUAN_OK;
}

// Input gradient of the pre-epilogue convolution (full form or separable).
quan_status_t run_bwd_data(const void* dy, const void* const w[4], int N, int H, int W, int Cin,
                           int Cout, int kh, int kw, int stride, int pad, bool separable,
                           void* workspace, size_t workspace_bytes, void* dx,
                           quan_stream_t stream) {
    if (!dy || !w[0] || !w[1] || !w[2] || !w[3] || !dx)
        return fail(QUAN_ERR_INVALID_ARG, "null tensor pointer");
    quan::ConvShape s;
    quan_status_t st = geometry(&s, N, H, W, Cin, Cout, kh, kw, stride, pad);
    if (st != QUAN_OK) return st;
    s.sep = separable ? 1 : 0;
    const size_t need = quan::bwd_data_workspace_bytes(Cin, Cout, kh, kw);
    if (!workspace || workspace_bytes < need)
        return fail(QUAN_ERR_INVALID_ARG, "workspace must hold %zu bytes (got %zu%s)", need,
                    workspace_bytes, workspace ? "" : ", NULL");
    const size_t dxb = x_bytes(s, 2), dyb = y_bytes(s, 2), wb = w_bytes(s, 2);
    for (int L = 0; L < 4; ++L)
        if (overlaps(dx, dxb, w[L], wb) || overlaps(workspace, workspace_bytes, w[L], wb))
            return fail(QUAN_ERR_INVALID_ARG, "dx or workspace overlaps a weight tensor");
    if (overlaps(dx, dxb, dy, dyb) || overlaps(workspace, workspace_bytes, dy, dyb) ||
        overlaps(workspace, workspace_bytes, dx, dxb))
        return fail(QUAN_ERR_INVALID_ARG, "dx, dy and workspace must not overlap");
    int num_sms = 0, cc = 0;
    cudaError_t e;
    if (!device_info(&num_sms, &cc, &e)) return cuda_fail(e, "device query");
    cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
    // The input gradient is a forward convolution of dy with the transformed letters
    // (output channels Cin, input channels Cout, padding kh - 1 - pad, stride 1); for a
    // strided forward, of dy with zeros inserted (u, after the letters in the workspace),
    // when the workspace holds it.
    quan::ConvShape t;
    const quan::EpilogueArgs none{nullptr, nullptr, nullptr, nullptr};
    const size_t per = need / 4;
    const void* tw[4];
    for (int L = 0; L < 4; ++L) tw[L] = static_cast<const char*>(workspace) + L * per;
    const int Hu = H + 2 * pad - kh + 1, Wu = W + 2 * pad - kw + 1;
    void* u = static_cast<char*>(workspace) + (need + 255) / 256 * 256;
    const size_t ub = static_cast<size_t>(N) * Hu * Wu * Cout * 2;
    const bool strided = stride > 1;
    const void* src = strided ? u : dy;
    bool tc_ok = kh == kw && pad <= kh - 1 && cc == 103 &&
                 (!strided || workspace_bytes >= (need + 255) / 256 * 256 + ub) &&
                 geometry(&t, N, strided ? Hu : s.Ho, strided ? Wu : s.Wo, Cout, Cin, kh, kw, 1,
                          kh - 1 - pad) == QUAN_OK &&
                 t.Ho == H && t.Wo == W && quan::tc_supported(t, src, tw, dx, none);
    // separable form: the transposed-separable MMA mode (Qin, Qout multiples of 16)
    if (separable) t.sep = 2;
    if (separable && (Cin % 64 != 0 || Cout % 64 != 0)) tc_ok = false;
    const int path = g_path.load();
    if (path == QUAN_PATH_TC && !tc_ok)
        return fail(QUAN_ERR_UNSUPPORTED,
                    "tensor-core input gradient needs a square filter, pad < kh, sm_103, "
                    "Cin/4 and Cout/4 multiples of 16 with 16-byte aligned tensors, and for "
                    "a strided forward quan_qconv2d_bwd_data_workspace_size_ex bytes");
    if (tc_ok && path != QUAN_PATH_SIMT) {
        e = quan::launch_bwd_transform(Cin, Cout, kh, kw, w, !separable, workspace, num_sms,
                                       cs);
        if (e != cudaSuccess) return cuda_fail(e, "bwd_transform launch");
        if (strided) {
            e = quan::launch_bwd_upsample(dy, N, s.Ho, s.Wo, Cout, stride, Hu, Wu, u, num_sms,
                                          cs);
            if (e != cudaSuccess) return cuda_fail(e, "bwd_upsample launch");
        }
        quan::TcOptions opt;
        opt.kappa = g_kappa.load();
        opt.bnq = g_bnq.load();
        opt.max_ctas = g_max_ctas.load();
        opt.mode = separable ? 0 : g_mode.load();
        opt.ws_halo = g_ws_halo.load();
        opt.ws_issuers = g_ws_issuers.load();
        opt.vs_rows = g_vs_rows.load();
        opt.sk_ws = nullptr;
        opt.sk_ws_bytes = 0;
        opt.wait_limit_ns = g_wait_limit.load();
        opt.inject_stall = g_inject.load();
        char err[256] = "";
        e = quan::launch_qconv_tc(t, src, tw, none, dx, opt, num_sms, cs, err, sizeof(err));
        if (err[0] != '\0') return fail(QUAN_ERR_UNSUPPORTED, "%s", err);
        if (e != cudaSuccess) return cuda_fail(e, "qconv_tc launch");
        t_last_path = QUAN_PATH_TC;
        t_last_kernel = quan::last_tc_kernel();
        return QUAN_OK;
    }
    e = quan::launch_bwd_data_simt(s, dy, w, dx, cs);
    if (e != cudaSuccess) return cuda_fail(e, "bwd_data_simt launch");
    t_last_path = QUAN_PATH_SIMT;
    t_last_kernel = separable ? "bwd_data_simt_kernel<sep>" : "bwd_data_simt_kernel";
    return QUAN_OK;
}

// Weight gradients of the pre-epilogue convolution (full form or separable).
quan_status_t run_bwd_weight(const void* x, const void* dy, int N, int H, int W, int Cin,
                             int Cout, int kh, int kw, int stride, int pad, bool separable,
                             float* const dw[4], quan_stream_t stream) {
    if (!x || !dy || !dw[0] || !dw[1] || !dw[2] || !dw[3])
        return fail(QUAN_ERR_INVALID_ARG, "null tensor pointer");
    quan::ConvShape s;
    quan_status_t st = geometry(&s, N, H, W, Cin, Cout, kh, kw, stride, pad);
    if (st != QUAN_OK) return st;
    s.sep = separable ? 1 : 0;
    const size_t xb = x_bytes(s, 2), dyb = y_bytes(s, 2), wb = w_bytes(s, 4);
    for (int L = 0; L < 4; ++L) {
        if (overlaps(dw[L], wb, x, xb) || overlaps(dw[L], wb, dy, dyb))
            return fail(QUAN_ERR_INVALID_ARG, "a weight gradient overlaps x or dy");
        for (int K = 0; K < L; ++K)
            if (overlaps(dw[L], wb, dw[K], wb))
                return fail(QUAN_ERR_INVALID_ARG, "the weight gradients overlap");
        if (reinterpret_cast<uintptr_t>(dw[L]) % 4 != 0)
            return fail(QUAN_ERR_INVALID_ARG, "weight gradients must be 4-byte aligned");
    }
    // tensor cores at stride 1 or 2, both forms (the shape checks need no device)
    const bool tc_shape = quan::bwd_weight_tc_supported(s, x, dy);
    const int path = g_path.load();
    if (path == QUAN_PATH_TC && !tc_shape)
        return fail(QUAN_ERR_UNSUPPORTED,
                    "tensor-core weight gradient needs stride 1 or 2, Cin and Cout multiples of 64 "
                    "(Cout <= 256 or a multiple of 256) and 16-byte aligned x and dy");
    int num_sms = 0, cc = 0;
    cudaError_t e;
    if (!device_info(&num_sms, &cc, &e)) return cuda_fail(e, "device query");
    cudaStream_t cs = reinterpret_cast<cudaStream_t>(stream);
    if (path == QUAN_PATH_TC && cc != 103)
        return fail(QUAN_ERR_UNSUPPORTED, "tensor-core weight gradient needs sm_103 (cc %d)", cc);
    if (tc_shape && cc == 103 && path != QUAN_PATH_SIMT) {
        char err[256] = "";
        e = quan::launch_bwd_weight_tc(s, x, dy, dw, num_sms, g_wait_limit.load(), cs, err,
                                       sizeof(err));
        if (err[0] != '\0') return fail(QUAN_ERR_UNSUPPORTED, "%s", err);
        if (e != cudaSuccess) return cuda_fail(e, "qconv_dw launch");
        t_last_path = QUAN_PATH_TC;
        t_last_kernel = quan::last_tc_kernel();
        return QUAN_OK;
    }
    e = quan::launch_bwd_weight_simt(s, x, dy, dw, num_sms, cs);
    if (e != cudaSuccess) return cuda_fail(e, "bwd_weight_simt launch");
    t_last_path = QUAN_PATH_SIMT;
    t_last_kernel = separable ? "bwd_weight_simt_kernel<sep>" : "bwd_weight_simt_kernel";
    return QUAN_OK;
}

}  // namespace

extern "C" {

quan_status_t quan_qconv2d_fwd(const void* x, const void* wr, const void* wi, const void* wj,
                               const void* wk, const float* bias, const float* iqbn_scale,
                               const float* iqbn_shift, int N, int H, int W, int Cin, int Cout,
                               int kh, int kw, int stride, int pad, int act, void* out,
                               quan_stream_t stream) {
    return run_bf16(x, wr, wi, wj, wk, bias, iqbn_scale, iqbn_shift, N, H, W, Cin, Cout, kh, kw,
                    stride, pad, act, nullptr, out, stream);
}

size_t quan_qconv2d_fwd_workspace_size(void) {
    int num_sms = 0, cc = 0;
    cudaError_t e;
    if (!device_info(&num_sms, &cc, &e)) return 0;
    return quan::tc_split_workspace_bytes(num_sms);
}

quan_status_t quan_qconv2d_fwd_ex(const void* x, const void* wr, const void* wi, const void* wj,
                                  const void* wk, const float* bias, const float* iqbn_scale,
                                  const float* iqbn_shift, int N, int H, int W, int Cin,
                                  int Cout, int kh, int kw, int stride, int pad, int act,
                                  const void* residual, void* workspace, size_t workspace_bytes,
                                  void* out, quan_stream_t stream) {
    if (workspace_bytes > 0 && workspace == nullptr)
        return fail(QUAN_ERR_INVALID_ARG, "workspace is NULL with workspace_bytes > 0");
    if (workspace != nullptr && (reinterpret_cast<uintptr_t>(workspace) & 255u) != 0)
        return fail(QUAN_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
    return run_bf16(x, wr, wi, wj, wk, bias, iqbn_scale, iqbn_shift, N, H, W, Cin, Cout, kh, kw,
                    stride, pad, act, residual, out, stream, false, workspace, workspace_bytes);
}

quan_status_t quan_qconv2d_fwd_shortcut(
    const void* x, const void* wr, const void* wi, const void* wj, const void* wk,
    const float* bias, const float* iqbn_scale, const float* iqbn_shift, int N, int H, int W,
    int Cin, int Cout, int kh, int kw, int stride, int pad, int act, const void* sc_wr,
    const void* sc_wi, const void* sc_wj, const void* sc_wk, const float* sc_bias,
    const float* sc_iqbn_scale, const float* sc_iqbn_shift, int Cout_sc, int sc_act, void* out,
    void* out_sc, quan_stream_t stream) {
    const void* w[4] = {wr, wi, wj, wk};
    const void* wsc[4] = {sc_wr, sc_wi, sc_wj, sc_wk};
    quan::ConvShape s, s1;
    quan_status_t st = validate(&s, x, w, bias, iqbn_scale, iqbn_shift, N, H, W, Cin, Cout, kh,
                                kw, stride, pad, act, nullptr, out, 2);
    if (st != QUAN_OK) return st;
    st = validate(&s1, x, wsc, sc_bias, sc_iqbn_scale, sc_iqbn_shift, N, H, W, Cin, Cout_sc, 1,
                  1, stride, 0, sc_act, nullptr, out_sc, 2);
    if (st != QUAN_OK) return st;
    if (s1.Ho != s.Ho || s1.Wo != s.Wo)
        return fail(QUAN_ERR_INVALID_ARG,
                    "the 1x1 shortcut's output (%dx%d) differs from the convolution's (%dx%d)",
                    s1.Ho, s1.Wo, s.Ho, s.Wo);
    if (overlaps(out, y_bytes(s, 2), out_sc, y_bytes(s1, 2)))
        return fail(QUAN_ERR_INVALID_ARG, "out and out_sc overlap");
    const size_t wb = w_bytes(s1, 2);
    for (int L = 0; L < 4; ++L)
        if (overlaps(out, y_bytes(s, 2), wsc[L], wb))
            return fail(QUAN_ERR_INVALID_ARG, "out overlaps a shortcut weight tensor");
    int num_sms = 0, cc = 0;
    cudaError_t e;
    if (!device_info(&num_sms, &cc, &e)) return cuda_fail(e, "device query");
    const quan::EpilogueArgs ep{bias, iqbn_scale, iqbn_shift, nullptr};
    const quan::EpilogueArgs ep_sc{sc_bias, sc_iqbn_scale, sc_iqbn_shift, nullptr};
    quan::TcOptions opt;
    opt.kappa = g_kappa.load();
    opt.bnq = g_bnq.load();
    opt.max_ctas = g_max_ctas.load();
    opt.mode = g_mode.load();
    opt.ws_halo = g_ws_halo.load();
    opt.ws_issuers = g_ws_issuers.load();
    opt.vs_rows = g_vs_rows.load();
    opt.sk_ws = nullptr;
    opt.sk_ws_bytes = 0;
    opt.wait_limit_ns = g_wait_limit.load();
    opt.inject_stall = g_inject.load();
    if (g_path.load() != QUAN_PATH_SIMT && cc == 103 &&
        quan::tc_shortcut_supported(s, x, w, out, ep, wsc, s1.Qout, ep_sc, out_sc, opt)) {
        char err[256] = "";
        e = quan::launch_qconv_tc_shortcut(s, x, w, ep, out, wsc, s1.Qout, sc_act, ep_sc, out_sc,
                                           opt, num_sms, reinterpret_cast<cudaStream_t>(stream),
                                           err, sizeof(err));
        if (err[0] != '\0') return fail(QUAN_ERR_UNSUPPORTED, "%s", err);
        if (e != cudaSuccess) return cuda_fail(e, "qconv_tc shortcut launch");
        t_last_path = QUAN_PATH_TC;
        t_last_kernel = quan::last_tc_kernel();
        return QUAN_OK;
    }
    // no fused form for these shapes, path or device: the two layers as separate calls
    st = run_bf16(x, wr, wi, wj, wk, bias, iqbn_scale, iqbn_shift, N, H, W, Cin, Cout, kh, kw,
                  stride, pad, act, nullptr, out, stream);
    if (st != QUAN_OK) return st;
    return run_bf16(x, sc_wr, sc_wi, sc_wj, sc_wk, sc_bias, sc_iqbn_scale, sc_iqbn_shift, N, H,
                    W, Cin, Cout_sc, 1, 1, stride, 0, sc_act, nullptr, out_sc, stream);
}

quan_status_t quan_qconv2d_fwd_res(const void* x, const void* wr, const void* wi, const void* wj,
                                   const void* wk, const float* bias, const float* iqbn_scale,
                                   const float* iqbn_shift, int N, int H, int W, int Cin,
                                   int Cout, int kh, int kw, int stride, int pad, int act,
                                   const void* residual, void* out, quan_stream_t stream) {
    if (!residual) return fail(QUAN_ERR_INVALID_ARG, "residual is NULL");
    return run_bf16(x, wr, wi, wj, wk, bias, iqbn_scale, iqbn_shift, N, H, W, Cin, Cout, kh, kw,
                    stride, pad, act, residual, out, stream);
}

quan_status_t quan_qconv2d_sep_fwd(const void* x, const void* wr, const void* wi,
                                   const void* wj, const void* wk, const float* bias,
                                   const float* iqbn_scale, const float* iqbn_shift, int N, int H,
                                   int W, int Cin, int Cout, int kh, int kw, int stride, int pad,
                                   int act, void* out, quan_stream_t stream) {
    return run_bf16(x, wr, wi, wj, wk, bias, iqbn_scale, iqbn_shift, N, H, W, Cin, Cout, kh, kw,
                    stride, pad, act, nullptr, out, stream, true);
}

quan_status_t quan_qconv2d_fwd_f32(const float* x, const float* wr, const float* wi,
                                   const float* wj, const float* wk, const float* bias,
                                   const float* iqbn_scale, const float* iqbn_shift, int N, int H,
                                   int W, int Cin, int Cout, int kh, int kw, int stride, int pad,
                                   int act, float* out, quan_stream_t stream) {
    const void* w[4] = {wr, wi, wj, wk};
    quan::ConvShape s;
    quan_status_t st = validate(&s, x, w, bias, iqbn_scale, iqbn_shift, N, H, W, Cin, Cout, kh,
                                kw, stride, pad, act, nullptr, out, 4);
    if (st != QUAN_OK) return st;
    if (g_path.load() == QUAN_PATH_TC)
        return fail(QUAN_ERR_UNSUPPORTED, "fp32 convolution runs on CUDA cores only");
    const quan::EpilogueArgs ep{bias, iqbn_scale, iqbn_shift, nullptr};
    cudaError_t e = quan::launch_qconv_simt_f32(s, x, w, ep, out,
                                                reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "qconv_simt_f32 launch");
    t_last_path = QUAN_PATH_SIMT;
    t_last_kernel = "qconv_simt_kernel<f32>";
    return QUAN_OK;
}

quan_status_t quan_poincare_fwd(const float* rgb, long long npix, void* out,
                                quan_stream_t stream) {
    if (npix < 0) return fail(QUAN_ERR_INVALID_ARG, "npix must be >= 0");
    if (npix == 0) return QUAN_OK;
    if (!rgb || !out) return fail(QUAN_ERR_INVALID_ARG, "null tensor pointer");
    if (npix > (1LL << 40)) return fail(QUAN_ERR_UNSUPPORTED, "tensor too large");
    if (reinterpret_cast<uintptr_t>(rgb) % 4 != 0 || reinterpret_cast<uintptr_t>(out) % 2 != 0)
        return fail(QUAN_ERR_INVALID_ARG, "rgb must be 4-byte and out 2-byte aligned");
    if (overlaps(rgb, static_cast<size_t>(npix) * 12, out, static_cast<size_t>(npix) * 8))
        return fail(QUAN_ERR_INVALID_ARG, "out overlaps rgb");
    int num_sms = 0, cc = 0;
    cudaError_t e;
    if (!device_info(&num_sms, &cc, &e)) return cuda_fail(e, "device query");
    e = quan::launch_poincare(rgb, npix, out, num_sms, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "poincare launch");
    return QUAN_OK;
}

size_t quan_qconv2d_bwd_data_workspace_size(int Cin, int Cout, int kh, int kw) {
    if (Cin < 4 || Cout < 4 || kh < 1 || kw < 1 || Cin % 4 || Cout % 4) return 0;
    return quan::bwd_data_workspace_bytes(Cin, Cout, kh, kw);
}

size_t quan_qconv2d_bwd_data_workspace_size_ex(int N, int H, int W, int Cin, int Cout, int kh,
                                               int kw, int stride, int pad) {
    quan::ConvShape s;
    if (geometry(&s, N, H, W, Cin, Cout, kh, kw, stride, pad) != QUAN_OK) return 0;
    const size_t letters = quan::bwd_data_workspace_bytes(Cin, Cout, kh, kw);
    if (stride == 1) return letters;
    const size_t Hu = static_cast<size_t>(H) + 2 * pad - kh + 1;
    const size_t Wu = static_cast<size_t>(W) + 2 * pad - kw + 1;
    return (letters + 255) / 256 * 256 + static_cast<size_t>(N) * Hu * Wu * Cout * 2;
}

quan_status_t quan_qconv2d_bwd_data(const void* dy, const void* wr, const void* wi,
                                    const void* wj, const void* wk, int N, int H, int W, int Cin,
                                    int Cout, int kh, int kw, int stride, int pad,
                                    void* workspace, size_t workspace_bytes, void* dx,
                                    quan_stream_t stream) {
    const void* w[4] = {wr, wi, wj, wk};
    return run_bwd_data(dy, w, N, H, W, Cin, Cout, kh, kw, stride, pad, false, workspace,
                        workspace_bytes, dx, stream);
}

quan_status_t quan_qconv2d_bwd_data_static(const void* dy, const void* wr, const void* wi,
                                           const void* wj, const void* wk, int N, int H, int W,
                                           int Cin, int Cout, int kh, int kw, int stride,
                                           int pad, void* dx, quan_stream_t stream) {
    quan::ConvShape s;
    quan_status_t st = geometry(&s, N, H, W, Cin, Cout, kh, kw, stride, pad);
    if (st != QUAN_OK) return st;
    if (!dy || !wr || !wi || !wj || !wk || !dx)
        return fail(QUAN_ERR_INVALID_ARG, "null tensor pointer");
    const size_t need = quan::bwd_data_workspace_bytes(Cin, Cout, kh, kw);
    if (need > quan::BWD_STATIC_SCRATCH_BYTES)
        return fail(QUAN_ERR_UNSUPPORTED,
                    "the transformed letters (%zu bytes) exceed the %zu-byte static scratch; "
                    "use quan_qconv2d_bwd_data with a workspace",
                    need, quan::BWD_STATIC_SCRATCH_BYTES);
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "device query");
    if (dev < 0 || dev >= kMaxDevices) return cuda_fail(cudaErrorInvalidDevice, "device query");
    void* scratch = nullptr;
    {
        std::lock_guard<std::mutex> lk(g_dev_mu);
        if (!g_static_scratch[dev]) {
            // once per device, with that device current
            void* p = nullptr;
            e = quan::bwd_static_scratch_address(&p);
            if (e != cudaSuccess || !p)
                return cuda_fail(e != cudaSuccess ? e : cudaErrorInvalidSymbol,
                                 "static scratch address");
            g_static_scratch[dev] = p;
        }
        scratch = g_static_scratch[dev];
    }
    const void* w[4] = {wr, wi, wj, wk};
    return run_bwd_data(dy, w, N, H, W, Cin, Cout, kh, kw, stride, pad, false, scratch,
                        quan::BWD_STATIC_SCRATCH_BYTES, dx, stream);
}

quan_status_t quan_qconv2d_sep_bwd_data(const void* dy, const void* wr, const void* wi,
                                        const void* wj, const void* wk, int N, int H, int W,
                                        int Cin, int Cout, int kh, int kw, int stride, int pad,
                                        void* workspace, size_t workspace_bytes, void* dx,
                                        quan_stream_t stream) {
    const void* w[4] = {wr, wi, wj, wk};
    return run_bwd_data(dy, w, N, H, W, Cin, Cout, kh, kw, stride, pad, true, workspace,
                        workspace_bytes, dx, stream);
}

quan_status_t quan_qconv2d_bwd_weight(const void* x, const void* dy, int N, int H, int W,
                                      int Cin, int Cout, int kh, int kw, int stride, int pad,
                                      float* dwr, float* dwi, float* dwj, float* dwk,
                                      quan_stream_t stream) {
    float* const dw[4] = {dwr, dwi, dwj, dwk};
    return run_bwd_weight(x, dy, N, H, W, Cin, Cout, kh, kw, stride, pad, false, dw, stream);
}

quan_status_t quan_qconv2d_sep_bwd_weight(const void* x, const void* dy, int N, int H, int W,
                                          int Cin, int Cout, int kh, int kw, int stride,
                                          int pad, float* dwr, float* dwi, float* dwj,
                                          float* dwk, quan_stream_t stream) {
    float* const dw[4] = {dwr, dwi, dwj, dwk};
    return run_bwd_weight(x, dy, N, H, W, Cin, Cout, kh, kw, stride, pad, true, dw, stream);
}

size_t quan_iqbn_batch_stats_workspace_size(int C) { return quan::iqbn_stats_workspace_bytes(C); }

quan_status_t quan_iqbn_batch_stats(const void* x, long long npix, int C, void* workspace,
                                    size_t workspace_bytes, float* mean, float* var,
                                    quan_stream_t stream) {
    if (!x || !mean || !var) return fail(QUAN_ERR_INVALID_ARG, "null tensor pointer");
    if (npix < 1 || C < 1) return fail(QUAN_ERR_INVALID_ARG, "npix and C must be >= 1");
    if (npix > (1LL << 40) / C) return fail(QUAN_ERR_UNSUPPORTED, "tensor too large");
    const size_t need = quan::iqbn_stats_workspace_bytes(C);
    if (!workspace || workspace_bytes < need)
        return fail(QUAN_ERR_INVALID_ARG, "workspace must hold %zu bytes (got %zu%s)", need,
                    workspace_bytes, workspace ? "" : ", NULL");
    if (reinterpret_cast<uintptr_t>(x) % 2 != 0 || reinterpret_cast<uintptr_t>(mean) % 4 != 0 ||
        reinterpret_cast<uintptr_t>(var) % 4 != 0 ||
        reinterpret_cast<uintptr_t>(workspace) % 4 != 0)
        return fail(QUAN_ERR_INVALID_ARG,
                    "x must be 2-byte, mean, var and the workspace 4-byte aligned");
    const size_t xb = static_cast<size_t>(npix) * C * 2, vb = static_cast<size_t>(C) * 4;
    if (overlaps(mean, vb, var, vb) || overlaps(mean, vb, x, xb) || overlaps(var, vb, x, xb) ||
        overlaps(workspace, need, x, xb) || overlaps(workspace, need, mean, vb) ||
        overlaps(workspace, need, var, vb))
        return fail(QUAN_ERR_INVALID_ARG, "mean, var, the workspace and x must not overlap");
    if (!quan::iqbn_supported(C, x, x))
        return fail(QUAN_ERR_UNSUPPORTED,
                    "C=%d: needs C <= 256, or C a multiple of 8 up to 2048 with x 16-byte "
                    "aligned", C);
    int num_sms = 0, cc = 0;
    cudaError_t e;
    if (!device_info(&num_sms, &cc, &e)) return cuda_fail(e, "device query");
    e = quan::launch_iqbn_stats(x, npix, C, workspace, mean, var, num_sms,
                                reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "iqbn_stats launch");
    return QUAN_OK;
}

quan_status_t quan_iqbn_train_fwd(const void* x, long long npix, int C, const float* mean,
                                  const float* var, const float* gamma, const float* beta,
                                  float eps, int act, void* out, quan_stream_t stream) {
    if (!x || !mean || !var || !out) return fail(QUAN_ERR_INVALID_ARG, "null tensor pointer");
    if (npix < 1 || C < 1) return fail(QUAN_ERR_INVALID_ARG, "npix and C must be >= 1");
    if (!(eps >= 0.0f) || !std::isfinite(eps))
        return fail(QUAN_ERR_INVALID_ARG, "eps must be finite and >= 0");
    if (act < QUAN_ACT_NONE || act > QUAN_ACT_SILU)
        return fail(QUAN_ERR_INVALID_ARG, "unknown activation %d", act);
    if (npix > (1LL << 40) / C) return fail(QUAN_ERR_UNSUPPORTED, "tensor too large");
    if (reinterpret_cast<uintptr_t>(x) % 2 != 0 || reinterpret_cast<uintptr_t>(out) % 2 != 0)
        return fail(QUAN_ERR_INVALID_ARG, "x and out must be 2-byte aligned");
    const size_t xb = static_cast<size_t>(npix) * C * 2, vb = static_cast<size_t>(C) * 4;
    if (out != x && overlaps(out, xb, x, xb))
        return fail(QUAN_ERR_INVALID_ARG, "out must be x itself or not overlap it");
    if (overlaps(out, xb, mean, vb) || overlaps(out, xb, var, vb) ||
        overlaps(out, xb, gamma, vb) || overlaps(out, xb, beta, vb))
        return fail(QUAN_ERR_INVALID_ARG, "out overlaps a per-channel vector");
    if (!quan::iqbn_supported(C, x, out))
        return fail(QUAN_ERR_UNSUPPORTED,
                    "C=%d: needs C <= 256, or C a multiple of 8 up to 2048 with x and out "
                    "16-byte aligned", C);
    int num_sms = 0, cc = 0;
    cudaError_t e;
    if (!device_info(&num_sms, &cc, &e)) return cuda_fail(e, "device query");
    e = quan::launch_iqbn_apply(x, npix, C, mean, var, gamma, beta, eps, act, out, num_sms,
                                reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "iqbn_apply launch");
    return QUAN_OK;
}

size_t quan_qconv2d_maxpool_workspace_size(int N, int H, int W, int Cout, int kh, int kw,
                                           int stride, int pad) {
    (void)N; (void)H; (void)W; (void)Cout; (void)kh; (void)kw; (void)stride; (void)pad;
    return 0;  // one kernel writes the pooled tensor directly
}

quan_status_t quan_qconv2d_maxpool_fwd(const void* x, const void* wr, const void* wi,
                                       const void* wj, const void* wk, const float* bias,
                                       const float* iqbn_scale, const float* iqbn_shift, int N,
                                       int H, int W, int Cin, int Cout, int kh, int kw,
                                       int stride, int pad, int act, void* workspace,
                                       size_t workspace_bytes, void* out,
                                       quan_stream_t stream) {
    (void)workspace;
    (void)workspace_bytes;
    const void* w[4] = {wr, wi, wj, wk};
    if (!x || !wr || !wi || !wj || !wk || !out)
        return fail(QUAN_ERR_INVALID_ARG, "null tensor pointer");
    quan::ConvShape s;
    quan_status_t st = geometry(&s, N, H, W, Cin, Cout, kh, kw, stride, pad);
    if (st != QUAN_OK) return st;
    if ((iqbn_scale == nullptr) != (iqbn_shift == nullptr))
        return fail(QUAN_ERR_INVALID_ARG, "iqbn_scale and iqbn_shift must both be given or both NULL");
    if (act < QUAN_ACT_NONE || act > QUAN_ACT_SILU)
        return fail(QUAN_ERR_INVALID_ARG, "unknown activation %d", act);
    s.act = act;
    const int pw = (s.Wo - 1) / 2 + 1, ph = (s.Ho - 1) / 2 + 1;
    const size_t ob = static_cast<size_t>(N) * ph * pw * Cout * 2;
    // the written tensor against every input
    const size_t xb = x_bytes(s, 2), wb = w_bytes(s, 2), vb = static_cast<size_t>(Cout) * 4;
    if (overlaps(out, ob, x, xb) || overlaps(out, ob, wr, wb) || overlaps(out, ob, wi, wb) ||
        overlaps(out, ob, wj, wb) || overlaps(out, ob, wk, wb) || overlaps(out, ob, bias, vb) ||
        overlaps(out, ob, iqbn_scale, vb) || overlaps(out, ob, iqbn_shift, vb))
        return fail(QUAN_ERR_INVALID_ARG, "out overlaps an input");
    int num_sms = 0, cc = 0;
    cudaError_t e;
    if (!device_info(&num_sms, &cc, &e)) return cuda_fail(e, "device query");
    const quan::EpilogueArgs ep{bias, iqbn_scale, iqbn_shift, nullptr};
    if (cc != 103 || !quan::tc_stem_pool_supported(s, x, w, out, ep))
        return fail(QUAN_ERR_UNSUPPORTED,
                    "the fused stem pooling needs sm_103, Cin = 4, Cout = 64, stride 2, an even "
                    "W, Wo <= 128, (kh + 2) * ceil-even((kw + pad %% 2) / 2) <= 36 and 16-byte "
                    "aligned tensors");
    quan::TcOptions opt;
    opt.kappa = 0;
    opt.bnq = 0;
    opt.max_ctas = g_max_ctas.load();
    opt.mode = 0;
    opt.ws_halo = 1;
    opt.ws_issuers = 0;
    opt.vs_rows = 0;
    opt.sk_ws = nullptr;
    opt.sk_ws_bytes = 0;
    opt.wait_limit_ns = g_wait_limit.load();
    opt.inject_stall = g_inject.load();
    char err[256] = "";
    e = quan::launch_qconv_stem_pool(s, x, w, ep, out, opt, num_sms,
                                     reinterpret_cast<cudaStream_t>(stream), err, sizeof(err));
    if (err[0] != '\0') return fail(QUAN_ERR_UNSUPPORTED, "%s", err);
    if (e != cudaSuccess) return cuda_fail(e, "qconv_stem_pool launch");
    t_last_path = QUAN_PATH_TC;
    t_last_kernel = quan::last_tc_kernel();
    return QUAN_OK;
}

quan_status_t quan_qconv2d_maxpool_rgb_fwd(const float* rgb, const void* wr, const void* wi,
                                           const void* wj, const void* wk, const float* bias,
                                           const float* iqbn_scale, const float* iqbn_shift,
                                           int N, int H, int W, int Cout, int kh, int kw,
                                           int stride, int pad, int act, void* out,
                                           quan_stream_t stream) {
    const void* w[4] = {wr, wi, wj, wk};
    if (!rgb || !wr || !wi || !wj || !wk || !out)
        return fail(QUAN_ERR_INVALID_ARG, "null tensor pointer");
    quan::ConvShape s;
    quan_status_t st = geometry(&s, N, H, W, 4, Cout, kh, kw, stride, pad);
    if (st != QUAN_OK) return st;
    if ((iqbn_scale == nullptr) != (iqbn_shift == nullptr))
        return fail(QUAN_ERR_INVALID_ARG, "iqbn_scale and iqbn_shift must both be given or both NULL");
    if (act < QUAN_ACT_NONE || act > QUAN_ACT_SILU)
        return fail(QUAN_ERR_INVALID_ARG, "unknown activation %d", act);
    s.act = act;
    const int pw = (s.Wo - 1) / 2 + 1, ph = (s.Ho - 1) / 2 + 1;
    const size_t ob = static_cast<size_t>(N) * ph * pw * Cout * 2;
    const size_t rb = static_cast<size_t>(N) * H * W * 12, wb = w_bytes(s, 2);
    const size_t vb = static_cast<size_t>(Cout) * 4;
    if (overlaps(out, ob, rgb, rb) || overlaps(out, ob, wr, wb) || overlaps(out, ob, wi, wb) ||
        overlaps(out, ob, wj, wb) || overlaps(out, ob, wk, wb) || overlaps(out, ob, bias, vb) ||
        overlaps(out, ob, iqbn_scale, vb) || overlaps(out, ob, iqbn_shift, vb))
        return fail(QUAN_ERR_INVALID_ARG, "out overlaps an input");
    int num_sms = 0, cc = 0;
    cudaError_t e;
    if (!device_info(&num_sms, &cc, &e)) return cuda_fail(e, "device query");
    const quan::EpilogueArgs ep{bias, iqbn_scale, iqbn_shift, nullptr};
    if (cc != 103 || !quan::tc_stem_pool_rgb_supported(s, rgb, w, out, ep))
        return fail(QUAN_ERR_UNSUPPORTED,
                    "the RGB stem pooling needs sm_103, Cout = 64, stride 2, W a multiple of "
                    "32, Wo <= 128, the stem's filter limits and 16-byte aligned tensors");
    quan::TcOptions opt;
    opt.kappa = 0;
    opt.bnq = 0;
    opt.max_ctas = g_max_ctas.load();
    opt.mode = 0;
    opt.ws_halo = 1;
    opt.ws_issuers = 0;
    opt.vs_rows = 0;
    opt.sk_ws = nullptr;
    opt.sk_ws_bytes = 0;
    opt.wait_limit_ns = g_wait_limit.load();
    opt.inject_stall = g_inject.load();
    char err[256] = "";
    e = quan::launch_qconv_stem_pool_rgb(s, rgb, w, ep, out, opt, num_sms,
                                         reinterpret_cast<cudaStream_t>(stream), err,
                                         sizeof(err));
    if (err[0] != '\0') return fail(QUAN_ERR_UNSUPPORTED, "%s", err);
    if (e != cudaSuccess) return cuda_fail(e, "qconv_stem_pool launch");
    t_last_path = QUAN_PATH_TC;
    t_last_kernel = quan::last_tc_kernel();
    return QUAN_OK;
}

quan_status_t quan_maxpool2d_fwd(const void* x, int N, int H, int W, int C, int k, int stride,
                                 int pad, void* out, quan_stream_t stream) {
    if (!x || !out) return fail(QUAN_ERR_INVALID_ARG, "null tensor pointer");
    if (N < 1 || H < 1 || W < 1 || C < 1 || k < 1 || stride < 1 || pad < 0)
        return fail(QUAN_ERR_INVALID_ARG, "sizes must be positive and pad >= 0");
    if (2 * pad > k)
        return fail(QUAN_ERR_INVALID_ARG, "pad=%d must be at most k/2 (k=%d)", pad, k);
    if (H + 2 * pad < k || W + 2 * pad < k)
        return fail(QUAN_ERR_INVALID_ARG, "window larger than the padded input");
    const long long Ho = (H + 2LL * pad - k) / stride + 1, Wo = (W + 2LL * pad - k) / stride + 1;
    const size_t xb = static_cast<size_t>(N) * H * W * C * 2;
    const size_t yb = static_cast<size_t>(N) * Ho * Wo * C * 2;
    if (overlaps(x, xb, out, yb)) return fail(QUAN_ERR_INVALID_ARG, "out overlaps x");
    int num_sms = 0, cc = 0;
    cudaError_t e;
    if (!device_info(&num_sms, &cc, &e)) return cuda_fail(e, "device query");
    e = quan::launch_maxpool_bf16(x, N, H, W, C, k, stride, pad, out, num_sms,
                                  reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "maxpool launch");
    return QUAN_OK;
}

quan_status_t quan_set_path(int path) {
    if (path < QUAN_PATH_AUTO || path > QUAN_PATH_SIMT)
        return fail(QUAN_ERR_INVALID_ARG, "unknown path %d", path);
    g_path.store(path);
    return QUAN_OK;
}

int quan_last_path(void) { return t_last_path; }

const char* quan_last_kernel(void) { return t_last_kernel; }

quan_status_t quan_set_tc_tiles(int kappa, int bnq, int max_ctas, int mode) {
    auto okv = [](int v) { return v == 0 || v == 16 || v == 32 || v == 64; };
    if (!okv(kappa) || !okv(bnq) || max_ctas < 0 || mode < 0 || mode > 7)
        return fail(QUAN_ERR_INVALID_ARG,
                    "kappa and bnq must be 0, 16, 32 or 64; max_ctas >= 0; mode 0 to 7");
    g_kappa.store(kappa);
    g_bnq.store(bnq);
    g_max_ctas.store(max_ctas);
    g_mode.store(mode);
    return QUAN_OK;
}

quan_status_t quan_set_tc_halo(int enable) {
    g_ws_halo.store(enable ? 1 : 0);
    return QUAN_OK;
}

quan_status_t quan_set_tc_issuers(int issuers) {
    if (issuers != 0 && issuers != 2 && issuers != 3)
        return fail(QUAN_ERR_INVALID_ARG, "issuers must be 0 (automatic), 2 or 3");
    g_ws_issuers.store(issuers);
    return QUAN_OK;
}

quan_status_t quan_set_tc_band_rows(int rows) {
    if (rows < 0 || rows > 4)
        return fail(QUAN_ERR_INVALID_ARG, "band rows must be 0 (automatic) or 1 to 4");
    g_vs_rows.store(rows);
    return QUAN_OK;
}

quan_status_t quan_set_wait_limit_ns(unsigned long long ns) {
    g_wait_limit.store(ns == 0 ? 2000000000ull : ns);
    return QUAN_OK;
}

quan_status_t quan_set_fault_injection(int enable) {
    g_inject.store(enable ? 1 : 0);
    return QUAN_OK;
}

quan_status_t quan_device_status(quan_stream_t stream, unsigned int* bits) {
    unsigned v = 0;
    cudaError_t e = quan::read_and_clear_status(&v, reinterpret_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "device status");
    if (bits) *bits = v;
    if (v) return fail(QUAN_ERR_DEVICE_TIMEOUT, "kernel wait timed out (status bits 0x%x)", v);
    return QUAN_OK;
}

const char* quan_status_string(quan_status_t status) {
    switch (status) {
        case QUAN_OK: return "QUAN_OK";
        case QUAN_ERR_INVALID_ARG: return "QUAN_ERR_INVALID_ARG";
        case QUAN_ERR_UNSUPPORTED: return "QUAN_ERR_UNSUPPORTED";
        case QUAN_ERR_CUDA: return "QUAN_ERR_CUDA";
        case QUAN_ERR_DEVICE_TIMEOUT: return "QUAN_ERR_DEVICE_TIMEOUT";
    }
    return "QUAN_ERR_UNKNOWN";
}

const char* quan_last_error_message(void) { return t_errmsg; }

int quan_version(void) { return 100; }

}  // extern "C"
