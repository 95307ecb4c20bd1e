// qconv_bwd.cu -- gradients of the quaternion convolution before its epilogue, given
// dy = dL/dy for y = the convolution's accumulator (bias, IQBN and activation excluded).
//
// Full Hamilton form (Eq. 5): the Jacobians of the Hamilton product (Eq. 3) give, for
// every tap and channel pair,
//   dL/dX = conj(W) (x) dy,     dL/dW = dy (x) conj(X),
// conj(W) = (W_r, -W_i, -W_j, -W_k).  So
//   * the input gradient is itself a quaternion convolution: of dy, with the letters
//     conjugated, their channel axes swapped and the filter rotated by 180 degrees, padding
//     kh - 1 - pad, stride 1 (for a stride-1 forward).  bwd_transform_kernel writes those
//     letters into a caller workspace and the forward tensor-core kernels run the rest.
//     A stride-s forward's input gradient is the same stride-1 convolution of dy with
//     s - 1 zero rows and columns inserted between its pixels (bwd_upsample_kernel, into
//     the workspace after the letters), when the caller's workspace holds it; otherwise
//     the direct CUDA-core kernel below runs;
//   * the weight gradient is a reduction over output pixels, done on CUDA cores: every
//     thread owns one (co, tap, ci) quaternion of dW for a chunk of pixels and adds its
//     fp32 partial sum to the zeroed output with atomicAdd.
// Separable form (Eq. 7): Eq. 8-10 -- the output gradients are first mixed by the matrix M
// of Eq. 9 (g_p = sum_m M[p][m] dy_m, M transposed equal to Eq. 7's sign table), then
// dL/dx_p is the transposed convolution of g_p with W_p alone and dL/dW_p the correlation
// of g_p with x_p alone.  On the tensor cores (stride 1) the input gradient is one
// convolution of dy whose block (q, p) is M[q][p] W'_q (W' the letters transposed and
// rotated, not conjugated): the forward kernel's transposed-separable mode.
#include <cuda_bf16.h>

#include "internal.h"

namespace quan {
namespace {

__device__ __forceinline__ float bf(const __nv_bfloat16* p) { return __bfloat162float(*p); }

// g = M dy for one output channel, M of Eq. 9 (rows p, columns m):
//   [ 1  1  1  1 ]
//   [-1  1 -1  1 ]
//   [-1  1  1 -1 ]
//   [-1 -1  1  1 ]
__device__ __forceinline__ void mix_eq9(float dr, float di, float dj, float dk, float& gr,
                                        float& gi, float& gj, float& gk) {
    gr = dr + di + dj + dk;
    gi = -dr + di - dj + dk;
    gj = -dr + di + dj - dk;
    gk = -dr - di + dj + dk;
}

// out_L[ci][dh][dw][co] = s_L * W_L[co][kh-1-dh][kw-1-dw][ci], s = (+1, -1, -1, -1) when
// conj, else +1.  Its output is the next kernel's weight operand, which the forward
// tensor-core kernels read before their dependency wait: this kernel does not trigger its
// dependents early, so the next one starts only once it has completed.
__global__ void __launch_bounds__(256) bwd_transform_kernel(
    int Qin, int Qout, int kh, int kw, int conj, const __nv_bfloat16* __restrict__ wr,
    const __nv_bfloat16* __restrict__ wi, const __nv_bfloat16* __restrict__ wj,
    const __nv_bfloat16* __restrict__ wk, __nv_bfloat16* __restrict__ out) {
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const long long per = static_cast<long long>(Qin) * kh * kw * Qout;
    const __nv_bfloat16* w[4] = {wr, wi, wj, wk};
    for (long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
         i < 4 * per; i += static_cast<long long>(gridDim.x) * blockDim.x) {
        const int L = static_cast<int>(i / per);
        long long r = i - L * per;
        const int co = static_cast<int>(r % Qout);
        r /= Qout;
        const int dw = static_cast<int>(r % kw);
        r /= kw;
        const int dh = static_cast<int>(r % kh);
        const int ci = static_cast<int>(r / kh);
        const long long src =
            ((static_cast<long long>(co) * kh + (kh - 1 - dh)) * kw + (kw - 1 - dw)) * Qin + ci;
        const __nv_bfloat16 v = w[L][src];
        out[i] = (L == 0 || !conj) ? v : __hneg(v);
    }
}

// dx for one (pixel, input quaternion channel), any stride and padding: the sum over taps
// and output channels of conj(W) (x) dy (full form), or of W_p g_p per component p
// (separable form, g = M dy).
template <bool SEP>
__global__ void __launch_bounds__(256) bwd_data_simt_kernel(
    ConvShape s, const __nv_bfloat16* __restrict__ dy, const __nv_bfloat16* __restrict__ wr,
    const __nv_bfloat16* __restrict__ wi, const __nv_bfloat16* __restrict__ wj,
    const __nv_bfloat16* __restrict__ wk, __nv_bfloat16* __restrict__ dx) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const long long total = static_cast<long long>(s.N) * s.H * s.W * s.Qin;
    const long long idx = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= total) return;
    const int ci = static_cast<int>(idx % s.Qin);
    const long long pix = idx / s.Qin;
    const int w = static_cast<int>(pix % s.W);
    const int h = static_cast<int>((pix / s.W) % s.H);
    const int n = static_cast<int>(pix / (static_cast<long long>(s.W) * s.H));
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
    for (int dh = 0; dh < s.kh; ++dh) {
        const int th = h + s.pad - dh;  // ho * stride
        if (th < 0 || th % s.stride != 0) continue;
        const int ho = th / s.stride;
        if (ho >= s.Ho) continue;
        for (int dw = 0; dw < s.kw; ++dw) {
            const int tw = w + s.pad - dw;
            if (tw < 0 || tw % s.stride != 0) continue;
            const int wo = tw / s.stride;
            if (wo >= s.Wo) continue;
            const __nv_bfloat16* g = dy + ((static_cast<long long>(n) * s.Ho + ho) * s.Wo + wo) *
                                              s.Cout;
            for (int co = 0; co < s.Qout; ++co) {
                const long long widx = ((static_cast<long long>(co) * s.kh + dh) * s.kw + dw) *
                                           s.Qin + ci;
                const float dr = bf(g + co), di = bf(g + s.Qout + co);
                const float dj = bf(g + 2 * s.Qout + co), dk = bf(g + 3 * s.Qout + co);
                if constexpr (SEP) {
                    float gr, gi, gj, gk;
                    mix_eq9(dr, di, dj, dk, gr, gi, gj, gk);
                    a0 += bf(wr + widx) * gr;
                    a1 += bf(wi + widx) * gi;
                    a2 += bf(wj + widx) * gj;
                    a3 += bf(wk + widx) * gk;
                } else {
                    // conj(W) = (a, -b, -c, -d); conj(W) (x) dy by Eq. 3
                    const float a = bf(wr + widx), b = -bf(wi + widx);
                    const float c = -bf(wj + widx), d = -bf(wk + widx);
                    a0 += a * dr - b * di - c * dj - d * dk;
                    a1 += a * di + b * dr + c * dk - d * dj;
                    a2 += a * dj - b * dk + c * dr + d * di;
                    a3 += a * dk + b * dj - c * di + d * dr;
                }
            }
        }
    }
    __nv_bfloat16* o = dx + pix * s.Cin;
    o[ci] = __float2bfloat16_rn(a0);
    o[s.Qin + ci] = __float2bfloat16_rn(a1);
    o[2 * s.Qin + ci] = __float2bfloat16_rn(a2);
    o[3 * s.Qin + ci] = __float2bfloat16_rn(a3);
}

// dW for one (co, tap, ci) quaternion over the output pixels of chunk blockIdx.y: the sum
// of dy (x) conj(X) (full form), or of g_p x_p per component p (separable form, g = M dy),
// added to the fp32 outputs.
template <bool SEP>
__global__ void __launch_bounds__(256) bwd_weight_simt_kernel(
    ConvShape s, const __nv_bfloat16* __restrict__ x, const __nv_bfloat16* __restrict__ dy,
    long long chunk, float* __restrict__ dwr, float* __restrict__ dwi, float* __restrict__ dwj,
    float* __restrict__ dwk) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const int taps = s.kh * s.kw;
    const long long outs = static_cast<long long>(s.Qout) * taps * s.Qin;
    const long long o = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (o >= outs) return;
    // o = (co * taps + tap) * Qin + ci, the layout of the letter tensors
    const int ci = static_cast<int>(o % s.Qin);
    const int tap = static_cast<int>((o / s.Qin) % taps);
    const int co = static_cast<int>(o / (static_cast<long long>(s.Qin) * taps));
    const int dh = tap / s.kw, dw = tap - (tap / s.kw) * s.kw;
    const long long p0 = blockIdx.y * chunk;
    long long p1 = p0 + chunk;
    if (p1 > s.M) p1 = s.M;
    float a0 = 0.f, a1 = 0.f, a2 = 0.f, a3 = 0.f;
    for (long long p = p0; p < p1; ++p) {
        const int wo = static_cast<int>(p % s.Wo);
        const int ho = static_cast<int>((p / s.Wo) % s.Ho);
        const int n = static_cast<int>(p / (static_cast<long long>(s.Wo) * s.Ho));
        const int h = ho * s.stride - s.pad + dh, w = wo * s.stride - s.pad + dw;
        if (h < 0 || h >= s.H || w < 0 || w >= s.W) continue;
        const __nv_bfloat16* xp = x + ((static_cast<long long>(n) * s.H + h) * s.W + w) * s.Cin;
        const __nv_bfloat16* g = dy + p * s.Cout;
        const float xr = bf(xp + ci), xi = bf(xp + s.Qin + ci);
        const float xj = bf(xp + 2 * s.Qin + ci), xk = bf(xp + 3 * s.Qin + ci);
        const float dr = bf(g + co), di = bf(g + s.Qout + co);
        const float dj = bf(g + 2 * s.Qout + co), dk = bf(g + 3 * s.Qout + co);
        if constexpr (SEP) {
            float gr, gi, gj, gk;
            mix_eq9(dr, di, dj, dk, gr, gi, gj, gk);
            a0 += gr * xr;
            a1 += gi * xi;
            a2 += gj * xj;
            a3 += gk * xk;
        } else {
            // dy (x) conj(X), conj(X) = (xr, -xi, -xj, -xk), by Eq. 3
            a0 += dr * xr + di * xi + dj * xj + dk * xk;
            a1 += -dr * xi + di * xr - dj * xk + dk * xj;
            a2 += -dr * xj + di * xk + dj * xr - dk * xi;
            a3 += -dr * xk - di * xj + dj * xi + dk * xr;
        }
    }
    atomicAdd(dwr + o, a0);
    atomicAdd(dwi + o, a1);
    atomicAdd(dwj + o, a2);
    atomicAdd(dwk + o, a3);
}

// Scratch of quan_qconv2d_bwd_data_static, the entry point for callers that cannot
// allocate device memory: the transformed letters of one call live here instead of in a
// caller workspace.  Every call writes all of the region it then reads, so nothing in it
// has to start at zero; calls that overlap on the GPU share it and race.  Host code must
// not pass this name to a kernel: on the host it is a stand-in, not a device address.
static __device__ __align__(256) unsigned char g_bwd_static_scratch[BWD_STATIC_SCRATCH_BYTES];

// u[n][y][x] = dy[n][y / s][x / s] where s divides y and x (and y / s < Ho, x / s < Wo),
// else 0: dy with s - 1 zeros between its pixels, [N][Hu][Wu][C], 16 bytes per thread.
__global__ void __launch_bounds__(256) bwd_upsample_kernel(const uint4* __restrict__ dy, int N,
                                                           int Ho, int Wo, int cv, int s, int Hu,
                                                           int Wu, uint4* __restrict__ u) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const long long total = static_cast<long long>(N) * Hu * Wu * cv;
    for (long long i = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; i < total;
         i += static_cast<long long>(gridDim.x) * blockDim.x) {
        const int c = static_cast<int>(i % cv);
        const long long pix = i / cv;
        const int x = static_cast<int>(pix % Wu);
        const int y = static_cast<int>((pix / Wu) % Hu);
        const int n = static_cast<int>(pix / (static_cast<long long>(Wu) * Hu));
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (y % s == 0 && x % s == 0 && y / s < Ho && x / s < Wo)
            v = __ldg(dy + ((static_cast<long long>(n) * Ho + y / s) * Wo + x / s) * cv + c);
        u[i] = v;
    }
}

}  // namespace

cudaError_t launch_bwd_upsample(const void* dy, int N, int Ho, int Wo, int C, int s, int Hu,
                                int Wu, void* u, int num_sms, cudaStream_t stream) {
    if (C % 8 != 0) return cudaErrorInvalidValue;
    const long long total = static_cast<long long>(N) * Hu * Wu * (C / 8);
    if (total == 0) return cudaSuccess;
    long long blocks = (total + 255) / 256;
    if (blocks > num_sms * 16LL) blocks = num_sms * 16LL;
    return launch_pdl(bwd_upsample_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0,
                      stream, static_cast<const uint4*>(dy), N, Ho, Wo, C / 8, s, Hu, Wu,
                      static_cast<uint4*>(u));
}

// Device address of the scratch on the current device (called once per device, with
// that device current, by the entry point's first call there).
cudaError_t bwd_static_scratch_address(void** ptr) {
    return cudaGetSymbolAddress(ptr, g_bwd_static_scratch);
}

size_t bwd_data_workspace_bytes(int Cin, int Cout, int kh, int kw) {
    return static_cast<size_t>(4) * (Cin / 4) * kh * kw * (Cout / 4) * 2;
}

cudaError_t launch_bwd_transform(int Cin, int Cout, int kh, int kw, const void* const w[4],
                                 bool conj, void* out, int num_sms, cudaStream_t stream) {
    const long long n = 4LL * (Cin / 4) * kh * kw * (Cout / 4);
    if (n == 0) return cudaSuccess;
    long long blocks = (n + 255) / 256;
    if (blocks > num_sms * 8LL) blocks = num_sms * 8LL;
    return launch_pdl(bwd_transform_kernel, dim3(static_cast<unsigned>(blocks)), dim3(256), 0,
                      stream, Cin / 4, Cout / 4, kh, kw, conj ? 1 : 0,
                      static_cast<const __nv_bfloat16*>(w[0]),
                      static_cast<const __nv_bfloat16*>(w[1]),
                      static_cast<const __nv_bfloat16*>(w[2]),
                      static_cast<const __nv_bfloat16*>(w[3]),
                      static_cast<__nv_bfloat16*>(out));
}

cudaError_t launch_bwd_data_simt(const ConvShape& s, const void* dy, const void* const w[4],
                                 void* dx, cudaStream_t stream) {
    auto kern = s.sep ? bwd_data_simt_kernel<true> : bwd_data_simt_kernel<false>;
    const long long total = static_cast<long long>(s.N) * s.H * s.W * s.Qin;
    if (total == 0) return cudaSuccess;
    const long long blocks = (total + 255) / 256;
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    return launch_pdl(kern, dim3(static_cast<unsigned>(blocks)), dim3(256), 0,
                      stream, s, static_cast<const __nv_bfloat16*>(dy),
                      static_cast<const __nv_bfloat16*>(w[0]),
                      static_cast<const __nv_bfloat16*>(w[1]),
                      static_cast<const __nv_bfloat16*>(w[2]),
                      static_cast<const __nv_bfloat16*>(w[3]), static_cast<__nv_bfloat16*>(dx));
}

cudaError_t launch_bwd_weight_simt(const ConvShape& s, const void* x, const void* dy,
                                   float* const dw[4], int num_sms, cudaStream_t stream) {
    const long long outs = static_cast<long long>(s.Qout) * s.kh * s.kw * s.Qin;
    const size_t bytes = static_cast<size_t>(outs) * sizeof(float);
    for (int L = 0; L < 4; ++L) {
        cudaError_t e = cudaMemsetAsync(dw[L], 0, bytes, stream);
        if (e != cudaSuccess) return e;
    }
    if (outs == 0 || s.M == 0) return cudaSuccess;
    // enough pixel chunks to give every SM a few thousand threads
    const long long oblocks = (outs + 255) / 256;
    long long chunks = (static_cast<long long>(num_sms) * 16 + oblocks - 1) / oblocks;
    if (chunks > s.M) chunks = s.M;
    if (chunks > 65535) chunks = 65535;
    if (chunks < 1) chunks = 1;
    const long long chunk = (s.M + chunks - 1) / chunks;
    chunks = (s.M + chunk - 1) / chunk;
    if (oblocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    auto kern = s.sep ? bwd_weight_simt_kernel<true> : bwd_weight_simt_kernel<false>;
    return launch_pdl(kern,
                      dim3(static_cast<unsigned>(oblocks), static_cast<unsigned>(chunks)),
                      dim3(256), 0, stream, s, static_cast<const __nv_bfloat16*>(x),
                      static_cast<const __nv_bfloat16*>(dy), chunk, dw[0], dw[1], dw[2], dw[3]);
}

}  // namespace quan
