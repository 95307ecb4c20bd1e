// qconv_simt.cu -- CUDA-core quaternion convolution (fp32 FFMA accumulation).
//
// Handles every shape the tensor-core path does not: fp32 tensors, quaternion channel
// counts that are not multiples of 16, unaligned pointers and the 4-channel stem.
// One thread computes one output quaternion (4 real outputs) of one pixel from the
// Hamilton-product expansion of Eq. 5 (Sec. III-B):
//   y_r = W_r x_r - W_i x_i - W_j x_j - W_k x_k
//   y_i = W_r x_i + W_i x_r + W_j x_k - W_k x_j
//   y_j = W_r x_j - W_i x_k + W_j x_r + W_k x_i
//   y_k = W_r x_k + W_i x_j - W_j x_i + W_k x_r
// summed over taps and input quaternion channels, followed by the fused epilogue
// act(scale * (acc + bias) + shift + residual) (IQBN inference form of Eq. 11-12).
// The separable form of Eq. 7 (s.sep) keeps only the diagonal convolutions
// c_p = W_p x_p and mixes them with that equation's signs:
//   y_r = c_r - c_i - c_j - c_k,  y_i = c_r + c_i + c_j - c_k,
//   y_j = c_r - c_i + c_j + c_k,  y_k = c_r + c_i - c_j + c_k.
#include <cuda_bf16.h>

#include "internal.h"

namespace quan {
namespace {

__device__ __forceinline__ float to_f32(float v) { return v; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 v) { return __bfloat162float(v); }
__device__ __forceinline__ void store(float* p, float v) { *p = v; }
__device__ __forceinline__ void store(__nv_bfloat16* p, float v) { *p = __float2bfloat16_rn(v); }

__device__ __forceinline__ float activate(float z, int act) {
    if (act == 1) return fmaxf(z, 0.0f);
    if (act == 2) return z / (1.0f + __expf(-z));
    return z;
}

template <typename T>
__global__ void __launch_bounds__(256) qconv_simt_kernel(ConvShape s, const T* __restrict__ x,
                                                         const T* __restrict__ wr,
                                                         const T* __restrict__ wi,
                                                         const T* __restrict__ wj,
                                                         const T* __restrict__ wk,
                                                         EpilogueArgs ep, T* __restrict__ out) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");  // inputs from the previous kernel
    const long long total = s.M * s.Qout;
    const long long idx = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= total) return;
    const int co = static_cast<int>(idx % s.Qout);
    const long long m = idx / s.Qout;
    const int hw = s.Ho * s.Wo;
    const int n = static_cast<int>(m / hw);
    const int rem = static_cast<int>(m % hw);
    const int ho = rem / s.Wo, wo = rem % s.Wo;
    const int Qin = s.Qin;

    float ar = 0.f, ai = 0.f, aj = 0.f, ak = 0.f;
    for (int dh = 0; dh < s.kh; ++dh) {
        const int h = ho * s.stride - s.pad + dh;
        if (h < 0 || h >= s.H) continue;
        for (int dw = 0; dw < s.kw; ++dw) {
            const int w = wo * s.stride - s.pad + dw;
            if (w < 0 || w >= s.W) continue;
            const T* xp = x + ((static_cast<long long>(n) * s.H + h) * s.W + w) * s.Cin;
            const long long wofs = (static_cast<long long>(co) * s.kh + dh) * s.kw + dw;
            const T* pr = wr + wofs * Qin;
            const T* pi = wi + wofs * Qin;
            const T* pj = wj + wofs * Qin;
            const T* pk = wk + wofs * Qin;
            if (s.sep) {
                // c_r .. c_k accumulate in ar .. ak
                for (int ci = 0; ci < Qin; ++ci) {
                    ar = fmaf(to_f32(__ldg(pr + ci)), to_f32(xp[ci]), ar);
                    ai = fmaf(to_f32(__ldg(pi + ci)), to_f32(xp[Qin + ci]), ai);
                    aj = fmaf(to_f32(__ldg(pj + ci)), to_f32(xp[2 * Qin + ci]), aj);
                    ak = fmaf(to_f32(__ldg(pk + ci)), to_f32(xp[3 * Qin + ci]), ak);
                }
                continue;
            }
            for (int ci = 0; ci < Qin; ++ci) {
                const float xr = to_f32(xp[ci]), xi = to_f32(xp[Qin + ci]);
                const float xj = to_f32(xp[2 * Qin + ci]), xk = to_f32(xp[3 * Qin + ci]);
                const float a = to_f32(__ldg(pr + ci)), b = to_f32(__ldg(pi + ci));
                const float c = to_f32(__ldg(pj + ci)), d = to_f32(__ldg(pk + ci));
                ar = fmaf(a, xr, ar); ar = fmaf(-b, xi, ar); ar = fmaf(-c, xj, ar); ar = fmaf(-d, xk, ar);
                ai = fmaf(a, xi, ai); ai = fmaf(b, xr, ai); ai = fmaf(c, xk, ai); ai = fmaf(-d, xj, ai);
                aj = fmaf(a, xj, aj); aj = fmaf(-b, xk, aj); aj = fmaf(c, xr, aj); aj = fmaf(d, xi, aj);
                ak = fmaf(a, xk, ak); ak = fmaf(b, xj, ak); ak = fmaf(-c, xi, ak); ak = fmaf(d, xr, ak);
            }
        }
    }
    float acc[4] = {ar, ai, aj, ak};
    if (s.sep) {
        acc[0] = ar - ai - aj - ak;
        acc[1] = ar + ai + aj - ak;
        acc[2] = ar - ai + aj + ak;
        acc[3] = ar + ai - aj + ak;
    }
    T* op = out + m * s.Cout;
    const T* rp = ep.residual ? static_cast<const T*>(ep.residual) + m * s.Cout : nullptr;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int c = q * s.Qout + co;
        float z = acc[q];
        if (ep.bias) z += __ldg(ep.bias + c);
        if (ep.scale) z = fmaf(__ldg(ep.scale + c), z, __ldg(ep.shift + c));
        if (rp) z += to_f32(rp[c]);
        store(op + c, activate(z, s.act));
    }
}

template <typename T>
cudaError_t launch(const ConvShape& s, const void* x, const void* const w[4],
                   const EpilogueArgs& ep, void* out, cudaStream_t stream) {
    const long long total = s.M * s.Qout;
    if (total == 0) return cudaSuccess;
    const int threads = 256;
    const long long blocks = (total + threads - 1) / threads;
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    return launch_pdl(qconv_simt_kernel<T>, dim3(static_cast<unsigned>(blocks)), dim3(threads),
                      0, stream, s, static_cast<const T*>(x), static_cast<const T*>(w[0]),
                      static_cast<const T*>(w[1]), static_cast<const T*>(w[2]),
                      static_cast<const T*>(w[3]), ep, static_cast<T*>(out));
}

}  // namespace

cudaError_t launch_qconv_simt_bf16(const ConvShape& s, const void* x, const void* const w[4],
                                   const EpilogueArgs& ep, void* out, cudaStream_t stream) {
    return launch<__nv_bfloat16>(s, x, w, ep, out, stream);
}

cudaError_t launch_qconv_simt_f32(const ConvShape& s, const void* x, const void* const w[4],
                                  const EpilogueArgs& ep, void* out, cudaStream_t stream) {
    return launch<float>(s, x, w, ep, out, stream);
}

}  // namespace quan
