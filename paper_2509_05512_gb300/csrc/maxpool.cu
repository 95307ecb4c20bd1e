// maxpool.cu -- max pooling applied to every real channel independently, the
// component-wise pooling rule of QSPPF (Sec. III-D): each of the r, i, j, k
// blocks is pooled on its own, so the quaternion channel layout is unchanged.
// bf16 NHWC; 8 channels (16 bytes) per thread when C % 8 == 0, else 1.
#include <cuda_bf16.h>

#include "internal.h"

namespace quan {
namespace {

template <int VEC>
__global__ void __launch_bounds__(256) maxpool_kernel(const __nv_bfloat16* __restrict__ x, int N,
                                                      int H, int W, int C, int k, int stride,
                                                      int pad, int Ho, int Wo,
                                                      __nv_bfloat16* __restrict__ y) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");  // inputs from the previous kernel
    const int cv = C / VEC;
    const long long total = static_cast<long long>(N) * Ho * Wo * cv;
    for (long long idx = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x;
         idx < total; idx += static_cast<long long>(gridDim.x) * blockDim.x) {
        const int c = static_cast<int>(idx % cv) * VEC;
        const long long pix = idx / cv;
        const int wo = static_cast<int>(pix % Wo);
        const int ho = static_cast<int>((pix / Wo) % Ho);
        const int n = static_cast<int>(pix / (static_cast<long long>(Wo) * Ho));
        float m[VEC];
#pragma unroll
        for (int v = 0; v < VEC; ++v) m[v] = -INFINITY;
        for (int dh = 0; dh < k; ++dh) {
            const int h = ho * stride - pad + dh;
            if (h < 0 || h >= H) continue;
            for (int dw = 0; dw < k; ++dw) {
                const int w = wo * stride - pad + dw;
                if (w < 0 || w >= W) continue;
                const __nv_bfloat16* p =
                    x + ((static_cast<long long>(n) * H + h) * W + w) * C + c;
                if constexpr (VEC == 8) {
                    const uint4 raw = __ldg(reinterpret_cast<const uint4*>(p));
                    const __nv_bfloat162* b2 = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
                    for (int v = 0; v < 4; ++v) {
                        const float2 f = __bfloat1622float2(b2[v]);
                        m[2 * v] = fmaxf(m[2 * v], f.x);
                        m[2 * v + 1] = fmaxf(m[2 * v + 1], f.y);
                    }
                } else {
                    m[0] = fmaxf(m[0], __bfloat162float(p[0]));
                }
            }
        }
        __nv_bfloat16* q = y + pix * C + c;
        if constexpr (VEC == 8) {
            uint4 raw;
            __nv_bfloat162* b2 = reinterpret_cast<__nv_bfloat162*>(&raw);
#pragma unroll
            for (int v = 0; v < 4; ++v) b2[v] = __floats2bfloat162_rn(m[2 * v], m[2 * v + 1]);
            *reinterpret_cast<uint4*>(q) = raw;
        } else {
            q[0] = __float2bfloat16_rn(m[0]);
        }
    }
}

// One CTA per output row (n, ho); thread t covers column wo = t / cv and channels
// 8 (t % cv) .. +7 (cv = C / 8), with a block-stride loop when Wo * cv exceeds the block.
// All index arithmetic is 32-bit and done once per output; neighbouring columns share
// their input columns through L1.
__global__ void __launch_bounds__(512) maxpool_rows_kernel(const __nv_bfloat16* __restrict__ x,
                                                           int H, int W, int C, int k,
                                                           int stride, int pad, int Ho, int Wo,
                                                           __nv_bfloat16* __restrict__ y) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");  // inputs from the previous kernel
    const int cv = C / 8;
    const int row = blockIdx.x;  // n * Ho + ho
    const int n = row / Ho, ho = row - (row / Ho) * Ho;
    const uint4* xr = reinterpret_cast<const uint4*>(x) + static_cast<long long>(n) * H * W * cv;
    uint4* yr = reinterpret_cast<uint4*>(y) + static_cast<long long>(row) * Wo * cv;
    const int h0 = ho * stride - pad;
    for (int t = threadIdx.x; t < Wo * cv; t += blockDim.x) {
        const int wo = t / cv, c = t - (t / cv) * cv;
        const int w0 = wo * stride - pad;
        float m[8];
#pragma unroll
        for (int v = 0; v < 8; ++v) m[v] = -INFINITY;
        for (int dh = 0; dh < k; ++dh) {
            const int h = h0 + dh;
            if (h < 0 || h >= H) continue;
            for (int dw = 0; dw < k; ++dw) {
                const int w = w0 + dw;
                if (w < 0 || w >= W) continue;
                const uint4 raw = __ldg(xr + (h * W + w) * cv + c);
                const __nv_bfloat162* b2 = reinterpret_cast<const __nv_bfloat162*>(&raw);
#pragma unroll
                for (int v = 0; v < 4; ++v) {
                    const float2 f = __bfloat1622float2(b2[v]);
                    m[2 * v] = fmaxf(m[2 * v], f.x);
                    m[2 * v + 1] = fmaxf(m[2 * v + 1], f.y);
                }
            }
        }
        uint4 raw;
        __nv_bfloat162* b2 = reinterpret_cast<__nv_bfloat162*>(&raw);
#pragma unroll
        for (int v = 0; v < 4; ++v) b2[v] = __floats2bfloat162_rn(m[2 * v], m[2 * v + 1]);
        yr[t] = raw;
    }
}

}  // namespace

cudaError_t launch_maxpool_bf16(const void* x, int N, int H, int W, int C, int k, int stride,
                                int pad, void* out, int num_sms, cudaStream_t stream) {
    const int Ho = (H + 2 * pad - k) / stride + 1;
    const int Wo = (W + 2 * pad - k) / stride + 1;
    const bool vec = (C % 8 == 0) && (reinterpret_cast<uintptr_t>(x) % 16 == 0) &&
                     (reinterpret_cast<uintptr_t>(out) % 16 == 0);
    const long long total = static_cast<long long>(N) * Ho * Wo * (vec ? C / 8 : C);
    if (total == 0) return cudaSuccess;
    const int threads = 256;
    long long blocks = (total + threads - 1) / threads;
    const long long cap = static_cast<long long>(num_sms) * 8 * 4;
    if (blocks > cap) blocks = cap;
    const auto* xb = static_cast<const __nv_bfloat16*>(x);
    auto* yb = static_cast<__nv_bfloat16*>(out);
    const long long rows = static_cast<long long>(N) * Ho;
    // 32-bit per-image offsets for the row kernel
    if (vec && rows <= 0x7fffffffLL && static_cast<long long>(H) * W * (C / 8) <= 0x7fffffffLL) {
        const int work = Wo * (C / 8);
        const int t = work >= 512 ? 512 : ((work + 31) / 32) * 32;
        return launch_pdl(maxpool_rows_kernel, dim3(static_cast<unsigned>(rows)), dim3(t), 0,
                          stream, xb, H, W, C, k, stride, pad, Ho, Wo, yb);
    }
    if (vec)
        return launch_pdl(maxpool_kernel<8>, dim3(static_cast<unsigned>(blocks)), dim3(threads),
                          0, stream, xb, N, H, W, C, k, stride, pad, Ho, Wo, yb);
    return launch_pdl(maxpool_kernel<1>, dim3(static_cast<unsigned>(blocks)), dim3(threads), 0,
                      stream, xb, N, H, W, C, k, stride, pad, Ho, Wo, yb);
}

}  // namespace quan
