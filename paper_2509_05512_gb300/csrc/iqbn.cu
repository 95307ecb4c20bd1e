// iqbn.cu -- Independent Quaternion Batch Normalization in training mode (Eq. 11-12,
// Sec. III-C): the batch statistics of every real channel (one component of one
// quaternion channel) over N, H, W, and the normalisation with them.
//
// x is bf16 [npix][C] (NHWC flattened).  Both kernels are HBM-bound streams; every thread
// keeps one fixed group of channels (8 channels read as one 16-byte vector, or a single
// channel when C is not a multiple of 8) and walks the pixels with a grid-wide stride, so
// its per-channel state stays in registers.
//
// Statistics: each thread sums d = x - K_c and d^2 in fp32 over its pixels, with the shift
// K_c = x[0][c] (the first pixel's value, read by every thread) keeping E[d^2] - E[d]^2 free
// of cancellation when the mean is large; the block reduces in shared memory and writes its
// partial sums to its own row of a caller workspace; a second kernel adds the rows in a
// fixed order with compensated fp32 sums (no atomics: the result does not depend on
// timing) and forms
// mean = K + S1 / n and the biased variance S2 / n - (S1 / n)^2 of Eq. 11.
#include <cuda_bf16.h>

#include "internal.h"

namespace quan {
namespace {

__device__ __forceinline__ void unpack8(const uint4 v, float (&f)[8]) {
    const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&v);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float2 t = __bfloat1622float2(h[i]);
        f[2 * i] = t.x;
        f[2 * i + 1] = t.y;
    }
}

// W channels per thread (8: one 16-byte vector, 1: scalar); G = C / W channel groups;
// blockDim.x = G * R, R pixel rows per block.
template <int W>
__global__ void __launch_bounds__(256) iqbn_stats_kernel(const __nv_bfloat16* __restrict__ x,
                                                         long long npix, int C, int G,
                                                         float* __restrict__ part) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    extern __shared__ float red[];  // [2][blockDim.x][W]
    const int slot = threadIdx.x % G, row = threadIdx.x / G;
    const int R = blockDim.x / G;
    const int c0 = slot * W;
    float K[W], a1[W], a2[W];
    if constexpr (W == 8) {
        unpack8(__ldg(reinterpret_cast<const uint4*>(x + c0)), K);
    } else {
        K[0] = __bfloat162float(x[c0]);
    }
#pragma unroll
    for (int i = 0; i < W; ++i) a1[i] = a2[i] = 0.f;
    const long long stride = static_cast<long long>(gridDim.x) * R;
    auto load = [&](long long p, float (&v)[W]) {
        if constexpr (W == 8) {
            unpack8(__ldg(reinterpret_cast<const uint4*>(x + p * C + c0)), v);
        } else {
            v[0] = __bfloat162float(x[p * C + c0]);
        }
    };
    auto add = [&](const float (&v)[W]) {
#pragma unroll
        for (int i = 0; i < W; ++i) {
            const float d = v[i] - K[i];
            a1[i] += d;
            a2[i] = fmaf(d, d, a2[i]);
        }
    };
    long long p = static_cast<long long>(blockIdx.x) * R + row;
    // eight independent loads in flight per thread, then the remainder one at a time
    if constexpr (W == 8) {
        for (; p + 7 * stride < npix; p += 8 * stride) {
            uint4 raw[8];
#pragma unroll
            for (int k = 0; k < 8; ++k)
                raw[k] = __ldg(reinterpret_cast<const uint4*>(x + (p + k * stride) * C + c0));
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                float v[8];
                unpack8(raw[k], v);
                add(v);
            }
        }
    } else {
        for (; p + 3 * stride < npix; p += 4 * stride) {
            float v0[W], v1[W], v2[W], v3[W];
            load(p, v0);
            load(p + stride, v1);
            load(p + 2 * stride, v2);
            load(p + 3 * stride, v3);
            add(v0);
            add(v1);
            add(v2);
            add(v3);
        }
    }
    for (; p < npix; p += stride) {
        float v[W];
        load(p, v);
        add(v);
    }
    float* r1 = red;
    float* r2 = red + blockDim.x * W;
#pragma unroll
    for (int i = 0; i < W; ++i) {
        r1[threadIdx.x * W + i] = a1[i];
        r2[threadIdx.x * W + i] = a2[i];
    }
    __syncthreads();
    if (row == 0) {
        for (int r = 1; r < R; ++r) {
#pragma unroll
            for (int i = 0; i < W; ++i) {
                a1[i] += r1[(r * G + slot) * W + i];
                a2[i] += r2[(r * G + slot) * W + i];
            }
        }
        float* row1 = part + static_cast<size_t>(blockIdx.x) * 2 * C;
#pragma unroll
        for (int i = 0; i < W; ++i) {
            row1[c0 + i] = a1[i];
            row1[C + c0 + i] = a2[i];
        }
    }
}

// Compensated (Kahan) fp32 addition: the running sum and its lost low-order part.
__device__ __forceinline__ void kahan_add(float& sum, float& comp, float v) {
    const float y = v - comp;
    const float t = sum + y;
    comp = (t - sum) - y;
    sum = t;
}

// Sum of the partial rows per channel in a fixed order (row lane rl takes rows rl, rl + 32,
// ..., compensated fp32; then the 32 lanes in order), then mean = K + S1 / n and
// var = max(S2 / n - (S1 / n)^2, 0) (these last few operations per channel in fp64; the
// row sums stay in fp32, the double-precision rate of this part being low).
// Block: 32 channels x 32 row lanes.
__global__ void __launch_bounds__(1024) iqbn_finalize_kernel(const __nv_bfloat16* __restrict__ x,
                                                             long long npix, int C, int rows,
                                                             const float* __restrict__ part,
                                                             float* __restrict__ mean,
                                                             float* __restrict__ var) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    __shared__ float red[2][32][33];
    const int cl = threadIdx.x % 32, rl = threadIdx.x / 32;
    const int c = blockIdx.x * 32 + cl;
    float t1 = 0.f, t2 = 0.f, e1 = 0.f, e2 = 0.f;
    if (c < C) {
#pragma unroll 4
        for (int r = rl; r < rows; r += 32) {
            kahan_add(t1, e1, part[static_cast<size_t>(r) * 2 * C + c]);
            kahan_add(t2, e2, part[static_cast<size_t>(r) * 2 * C + C + c]);
        }
    }
    red[0][rl][cl] = t1 - e1;
    red[1][rl][cl] = t2 - e2;
    __syncthreads();
    if (rl == 0 && c < C) {
        float s1 = 0.f, s2 = 0.f, f1 = 0.f, f2 = 0.f;
        for (int k = 0; k < 32; ++k) {
            kahan_add(s1, f1, red[0][k][cl]);
            kahan_add(s2, f2, red[1][k][cl]);
        }
        const double inv_n = 1.0 / static_cast<double>(npix);
        const double d1 = (static_cast<double>(s1) - f1) * inv_n;
        const double m2 = (static_cast<double>(s2) - f2) * inv_n - d1 * d1;
        mean[c] = static_cast<float>(static_cast<double>(__bfloat162float(x[c])) + d1);
        var[c] = m2 > 0.0 ? static_cast<float>(m2) : 0.0f;
    }
}

__device__ __forceinline__ float act_fn(float z, int act) {
    if (act == 1) return fmaxf(z, 0.0f);
    if (act == 2) return z / (1.0f + __expf(-z));
    return z;
}

// out = act(gamma (x - mean) / sqrt(var + eps) + beta) (Eq. 11-12), as scale * x + shift.
template <int W>
__global__ void __launch_bounds__(256) iqbn_apply_kernel(
    const __nv_bfloat16* x, long long npix, int C, int G, const float* __restrict__ mean,
    const float* __restrict__ var, const float* __restrict__ gamma,
    const float* __restrict__ beta, float eps, int act, __nv_bfloat16* out) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");
    const int slot = threadIdx.x % G, row = threadIdx.x / G;
    const int R = blockDim.x / G;
    const int c0 = slot * W;
    float sc[W], sh[W];
#pragma unroll
    for (int i = 0; i < W; ++i) {
        const int c = c0 + i;
        const float g = gamma ? gamma[c] : 1.0f;
        const float b = beta ? beta[c] : 0.0f;
        sc[i] = g / sqrtf(var[c] + eps);
        sh[i] = fmaf(-mean[c], sc[i], b);
    }
    const long long stride = static_cast<long long>(gridDim.x) * R;
    auto one = [&](long long p) {
        if constexpr (W == 8) {
            float v[8];
            unpack8(*reinterpret_cast<const uint4*>(x + p * C + c0), v);
            uint4 o;
            uint32_t* ow = reinterpret_cast<uint32_t*>(&o);
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const __nv_bfloat162 t =
                    __floats2bfloat162_rn(act_fn(fmaf(v[2 * i], sc[2 * i], sh[2 * i]), act),
                                          act_fn(fmaf(v[2 * i + 1], sc[2 * i + 1], sh[2 * i + 1]), act));
                ow[i] = *reinterpret_cast<const uint32_t*>(&t);
            }
            *reinterpret_cast<uint4*>(out + p * C + c0) = o;
        } else {
            const float v = __bfloat162float(x[p * C + c0]);
            out[p * C + c0] = __float2bfloat16_rn(act_fn(fmaf(v, sc[0], sh[0]), act));
        }
    };
    long long p = static_cast<long long>(blockIdx.x) * R + row;
    if constexpr (W == 8) {
        // four loads in flight before the first store (each thread reads only the
        // elements it writes, so an in-place call is still safe)
        for (; p + 3 * stride < npix; p += 4 * stride) {
            uint4 raw[4];
#pragma unroll
            for (int k = 0; k < 4; ++k)
                raw[k] = *reinterpret_cast<const uint4*>(x + (p + k * stride) * C + c0);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                float v[8];
                unpack8(raw[k], v);
                uint4 o;
                uint32_t* ow = reinterpret_cast<uint32_t*>(&o);
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const __nv_bfloat162 t = __floats2bfloat162_rn(
                        act_fn(fmaf(v[2 * i], sc[2 * i], sh[2 * i]), act),
                        act_fn(fmaf(v[2 * i + 1], sc[2 * i + 1], sh[2 * i + 1]), act));
                    ow[i] = *reinterpret_cast<const uint32_t*>(&t);
                }
                *reinterpret_cast<uint4*>(out + (p + k * stride) * C + c0) = o;
            }
        }
    }
    for (; p < npix; p += stride) one(p);
}

// Channel groups, block size and grid of one launch; false if C has no layout.
bool iqbn_layout(int C, bool vec, long long npix, int num_sms, int per_sm, int* G, int* block,
                 int* grid) {
    const int W = vec ? 8 : 1;
    const int g = C / W;
    if (g < 1 || g > 256) return false;
    const int R = 256 / g;
    *G = g;
    *block = g * R;
    long long blocks = (npix + R - 1) / R;
    const long long cap = static_cast<long long>(num_sms) * per_sm;
    if (blocks > cap) blocks = cap;
    *grid = static_cast<int>(blocks);
    return true;
}

}  // namespace

bool iqbn_vec_ok(int C, const void* a, const void* b) {
    return C % 8 == 0 && C / 8 <= 256 && reinterpret_cast<uintptr_t>(a) % 16 == 0 &&
           reinterpret_cast<uintptr_t>(b) % 16 == 0;
}

bool iqbn_supported(int C, const void* a, const void* b) {
    return iqbn_vec_ok(C, a, b) || (C >= 1 && C <= 256);
}

size_t iqbn_stats_workspace_bytes(int C) {
    return C < 1 ? 0 : static_cast<size_t>(IQBN_MAX_PARTIALS) * 2 * C * sizeof(float);
}

cudaError_t launch_iqbn_stats(const void* x, long long npix, int C, void* workspace,
                              float* mean, float* var, int num_sms, cudaStream_t stream) {
    const bool vec = iqbn_vec_ok(C, x, x);
    int G = 0, block = 0, grid = 0;
    if (!iqbn_layout(C, vec, npix, num_sms, 4, &G, &block, &grid)) return cudaErrorInvalidValue;
    if (grid > IQBN_MAX_PARTIALS) grid = IQBN_MAX_PARTIALS;
    const auto* xb = static_cast<const __nv_bfloat16*>(x);
    auto* part = static_cast<float*>(workspace);
    const size_t smem = static_cast<size_t>(2) * block * (vec ? 8 : 1) * sizeof(float);
    cudaError_t e = vec ? launch_pdl(iqbn_stats_kernel<8>, dim3(grid), dim3(block), smem, stream,
                                     xb, npix, C, G, part)
                        : launch_pdl(iqbn_stats_kernel<1>, dim3(grid), dim3(block), smem, stream,
                                     xb, npix, C, G, part);
    if (e != cudaSuccess) return e;
    return launch_pdl(iqbn_finalize_kernel, dim3((C + 31) / 32), dim3(1024), 0, stream, xb,
                      npix, C, grid, static_cast<const float*>(part), mean, var);
}

cudaError_t launch_iqbn_apply(const void* x, long long npix, int C, const float* mean,
                              const float* var, const float* gamma, const float* beta, float eps,
                              int act, void* out, int num_sms, cudaStream_t stream) {
    const bool vec = iqbn_vec_ok(C, x, out);
    int G = 0, block = 0, grid = 0;
    if (!iqbn_layout(C, vec, npix, num_sms, 8, &G, &block, &grid)) return cudaErrorInvalidValue;
    const auto* xb = static_cast<const __nv_bfloat16*>(x);
    auto* ob = static_cast<__nv_bfloat16*>(out);
    return vec ? launch_pdl(iqbn_apply_kernel<8>, dim3(grid), dim3(block), 0, stream, xb, npix,
                            C, G, mean, var, gamma, beta, eps, act, ob)
               : launch_pdl(iqbn_apply_kernel<1>, dim3(grid), dim3(block), 0, stream, xb, npix,
                            C, G, mean, var, gamma, beta, eps, act, ob);
}

}  // namespace quan
