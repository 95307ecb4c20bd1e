// poincare.cu -- the Poincare mapping of RGB pixels onto the unit quaternion sphere
// (Eq. 4, Sec. III-A), the input mapping in front of the 4-channel stem:
//   n2 = r^2 + g^2 + b^2,  q = ((1 - n2), 2 r, 2 g, 2 b) / (1 + n2),
// fp32 RGB [npix][3] -> bf16 [npix][4] in the component-major channel order [r|i|j|k]
// the convolutions read (one quaternion channel: the four components of a pixel).
// Elementwise and HBM-bound (12 bytes read, 8 written per pixel): one pixel per thread,
// coalesced 4-byte loads, one 8-byte store.  The reciprocal is the fast one (__fdividef,
// within a few fp32 ulps: far below the bf16 result's rounding); the stem kernel's fused
// mapping uses the same arithmetic, so mapping first and mapping in the stem agree bit for
// bit.
#include <cuda_bf16.h>

#include "internal.h"

namespace quan {
namespace {

template <bool VEC>
__global__ void __launch_bounds__(256) poincare_kernel(const float* __restrict__ rgb,
                                                        long long npix,
                                                        __nv_bfloat16* __restrict__ q) {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    asm volatile("griddepcontrol.wait;" ::: "memory");  // inputs from the previous kernel
    for (long long p = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; p < npix;
         p += static_cast<long long>(gridDim.x) * blockDim.x) {
        const float r = __ldg(rgb + 3 * p), g = __ldg(rgb + 3 * p + 1), b = __ldg(rgb + 3 * p + 2);
        const float n2 = fmaf(r, r, fmaf(g, g, b * b));
        const float inv = __fdividef(1.0f, 1.0f + n2);
        const float two_inv = 2.0f * inv;
        const __nv_bfloat162 ri = __floats2bfloat162_rn((1.0f - n2) * inv, r * two_inv);
        const __nv_bfloat162 jk = __floats2bfloat162_rn(g * two_inv, b * two_inv);
        if constexpr (VEC) {
            uint2 v;
            v.x = *reinterpret_cast<const uint32_t*>(&ri);
            v.y = *reinterpret_cast<const uint32_t*>(&jk);
            *reinterpret_cast<uint2*>(q + 4 * p) = v;
        } else {
            q[4 * p] = ri.x;
            q[4 * p + 1] = ri.y;
            q[4 * p + 2] = jk.x;
            q[4 * p + 3] = jk.y;
        }
    }
}

}  // namespace

cudaError_t launch_poincare(const float* rgb, long long npix, void* out, int num_sms,
                            cudaStream_t stream) {
    if (npix == 0) return cudaSuccess;
    const int threads = 256;
    long long blocks = (npix + threads - 1) / threads;
    const long long cap = static_cast<long long>(num_sms) * 16;  // grid-stride beyond this
    if (blocks > cap) blocks = cap;
    auto* q = static_cast<__nv_bfloat16*>(out);
    if (reinterpret_cast<uintptr_t>(out) % 8 == 0)
        return launch_pdl(poincare_kernel<true>, dim3(static_cast<unsigned>(blocks)),
                          dim3(threads), 0, stream, rgb, npix, q);
    return launch_pdl(poincare_kernel<false>, dim3(static_cast<unsigned>(blocks)), dim3(threads),
                      0, stream, rgb, npix, q);
}

}  // namespace quan
