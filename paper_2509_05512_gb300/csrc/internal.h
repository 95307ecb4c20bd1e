// internal.h -- launch interfaces shared by the C-ABI front end (quan_api.cu) and the
// kernels.  Not part of the public header.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

namespace quan {

// Geometry and epilogue of one quaternion convolution call.  Channels are real
// channels; Q = C / 4 quaternion channels per component block.
struct ConvShape {
    int N, H, W, Cin, Cout, kh, kw, stride, pad, act;
    int Ho, Wo, Qin, Qout;
    long long M;  // N * Ho * Wo output pixels
    int sep;      // 1: the separable form of Eq. 7 (per-component convolutions, sign mix);
                  // 2 (tensor-core path only): its transpose, the input gradient's
                  // convolution (block (q, p) = sign(p, q) W_q)
};

struct EpilogueArgs {
    const float* bias;   // [Cout] or null
    const float* scale;  // [Cout] or null (IQBN scale, with shift)
    const float* shift;  // [Cout] or null
    const void* residual;  // [M][Cout] (same dtype as out) or null
};

// Device status word bits (set by kernels whose bounded waits ran out).
enum : unsigned {
    STATUS_TIMEOUT_PRODUCER = 1u,
    STATUS_TIMEOUT_MMA = 2u,
    STATUS_TIMEOUT_EPILOGUE = 4u,
    STATUS_TIMEOUT_DRAIN = 8u,
};

struct TcOptions {
    int kappa;                    // quaternion input channels per K block (16, 32 or 64); 0 = auto
    int bnq;                      // quaternion output channels per tile (16, 32 or 64); 0 = auto
    int max_ctas;                 // persistent grid cap; 0 = number of SMs
    int mode;                     // 0 auto, 1 one MMA per (q, p), 2 paired output components,
                                  // 3 weight-stationary
    int ws_halo;                  // weight-stationary: stage row blocks with halos (1) when
                                  // the shape allows it, else one im2col box per tap (0)
    int ws_issuers;               // weight-stationary MMA issuers: 0 auto, 2 or 3
    int vs_rows;                  // vertical-tap kernel: output rows per band, 0 auto, 1..4
    void* sk_ws;                  // caller workspace for K ranges split over the CTAs (the
    size_t sk_ws_bytes;           // quad/pair kernel's partial tiles and flags), or null
    unsigned long long wait_limit_ns;
    int inject_stall;             // failure-injection: the MMA role never consumes
};

// Tensor-core path (tcgen05 + TMA), bf16 in/out, fp32 accumulation.
bool tc_supported(const ConvShape& s, const void* x, const void* const w[4], const void* out,
                  const EpilogueArgs& ep);
cudaError_t launch_qconv_tc(const ConvShape& s, const void* x, const void* const w[4],
                            const EpilogueArgs& ep, void* out, const TcOptions& opt,
                            int num_sms, cudaStream_t stream, char* err, size_t errlen);
cudaError_t read_and_clear_status(unsigned* status, cudaStream_t stream);
// Workspace bytes that let a quad/pair-kernel launch on a device of num_sms SMs split its
// K ranges evenly over its CTAs (one fp32 partial tile and one flag per CTA).
size_t tc_split_workspace_bytes(int num_sms);
// The convolution s and a 1x1 shortcut (Qout_sc quaternion output channels, no padding, the
// same stride) on the same input x in one tensor-core launch; its own letters, epilogue
// vectors (no residual), activation and output.
bool tc_shortcut_supported(const ConvShape& s, const void* x, const void* const w[4],
                           const void* out, const EpilogueArgs& ep, const void* const wsc[4],
                           int qout_sc, const EpilogueArgs& ep_sc, const void* out_sc,
                           const TcOptions& opt);
cudaError_t launch_qconv_tc_shortcut(const ConvShape& s, const void* x, const void* const w[4],
                                     const EpilogueArgs& ep, void* out,
                                     const void* const wsc[4], int qout_sc, int act_sc,
                                     const EpilogueArgs& ep_sc, void* out_sc,
                                     const TcOptions& opt, int num_sms, cudaStream_t stream,
                                     char* err, size_t errlen);
// Name of the tensor-core kernel the calling thread's last launch_qconv_tc used.
const char* last_tc_kernel();

// CUDA-core path, any shape; T = __nv_bfloat16 or float.
cudaError_t launch_qconv_simt_bf16(const ConvShape& s, const void* x, const void* const w[4],
                                   const EpilogueArgs& ep, void* out, cudaStream_t stream);
cudaError_t launch_qconv_simt_f32(const ConvShape& s, const void* x, const void* const w[4],
                                  const EpilogueArgs& ep, void* out, cudaStream_t stream);

// Launch with programmatic stream serialization: the kernel may start while the previous
// kernel in the stream is finishing (once all of that grid's CTAs have signalled), runs its
// prologue (barriers, TMEM, descriptor prefetch) and waits with griddepcontrol.wait before
// its first global access.  Every kernel of this library follows that rule.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                       cudaStream_t stream, Args&&... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// Poincare RGB -> quaternion mapping (Eq. 4): fp32 [npix][3] -> bf16 [npix][4].
cudaError_t launch_poincare(const float* rgb, long long npix, void* out, int num_sms,
                            cudaStream_t stream);

// Backward of the pre-epilogue convolution (s.sep selects the separable form, Eq. 8-10).
// Bytes of the transformed letters bwd_transform writes: 4 x [Qin][kh][kw][Qout] bf16.
size_t bwd_data_workspace_bytes(int Cin, int Cout, int kh, int kw);
// out_L[ci][kh-1-dh][kw-1-dw][co] = s_L * w_L[co][dh][dw][ci], the four letters one after
// the other: the forward weights of the stride-1 input gradient; s = (+1, -1, -1, -1)
// (the conjugate, full form) when conj, else +1 (the separable form's signs are applied
// by the MMA table).
cudaError_t launch_bwd_transform(int Cin, int Cout, int kh, int kw, const void* const w[4],
                                 bool conj, void* out, int num_sms, cudaStream_t stream);
// dy [N][Ho][Wo][C] with s - 1 zeros inserted between pixels, [N][Hu][Wu][C] (C % 8 == 0,
// 16-byte aligned): the input of a strided forward's input-gradient convolution.
cudaError_t launch_bwd_upsample(const void* dy, int N, int Ho, int Wo, int C, int s, int Hu,
                                int Wu, void* u, int num_sms, cudaStream_t stream);
// dx [N][H][W][Cin] from dy [N][Ho][Wo][Cout] on CUDA cores, any stride.
cudaError_t launch_bwd_data_simt(const ConvShape& s, const void* dy, const void* const w[4],
                                 void* dx, cudaStream_t stream);
// Library-owned device scratch of quan_qconv2d_bwd_data_static (one per device, in the
// module's static device memory): its size, and its address on the current device.
constexpr size_t BWD_STATIC_SCRATCH_BYTES = size_t(2) << 20;
cudaError_t bwd_static_scratch_address(void** ptr);
// Tensor-core weight gradient, both forms (s.sep) (stride 1 or 2, Cin and Cout multiples of 64,
// Cout <= 256 or a multiple of 256, 16-byte aligned x and dy).  Zeroes dW_L, then adds.
bool bwd_weight_tc_supported(const ConvShape& s, const void* x, const void* dy);
cudaError_t launch_bwd_weight_tc(const ConvShape& s, const void* x, const void* dy,
                                 float* const dw[4], int num_sms,
                                 unsigned long long wait_limit_ns, cudaStream_t stream,
                                 char* err, size_t errlen);
// dW_L fp32 [Qout][kh][kw][Qin] (zeroed, then accumulated) on CUDA cores.
cudaError_t launch_bwd_weight_simt(const ConvShape& s, const void* x, const void* dy,
                                   float* const dw[4], int num_sms, cudaStream_t stream);

// Training-mode IQBN (Eq. 11-12) over bf16 [npix][C].  The 16-byte vector path needs C a
// multiple of 8 (at most 2048) and 16-byte aligned tensors; otherwise C <= 256.
bool iqbn_vec_ok(int C, const void* a, const void* b);
bool iqbn_supported(int C, const void* a, const void* b);
// Partial sums of at most IQBN_MAX_PARTIALS blocks: workspace fp32 [blocks][2][C].
constexpr int IQBN_MAX_PARTIALS = 1024;
size_t iqbn_stats_workspace_bytes(int C);
cudaError_t launch_iqbn_stats(const void* x, long long npix, int C, void* workspace,
                              float* mean, float* var, int num_sms, cudaStream_t stream);
cudaError_t launch_iqbn_apply(const void* x, long long npix, int C, const float* mean,
                              const float* var, const float* gamma, const float* beta, float eps,
                              int act, void* out, int num_sms, cudaStream_t stream);

// The 4-channel stem convolution and its 3x3/2, padding-1 max pooling in one kernel:
// out [N][(Ho - 1) / 2 + 1][(Wo - 1) / 2 + 1][64] bf16 (Cin = 4, Cout = 64, stride 2, even W,
// Wo <= 128).
bool tc_stem_pool_supported(const ConvShape& s, const void* x, const void* const w[4],
                            const void* out, const EpilogueArgs& ep);
cudaError_t launch_qconv_stem_pool(const ConvShape& s, const void* x, const void* const w[4],
                                   const EpilogueArgs& ep, void* out, const TcOptions& opt,
                                   int num_sms, cudaStream_t stream, char* err, size_t errlen);

// The same from fp32 RGB pixels [N][H][W][3] (W a multiple of 32), the Poincare mapping of
// Eq. 4 done in the kernel's loader; s is the convolution's shape (Cin = 4).
bool tc_stem_pool_rgb_supported(const ConvShape& s, const float* rgb, const void* const w[4],
                                const void* out, const EpilogueArgs& ep);
cudaError_t launch_qconv_stem_pool_rgb(const ConvShape& s, const float* rgb,
                                       const void* const w[4], const EpilogueArgs& ep, void* out,
                                       const TcOptions& opt, int num_sms, cudaStream_t stream,
                                       char* err, size_t errlen);

// Per-real-channel max pooling, bf16 NHWC.
cudaError_t launch_maxpool_bf16(const void* x, int N, int H, int W, int C, int k, int stride,
                                int pad, void* out, int num_sms, cudaStream_t stream);

}  // namespace quan
