/*
 * quan.h -- libquan: quaternion convolution for NVIDIA GB300 (sm_103a).
 *
 * Implements the QUAN quaternion convolution (Grant & Wang,
 * "Quaternion Approximate Networks for Enhanced Image Classification and Oriented
 * Object Detection", arXiv 2509.05512):
 *   - the full Hamilton-product convolution of Sec. III-B, Eq. 5, whose real
 *     weight is the signed 4x4 block matrix of Eq. 6 built from four letter tensors
 *     W_r, W_i, W_j, W_k (weight on the left: Y = W (x) X, Hamilton product of Eq. 3);
 *   - Independent Quaternion Batch Normalization in inference form (Sec. III-C,
 *     Eq. 11-12), folded by the caller into one scale and one shift per real channel;
 *   - a split (per real component) activation (ReLU or SiLU, Sec. IV-E ablation);
 *   - component-wise max pooling (the QSPPF pooling rule of Sec. III-D);
 *   - the Poincare RGB mapping of Eq. 4 (Sec. III-A);
 *   - the separable form of Eq. 7 and its backward pass (Eq. 8-10), and the backward
 *     pass of the full form (input and weight gradients before the epilogue);
 *   - IQBN in training mode: batch statistics (Eq. 11) and normalisation (Eq. 12).
 *
 * Conventions shared by every entry point
 *   Layout      x is NHWC [N][H][W][C_in]; the C_in real channels are four
 *               component-major blocks [r | i | j | k] of Q_in = C_in / 4 channels, so
 *               channel c = comp * Q_in + ci.  The output is [N][Ho][Wo][C_out] with
 *               the same component-major order.  Each letter tensor w_L is
 *               [Q_out][kh][kw][Q_in], contiguous.  Ho = (H + 2 pad - kh) / stride + 1
 *               (floor), likewise Wo.
 *   Convolution "convolution" is a cross-correlation (no kernel flip) with zero padding.
 *   Epilogue    out = act(scale[c] * (acc + bias[c]) + shift[c] (+ residual)), every
 *               per-channel vector fp32 [C_out]; a NULL bias is 0, a NULL scale/shift pair
 *               is the identity (scale and shift must both be NULL or both non-NULL).
 *   Memory      every tensor pointer is a DEVICE pointer owned by the caller; the library
 *               keeps no reference after the call and allocates nothing per call.
 *               `out` must not overlap any input.
 *   Streams     calls are asynchronous on `stream` (a cudaStream_t; NULL is the legacy
 *               default stream) and do not synchronise.  Kernels are launched with
 *               programmatic stream serialization: a convolution kernel may start while
 *               the preceding library kernel on the stream finishes, and waits for it
 *               before touching activations (input, residual, output).  Its weights and
 *               per-channel vectors may be read before that wait, so they must not be
 *               written by the immediately preceding call on the stream when that call is
 *               a forward convolution or quan_qconv2d_bwd_weight (any other producer, e.g.
 *               a framework kernel or a copy, completes before the call's kernels start).
 *   Errors      argument errors are detected on the host before anything is launched and
 *               return QUAN_ERR_INVALID_ARG or QUAN_ERR_UNSUPPORTED; a launch failure
 *               returns QUAN_ERR_CUDA.  quan_last_error_message() describes the last error
 *               of the calling thread.  Kernel-side timeouts are reported by
 *               quan_device_status().
 */
#ifndef QUAN_H_
#define QUAN_H_

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t. */
typedef struct CUstream_st* quan_stream_t;

typedef enum {
    QUAN_OK = 0,
    QUAN_ERR_INVALID_ARG = 1,     /* null pointer, bad size, C % 4 != 0, overlap, ... */
    QUAN_ERR_UNSUPPORTED = 2,     /* valid arguments no compiled path can run */
    QUAN_ERR_CUDA = 3,            /* CUDA runtime or launch error */
    QUAN_ERR_DEVICE_TIMEOUT = 4   /* a kernel's bounded wait ran out (quan_device_status) */
} quan_status_t;

typedef enum { QUAN_ACT_NONE = 0, QUAN_ACT_RELU = 1, QUAN_ACT_SILU = 2 } quan_act_t;

typedef enum {
    QUAN_PATH_AUTO = 0, /* tensor-core path when the shape allows it, else CUDA cores */
    QUAN_PATH_TC = 1,   /* tcgen05 implicit GEMM; UNSUPPORTED if the shape does not allow it */
    QUAN_PATH_SIMT = 2  /* CUDA-core direct convolution */
} quan_path_t;

/*
 * Quaternion convolution forward, bfloat16 tensors, fp32 accumulation.
 * Sec. III-B Eq. 5 (Hamilton product of Eq. 3 per tap and channel), Eq. 6 block weight,
 * IQBN inference epilogue of Eq. 11-12.
 *   x            bf16 [N][H][W][Cin]           (device)
 *   wr,wi,wj,wk  bf16 [Cout/4][kh][kw][Cin/4]  (device), the letter tensors of Eq. 5
 *   bias         fp32 [Cout] or NULL           (device)
 *   iqbn_scale   fp32 [Cout] or NULL           (device)  gamma / sqrt(var + eps)
 *   iqbn_shift   fp32 [Cout] or NULL           (device)  beta - mean * scale
 *   N,H,W        batch and input size, >= 1
 *   Cin, Cout    real channel counts, multiples of 4
 *   kh,kw        filter size >= 1; stride >= 1; pad >= 0; Ho, Wo >= 1
 *   act          quan_act_t
 *   out          bf16 [N][Ho][Wo][Cout]        (device), rounded to nearest even
 * The tensor-core path needs 16-byte aligned pointers (every tensor, the residual and the
 * per-channel vectors), fewer than 2^31 output
 * pixels and either Cin/4 and Cout/4 multiples of 16, or Cin = 4, Cout = 64, stride 2
 * and an even W (the 4-channel stem: kh * P <= 32, where P = ceil((kw + pad mod 2) / 2)
 * rounded up to even is the number of 2-pixel pairs a filter row spans); other shapes
 * run on CUDA cores.  Returns QUAN_OK once launched.
 */
quan_status_t quan_qconv2d_fwd(const void* x, const void* wr, const void* wi, const void* wj,
                               const void* wk, const float* bias, const float* iqbn_scale,
                               const float* iqbn_shift, int N, int H, int W, int Cin, int Cout,
                               int kh, int kw, int stride, int pad, int act, void* out,
                               quan_stream_t stream);

/* Same operation with fp32 x, weights and out (CUDA-core fp32 FFMA path). */
quan_status_t quan_qconv2d_fwd_f32(const float* x, const float* wr, const float* wi,
                                   const float* wj, const float* wk, const float* bias,
                                   const float* iqbn_scale, const float* iqbn_shift, int N, int H,
                                   int W, int Cin, int Cout, int kh, int kw, int stride, int pad,
                                   int act, float* out, quan_stream_t stream);

/*
 * bf16 quaternion convolution that adds `residual` (bf16 [N][Ho][Wo][Cout], device, same
 * layout as out; may not overlap out) after the IQBN affine and before the activation:
 *   out = act(scale * (acc + bias) + shift + residual).
 * This is the second convolution of a residual basic block in the ResNet-style backbone.
 */
quan_status_t quan_qconv2d_fwd_res(const void* x, const void* wr, const void* wi, const void* wj,
                                   const void* wk, const float* bias, const float* iqbn_scale,
                                   const float* iqbn_shift, int N, int H, int W, int Cin,
                                   int Cout, int kh, int kw, int stride, int pad, int act,
                                   const void* residual, void* out, quan_stream_t stream);

/*
 * quan_qconv2d_fwd (residual NULL) or quan_qconv2d_fwd_res (residual given) with a caller
 * workspace that lets the tensor-core kernel split its work evenly over the SMs (Eq. 5/6,
 * the same convolution and epilogue).  A layer whose output tiles make between one and two
 * waves of CTAs (the backbone's 7 x 7 layers: 196 tiles on 152 SMs) otherwise leaves most
 * SMs idle in its second wave; with the workspace each CTA takes an equal contiguous range
 * of the (tile, K block) iterations, a tile shared by two CTAs being finished by one of
 * them after adding the other's fp32 partial sums from the workspace.  Other layers run as
 * without the workspace.
 * The summation order differs from quan_qconv2d_fwd's, so results agree within rounding,
 * not bit for bit.
 *   workspace        device memory of at least quan_qconv2d_fwd_workspace_size() bytes,
 *                    256-byte aligned, owned by the caller, overlapping no tensor of the
 *                    call; ZERO-FILLED before its first use: every call leaves it as zero
 *                    again (after a QUAN_ERR_DEVICE_TIMEOUT, zero it once more).  Calls that
 *                    may run at the same time on the GPU need separate workspaces.  NULL
 *                    (with workspace_bytes 0) or a smaller workspace: no split, the call runs
 *                    as quan_qconv2d_fwd / quan_qconv2d_fwd_res.
 * Errors as quan_qconv2d_fwd; a NULL workspace with workspace_bytes > 0 or a workspace not
 * 256-byte aligned is QUAN_ERR_INVALID_ARG.
 */
size_t quan_qconv2d_fwd_workspace_size(void);
quan_status_t quan_qconv2d_fwd_ex(const void* x, const void* wr, const void* wi, const void* wj,
                                  const void* wk, const float* bias, const float* iqbn_scale,
                                  const float* iqbn_shift, int N, int H, int W, int Cin,
                                  int Cout, int kh, int kw, int stride, int pad, int act,
                                  const void* residual, void* workspace, size_t workspace_bytes,
                                  void* out, quan_stream_t stream);

/*
 * A convolution (Eq. 5/6, as quan_qconv2d_fwd: x, its letters, bias / IQBN scale / shift,
 * act -> out) and a 1x1 quaternion convolution of the same input x with the same stride and
 * no padding (the residual shortcut of a downsampling block, Sec. III-D: letters sc_w*
 * [Cout_sc/4][1][1][Cin/4], its own bias / IQBN scale / shift and activation -> out_sc
 * [N][Ho][Wo][Cout_sc]), both bf16, in one call.  The shortcut reads x at (ho stride,
 * wo stride), the pixel the convolution's filter tap (pad, pad) reads, so on the tensor
 * path the two run as one launch: the shortcut's output-channel tiles follow the
 * convolution's and run the K blocks of that tap only, with their own letters and
 * epilogue (quan_last_kernel() then names a "shortcut" instance).  Shapes without that form
 * (or the CUDA-core path) run as the two separate calls.  Each output equals, within
 * rounding, what quan_qconv2d_fwd gives for its layer; with the same tile overrides the
 * fused launch is bit-identical to separate calls on the quad/pair kernel.
 *   Requirements: pad < kh and pad < kw; (H - 1) / stride + 1 == Ho and likewise for W
 *   (the two outputs have one size); out and out_sc disjoint from each other and from every
 *   input.  No residual input, no split workspace.
 * Errors: QUAN_ERR_INVALID_ARG for argument errors of either layer or mismatched output
 * sizes; otherwise as quan_qconv2d_fwd.
 */
quan_status_t quan_qconv2d_fwd_shortcut(
    const void* x, const void* wr, const void* wi, const void* wj, const void* wk,
    const float* bias, const float* iqbn_scale, const float* iqbn_shift, int N, int H, int W,
    int Cin, int Cout, int kh, int kw, int stride, int pad, int act, const void* sc_wr,
    const void* sc_wi, const void* sc_wj, const void* sc_wk, const float* sc_bias,
    const float* sc_iqbn_scale, const float* sc_iqbn_shift, int Cout_sc, int sc_act, void* out,
    void* out_sc, quan_stream_t stream);

/*
 * The separable QUAN convolution of Eq. 7 (Sec. III-B), bf16, same arguments, layouts,
 * epilogue and errors as quan_qconv2d_fwd.  Each output component is a signed sum of the
 * four per-component convolutions c_p = W_p (*) x_p (p = r, i, j, k):
 *   y_r = c_r - c_i - c_j - c_k,   y_i = c_r + c_i + c_j - c_k,
 *   y_j = c_r - c_i + c_j + c_k,   y_k = c_r + c_i - c_j + c_k,
 * a quarter of the full form's multiply-adds (the cross-component terms W_L x_p, L != p,
 * are dropped, as the paper describes).  The tensor-core path needs Cin/4 and Cout/4
 * multiples of 16 and 16-byte aligned pointers; other shapes run on CUDA cores.  MMA-mode
 * overrides (quan_set_tc_tiles' mode) must be 0: UNSUPPORTED otherwise.
 */
quan_status_t quan_qconv2d_sep_fwd(const void* x, const void* wr, const void* wi,
                                   const void* wj, const void* wk, const float* bias,
                                   const float* iqbn_scale, const float* iqbn_shift, int N, int H,
                                   int W, int Cin, int Cout, int kh, int kw, int stride, int pad,
                                   int act, void* out, quan_stream_t stream);

/*
 * Poincare mapping of RGB pixels onto the unit quaternion sphere (Eq. 4, Sec. III-A), the
 * input mapping in front of the quaternion stem:
 *   n2 = r^2 + g^2 + b^2,   q = ((1 - n2), 2 r, 2 g, 2 b) / (1 + n2),
 * computed in fp32 and rounded to bf16 (nearest even).
 *   rgb   fp32 [npix][3] (device; e.g. NHWC with C = 3, npix = N H W), 4-byte aligned
 *   out   bf16 [npix][4] (device): channels [r|i|j|k] of one quaternion channel, the
 *         layout quan_qconv2d_fwd reads for Cin = 4; must not overlap rgb
 * npix = 0 is a no-op; npix < 0, a NULL pointer or a misaligned pointer returns
 * QUAN_ERR_INVALID_ARG.
 */
quan_status_t quan_poincare_fwd(const float* rgb, long long npix, void* out,
                                quan_stream_t stream);

/*
 * Backward pass of the convolution before its epilogue.  dy is dL/d(acc), the gradient of
 * the convolution's accumulator (the caller applies the activation, IQBN scale and bias
 * gradients first).  Layouts as in quan_qconv2d_fwd; dy is bf16 [N][Ho][Wo][Cout].
 *
 * Full form (Eq. 5): from the Jacobians of the Hamilton product (Eq. 3), per tap and
 * channel pair, dL/dX = conj(W) (x) dy and dL/dW = dy (x) conj(X), with
 * conj(q) = (q_r, -q_i, -q_j, -q_k).
 * Separable form (Eq. 7): Eq. 8-10.  The output gradients are mixed by the matrix M of
 * Eq. 9, g_p = sum_m M[p][m] dy_m (M transposed is Eq. 7's sign table), and then
 * dL/dx_p is the transposed convolution of g_p with W_p and dL/dW_p the correlation of g_p
 * with x_p, per component p.
 */

/*
 * Bytes of device workspace quan_qconv2d_bwd_data and quan_qconv2d_sep_bwd_data need:
 * the four transformed letter tensors, 4 * (Cin/4) * kh * kw * (Cout/4) bf16.  Returns 0
 * for sizes that are not positive or channel counts that are not multiples of 4.
 */
size_t quan_qconv2d_bwd_data_workspace_size(int Cin, int Cout, int kh, int kw);

/*
 * Workspace that lets quan_qconv2d_bwd_data (and _sep_) run a STRIDED forward's input
 * gradient on the tensor cores: the transformed letters, then dy with stride - 1 zeros
 * between its pixels, [N][H + 2 pad - kh + 1][W + 2 pad - kw + 1][Cout] bf16 (256-byte
 * aligned after the letters).  Equals quan_qconv2d_bwd_data_workspace_size for stride 1;
 * 0 for invalid sizes.  Arguments are the forward convolution's.
 */
size_t quan_qconv2d_bwd_data_workspace_size_ex(int N, int H, int W, int Cin, int Cout, int kh,
                                               int kw, int stride, int pad);

/*
 * Input gradient dx = dL/dx, bf16 [N][H][W][Cin] (device), rounded to nearest even from an
 * fp32 accumulation.  N..pad are the FORWARD convolution's arguments.
 *   workspace        device scratch of at least quan_qconv2d_bwd_data_workspace_size
 *                    bytes, 16-byte aligned for the tensor-core path, owned by the caller;
 *                    NULL or too small returns QUAN_ERR_INVALID_ARG.  Its contents are
 *                    overwritten; concurrent calls need separate workspaces.
 * dx must not overlap dy, the weights or the workspace.  For a square filter, pad < kh and
 * Cin/4, Cout/4 multiples of 16 on sm_103, the tensor-core path runs: one kernel writes
 * conj(W) with its channel axes swapped and the filter rotated by 180 degrees into the
 * workspace, then the forward tensor-core kernel convolves dy with it (stride 1, padding
 * kh - 1 - pad).  For a strided forward this needs the larger workspace of
 * quan_qconv2d_bwd_data_workspace_size_ex: dy is first spread out with zeros between its
 * pixels (stride - 1 of them), which multiplies the MMAs by stride^2 but keeps them on the
 * tensor cores.  Other shapes, or a strided forward with the smaller workspace, run a
 * direct CUDA-core kernel.
 * quan_set_path(QUAN_PATH_TC) makes a shape the tensor-core path cannot run fail with
 * QUAN_ERR_UNSUPPORTED.
 */
quan_status_t quan_qconv2d_bwd_data(const void* dy, const void* wr, const void* wi,
                                    const void* wj, const void* wk, int N, int H, int W, int Cin,
                                    int Cout, int kh, int kw, int stride, int pad,
                                    void* workspace, size_t workspace_bytes, void* dx,
                                    quan_stream_t stream);

/*
 * quan_qconv2d_bwd_data without the workspace argument, for callers that cannot allocate
 * device memory: code running where cudaMalloc is off limits (its implicit device-wide
 * synchronisation would stall other work, or a framework owns all device memory through
 * its own pool), or a plain C caller with no allocator at hand.  The paper has no
 * counterpart.  The transformed letters (and, for a strided forward, the spread-out dy
 * when both fit) go to a scratch buffer of 2 MiB (2097152 bytes) that the library keeps in
 * static device memory: every GPU that loads the library holds it until the process
 * exits; the call itself allocates and frees nothing.
 * Same arguments (minus the workspace), results and errors as quan_qconv2d_bwd_data with
 * a 2 MiB workspace, and the paths that workspace allows, plus QUAN_ERR_UNSUPPORTED when
 * quan_qconv2d_bwd_data_workspace_size exceeds 2 MiB (e.g. 1024 -> 1024 real channels
 * with a 3x3 filter: use quan_qconv2d_bwd_data with a workspace there).
 *   Sharing  every call on a device uses the same buffer, which keeps the last call's
 *            contents (each call rewrites all of it that it reads, so nothing has to start
 *            at zero).  Calls whose kernels overlap on the GPU (other streams, other host
 *            threads) race on it: order them (one stream, or events).
 *   Set-up   the first call on each device looks up the buffer's device address, with
 *            that device current; make that first call before any stream capture.  The
 *            address is kept for the life of the process: do not call cudaDeviceReset on a
 *            device between calls of this entry point (the library's module is then loaded
 *            again and the buffer may move).
 */
quan_status_t quan_qconv2d_bwd_data_static(const void* dy, const void* wr, const void* wi,
                                           const void* wj, const void* wk, int N, int H, int W,
                                           int Cin, int Cout, int kh, int kw, int stride,
                                           int pad, void* dx, quan_stream_t stream);

/* Separable form (Eq. 8-9) of the input gradient; same arguments and paths.  The
 * tensor-core path (a square filter, pad < kh, Cin/4 and Cout/4 multiples of 16) writes the
 * letters transposed and rotated (not conjugated) into the workspace and runs one
 * convolution of dy whose block (q, p) is M[q][p] W'_q, M of Eq. 9; other shapes run on
 * CUDA cores (the workspace is then checked but not used). */
quan_status_t quan_qconv2d_sep_bwd_data(const void* dy, const void* wr, const void* wi,
                                        const void* wj, const void* wk, int N, int H, int W,
                                        int Cin, int Cout, int kh, int kw, int stride, int pad,
                                        void* workspace, size_t workspace_bytes, void* dx,
                                        quan_stream_t stream);

/*
 * Weight gradients dwr..dwk = dL/dW_L, fp32 [Cout/4][kh][kw][Cin/4] each (device, 4-byte
 * aligned, pairwise disjoint and disjoint from x and dy): zeroed on the stream, then
 * accumulated over all N * Ho * Wo output pixels (fp32 partial sums added with atomics,
 * so the summation order, and the last bits, vary from run to run).  Stride 1 or 2 with Cin
 * and Cout multiples of 64 (Cout <= 256 or a multiple of 256) and 16-byte aligned x and dy
 * runs on the tensor cores (the real weight gradient of every tap as one product over
 * the pixels, folded into the four letters), other shapes on CUDA cores;
 * quan_set_path(QUAN_PATH_TC) makes those fail with QUAN_ERR_UNSUPPORTED.
 * x is the forward input, bf16 [N][H][W][Cin].
 */
quan_status_t quan_qconv2d_bwd_weight(const void* x, const void* dy, int N, int H, int W,
                                      int Cin, int Cout, int kh, int kw, int stride, int pad,
                                      float* dwr, float* dwi, float* dwj, float* dwk,
                                      quan_stream_t stream);

/* Separable form (Eq. 10) of the weight gradients; same arguments and paths (the
 * tensor-core kernel folds its blocks by Eq. 7's sign table). */
quan_status_t quan_qconv2d_sep_bwd_weight(const void* x, const void* dy, int N, int H, int W,
                                          int Cin, int Cout, int kh, int kw, int stride,
                                          int pad, float* dwr, float* dwi, float* dwj,
                                          float* dwk, quan_stream_t stream);

/*
 * Independent Quaternion Batch Normalization in training mode (Sec. III-C, Eq. 11-12):
 * every real channel (one component of one quaternion channel) is normalised with its own
 * statistics over the batch and the spatial positions.  x is bf16 [npix][C] (NHWC with
 * npix = N H W), device.  The CUDA-core kernels take C a multiple of 8 up to 2048 with
 * 16-byte aligned x (and out), or any C up to 256; other C return QUAN_ERR_UNSUPPORTED.
 *
 * quan_iqbn_batch_stats: mean[c] = E[x_c] and var[c] = E[(x_c - mean[c])^2] (the biased
 * variance of Eq. 11; the unbiased running estimate is var * npix / (npix - 1)), fp32 [C]
 * each, device, 4-byte aligned, disjoint from each other and from x.  `workspace` is
 * device scratch of at least quan_iqbn_batch_stats_workspace_size(C) bytes (4-byte
 * aligned, owned by the caller, overwritten; NULL or too small is QUAN_ERR_INVALID_ARG):
 * one row of per-block partial sums, added in a fixed order, so repeated calls on the
 * same input give the same bits.
 */
size_t quan_iqbn_batch_stats_workspace_size(int C);
quan_status_t quan_iqbn_batch_stats(const void* x, long long npix, int C, void* workspace,
                                    size_t workspace_bytes, float* mean, float* var,
                                    quan_stream_t stream);

/*
 * quan_iqbn_train_fwd: out = act(gamma[c] (x - mean[c]) / sqrt(var[c] + eps) + beta[c])
 * (Eq. 12 followed by the split activation), bf16 [npix][C], rounded to nearest even.
 * mean and var are typically quan_iqbn_batch_stats' outputs; gamma and beta fp32 [C] or
 * NULL (1 and 0).  out may be x itself (in place) but must not overlap it otherwise.
 * eps must be finite and >= 0.
 */
quan_status_t quan_iqbn_train_fwd(const void* x, long long npix, int C, const float* mean,
                                  const float* var, const float* gamma, const float* beta,
                                  float eps, int act, void* out, quan_stream_t stream);

/*
 * The 4-channel stem convolution followed by a 3x3, stride-2, padding-1 max pooling of
 * every real channel (Sec. III-D pooling rule), in one kernel that writes only the pooled
 * tensor: each CTA takes a band of pooled rows, computes the two convolution rows of each
 * (an MMA whose rows are the signed block weight of Eq. 6 stacked for both rows and whose
 * columns are the row's pixels) and takes the 3x3 max in registers.
 * The result is bit-identical to quan_qconv2d_fwd followed by quan_maxpool2d_fwd(k = 3,
 * stride 2, pad 1) (max commutes with the monotone bf16 rounding and, for ReLU or no
 * activation, with the monotone affine IQBN step).
 *   arguments   those of quan_qconv2d_fwd; out is bf16 [N][Hp][Wp][Cout] with
 *               Hp = (Ho - 1) / 2 + 1, Wp = (Wo - 1) / 2 + 1 (Ho, Wo of the convolution)
 *   workspace   not used (may be NULL, workspace_bytes 0): quan_qconv2d_maxpool_workspace_size
 *               returns 0 for every shape
 * Only the tensor-core pixel-pair shapes: sm_103, Cin = 4, Cout = 64, stride 2, even W,
 * Wo <= 128, (kh + 2) x (filter pixel pairs per row, rounded up to even) <= 36 (the 7x7
 * stem: 9 x 4), 16-byte aligned tensors; otherwise QUAN_ERR_UNSUPPORTED.  out must not
 * overlap an input (QUAN_ERR_INVALID_ARG).
 */
size_t quan_qconv2d_maxpool_workspace_size(int N, int H, int W, int Cout, int kh, int kw,
                                           int stride, int pad);
quan_status_t quan_qconv2d_maxpool_fwd(const void* x, const void* wr, const void* wi,
                                       const void* wj, const void* wk, const float* bias,
                                       const float* iqbn_scale, const float* iqbn_shift, int N,
                                       int H, int W, int Cin, int Cout, int kh, int kw,
                                       int stride, int pad, int act, void* workspace,
                                       size_t workspace_bytes, void* out,
                                       quan_stream_t stream);

/*
 * quan_qconv2d_maxpool_fwd from RGB pixels: the Poincare mapping of Eq. 4 (Sec. III-A),
 * q = ((1 - n2), 2 r, 2 g, 2 b) / (1 + n2) with n2 = r^2 + g^2 + b^2, fused into the stem
 * kernel's loader (each tile's input rows are loaded as fp32 RGB and turned into the bf16
 * quaternion pixels the MMAs read; the padding around the image is zero quaternions).
 * The result is bit-identical to quan_poincare_fwd followed by quan_qconv2d_maxpool_fwd.
 *   rgb         fp32 [N][H][W][3], 16-byte aligned, owned by the caller
 *   the rest    as quan_qconv2d_maxpool_fwd with Cin = 4 (no workspace)
 * Only W a multiple of 32 (and at most 2730) on top of quan_qconv2d_maxpool_fwd's shape
 * limits; otherwise QUAN_ERR_UNSUPPORTED.
 */
quan_status_t quan_qconv2d_maxpool_rgb_fwd(const float* rgb, const void* wr, const void* wi,
                                           const void* wj, const void* wk, const float* bias,
                                           const float* iqbn_scale, const float* iqbn_shift,
                                           int N, int H, int W, int Cout, int kh, int kw,
                                           int stride, int pad, int act, void* out,
                                           quan_stream_t stream);

/*
 * Max pooling of every real channel on its own (component-wise pooling of Sec. III-D,
 * QSPPF), bf16 NHWC [N][H][W][C] -> [N][Ho][Wo][C], window k x k, stride, zero-size
 * padding that never wins.  C is any positive count.
 */
quan_status_t quan_maxpool2d_fwd(const void* x, int N, int H, int W, int C, int k, int stride,
                                 int pad, void* out, quan_stream_t stream);

/* Select the path of later quan_qconv2d_fwd / _res calls in this process (default AUTO). */
quan_status_t quan_set_path(int path);
/* Path (quan_path_t, TC or SIMT) the last successful convolution call of this thread ran. */
int quan_last_path(void);
/* Name of the kernel (with its template variant) the last successful convolution call of
 * this thread launched, e.g. "qconv_ws_kernel<halo>"; "" before the first call.  The
 * string is owned by the library and stays valid until the thread's next call. */
const char* quan_last_kernel(void);

/*
 * Tensor-core tile override for later calls (0 = automatic): kappa = quaternion input
 * channels per K block (16, 32 or 64), bnq = quaternion output channels per tile
 * (16, 32 or 64), max_ctas = persistent grid size cap, mode = MMA decomposition
 * (1: one MMA per output/input component pair, N = bnq; 2: output components paired,
 * N = 2 bnq; 3: weight-stationary, the whole signed block weight expanded once per CTA
 * in shared memory, only for Cin = Cout = 64 and at most 9 taps; 4: pixel pairs,
 * weight-stationary with the input loaded as 16-byte pairs of adjacent pixels, one TMA
 * box per filter row, only for the Cin = 4 stem shapes above; mode 0 picks it for
 * those; 5: pointwise, the MMA's rows the expanded block weight of 32 quaternion output
 * channels and its columns 256 streamed pixels, only for 1x1 filters with pad 0, stride 1
 * or 2 (even H and W), Cin a multiple of 64 up to 512, Cout a multiple of 128 and no
 * residual; mode 0 picks it for those; 6: CTA pairs (tcgen05 cta_group::2), M = 256 MMAs
 * over two CTAs' pixels, each CTA keeping half of the signed block weight, only for
 * Cout = 128, Cin a multiple of 64 and kh x kw x Cin <= 1152; mode 0 picks it for 3x3
 * filters of stride 1 or 2 where a tile of whole output rows and its input rows (stride 2:
 * four boxes, one per parity of the input row and column) fit twice in shared memory;
 * 7: vertical taps stacked, for 3x3 stride-1 layers with Cin = Cout = 64 (pad <= 2): one
 * MMA multiplies a row of input pixels by the block weights of the three vertical taps of
 * one horizontal tap (N = 192), its three results going to three consecutive output rows
 * kept side by side in the accumulator; mode 0 picks it for those shapes, mode 3 keeps the
 * older weight-stationary kernel).  Values that do not
 * divide the layer, or a tile that does not fit in shared memory, make the call fail
 * with QUAN_ERR_UNSUPPORTED.
 */
quan_status_t quan_set_tc_tiles(int kappa, int bnq, int max_ctas, int mode);

/*
 * Weight-stationary pixel staging (default 1): for stride-1 layers whose output keeps the
 * input size and whose width is a multiple of 8 (at most 128), a tile is a block of whole
 * output rows and one TMA box per horizontal filter offset holds those rows plus their
 * vertical halo, shared by the vertical filter offsets.  0 stages one im2col box per
 * filter tap instead (same results).
 */
quan_status_t quan_set_tc_halo(int enable);

/*
 * MMA-issuing threads of the weight-stationary kernel (16 -> 16 quaternion channels):
 * 0 (default) chooses three when that still leaves every issuer as many pixel stages as
 * a tile has K blocks (at most three), else two; 2 or 3 force the count.  Any other
 * value returns QUAN_ERR_INVALID_ARG.  Results do not depend on it.  Process-wide, like
 * the other tile options.
 */
quan_status_t quan_set_tc_issuers(int issuers);

/*
 * Output rows per band of the vertical-tap kernel (mode 7): 0 (default) picks the height
 * with the fewest estimated MMA clocks over the grid's waves; 1 to 4 force it.  Any other
 * value returns QUAN_ERR_INVALID_ARG.  Results do not depend on it.  Process-wide.
 */
quan_status_t quan_set_tc_band_rows(int rows);

/* Time limit of every bounded wait inside the tensor-core kernel, in nanoseconds
 * (default 2e9).  0 restores the default. */
quan_status_t quan_set_wait_limit_ns(unsigned long long ns);

/*
 * Synchronises `stream`, then reads and clears the device status word that kernels set
 * when a bounded wait runs out.  Returns QUAN_ERR_DEVICE_TIMEOUT if any bit was set
 * (the bits are stored in *bits when bits != NULL), QUAN_ERR_CUDA on a CUDA error.
 */
quan_status_t quan_device_status(quan_stream_t stream, unsigned int* bits);

/* Test hook: when enabled, the tensor-core kernel's MMA role waits on a barrier nothing
 * arrives on, so every role's bounded wait runs out and the kernel reports a timeout
 * through quan_device_status() while leaving the context usable. */
quan_status_t quan_set_fault_injection(int enable);

const char* quan_status_string(quan_status_t status);
const char* quan_last_error_message(void);
/* Library version as major * 10000 + minor * 100 + patch. */
int quan_version(void);

#ifdef __cplusplus
}
#endif

#endif /* QUAN_H_ */
