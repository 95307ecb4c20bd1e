// qconv_tc.cu -- tensor-core quaternion convolution for sm_103a (tcgen05 + TMA).
//
// The quaternion convolution of Eq. 5 (Sec. III-B) is an implicit GEMM
//   Y[pixel][q, co] = sum_{tap, p, ci} X[pixel + tap][p, ci] * B[tap][p, ci][q, co]
// whose weight B is the signed 4x4 block (Hamilton) matrix of Eq. 6 built from four
// compact letter tensors W_r, W_i, W_j, W_k.  This kernel never materialises B, not
// even in shared memory: each K block stages the four input-component tiles X_p and
// the four compact letter tiles W_L, and issues 16 sub-MMAs
//   D_q += sign(q, p) * X_p * W_{L(q, p)}^T
// where the letter is picked by choosing the shared-memory descriptor and the sign by
// the instruction descriptor's negate bit.  Weight traffic is therefore 1/4 of the
// real-equivalent layer, and the sign flips are exact.
//
// Structure (one persistent CTA per SM, 6 warps):
//   warp 0      TMA producer: per K block (tap, chunk of KAPPA quaternion input channels)
//               4 im2col loads of X (zero padding comes from out-of-bounds fill) and
//               4 tiled loads of W_L, into a STAGES-deep ring;
//   warp 1      owns TMEM (2 accumulator buffers x 4 components x BNQ columns) and one
//               lane issues the tcgen05.mma / tcgen05.commit stream;
//   warps 2..5  epilogue: tcgen05.ld TMEM -> registers, act(scale*(acc+bias)+shift+res)
//               (IQBN inference form of Eq. 11-12), bf16 round-to-nearest, 16-byte stores
//               into the component-major NHWC output.  Double-buffered accumulators let
//               the epilogue of tile i overlap the main loop of tile i+1.
// Every mbarrier wait is bounded in time; a wait that runs out sets a bit in the device
// status word, raises a CTA-wide abort flag, drains the copies and MMAs still in flight,
// frees TMEM and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <cstdio>
#include <mutex>

#include "internal.h"
#include "ptx.cuh"

namespace quan {

__device__ unsigned int g_status;

namespace {

constexpr int BM = 128;           // output pixels per tile (MMA M)
constexpr int NUM_THREADS = 192;  // 6 warps
constexpr int UMMA_K = 16;        // K of one kind::f16 MMA

// Output component q takes input component p through letter L = q xor p, read off Eq. 5:
//   y_r: +W_r X_r  -W_i X_i  -W_j X_j  -W_k X_k
//   y_i: +W_i X_r  +W_r X_i  -W_k X_j  +W_j X_k
//   y_j: +W_j X_r  +W_k X_i  +W_r X_j  -W_i X_k
//   y_k: +W_k X_r  -W_j X_i  +W_i X_j  +W_r X_k
// Bit (4 q + p) of NEG_MASK marks the negative terms.
constexpr uint32_t NEG_MASK = (1u << 1) | (1u << 2) | (1u << 3)  // y_r: X_i, X_j, X_k
                              | (1u << 6)                        // y_i: X_j
                              | (1u << 11)                       // y_j: X_k
                              | (1u << 13);                      // y_k: X_i

struct TcParams {
    ConvShape s;
    EpilogueArgs ep;
    __nv_bfloat16* out;
    int kchunks;      // Qin / KAPPA
    int ktiles;       // kh * kw * kchunks K blocks per tile
    int num_n_tiles;  // Qout / BNQ
    int num_tiles;
    unsigned long long wait_limit_ns;
    int inject_stall;
    int a_reuse;      // keep each X_p tile in the A collector across its 4 sub-MMAs
};

template <int KAPPA, int BNQ>
struct Cfg {
    static constexpr int A_TILE = BM * KAPPA * 2;   // one component of the pixel tile
    static constexpr int B_TILE = BNQ * KAPPA * 2;  // one letter of the weight tile
    static constexpr int STAGE_BYTES = 4 * A_TILE + 4 * B_TILE;
    static constexpr int STAGES_RAW = (200 * 1024) / STAGE_BYTES;
    static constexpr int STAGES = STAGES_RAW > 8 ? 8 : (STAGES_RAW < 2 ? 2 : STAGES_RAW);
    static constexpr int TILES_BYTES = STAGES * STAGE_BYTES;
    static constexpr int NUM_BARS = 2 * STAGES + 5;  // full, empty, acc_full[2], acc_empty[2], drain
    static constexpr int SMEM_BYTES = 1024 + TILES_BYTES + NUM_BARS * 8 + 16;
    static constexpr uint32_t TMEM_COLS = 8 * BNQ;  // 2 buffers x 4 components x BNQ fp32 columns
    static constexpr int KSTEPS = KAPPA / UMMA_K;
    static constexpr uint32_t ROW_BYTES = KAPPA * 2;
    static constexpr uint32_t SBO = 8 * ROW_BYTES;  // pitch of 8-row core-matrix groups
    // smem descriptor layout type: 128B, 64B or 32B swizzle (rows of KAPPA bf16)
    static constexpr uint64_t LAYOUT = KAPPA == 64 ? 2ull : (KAPPA == 32 ? 4ull : 6ull);
    static_assert(KAPPA == 16 || KAPPA == 32 || KAPPA == 64, "KAPPA");
    static_assert(BNQ == 16 || BNQ == 32 || BNQ == 64, "BNQ");
    static_assert(SMEM_BYTES <= 227 * 1024, "shared memory");
};

// tcgen05 shared-memory matrix descriptor for a K-major, swizzled operand tile.
__device__ __forceinline__ uint64_t make_sdesc(uint32_t saddr, uint32_t sbo, uint64_t layout) {
    uint64_t d = 0;
    d |= static_cast<uint64_t>((saddr & 0x3FFFFu) >> 4);             // start address
    d |= static_cast<uint64_t>(1) << 16;                               // LBO (unused here)
    d |= static_cast<uint64_t>((sbo >> 4) & 0x3FFFu) << 32;            // SBO
    d |= static_cast<uint64_t>(1) << 46;                               // descriptor version
    d |= layout << 61;                                                 // swizzle mode
    return d;
}

// Instruction descriptor, kind::f16: bf16 A and B, fp32 D, both operands K-major.
__host__ __device__ constexpr uint32_t make_idesc(int M, int N, int negate) {
    return (1u << 4)                                   // D format: f32
           | (1u << 7)                                 // A format: bf16
           | (1u << 10)                                // B format: bf16
           | (static_cast<uint32_t>(negate) << 13)     // negate A
           | (static_cast<uint32_t>(N >> 3) << 17)     // N / 8
           | (static_cast<uint32_t>(M >> 4) << 24);    // M / 16
}

__device__ __forceinline__ float activate(float z, int act) {
    if (act == 1) return fmaxf(z, 0.0f);
    if (act == 2) return z / (1.0f + __expf(-z));
    return z;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&v);
}

__device__ __forceinline__ bool wait_or_abort(uint32_t bar, uint32_t parity, uint64_t limit,
                                              volatile int* abort_flag, unsigned code) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    while (true) {
        if (mbar_try_wait(bar, parity)) return true;
        if (*abort_flag) return false;
        if (global_timer_ns() - t0 > limit) {
            atomicOr(&g_status, code);
            *abort_flag = 1;
            return false;
        }
    }
}

template <int KAPPA, int BNQ>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    qconv_tc_kernel(const __grid_constant__ CUtensorMap tmap_x,
                    const __grid_constant__ CUtensorMap tmap_wr,
                    const __grid_constant__ CUtensorMap tmap_wi,
                    const __grid_constant__ CUtensorMap tmap_wj,
                    const __grid_constant__ CUtensorMap tmap_wk, const TcParams p) {
    using C = Cfg<KAPPA, BNQ>;
    constexpr int STAGES = C::STAGES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::TILES_BYTES);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::NUM_BARS);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
    auto accf_bar = [&](int b) { return bar0 + 8u * (2 * STAGES + b); };
    auto acce_bar = [&](int b) { return bar0 + 8u * (2 * STAGES + 2 + b); };
    const uint32_t drain_bar = bar0 + 8u * (2 * STAGES + 4);

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const ConvShape& s = p.s;
    const uint64_t limit = p.wait_limit_ns;

    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            mbar_init(full_bar(i), 1);
            mbar_init(empty_bar(i), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(accf_bar(b), 1);
            mbar_init(acce_bar(b), 4 * 32);
        }
        mbar_init(drain_bar, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmap_x);
        tma_prefetch_desc(&tmap_wr);
        tma_prefetch_desc(&tmap_wi);
        tma_prefetch_desc(&tmap_wj);
        tma_prefetch_desc(&tmap_wk);
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    const int hw = s.Ho * s.Wo;

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint64_t pol_x = l2_policy_evict_normal();
            const uint64_t pol_w = l2_policy_evict_last();
            int stage = 0;
            uint32_t phase = 0;
            uint32_t filled = 0, fill_parity = 0;  // per-stage: ever filled, parity of last fill
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < p.num_tiles; tile += gridDim.x) {
                const int m_tile = tile / p.num_n_tiles;
                const int n_tile = tile - m_tile * p.num_n_tiles;
                const long long m0 = static_cast<long long>(m_tile) * BM;
                const int img = static_cast<int>(m0 / hw);
                const int rem = static_cast<int>(m0 - static_cast<long long>(img) * hw);
                const int ho = rem / s.Wo, wo = rem - (rem / s.Wo) * s.Wo;
                const int wbase = wo * s.stride - s.pad, hbase = ho * s.stride - s.pad;
                for (int kt = 0; kt < p.ktiles; ++kt) {
                    const int tap = kt / p.kchunks, chunk = kt - tap * p.kchunks;
                    const int dh = tap / s.kw, dw = tap - (tap / s.kw) * s.kw;
                    if (!wait_or_abort(empty_bar(stage), phase ^ 1u, limit, abort_flag,
                                       STATUS_TIMEOUT_PRODUCER)) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(full_bar(stage), C::STAGE_BYTES);
                    filled |= 1u << stage;
                    fill_parity = (fill_parity & ~(1u << stage)) | (phase << stage);
                    const uint32_t a0 = sbase + stage * C::STAGE_BYTES;
                    const uint32_t b0 = a0 + 4 * C::A_TILE;
                    const int cin0 = chunk * KAPPA;
#pragma unroll
                    for (int comp = 0; comp < 4; ++comp)
                        tma_load_im2col_4d(a0 + comp * C::A_TILE, &tmap_x, full_bar(stage),
                                           comp * s.Qin + cin0, wbase, hbase, img,
                                           static_cast<uint16_t>(dw), static_cast<uint16_t>(dh),
                                           pol_x);
                    const int wcol = tap * s.Qin + cin0, wrow = n_tile * BNQ;
                    tma_load_2d(b0 + 0 * C::B_TILE, &tmap_wr, full_bar(stage), wcol, wrow, pol_w);
                    tma_load_2d(b0 + 1 * C::B_TILE, &tmap_wi, full_bar(stage), wcol, wrow, pol_w);
                    tma_load_2d(b0 + 2 * C::B_TILE, &tmap_wj, full_bar(stage), wcol, wrow, pol_w);
                    tma_load_2d(b0 + 3 * C::B_TILE, &tmap_wk, full_bar(stage), wcol, wrow, pol_w);
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (!ok) {
                // Copies already issued complete on their own; wait for each stage's most
                // recent fill so that no copy targets this CTA's memory after it exits.
                for (int i = 0; i < STAGES; ++i) {
                    if (!(filled & (1u << i))) continue;
                    const uint64_t t0 = global_timer_ns();
                    while (!mbar_try_wait(full_bar(i), (fill_parity >> i) & 1u)) {
                        if (global_timer_ns() - t0 > limit) {
                            atomicOr(&g_status, STATUS_TIMEOUT_DRAIN);
                            break;
                        }
                    }
                }
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t IDESC_POS = make_idesc(BM, BNQ, 0);
            constexpr uint32_t IDESC_NEG = make_idesc(BM, BNQ, 1);
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            int issued = 0;
            if (p.inject_stall) {
                // Failure injection: wait on a barrier nothing arrives on, so that every
                // role runs into its bounded wait and the kernel reports a timeout.
                ok = wait_or_abort(drain_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
                ok = false;
            }
            int local = 0;
            for (int tile = blockIdx.x; ok && tile < p.num_tiles; tile += gridDim.x, ++local) {
                const int buf = local & 1;
                const uint32_t use = static_cast<uint32_t>(local >> 1) & 1u;
                if (!wait_or_abort(acce_bar(buf), use ^ 1u, limit, abort_flag,
                                   STATUS_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t dbase = tmem_base + static_cast<uint32_t>(buf * 4 * BNQ);
                for (int kt = 0; kt < p.ktiles; ++kt) {
                    if (!wait_or_abort(full_bar(stage), phase, limit, abort_flag,
                                       STATUS_TIMEOUT_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a0 = sbase + stage * C::STAGE_BYTES;
                    const uint32_t b0 = a0 + 4 * C::A_TILE;
#pragma unroll
                    for (int pc = 0; pc < 4; ++pc) {
#pragma unroll
                        for (int ks = 0; ks < C::KSTEPS; ++ks) {
                            const uint64_t adesc = make_sdesc(
                                a0 + pc * C::A_TILE + ks * (UMMA_K * 2), C::SBO, C::LAYOUT);
                            const uint32_t acc = (kt | pc | ks) != 0 ? 1u : 0u;
#pragma unroll
                            for (int q = 0; q < 4; ++q) {
                                const int L = q ^ pc;
                                const uint64_t bdesc = make_sdesc(
                                    b0 + L * C::B_TILE + ks * (UMMA_K * 2), C::SBO, C::LAYOUT);
                                const bool neg = (NEG_MASK >> (4 * q + pc)) & 1u;
                                const uint32_t idesc = neg ? IDESC_NEG : IDESC_POS;
                                if (p.a_reuse)
                                    umma_f16_collect(dbase + q * BNQ, adesc, bdesc, idesc, acc,
                                                     q == 0 ? 0 : (q == 3 ? 2 : 1));
                                else
                                    umma_f16(dbase + q * BNQ, adesc, bdesc, idesc, acc);
                            }
                        }
                    }
                    ++issued;
                    umma_commit(empty_bar(stage));  // frees the stage when these MMAs finish
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (!ok) break;
                umma_commit(accf_bar(buf));  // accumulator buffer ready for the epilogue
            }
            if (!ok && issued > 0) {
                // Let every MMA already issued finish before TMEM is released.
                umma_commit(drain_bar);
                const uint64_t t0 = global_timer_ns();
                while (!mbar_try_wait(drain_bar, 0u)) {
                    if (global_timer_ns() - t0 > limit) {
                        atomicOr(&g_status, STATUS_TIMEOUT_DRAIN);
                        break;
                    }
                }
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue
        const int quad = warp & 3;  // TMEM lane quadrant this warp may access
        const int row = quad * 32 + lane;
        const int Cout = s.Cout;
        const __nv_bfloat16* res = static_cast<const __nv_bfloat16*>(p.ep.residual);
        int local = 0;
        for (int tile = blockIdx.x; tile < p.num_tiles; tile += gridDim.x, ++local) {
            const int buf = local & 1;
            const uint32_t use = static_cast<uint32_t>(local >> 1) & 1u;
            if (!wait_or_abort(accf_bar(buf), use, limit, abort_flag, STATUS_TIMEOUT_EPILOGUE))
                break;
            tc_fence_after();
            const int m_tile = tile / p.num_n_tiles;
            const int n_tile = tile - m_tile * p.num_n_tiles;
            const long long m = static_cast<long long>(m_tile) * BM + row;
            const bool valid = m < s.M;
            const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                                   static_cast<uint32_t>(buf * 4 * BNQ);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
#pragma unroll
                for (int j0 = 0; j0 < BNQ; j0 += 16) {
                    uint32_t v[16];
                    tmem_ld_32x32b_x16(taddr + q * BNQ + j0, v);
                    tmem_ld_wait();
                    if (valid) {
                        const int c0 = q * s.Qout + n_tile * BNQ + j0;
                        float z[16];
#pragma unroll
                        for (int t = 0; t < 16; ++t) z[t] = __uint_as_float(v[t]);
                        if (p.ep.bias) {
#pragma unroll
                            for (int t = 0; t < 16; ++t) z[t] += __ldg(p.ep.bias + c0 + t);
                        }
                        if (p.ep.scale) {
#pragma unroll
                            for (int t = 0; t < 16; ++t)
                                z[t] = fmaf(__ldg(p.ep.scale + c0 + t), z[t],
                                            __ldg(p.ep.shift + c0 + t));
                        }
                        if (res) {
                            const uint4* rp =
                                reinterpret_cast<const uint4*>(res + m * Cout + c0);
                            const uint4 r0 = __ldg(rp), r1 = __ldg(rp + 1);
                            const __nv_bfloat162* h0 = reinterpret_cast<const __nv_bfloat162*>(&r0);
                            const __nv_bfloat162* h1 = reinterpret_cast<const __nv_bfloat162*>(&r1);
#pragma unroll
                            for (int t = 0; t < 4; ++t) {
                                const float2 f0 = __bfloat1622float2(h0[t]);
                                const float2 f1 = __bfloat1622float2(h1[t]);
                                z[2 * t] += f0.x;
                                z[2 * t + 1] += f0.y;
                                z[8 + 2 * t] += f1.x;
                                z[8 + 2 * t + 1] += f1.y;
                            }
                        }
                        uint4 o0, o1;
                        o0.x = pack_bf16x2(activate(z[0], s.act), activate(z[1], s.act));
                        o0.y = pack_bf16x2(activate(z[2], s.act), activate(z[3], s.act));
                        o0.z = pack_bf16x2(activate(z[4], s.act), activate(z[5], s.act));
                        o0.w = pack_bf16x2(activate(z[6], s.act), activate(z[7], s.act));
                        o1.x = pack_bf16x2(activate(z[8], s.act), activate(z[9], s.act));
                        o1.y = pack_bf16x2(activate(z[10], s.act), activate(z[11], s.act));
                        o1.z = pack_bf16x2(activate(z[12], s.act), activate(z[13], s.act));
                        o1.w = pack_bf16x2(activate(z[14], s.act), activate(z[15], s.act));
                        uint4* op = reinterpret_cast<uint4*>(p.out + m * Cout + c0);
                        op[0] = o0;
                        op[1] = o1;
                    }
                }
            }
            tc_fence_before();
            mbar_arrive(acce_bar(buf));
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, C::TMEM_COLS);
    }
}

// ---------------------------------------------------------------- host side
PFN_cuTensorMapEncodeTiled_v12000 g_encode_tiled = nullptr;
PFN_cuTensorMapEncodeIm2col_v12000 g_encode_im2col = nullptr;
std::once_flag g_encode_once;

bool load_encoders() {
    std::call_once(g_encode_once, [] {
        cudaDriverEntryPointQueryResult q1, q2;
        void* f1 = nullptr;
        void* f2 = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f1, 12000,
                                             cudaEnableDefault, &q1) == cudaSuccess &&
            q1 == cudaDriverEntryPointSuccess)
            g_encode_tiled = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f1);
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeIm2col", &f2, 12000,
                                             cudaEnableDefault, &q2) == cudaSuccess &&
            q2 == cudaDriverEntryPointSuccess)
            g_encode_im2col = reinterpret_cast<PFN_cuTensorMapEncodeIm2col_v12000>(f2);
    });
    return g_encode_tiled != nullptr && g_encode_im2col != nullptr;
}

CUtensorMapSwizzle swizzle_for(int kappa) {
    return kappa == 64 ? CU_TENSOR_MAP_SWIZZLE_128B
                       : (kappa == 32 ? CU_TENSOR_MAP_SWIZZLE_64B : CU_TENSOR_MAP_SWIZZLE_32B);
}

bool encode_x(CUtensorMap* map, const ConvShape& s, const void* x, int kappa) {
    const cuuint64_t dims[4] = {static_cast<cuuint64_t>(s.Cin), static_cast<cuuint64_t>(s.W),
                                static_cast<cuuint64_t>(s.H), static_cast<cuuint64_t>(s.N)};
    const cuuint64_t strides[3] = {static_cast<cuuint64_t>(s.Cin) * 2,
                                   static_cast<cuuint64_t>(s.Cin) * 2 * s.W,
                                   static_cast<cuuint64_t>(s.Cin) * 2 * s.W * s.H};
    // Bounding box of filter origins: from -pad to (dim - 1) + pad - (k - 1), per
    // spatial dimension, innermost (W) first.
    const int lower[2] = {-s.pad, -s.pad};
    const int upper[2] = {s.pad - (s.kw - 1), s.pad - (s.kh - 1)};
    const cuuint32_t estr[4] = {1, static_cast<cuuint32_t>(s.stride),
                                static_cast<cuuint32_t>(s.stride), 1};
    const CUresult r = g_encode_im2col(
        map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(x), dims, strides, lower,
        upper, static_cast<cuuint32_t>(kappa), BM, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
        swizzle_for(kappa), CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool encode_w(CUtensorMap* map, const ConvShape& s, const void* w, int kappa, int bnq) {
    const cuuint64_t kw_cols = static_cast<cuuint64_t>(s.kh) * s.kw * s.Qin;
    const cuuint64_t dims[2] = {kw_cols, static_cast<cuuint64_t>(s.Qout)};
    const cuuint64_t strides[1] = {kw_cols * 2};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(kappa), static_cast<cuuint32_t>(bnq)};
    const cuuint32_t estr[2] = {1, 1};
    const CUresult r = g_encode_tiled(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2,
                                      const_cast<void*>(w), dims, strides, box, estr,
                                      CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle_for(kappa),
                                      CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                                      CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

template <int KAPPA, int BNQ>
cudaError_t launch_cfg(const CUtensorMap maps[5], const TcParams& prm, int grid,
                       cudaStream_t stream) {
    using C = Cfg<KAPPA, BNQ>;
    auto kern = qconv_tc_kernel<KAPPA, BNQ>;
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, C::SMEM_BYTES);
    if (e != cudaSuccess) return e;
    kern<<<grid, NUM_THREADS, C::SMEM_BYTES, stream>>>(maps[0], maps[1], maps[2], maps[3],
                                                       maps[4], prm);
    return cudaGetLastError();
}

int pick_kappa(int Qin, int req) {
    if (req == 16 || req == 32 || req == 64) return Qin % req == 0 ? req : 0;
    if (Qin % 32 == 0) return 32;
    return 16;
}

int pick_bnq(int Qout, int req) {
    if (req == 16 || req == 32 || req == 64) return Qout % req == 0 ? req : 0;
    if (Qout % 64 == 0) return 64;
    if (Qout % 32 == 0) return 32;
    return 16;
}

}  // namespace

bool tc_supported(const ConvShape& s, const void* x, const void* const w[4], const void* out,
                  const void* residual) {
    auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
    if (s.Qin % 16 != 0 || s.Qout % 16 != 0) return false;
    if (!al16(x) || !al16(out) || !al16(w[0]) || !al16(w[1]) || !al16(w[2]) || !al16(w[3]))
        return false;
    if (residual && !al16(residual)) return false;
    if (s.stride > 8) return false;
    // im2col bounding-box corner offsets must fit the 4-D encoding range [-128, 127]
    if (s.pad > 127 || s.pad - (s.kh - 1) < -128 || s.pad - (s.kw - 1) < -128) return false;
    if (s.kh * s.kw > 65535) return false;
    if (s.kh > 65536 || s.kw > 65536) return false;
    return true;
}

cudaError_t launch_qconv_tc(const ConvShape& s, const void* x, const void* const w[4],
                            const EpilogueArgs& ep, void* out, const TcOptions& opt,
                            int num_sms, cudaStream_t stream, char* err, size_t errlen) {
    if (!load_encoders()) {
        snprintf(err, errlen, "tensor-map encoders unavailable from the CUDA driver");
        return cudaErrorNotSupported;
    }
    const int kappa = pick_kappa(s.Qin, opt.kappa);
    const int bnq = pick_bnq(s.Qout, opt.bnq);
    if (kappa == 0 || bnq == 0) {
        snprintf(err, errlen, "requested tile (kappa=%d, bnq=%d) does not divide Qin=%d/Qout=%d",
                 opt.kappa, opt.bnq, s.Qin, s.Qout);
        return cudaErrorInvalidValue;
    }
    CUtensorMap maps[5];
    if (!encode_x(&maps[0], s, x, kappa)) {
        snprintf(err, errlen, "cuTensorMapEncodeIm2col failed for the activation tensor");
        return cudaErrorInvalidValue;
    }
    for (int l = 0; l < 4; ++l)
        if (!encode_w(&maps[1 + l], s, w[l], kappa, bnq)) {
            snprintf(err, errlen, "cuTensorMapEncodeTiled failed for weight letter %d", l);
            return cudaErrorInvalidValue;
        }
    TcParams prm;
    prm.s = s;
    prm.ep = ep;
    prm.out = static_cast<__nv_bfloat16*>(out);
    prm.kchunks = s.Qin / kappa;
    prm.ktiles = s.kh * s.kw * prm.kchunks;
    prm.num_n_tiles = s.Qout / bnq;
    const long long m_tiles = (s.M + BM - 1) / BM;
    const long long tiles = m_tiles * prm.num_n_tiles;
    if (tiles > 0x7fffffffLL) {
        snprintf(err, errlen, "too many tiles");
        return cudaErrorInvalidValue;
    }
    prm.num_tiles = static_cast<int>(tiles);
    prm.wait_limit_ns = opt.wait_limit_ns;
    prm.inject_stall = opt.inject_stall;
    prm.a_reuse = opt.a_reuse;
    int grid = opt.max_ctas > 0 ? opt.max_ctas : num_sms;
    if (grid > prm.num_tiles) grid = prm.num_tiles;
    if (grid < 1) grid = 1;

#define QUAN_TC_CASE(K, B) \
    if (kappa == K && bnq == B) return launch_cfg<K, B>(maps, prm, grid, stream);
    QUAN_TC_CASE(16, 16)
    QUAN_TC_CASE(16, 32)
    QUAN_TC_CASE(16, 64)
    QUAN_TC_CASE(32, 16)
    QUAN_TC_CASE(32, 32)
    QUAN_TC_CASE(32, 64)
    QUAN_TC_CASE(64, 16)
    QUAN_TC_CASE(64, 32)
    QUAN_TC_CASE(64, 64)
#undef QUAN_TC_CASE
    snprintf(err, errlen, "no kernel instance for kappa=%d bnq=%d", kappa, bnq);
    return cudaErrorInvalidValue;
}

cudaError_t read_and_clear_status(unsigned* status, cudaStream_t stream) {
    cudaError_t e = cudaMemcpyFromSymbolAsync(status, g_status, sizeof(unsigned), 0,
                                              cudaMemcpyDeviceToHost, stream);
    if (e != cudaSuccess) return e;
    e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) return e;
    const unsigned zero = 0;
    e = cudaMemcpyToSymbolAsync(g_status, &zero, sizeof(unsigned), 0, cudaMemcpyHostToDevice,
                                stream);
    if (e != cudaSuccess) return e;
    return cudaStreamSynchronize(stream);
}

}  // namespace quan
