// qconv_tc.cu -- tensor-core quaternion convolution for sm_103a (tcgen05 + TMA).
//
// The quaternion convolution of Eq. 5 (Sec. III-B) is an implicit GEMM
//   Y[pixel][q, co] = sum_{tap, p, ci} X[pixel + tap][p, ci] * B[tap][p, ci][q, co]
// whose weight B is the signed 4x4 block (Hamilton) matrix of Eq. 6 built from four
// compact letter tensors W_r, W_i, W_j, W_k.  The block weight is never written to
// global memory: each K block stages the four input-component tiles X_p and the
// compact letter tiles, and the signed block structure is produced by choosing, per
// MMA, which letter tile the B descriptor points at and the instruction's negate bit.
// Weight traffic is therefore 1/4 of the real-equivalent layer.
//
// Two MMA decompositions (template MODE):
//   MODE_QUAD  16 MMAs per 16-wide K step, one per (output q, input p):
//                D_q += sign(q, p) * X_p * W_{q xor p}^T            (N = BNQ)
//   MODE_PAIR  8 MMAs per K step, each covering two output components:
//                [D_r | D_i] and [D_j | D_k] += +-X_p * S^T         (N = 2 BNQ)
//              where S is a stack of two letter blocks.  The four stacks Eq. 6 needs,
//              [W_r; W_i], [-W_i; W_r], [W_j; W_k], [W_k; -W_j] (up to an overall sign),
//              are all windows of the two 3-block sequences
//                [-W_i | W_r | W_i]  and  [W_j | W_k | -W_j],
//              so a stage holds 6 letter blocks (W_i and W_j are loaded twice) and a
//              helper warp flips the sign bits of the two negated copies.  The larger N
//              keeps the tensor pipe busy (an M=128 MMA costs at least ~45 cycles on
//              this part, a full N=64 one is 32 cycles of work, N=128 is 64).
//
//   MODE_WS    (16 -> 16 quaternion channels, at most 9 taps) weight-stationary: every CTA
//              expands the whole signed block weight of Eq. 6 into shared memory once
//              (read from the compact letters, 72 KB for 3x3), then streams one im2col
//              box per tap that holds all four input components (64 channels, 128-byte
//              rows); 4 MMAs of N = 64 per tap cover all four output components.
//
// Structure (one persistent CTA per SM, 12 warps):
//   warps 0, 3  TMA producers: per K block (tap, chunk of KAPPA quaternion input channels)
//               warp 0 issues the 4 im2col loads of X (zero padding comes from
//               out-of-bounds fill) and warp 3 the letter tiles, into a STAGES-deep ring
//               (a single thread issues TMA copies at a limited rate);
//   warp 1      owns TMEM (2 accumulator buffers x 4 components x BNQ columns); one lane
//               issues the tcgen05.mma / tcgen05.commit stream;
//   warp 2      MODE_PAIR only: writes the two sign-flipped letter copies of each stage;
//   warps 4..11 epilogue, two warps per TMEM lane quadrant, each half of them owning two
//               output components: tcgen05.ld TMEM -> registers,
//               act(scale*(acc+bias)+shift+res) (IQBN inference form of Eq. 11-12) with
//               the per-channel vectors staged in shared memory, bf16 round-to-nearest
//               into a swizzled shared-memory tile, TMA store into the component-major
//               NHWC output (rows past the last pixel are clipped by the tensor map).
//               Double-buffered accumulators let the epilogue of tile i overlap the
//               main loop of tile i+1.
// Every mbarrier wait is bounded in time; a wait that runs out sets a bit in the device
// status word, raises a CTA-wide abort flag, drains the copies and MMAs still in flight,
// frees TMEM and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <cstdio>
#include <mutex>

#include "internal.h"
#include "ptx.cuh"

namespace quan {

__device__ unsigned int g_status;

namespace {

constexpr int BM = 128;           // output pixels per tile (MMA M)
constexpr int NUM_THREADS = 384;  // 12 warps
constexpr int MODE_QUAD = 0;
constexpr int MODE_PAIR = 1;
constexpr int MODE_WS = 2;
constexpr int WS_MAX_TAPS = 9;
constexpr int EPI_WARP0 = 4;
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
    const __nv_bfloat16* w[4];  // compact letter tensors (read directly by MODE_WS)
};

template <int KAPPA, int BNQ, int MODE>
struct Cfg {
    // pixel-tile row: KAPPA channels of one component, or all four components (WS)
    static constexpr int A_ROW_BYTES = (MODE == MODE_WS ? 4 * KAPPA : KAPPA) * 2;
    static constexpr int A_TILE = BM * A_ROW_BYTES;
    static constexpr int A_TILES = MODE == MODE_WS ? 1 : 4;
    static constexpr int B_TILE = BNQ * KAPPA * 2;  // one letter block of the weight tile
    static constexpr int B_SLOTS = MODE == MODE_PAIR ? 6 : (MODE == MODE_QUAD ? 4 : 0);
    static constexpr int STAGE_BYTES = A_TILES * A_TILE + B_SLOTS * B_TILE;
    // bytes the TMA copies per stage (pair mode writes two slots itself)
    static constexpr int STAGE_TX = A_TILES * A_TILE + (B_SLOTS ? 4 : 0) * B_TILE;
    // resident expanded weight (WS): per tap a [4 BNQ rows x 4 KAPPA] K-major tile
    static constexpr int WSB_TAP = MODE == MODE_WS ? 4 * BNQ * 4 * KAPPA * 2 : 0;
    static constexpr int WSB_BYTES = MODE == MODE_WS ? WS_MAX_TAPS * WSB_TAP : 0;
    static constexpr int OUT_TILE = BM * BNQ * 2;        // one output component block, bf16
    static constexpr int STAGING_BYTES = 2 * OUT_TILE;   // one block per epilogue half
    static constexpr int PARAM_BYTES = 3 * 4 * BNQ * 4;  // bias, scale, shift of a tile
    static constexpr int FIXED_BYTES = 1024 + WSB_BYTES + STAGING_BYTES + PARAM_BYTES + 512;
    static constexpr int STAGES_RAW = (227 * 1024 - FIXED_BYTES) / STAGE_BYTES;
    static constexpr int STAGES = STAGES_RAW > 8 ? 8 : (STAGES_RAW < 2 ? 2 : STAGES_RAW);
    static constexpr int TILES_BYTES = STAGES * STAGE_BYTES;
    static constexpr int WSB_OFF = TILES_BYTES;
    static constexpr int STAGING_OFF = WSB_OFF + WSB_BYTES;
    static constexpr int PARAM_OFF = STAGING_OFF + STAGING_BYTES;
    static constexpr int BAR_OFF = PARAM_OFF + PARAM_BYTES;
    // output staging swizzle: rows of BNQ bf16 (128, 64 or 32 bytes)
    static constexpr uint32_t OUT_ROW = BNQ * 2;
    static constexpr uint32_t OUT_SW_MASK = BNQ == 64 ? 7u : (BNQ == 32 ? 3u : 1u);
    // full (pixels), full (letters), empty, ready (negated copies done), acc_full[2],
    // acc_empty[2], drain, expanded weight ready (WS)
    static constexpr int NUM_BARS = 4 * STAGES + 6;
    static constexpr int SMEM_BYTES = 1024 + BAR_OFF + NUM_BARS * 8 + 16;
    static constexpr bool FITS = SMEM_BYTES <= 227 * 1024;
    static constexpr uint32_t TMEM_COLS = 8 * BNQ;  // 2 buffers x 4 components x BNQ fp32 columns
    static constexpr int KSTEPS = KAPPA / UMMA_K;
    static constexpr uint32_t SBO = 8 * A_ROW_BYTES;  // pitch of 8-row core-matrix groups
    // smem descriptor layout type: 128B, 64B or 32B swizzle
    static constexpr uint64_t LAYOUT = A_ROW_BYTES == 128 ? 2ull : (A_ROW_BYTES == 64 ? 4ull : 6ull);
    // high 32 bits of every operand descriptor: SBO, descriptor version, swizzle mode
    static constexpr uint32_t DESC_HI =
        (SBO >> 4) | (1u << 14) | (static_cast<uint32_t>(LAYOUT) << 29);
    static_assert(KAPPA == 16 || KAPPA == 32 || KAPPA == 64, "KAPPA");
    static_assert(BNQ == 16 || BNQ == 32 || BNQ == 64, "BNQ");
    static_assert(MODE != MODE_WS || (KAPPA == 16 && BNQ == 16), "WS tile");
};

// tcgen05 shared-memory matrix descriptors (K-major, swizzled operand tiles) are built
// as two 32-bit words: the low word holds the start address >> 4 (bits 0-13) and the
// leading byte offset (bits 16-29, unused for these layouts, set to 1); the high word
// holds the stride byte offset >> 4 (pitch of 8-row core-matrix groups), the
// descriptor version (bit 46) and the swizzle mode (bits 61-63).
// Low 32 bits of the descriptor: start address and the (unused) leading byte offset.
__device__ __forceinline__ uint32_t desc_lo(uint32_t saddr) {
    return ((saddr & 0x3FFFFu) >> 4) | (1u << 16);
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

template <int KAPPA, int BNQ, int MODE>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    qconv_tc_kernel(const __grid_constant__ CUtensorMap tmap_x,
                    const __grid_constant__ CUtensorMap tmap_wr,
                    const __grid_constant__ CUtensorMap tmap_wi,
                    const __grid_constant__ CUtensorMap tmap_wj,
                    const __grid_constant__ CUtensorMap tmap_wk,
                    const __grid_constant__ CUtensorMap tmap_y, const TcParams p) {
    using C = Cfg<KAPPA, BNQ, MODE>;
    constexpr int STAGES = C::STAGES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::BAR_OFF);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::NUM_BARS);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
    auto ready_bar = [&](int s) { return bar0 + 8u * (2 * STAGES + s); };
    auto fullw_bar = [&](int s) { return bar0 + 8u * (3 * STAGES + s); };
    auto accf_bar = [&](int b) { return bar0 + 8u * (4 * STAGES + b); };
    auto acce_bar = [&](int b) { return bar0 + 8u * (4 * STAGES + 2 + b); };
    const uint32_t drain_bar = bar0 + 8u * (4 * STAGES + 4);
    const uint32_t wsready_bar = bar0 + 8u * (4 * STAGES + 5);

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const ConvShape& s = p.s;
    const uint64_t limit = p.wait_limit_ns;

    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            mbar_init(full_bar(i), 1);
            mbar_init(fullw_bar(i), 1);
            mbar_init(empty_bar(i), 1);
            mbar_init(ready_bar(i), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(accf_bar(b), 1);
            mbar_init(acce_bar(b), 8 * 32);
        }
        mbar_init(drain_bar, 1);
        mbar_init(wsready_bar, NUM_THREADS / 32 - 2);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmap_x);
        tma_prefetch_desc(&tmap_wr);
        tma_prefetch_desc(&tmap_wi);
        tma_prefetch_desc(&tmap_wj);
        tma_prefetch_desc(&tmap_wk);
        tma_prefetch_desc(&tmap_y);
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

    if constexpr (MODE == MODE_WS) {
        if (warp >= 2) {
            // Expand the signed block weight of Eq. 6 once (warps 2..11, while the producer
            // already streams pixels): for tap t, row n = (q, co) and K index k = (p, ci)
            // the value is sign(q, p) * W_{q xor p}[co][t][ci]; rows are 128 bytes (all four
            // input components) in the 128-byte swizzled K-major layout.
            constexpr int EXP_THREADS = NUM_THREADS - 64;
            constexpr int MAX_CHUNKS = WS_MAX_TAPS * 4 * BNQ * 8;
            constexpr int PER_THREAD = (MAX_CHUNKS + EXP_THREADS - 1) / EXP_THREADS;
            const int taps = s.kh * s.kw;
            const int chunks = taps * (4 * BNQ) * 8;  // 16-byte chunks
            const int et = threadIdx.x - 64;
            uint4 v[PER_THREAD];
#pragma unroll
            for (int k = 0; k < PER_THREAD; ++k) {
                const int idx = et + k * EXP_THREADS;
                if (idx < chunks) {
                    const int ch = idx & 7;                // chunk of the row: p = ch / 2
                    const int n = (idx >> 3) % (4 * BNQ);  // row: q = n / BNQ, co = n % BNQ
                    const int t = (idx >> 3) / (4 * BNQ);  // tap
                    const int q = n / BNQ, co = n % BNQ, pc = ch >> 1, ci0 = (ch & 1) * 8;
                    v[k] = __ldg(reinterpret_cast<const uint4*>(
                        p.w[q ^ pc] + (static_cast<size_t>(co) * taps + t) * KAPPA + ci0));
                }
            }
#pragma unroll
            for (int k = 0; k < PER_THREAD; ++k) {
                const int idx = et + k * EXP_THREADS;
                if (idx < chunks) {
                    const int ch = idx & 7;
                    const int n = (idx >> 3) % (4 * BNQ);
                    const int t = (idx >> 3) / (4 * BNQ);
                    const int q = n / BNQ, pc = ch >> 1;
                    uint4 u = v[k];
                    if ((NEG_MASK >> (4 * q + pc)) & 1u) {
                        u.x ^= 0x80008000u; u.y ^= 0x80008000u; u.z ^= 0x80008000u; u.w ^= 0x80008000u;
                    }
                    const uint32_t off = static_cast<uint32_t>(
                        C::WSB_OFF + t * C::WSB_TAP + n * 128 + ((ch ^ (n & 7)) << 4));
                    *reinterpret_cast<uint4*>(smem + off) = u;
                }
            }
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(wsready_bar);
        }
    }

    if (warp == 0 || warp == 3) {
        // ------------------------------------------------------------ TMA producers
        // One thread can only issue TMA copies at a limited rate, so two warps share the
        // work: warp 0 stages the pixel tiles and warp 3 the letter tiles of each K block
        // (WS mode: the two alternate K blocks).
        if (lane == 0) {
            const int role = warp == 0 ? 0 : 1;
            const uint64_t pol_x = l2_policy_evict_normal();
            const uint64_t pol_w = l2_policy_evict_last();
            int stage = 0;
            uint32_t phase = 0;
            uint32_t filled = 0, fill_parity = 0;  // per-stage: ever filled, parity of last fill
            bool ok = true;
            int kt_all = 0;
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
                    if (MODE == MODE_WS && (kt_all++ & 1) != role) {
                        if (++stage == STAGES) {
                            stage = 0;
                            phase ^= 1u;
                        }
                        continue;
                    }
                    if (!wait_or_abort(empty_bar(stage), phase ^ 1u, limit, abort_flag,
                                       STATUS_TIMEOUT_PRODUCER)) {
                        ok = false;
                        break;
                    }
                    // pixels complete full_bar, letters complete fullw_bar
                    const uint32_t fb = role == 0 || MODE == MODE_WS ? full_bar(stage)
                                                                     : fullw_bar(stage);
                    mbar_arrive_expect_tx(fb, MODE == MODE_WS ? C::STAGE_TX
                                              : (role == 0 ? C::A_TILES * C::A_TILE
                                                           : C::STAGE_TX - C::A_TILES * C::A_TILE));
                    filled |= 1u << stage;
                    fill_parity = (fill_parity & ~(1u << stage)) | (phase << stage);
                    const uint32_t a0 = sbase + stage * C::STAGE_BYTES;
                    const uint32_t b0 = a0 + C::A_TILES * C::A_TILE;
                    const int cin0 = chunk * KAPPA;
                    if constexpr (MODE == MODE_WS) {
                        // all four components of the pixel (channels 0 .. 4 KAPPA) at once
                        tma_load_im2col_4d(a0, &tmap_x, fb, 0, wbase, hbase, img,
                                           static_cast<uint16_t>(dw), static_cast<uint16_t>(dh),
                                           pol_x);
                    } else if (role == 0) {
#pragma unroll
                        for (int comp = 0; comp < 4; ++comp)
                            tma_load_im2col_4d(a0 + comp * C::A_TILE, &tmap_x, fb,
                                               comp * s.Qin + cin0, wbase, hbase, img,
                                               static_cast<uint16_t>(dw),
                                               static_cast<uint16_t>(dh), pol_x);
                    } else {
                        const int wcol = tap * s.Qin + cin0, wrow = n_tile * BNQ;
                        if constexpr (MODE == MODE_PAIR) {
                            // slots: [-W_i | W_r | W_i] [W_j | W_k | -W_j]; the sign-flip
                            // warp writes slots 0 and 5 from slots 2 and 3
                            tma_load_2d(b0 + 1 * C::B_TILE, &tmap_wr, fb, wcol, wrow, pol_w);
                            tma_load_2d(b0 + 2 * C::B_TILE, &tmap_wi, fb, wcol, wrow, pol_w);
                            tma_load_2d(b0 + 3 * C::B_TILE, &tmap_wj, fb, wcol, wrow, pol_w);
                            tma_load_2d(b0 + 4 * C::B_TILE, &tmap_wk, fb, wcol, wrow, pol_w);
                        } else {
                            // slots: [W_r | W_i | W_j | W_k]
                            tma_load_2d(b0 + 0 * C::B_TILE, &tmap_wr, fb, wcol, wrow, pol_w);
                            tma_load_2d(b0 + 1 * C::B_TILE, &tmap_wi, fb, wcol, wrow, pol_w);
                            tma_load_2d(b0 + 2 * C::B_TILE, &tmap_wj, fb, wcol, wrow, pol_w);
                            tma_load_2d(b0 + 3 * C::B_TILE, &tmap_wk, fb, wcol, wrow, pol_w);
                        }
                    }
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
                    const uint32_t own = role == 0 || MODE == MODE_WS ? full_bar(i) : fullw_bar(i);
                    const uint64_t t0 = global_timer_ns();
                    while (!mbar_try_wait(own, (fill_parity >> i) & 1u)) {
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
            constexpr int NMMA = MODE == MODE_PAIR ? 2 * BNQ : (MODE == MODE_WS ? 4 * BNQ : BNQ);
            constexpr uint32_t IDESC_POS = make_idesc(BM, NMMA, 0);
            constexpr uint32_t IDESC_NEG = make_idesc(BM, NMMA, 1);
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
            if constexpr (MODE == MODE_WS) {
                if (ok) ok = wait_or_abort(wsready_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
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
                    // pixels, then the letter tiles (pair mode: with their negated copies)
                    if (!wait_or_abort(full_bar(stage), phase, limit, abort_flag,
                                       STATUS_TIMEOUT_MMA)) {
                        ok = false;
                        break;
                    }
                    if constexpr (MODE != MODE_WS) {
                        const uint32_t wb = MODE == MODE_PAIR ? ready_bar(stage) : fullw_bar(stage);
                        if (!wait_or_abort(wb, phase, limit, abort_flag, STATUS_TIMEOUT_MMA)) {
                            ok = false;
                            break;
                        }
                    }
                    tc_fence_after();
                    // descriptor low words of this stage's first X_p and W_L tiles; every
                    // sub-MMA below only adds a compile-time offset to them
                    const uint32_t a_lo0 = desc_lo(sbase + stage * C::STAGE_BYTES);
                    const uint32_t first = kt != 0 ? 1u : 0u;
                    if constexpr (MODE == MODE_WS) {
                        // K step p = input component p (32 bytes into the 128-byte rows)
                        const uint32_t b_lo0 = desc_lo(sbase + C::WSB_OFF + kt * C::WSB_TAP);
#pragma unroll
                        for (int pc = 0; pc < 4; ++pc)
                            umma_f16_w(dbase, a_lo0 + pc * 2, C::DESC_HI, b_lo0 + pc * 2,
                                       C::DESC_HI, IDESC_POS, pc != 0 ? 1u : first);
                    } else {
                    const uint32_t b_lo0 = a_lo0 + (4 * C::A_TILE >> 4);
#pragma unroll
                    for (int pc = 0; pc < 4; ++pc) {
#pragma unroll
                        for (int ks = 0; ks < C::KSTEPS; ++ks) {
                            const uint32_t a_lo =
                                a_lo0 + ((pc * C::A_TILE + ks * (UMMA_K * 2)) >> 4);
                            const uint32_t acc = (pc | ks) != 0 ? 1u : first;
                            if constexpr (MODE == MODE_PAIR) {
                                // stack slot (first of two) and sign for [D_r|D_i], [D_j|D_k]
                                constexpr int SLOT1[4] = {1, 0, 3, 4};
                                constexpr int SLOT2[4] = {3, 4, 1, 0};
                                constexpr bool NEG1[4] = {false, false, true, true};
                                const uint32_t b1 =
                                    b_lo0 + ((SLOT1[pc] * C::B_TILE + ks * (UMMA_K * 2)) >> 4);
                                const uint32_t b2 =
                                    b_lo0 + ((SLOT2[pc] * C::B_TILE + ks * (UMMA_K * 2)) >> 4);
                                umma_f16_w(dbase, a_lo, C::DESC_HI, b1, C::DESC_HI,
                                           NEG1[pc] ? IDESC_NEG : IDESC_POS, acc);
                                umma_f16_w(dbase + 2 * BNQ, a_lo, C::DESC_HI, b2, C::DESC_HI,
                                           IDESC_POS, acc);
                            } else {
#pragma unroll
                                for (int q = 0; q < 4; ++q) {
                                    const int L = q ^ pc;
                                    const uint32_t b_lo =
                                        b_lo0 + ((L * C::B_TILE + ks * (UMMA_K * 2)) >> 4);
                                    const bool neg = (NEG_MASK >> (4 * q + pc)) & 1u;
                                    umma_f16_w(dbase + q * BNQ, a_lo, C::DESC_HI, b_lo,
                                               C::DESC_HI, neg ? IDESC_NEG : IDESC_POS, acc);
                                }
                            }
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
    } else if (warp == 2) {
        // ------------------------------------------------------------ sign flips
        if constexpr (MODE == MODE_PAIR) {
            // Write -W_i (slot 0) and -W_j (slot 5) of every stage from its copies of W_i
            // and W_j (slots 2, 3) once they have landed, then hand the stage to the MMA
            // issuer.  Slot sizes are multiples of the swizzle period, so a raw copy keeps
            // the layout.
            constexpr int WORDS = C::B_TILE / 16;  // uint4 per slot
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true;
            for (int tile = blockIdx.x; ok && tile < p.num_tiles; tile += gridDim.x) {
                for (int kt = 0; kt < p.ktiles; ++kt) {
                    if (!wait_or_abort(fullw_bar(stage), phase, limit, abort_flag,
                                       STATUS_TIMEOUT_PRODUCER)) {
                        ok = false;
                        break;
                    }
                    uint8_t* b0 = smem + stage * C::STAGE_BYTES + 4 * C::A_TILE;
                    const uint4* s2 = reinterpret_cast<const uint4*>(b0 + 2 * C::B_TILE);
                    const uint4* s3 = reinterpret_cast<const uint4*>(b0 + 3 * C::B_TILE);
                    uint4* s0 = reinterpret_cast<uint4*>(b0);
                    uint4* s5 = reinterpret_cast<uint4*>(b0 + 5 * C::B_TILE);
#pragma unroll 4
                    for (int i = lane; i < WORDS; i += 32) {
                        uint4 a = s2[i], b = s3[i];
                        a.x ^= 0x80008000u; a.y ^= 0x80008000u; a.z ^= 0x80008000u; a.w ^= 0x80008000u;
                        b.x ^= 0x80008000u; b.y ^= 0x80008000u; b.z ^= 0x80008000u; b.w ^= 0x80008000u;
                        s0[i] = a;
                        s5[i] = b;
                    }
                    // make the generic-proxy writes visible to the tensor core (async proxy)
                    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
                    __syncwarp();
                    if (lane == 0) mbar_arrive(ready_bar(stage));
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
        }
    } else if (warp >= EPI_WARP0) {
        // ------------------------------------------------------------ epilogue
        const int quad = warp & 3;                 // TMEM lane quadrant this warp may access
        const int half = (warp - EPI_WARP0) >> 2;  // output components 2*half, 2*half+1
        const int row = quad * 32 + lane;
        const bool leader = (warp == EPI_WARP0 + 4 * half) && lane == 0;
        const int etid = threadIdx.x - EPI_WARP0 * 32;  // 0..255
        const int Cout = s.Cout;
        const __nv_bfloat16* res = static_cast<const __nv_bfloat16*>(p.ep.residual);
        float* prm_s = reinterpret_cast<float*>(smem + C::PARAM_OFF);  // [3][4*BNQ]
        uint8_t* stg = smem + C::STAGING_OFF + half * C::OUT_TILE;
        const uint32_t stg_addr = smem_u32(stg);
        int cached_n = -1;
        int local = 0;
        for (int tile = blockIdx.x; tile < p.num_tiles; tile += gridDim.x, ++local) {
            const int buf = local & 1;
            const uint32_t use = static_cast<uint32_t>(local >> 1) & 1u;
            const bool ok = wait_or_abort(accf_bar(buf), use, limit, abort_flag,
                                          STATUS_TIMEOUT_EPILOGUE);
            // leave together: a warp that gave up must not strand the others at a barrier
            if (named_bar_or(1, 256, !ok)) break;
            tc_fence_after();
            const int m_tile = tile / p.num_n_tiles;
            const int n_tile = tile - m_tile * p.num_n_tiles;
            if (n_tile != cached_n) {
                // per-channel vectors of this tile's 4 x BNQ channels -> shared memory
                named_bar_sync(1, 256);
                for (int i = etid; i < 4 * BNQ; i += 256) {
                    const int c = (i / BNQ) * s.Qout + n_tile * BNQ + (i % BNQ);
                    prm_s[i] = p.ep.bias ? __ldg(p.ep.bias + c) : 0.0f;
                    prm_s[4 * BNQ + i] = p.ep.scale ? __ldg(p.ep.scale + c) : 1.0f;
                    prm_s[8 * BNQ + i] = p.ep.scale ? __ldg(p.ep.shift + c) : 0.0f;
                }
                named_bar_sync(1, 256);
                cached_n = n_tile;
            }
            const long long m = static_cast<long long>(m_tile) * BM + row;
            const bool valid = m < s.M;
            const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                                   static_cast<uint32_t>(buf * 4 * BNQ);
#pragma unroll
            for (int qq = 0; qq < 2; ++qq) {
                const int q = 2 * half + qq;
                // the staging block is free once the previous store has read it
                if (leader) bulk_wait_group_read<0>();
                named_bar_sync(2 + half, 128);
                constexpr int CH = BNQ < 32 ? BNQ : 32;  // columns per TMEM load
#pragma unroll
                for (int j0 = 0; j0 < BNQ; j0 += CH) {
                    uint32_t v[32];
                    if constexpr (CH == 32) {
                        tmem_ld_32x32b_x32(taddr + q * BNQ + j0, v);
                    } else {
                        uint32_t (&v16)[16] = *reinterpret_cast<uint32_t(*)[16]>(v);
                        tmem_ld_32x32b_x16(taddr + q * BNQ + j0, v16);
                    }
                    float rz[CH];
                    if (res != nullptr && valid) {
                        const uint4* rp = reinterpret_cast<const uint4*>(
                            res + m * Cout + q * s.Qout + n_tile * BNQ + j0);
#pragma unroll
                        for (int u = 0; u < CH / 8; ++u) {
                            const uint4 r4 = __ldg(rp + u);
                            const __nv_bfloat162* h = reinterpret_cast<const __nv_bfloat162*>(&r4);
#pragma unroll
                            for (int t = 0; t < 4; ++t) {
                                const float2 f = __bfloat1622float2(h[t]);
                                rz[8 * u + 2 * t] = f.x;
                                rz[8 * u + 2 * t + 1] = f.y;
                            }
                        }
                    } else {
#pragma unroll
                        for (int t = 0; t < CH; ++t) rz[t] = 0.0f;
                    }
                    tmem_ld_wait();
                    const float* pb = prm_s + q * BNQ + j0;
                    const float* ps = prm_s + 4 * BNQ + q * BNQ + j0;
                    const float* ph = prm_s + 8 * BNQ + q * BNQ + j0;
#pragma unroll
                    for (int u = 0; u < CH / 8; ++u) {
                        uint32_t w[4];
#pragma unroll
                        for (int t = 0; t < 4; ++t) {
                            const int e = 8 * u + 2 * t;
                            float z0 = __uint_as_float(v[e]) + pb[e];
                            float z1 = __uint_as_float(v[e + 1]) + pb[e + 1];
                            z0 = fmaf(ps[e], z0, ph[e]) + rz[e];
                            z1 = fmaf(ps[e + 1], z1, ph[e + 1]) + rz[e + 1];
                            w[t] = pack_bf16x2(activate(z0, s.act), activate(z1, s.act));
                        }
                        // 16-byte chunk (j0/8 + u) of this row, swizzled like the TMA map
                        const uint32_t chunk = static_cast<uint32_t>(j0 / 8 + u);
                        const uint32_t off = static_cast<uint32_t>(row) * C::OUT_ROW +
                                             ((chunk ^ ((static_cast<uint32_t>(row) *
                                                         C::OUT_ROW >> 7) & C::OUT_SW_MASK))
                                              << 4);
                        *reinterpret_cast<uint4*>(stg + off) = make_uint4(w[0], w[1], w[2], w[3]);
                    }
                }
                fence_proxy_async_smem();
                named_bar_sync(2 + half, 128);
                if (leader) {
                    tma_store_2d(&tmap_y, stg_addr, q * s.Qout + n_tile * BNQ,
                                 static_cast<int>(m_tile) * BM);
                    bulk_commit_group();
                }
            }
            tc_fence_before();
            mbar_arrive(acce_bar(buf));
        }
        if (leader) bulk_wait_group<0>();
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

// Output [M rows][Cout] bf16, stored in boxes of 128 rows x BNQ channels.
bool encode_y(CUtensorMap* map, const ConvShape& s, const void* y, int bnq) {
    const cuuint64_t dims[2] = {static_cast<cuuint64_t>(s.Cout), static_cast<cuuint64_t>(s.M)};
    const cuuint64_t strides[1] = {static_cast<cuuint64_t>(s.Cout) * 2};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(bnq), static_cast<cuuint32_t>(BM)};
    const cuuint32_t estr[2] = {1, 1};
    const CUtensorMapSwizzle sw = bnq == 64 ? CU_TENSOR_MAP_SWIZZLE_128B
                                            : (bnq == 32 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                         : CU_TENSOR_MAP_SWIZZLE_32B);
    const CUresult r = g_encode_tiled(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(y),
                                      dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw,
                                      CU_TENSOR_MAP_L2_PROMOTION_NONE,
                                      CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

template <int KAPPA, int BNQ, int MODE>
cudaError_t launch_cfg(const CUtensorMap maps[6], const TcParams& prm, int grid,
                       cudaStream_t stream) {
    using C = Cfg<KAPPA, BNQ, MODE>;
    if constexpr (!C::FITS) {
        return cudaErrorInvalidValue;
    } else {
    auto kern = qconv_tc_kernel<KAPPA, BNQ, MODE>;
    // The shared-memory opt-in is per device; set it once for each.
    static std::atomic<unsigned long long> attr_done{0};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = 1ull << (dev & 63);
    if (!(attr_done.load() & bit)) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 C::SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr_done.fetch_or(bit);
    }
    kern<<<grid, NUM_THREADS, C::SMEM_BYTES, stream>>>(maps[0], maps[1], maps[2], maps[3],
                                                       maps[4], maps[5], prm);
    return cudaGetLastError();
    }
}

template <int KAPPA, int BNQ, int MODE>
constexpr bool cfg_fits() {
    return Cfg<KAPPA, BNQ, MODE>::FITS;
}

// Encoded tensor maps of recent calls, keyed by every value that goes into them, so a
// layer called repeatedly on the same buffers skips the five host-side encodes.
struct MapKey {
    const void* ptr[6];
    int N, H, W, Cin, Cout, kh, kw, stride, pad, kappa, bnq;
    bool operator==(const MapKey& o) const {
        for (int i = 0; i < 6; ++i)
            if (ptr[i] != o.ptr[i]) return false;
        return N == o.N && H == o.H && W == o.W && Cin == o.Cin && Cout == o.Cout &&
               kh == o.kh && kw == o.kw && stride == o.stride && pad == o.pad &&
               kappa == o.kappa && bnq == o.bnq;
    }
};

struct MapEntry {
    MapKey key;
    CUtensorMap maps[6];
    bool valid;
};

constexpr int kMapCacheSize = 64;
MapEntry g_map_cache[kMapCacheSize];
int g_map_next = 0;
std::mutex g_map_mu;

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
    int kappa = pick_kappa(s.Qin, opt.kappa);
    int bnq = pick_bnq(s.Qout, opt.bnq);
    // Weight-stationary for 16 -> 16 quaternion channels (the whole expanded weight fits);
    // pair mode (N = 2 BNQ per MMA) otherwise, unless the tile is so narrow that even
    // pairs stay far below the tensor pipe's per-instruction cost.
    const bool ws_ok = s.Qin == 16 && s.Qout == 16 && s.kh * s.kw <= WS_MAX_TAPS;
    int mode;
    if (opt.mode == 1) mode = MODE_QUAD;
    else if (opt.mode == 2) mode = MODE_PAIR;
    else if (opt.mode == 3) mode = MODE_WS;
    else mode = ws_ok ? MODE_WS : (bnq >= 32 ? MODE_PAIR : MODE_QUAD);
    if (mode == MODE_WS) {
        if (!ws_ok) {
            snprintf(err, errlen, "weight-stationary mode needs Cin = Cout = 64 and <= %d taps",
                     WS_MAX_TAPS);
            return cudaErrorInvalidValue;
        }
        kappa = 16;
        bnq = 16;
    }
    // A 6-slot stage of 64 x 64 letter blocks plus 64-channel pixel tiles does not fit
    // twice in shared memory; use 32-channel K blocks then.
    if (mode == MODE_PAIR && kappa == 64 && bnq == 64 && opt.kappa == 0) kappa = 32;
    if (kappa == 0 || bnq == 0) {
        snprintf(err, errlen, "requested tile (kappa=%d, bnq=%d) does not divide Qin=%d/Qout=%d",
                 opt.kappa, opt.bnq, s.Qin, s.Qout);
        return cudaErrorInvalidValue;
    }
    MapKey key;
    key.ptr[0] = x;
    for (int l = 0; l < 4; ++l) key.ptr[1 + l] = w[l];
    key.ptr[5] = out;
    key.N = s.N; key.H = s.H; key.W = s.W; key.Cin = s.Cin; key.Cout = s.Cout;
    key.kh = s.kh; key.kw = s.kw; key.stride = s.stride; key.pad = s.pad;
    key.kappa = mode == MODE_WS ? -kappa : kappa; key.bnq = bnq;
    CUtensorMap maps[6];
    bool hit = false;
    {
        std::lock_guard<std::mutex> lk(g_map_mu);
        for (int i = 0; i < kMapCacheSize; ++i)
            if (g_map_cache[i].valid && g_map_cache[i].key == key) {
                for (int l = 0; l < 6; ++l) maps[l] = g_map_cache[i].maps[l];
                hit = true;
                break;
            }
    }
    if (!hit) {
        if (!encode_x(&maps[0], s, x, mode == MODE_WS ? 4 * kappa : kappa)) {
            snprintf(err, errlen, "cuTensorMapEncodeIm2col failed for the activation tensor");
            return cudaErrorInvalidValue;
        }
        for (int l = 0; l < 4; ++l)
            if (!encode_w(&maps[1 + l], s, w[l], kappa, bnq)) {
                snprintf(err, errlen, "cuTensorMapEncodeTiled failed for weight letter %d", l);
                return cudaErrorInvalidValue;
            }
        if (!encode_y(&maps[5], s, out, bnq)) {
            snprintf(err, errlen, "cuTensorMapEncodeTiled failed for the output tensor");
            return cudaErrorInvalidValue;
        }
        std::lock_guard<std::mutex> lk(g_map_mu);
        MapEntry& e = g_map_cache[g_map_next];
        g_map_next = (g_map_next + 1) % kMapCacheSize;
        e.key = key;
        for (int l = 0; l < 6; ++l) e.maps[l] = maps[l];
        e.valid = true;
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
    for (int l = 0; l < 4; ++l) prm.w[l] = static_cast<const __nv_bfloat16*>(w[l]);
    int grid = opt.max_ctas > 0 ? opt.max_ctas : num_sms;
    if (grid > prm.num_tiles) grid = prm.num_tiles;
    if (grid < 1) grid = 1;

    static_assert(Cfg<16, 16, MODE_WS>::FITS, "weight-stationary tile must fit");
    if (mode != MODE_WS) {
        bool fits = true;
#define QUAN_FIT_CASE(K, B)                                                        \
    if (kappa == K && bnq == B)                                                    \
        fits = mode == MODE_PAIR ? cfg_fits<K, B, MODE_PAIR>() : cfg_fits<K, B, MODE_QUAD>();
        QUAN_FIT_CASE(16, 16) QUAN_FIT_CASE(16, 32) QUAN_FIT_CASE(16, 64)
        QUAN_FIT_CASE(32, 16) QUAN_FIT_CASE(32, 32) QUAN_FIT_CASE(32, 64)
        QUAN_FIT_CASE(64, 16) QUAN_FIT_CASE(64, 32) QUAN_FIT_CASE(64, 64)
#undef QUAN_FIT_CASE
        if (!fits) {
            snprintf(err, errlen, "tile kappa=%d bnq=%d mode=%d exceeds shared memory", kappa,
                     bnq, mode);
            return cudaErrorInvalidValue;
        }
    }
    if (mode == MODE_WS) return launch_cfg<16, 16, MODE_WS>(maps, prm, grid, stream);
#define QUAN_TC_CASE(K, B)                                                       \
    if (kappa == K && bnq == B)                                                  \
        return mode == MODE_PAIR ? launch_cfg<K, B, MODE_PAIR>(maps, prm, grid, stream) \
                                 : launch_cfg<K, B, MODE_QUAD>(maps, prm, grid, stream);
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
    snprintf(err, errlen, "no kernel instance for kappa=%d bnq=%d mode=%d", kappa, bnq, mode);
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
