// qconv_tc.cu -- tensor-core quaternion convolution for sm_103a (tcgen05 + TMA).
//
// The quaternion convolution of Eq. 5 (Sec. III-B) is an implicit GEMM
//   Y[pixel][q, co] = sum_{tap, p, ci} X[pixel + tap][p, ci] * B[tap][p, ci][q, co]
// whose weight B is the signed 4x4 block (Hamilton) matrix of Eq. 6 built from four
// compact letter tensors W_r, W_i, W_j, W_k.  The block weight is never written to
// global memory: the signed block structure is produced on chip, so weight traffic
// is 1/4 of the real-equivalent layer.  Three MMA decompositions:
//
//   MODE_QUAD  16 MMAs per 16-wide K step, one per (output q, input p):
//                D_q += sign(q, p) * X_p * W_{q xor p}^T            (N = BNQ)
//              the letter is chosen by the B descriptor and the sign by the
//              instruction descriptor's negate bit.
//   MODE_PAIR  8 MMAs per K step, each covering two output components:
//                [D_r | D_i] and [D_j | D_k] += +-X_p * S^T         (N = 2 BNQ)
//              where S is a stack of two letter blocks.  The four stacks Eq. 6 needs,
//              [W_r; W_i], [-W_i; W_r], [W_j; W_k], [W_k; -W_j] (up to an overall sign),
//              are all windows of the two 3-block sequences
//                [-W_i | W_r | W_i]  and  [W_j | W_k | -W_j],
//              so a stage holds 6 letter blocks; TMA loads the 4 letters and a helper
//              warp writes the two negated copies.  The larger N keeps the tensor pipe
//              busy (an M=128 MMA costs at least ~45 cycles on this part, a full N=64 one
//              is 32 cycles of work, N=128 is 64).
//   MODE_SEP   the separable form of Eq. 7: 4 MMAs per K step, D_p += X_p * W_p^T
//              (N = BNQ), one per input component; the epilogue mixes the four D_p
//              with the signs of Eq. 7 (epilogue_direct_sep), so no negated letters.
//   MODE_WS    (16 -> 16 quaternion channels, at most 9 taps; qconv_ws.cuh)
//              weight-stationary: every CTA expands the whole signed block weight once
//              into shared memory and streams only pixels; N = 64 MMAs cover all four
//              output components.
//   pairs      (1 -> 16 quaternion channels, stride 2: the 4-channel stem;
//              qconv_gather.cuh) weight-stationary like MODE_WS; pixels are loaded as
//              16-byte horizontal pairs, one TMA box per filter row, and the filter taps
//              are descriptor offsets into those boxes.
//
// Structure of the QUAD/PAIR kernel (one persistent CTA per SM, 12 warps):
//   warps 0, 3  TMA producers: per K block (tap, chunk of KAPPA quaternion input channels)
//               warp 0 issues the 4 im2col loads of X (zero padding comes from
//               out-of-bounds fill) and warp 3 the letter tiles, into a STAGES-deep ring
//               (one thread issues TMA copies at a limited rate);
//   warp 1      owns TMEM (2 accumulator buffers x 4 components x BNQ columns); one lane
//               issues the tcgen05.mma / tcgen05.commit stream;
//   warp 2      waits for both fills of each stage (MODE_PAIR: writes the two
//               sign-flipped letter copies) and hands it to the issuer by a release store
//               of the stage's sequence word, which the issuer reads with an acquire load;
//   warps 4..11 epilogue (tc_common.cuh), overlapping the next tile's main loop.
// Every mbarrier wait is bounded in time; a wait that runs out sets a bit in the device
// status word, raises a CTA-wide abort flag, drains the copies and MMAs still in flight,
// frees TMEM and returns.
#include <cuda.h>
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <atomic>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "internal.h"
#include "ptx.cuh"
#include "tc_common.cuh"

namespace quan {
namespace {

using namespace tc;

thread_local char t_kernel_name[64] = "";

void set_kernel_name(const char* fmt, int a = 0, int b = 0) {
    snprintf(t_kernel_name, sizeof(t_kernel_name), fmt, a, b);
}

constexpr int MODE_QUAD = 0;
constexpr int MODE_PAIR = 1;
constexpr int MODE_WS = 2;
constexpr int MODE_SEP = 3;
// The separable form's input gradient (ConvShape::sep == 2): 16 MMAs per K step like
// MODE_QUAD, block (output q, input p) = the letter q with the sign of Eq. 7's term
// (output p, letter q) -- the transpose of the separable block weight.
constexpr int MODE_SEPT = 4;
constexpr int WS_MAX_TAPS = 9;
constexpr int MAX_STAGES = 8;

struct TcParams {
    ConvShape s;
    EpilogueArgs ep;
    int kchunks;      // Qin / KAPPA
    int ktiles;       // kh * kw * kchunks K blocks per tile
    int num_n_tiles;  // Qout / BNQ
    int num_tiles;
    void* y;          // output [M][Cout]
    unsigned long long wait_limit_ns;
    int inject_stall;
    SplitK sk;        // K ranges split evenly over the CTAs (QUAD/PAIR modes, caller workspace)
    ScParams sc;      // the fused 1x1 shortcut (the SC form of the kernel)
};

// The fused shortcut's four letter maps (SC form; unused otherwise).
struct ScMaps {
    CUtensorMap w[4];
};

template <int KAPPA, int BNQ, int MODE>
struct Cfg {
    static constexpr int A_ROW_BYTES = KAPPA * 2;
    static constexpr int A_TILE = BM * A_ROW_BYTES;  // one component of the pixel tile
    static constexpr int B_TILE = BNQ * KAPPA * 2;   // one letter block of the weight tile
    static constexpr int B_SLOTS = MODE == MODE_PAIR ? 6 : 4;
    static constexpr int STAGE_BYTES = 4 * A_TILE + B_SLOTS * B_TILE;
    static constexpr int TX_A = 4 * A_TILE;          // bytes TMA writes per stage: pixels
    static constexpr int TX_W = 4 * B_TILE;          //                               letters
    // 1024 bytes of alignment slack, then the stage ring and the barrier area (the
    // epilogue needs no shared memory)
    static constexpr int FIXED_BYTES = 1024 + 384;
    static constexpr int STAGES_RAW = (227 * 1024 - FIXED_BYTES) / STAGE_BYTES;
    static constexpr int STAGES =
        STAGES_RAW > MAX_STAGES ? MAX_STAGES : (STAGES_RAW < 2 ? 2 : STAGES_RAW);
    static constexpr int TILES_BYTES = STAGES * STAGE_BYTES;
    static constexpr int BAR_OFF = TILES_BYTES;
    // full (pixels), empty, full (letters), acc_full[2], acc_empty[2], drain; then the
    // TMEM address, the abort flag and one ready sequence word per stage
    static constexpr int NUM_BARS = 3 * STAGES + 5;
    static constexpr int SMEM_BYTES = 1024 + BAR_OFF + NUM_BARS * 8 + 16 + 4 * STAGES;
    static_assert(NUM_BARS * 8 + 16 + 4 * STAGES <= FIXED_BYTES - 1024, "barrier area");
    static constexpr bool FITS = SMEM_BYTES <= 227 * 1024;
    static constexpr uint32_t TMEM_COLS = 8 * BNQ;  // 2 buffers x 4 components x BNQ fp32 columns
    static constexpr int KSTEPS = KAPPA / UMMA_K;
    static constexpr uint32_t DESC_HI = desc_hi(8 * A_ROW_BYTES, desc_layout(A_ROW_BYTES));
    static_assert(KAPPA == 16 || KAPPA == 32 || KAPPA == 64, "KAPPA");
    static_assert(BNQ == 16 || BNQ == 32 || BNQ == 64, "BNQ");
};

// SC: N tiles from p.sc.n_conv on belong to a 1x1 shortcut on the same input, fused into
// the launch (ScParams): their K blocks are the filter tap p.sc.tap's only, their letters
// come from `scm`, and the epilogue writes them to the shortcut's output.
template <int KAPPA, int BNQ, int MODE, bool SC = false>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    qconv_tc_kernel(const __grid_constant__ CUtensorMap tmap_x,
                    const __grid_constant__ CUtensorMap tmap_wr,
                    const __grid_constant__ CUtensorMap tmap_wi,
                    const __grid_constant__ CUtensorMap tmap_wj,
                    const __grid_constant__ CUtensorMap tmap_wk, const TcParams p,
                    const __grid_constant__ ScMaps scm) {
    static_assert(!SC || MODE == MODE_PAIR || MODE == MODE_QUAD, "fused shortcut modes");
    using C = Cfg<KAPPA, BNQ, MODE>;
    constexpr int STAGES = C::STAGES;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::BAR_OFF);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::NUM_BARS);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    uint32_t* ready_seq = tmem_slot + 4;  // per stage: fills handed to the issuer so far
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (STAGES + s); };
    auto fullw_bar = [&](int s) { return bar0 + 8u * (2 * STAGES + s); };
    auto ready_word = [&](int s) { return smem_u32(ready_seq + s); };
    const uint32_t accf0 = bar0 + 8u * (3 * STAGES);
    const uint32_t acce0 = bar0 + 8u * (3 * STAGES + 2);
    const uint32_t drain_bar = bar0 + 8u * (3 * STAGES + 4);

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const ConvShape& s = p.s;
    const uint64_t limit = p.wait_limit_ns;

    griddep_launch_dependents();
    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            mbar_init(full_bar(i), 1);
            mbar_init(fullw_bar(i), 1);
            mbar_init(empty_bar(i), 1);
            ready_seq[i] = 0;
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(accf0 + 8u * b, 1);
            mbar_init(acce0 + 8u * b, 8 * 32);
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
        if constexpr (SC)
            for (int l = 0; l < 4; ++l) tma_prefetch_desc(&scm.w[l]);
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
    griddep_wait();  // the previous kernel's output (this layer's input) is complete

    if (warp == 0 || warp == 3) {
        // ------------------------------------------------------------ TMA producers
        if (lane == 0) {
            const int role = warp == 0 ? 0 : 1;  // 0: pixels, 1: letters
            const uint64_t pol_x = l2_policy_evict_normal();
            const uint64_t pol_w = l2_policy_evict_last();
            int stage = 0;
            uint32_t phase = 0;
            uint32_t filled = 0, fill_parity = 0;  // per stage: ever filled, parity of last fill
            bool ok = true;
            UnitIter units(p.sk.on, p.num_tiles, p.ktiles);
            Unit unit;
            while (ok && units.next(unit)) {
                const int tile = unit.tile;
                const int m_tile = tile / p.num_n_tiles;
                const int n_tile = tile - m_tile * p.num_n_tiles;
                const long long m0 = static_cast<long long>(m_tile) * BM;
                const int img = static_cast<int>(m0 / hw);
                const int rem = static_cast<int>(m0 - static_cast<long long>(img) * hw);
                const int ho = rem / s.Wo, wo = rem - (rem / s.Wo) * s.Wo;
                const int wbase = wo * s.stride - s.pad, hbase = ho * s.stride - s.pad;
                // K block kt = (tap, chunk), tap = dh * kw + dw: walked without divisions
                // from the unit's first block
                int tap = unit.k0 / p.kchunks;
                int chunk = unit.k0 - tap * p.kchunks;
                int dh = tap / s.kw, dw = tap - (tap / s.kw) * s.kw;
                int k1 = unit.k1;
                bool sct = false;  // a fused shortcut's tile: one tap, its own letters
                if constexpr (SC) {
                    sct = n_tile >= p.sc.n_conv;
                    if (sct) {
                        k1 = p.sc.ktiles;
                        tap = p.sc.tap;
                        dh = p.sc.dh;
                        dw = p.sc.dw;
                        chunk = 0;
                    }
                }
                for (int kt = unit.k0; kt < k1; ++kt) {
                    if (SC && sct) {
                        if (kt > unit.k0) ++chunk;
                    } else if (kt > unit.k0 && ++chunk == p.kchunks) {
                        chunk = 0;
                        ++tap;
                        if (++dw == s.kw) {
                            dw = 0;
                            ++dh;
                        }
                    }
                    if (!wait_or_abort(empty_bar(stage), phase ^ 1u, limit, abort_flag,
                                       STATUS_TIMEOUT_PRODUCER)) {
                        ok = false;
                        break;
                    }
                    // pixels complete full_bar, letters complete fullw_bar
                    const uint32_t fb = role == 0 ? full_bar(stage) : fullw_bar(stage);
                    mbar_arrive_expect_tx(fb, role == 0 ? C::TX_A : C::TX_W);
                    filled |= 1u << stage;
                    fill_parity = (fill_parity & ~(1u << stage)) | (phase << stage);
                    const uint32_t a0 = sbase + stage * C::STAGE_BYTES;
                    const uint32_t b0 = a0 + 4 * C::A_TILE;
                    const int cin0 = chunk * KAPPA;
                    if (role == 0) {
#pragma unroll
                        for (int comp = 0; comp < 4; ++comp)
                            tma_load_im2col_4d(a0 + comp * C::A_TILE, &tmap_x, fb,
                                               comp * s.Qin + cin0, wbase, hbase, img,
                                               static_cast<uint16_t>(dw),
                                               static_cast<uint16_t>(dh), pol_x);
                    } else {
                        const int wcol = tap * s.Qin + cin0, wrow = n_tile * BNQ;
                        if (SC && sct) {
                            // the shortcut's 1x1 letters [Qout_sc][Qin]
                            const int wr2 = (n_tile - p.sc.n_conv) * BNQ;
                            if constexpr (MODE == MODE_PAIR) {
                                tma_load_2d(b0 + 1 * C::B_TILE, &scm.w[0], fb, cin0, wr2, pol_w);
                                tma_load_2d(b0 + 2 * C::B_TILE, &scm.w[1], fb, cin0, wr2, pol_w);
                                tma_load_2d(b0 + 3 * C::B_TILE, &scm.w[2], fb, cin0, wr2, pol_w);
                                tma_load_2d(b0 + 4 * C::B_TILE, &scm.w[3], fb, cin0, wr2, pol_w);
                            } else {
                                tma_load_2d(b0 + 0 * C::B_TILE, &scm.w[0], fb, cin0, wr2, pol_w);
                                tma_load_2d(b0 + 1 * C::B_TILE, &scm.w[1], fb, cin0, wr2, pol_w);
                                tma_load_2d(b0 + 2 * C::B_TILE, &scm.w[2], fb, cin0, wr2, pol_w);
                                tma_load_2d(b0 + 3 * C::B_TILE, &scm.w[3], fb, cin0, wr2, pol_w);
                            }
                        } else if constexpr (MODE == MODE_PAIR) {
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
            // after an abort anywhere in the CTA, let every copy still in flight land
            // before the CTA can exit
            if (!ok || *abort_flag)
                drain_fills(role == 0 ? full_bar(0) : fullw_bar(0), STAGES, filled, fill_parity,
                            limit);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr int NMMA = MODE == MODE_PAIR ? 2 * BNQ : BNQ;
            constexpr uint32_t IDESC_POS = make_idesc(BM, NMMA, 0);
            constexpr uint32_t IDESC_NEG = make_idesc(BM, NMMA, 1);
            int stage = 0;
            uint32_t round = 0;  // completed passes over the stage ring
            bool ok = true;
            int issued = 0;
            if (p.inject_stall) {
                // Failure injection: wait on a barrier nothing arrives on, so that every
                // role runs into its bounded wait and the kernel reports a timeout.
                wait_or_abort(drain_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
                ok = false;
            }
            int local = 0;
            UnitIter units(p.sk.on, p.num_tiles, p.ktiles);
            Unit unit;
            while (ok && units.next(unit)) {
                const int buf = local & 1;
                const uint32_t use = static_cast<uint32_t>(local >> 1) & 1u;
                ++local;
                if (!wait_or_abort(acce0 + 8u * buf, use ^ 1u, limit, abort_flag,
                                   STATUS_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t dbase = tmem_base + static_cast<uint32_t>(buf * 4 * BNQ);
                int k1 = unit.k1;
                if constexpr (SC)
                    if (unit.tile % p.num_n_tiles >= p.sc.n_conv) k1 = p.sc.ktiles;
                for (int kt = unit.k0; kt < k1; ++kt) {
                    // pixels and letter tiles landed (pair mode: with the negated copies)
                    if (!flag_wait_or_abort(ready_word(stage), round + 1u, limit, abort_flag,
                                            STATUS_TIMEOUT_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    // descriptor low words of this stage's first X_p and W_L tiles; every
                    // sub-MMA below only adds a compile-time offset to them
                    const uint32_t a_lo0 = desc_lo(sbase + stage * C::STAGE_BYTES);
                    const uint32_t b_lo0 = a_lo0 + (4 * C::A_TILE >> 4);
                    const uint32_t first = kt != unit.k0 ? 1u : 0u;
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
                            } else if constexpr (MODE == MODE_SEP) {
                                // D_pc += X_pc * W_pc^T (letter pc sits in slot pc); D_pc's
                                // first MMA of a tile is its own ks = 0 of K block 0
                                const uint32_t b_lo =
                                    b_lo0 + ((pc * C::B_TILE + ks * (UMMA_K * 2)) >> 4);
                                umma_f16_w(dbase + pc * BNQ, a_lo, C::DESC_HI, b_lo, C::DESC_HI,
                                           IDESC_POS, ks != 0 ? 1u : first);
                            } else {
#pragma unroll
                                for (int q = 0; q < 4; ++q) {
                                    const int L = MODE == MODE_SEPT ? q : q ^ pc;
                                    const uint32_t b_lo =
                                        b_lo0 + ((L * C::B_TILE + ks * (UMMA_K * 2)) >> 4);
                                    const bool neg = MODE == MODE_SEPT
                                                         ? ((SEP_NEG >> (4 * pc + q)) & 1u)
                                                         : ((NEG_MASK >> (4 * q + pc)) & 1u);
                                    umma_f16_w(dbase + q * BNQ, a_lo, C::DESC_HI, b_lo,
                                               C::DESC_HI, neg ? IDESC_NEG : IDESC_POS, acc);
                                }
                            }
                        }
                    }
                    ++issued;
                    umma_commit(empty_bar(stage));  // frees the stage when these MMAs finish
                    if (++stage == STAGES) {
                        stage = 0;
                        ++round;
                    }
                }
                if (!ok) break;
                umma_commit(accf0 + 8u * buf);  // accumulator buffer ready for the epilogue
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
        // ------------------------------------------------------------ stage hand-off
        // Waits for both fills of every stage (and in pair mode writes -W_i (slot 0) and
        // -W_j (slot 5) from its copies of W_i and W_j (slots 2, 3); slot sizes are
        // multiples of the swizzle period, so a raw copy keeps the layout), then hands
        // the stage to the MMA issuer through its ready sequence word: every mbarrier wait
        // the issuing thread itself performs stalls the tensor pipe for hundreds of cycles,
        // an acquire load of that word for about a third of that.
        constexpr int WORDS = C::B_TILE / 16;  // uint4 per slot
        int stage = 0;
        uint32_t phase = 0, round = 0;
        bool ok = true;
        UnitIter units(p.sk.on, p.num_tiles, p.ktiles);
        Unit unit;
        while (ok && units.next(unit)) {
            int k1 = unit.k1;
            if constexpr (SC)
                if (unit.tile % p.num_n_tiles >= p.sc.n_conv) k1 = p.sc.ktiles;
            for (int kt = unit.k0; kt < k1; ++kt) {
                if (!wait_or_abort(fullw_bar(stage), phase, limit, abort_flag,
                                   STATUS_TIMEOUT_PRODUCER)) {
                    ok = false;
                    break;
                }
                if constexpr (MODE == MODE_PAIR) {
                    uint8_t* b0 = smem + stage * C::STAGE_BYTES + 4 * C::A_TILE;
                    const uint4* s2 = reinterpret_cast<const uint4*>(b0 + 2 * C::B_TILE);
                    const uint4* s3 = reinterpret_cast<const uint4*>(b0 + 3 * C::B_TILE);
                    uint4* s0 = reinterpret_cast<uint4*>(b0);
                    uint4* s5 = reinterpret_cast<uint4*>(b0 + 5 * C::B_TILE);
#pragma unroll 4
                    for (int i = lane; i < WORDS; i += 32) {
                        s0[i] = negate_bf16x8(s2[i]);
                        s5[i] = negate_bf16x8(s3[i]);
                    }
                    // make the generic-proxy writes visible to the tensor core (async proxy)
                    fence_proxy_async_smem();
                }
                if (!wait_or_abort(full_bar(stage), phase, limit, abort_flag,
                                   STATUS_TIMEOUT_PRODUCER)) {
                    ok = false;
                    break;
                }
                __syncwarp();
                if (lane == 0) st_release_shared(ready_word(stage), round + 1u);
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                    ++round;
                }
            }
        }
    } else if (warp >= EPI_WARP0) {
        // ------------------------------------------------------------ epilogue
        const int num_n = p.num_n_tiles;
        const long long M = s.M;
        auto geo = [num_n, M](int tile) {
            EpiTile g;
            const int m_tile = tile / num_n;
            g.n_tile = tile - m_tile * num_n;
            g.m0 = static_cast<long long>(m_tile) * BM;
            const long long left = M - g.m0;
            g.rows = left < BM ? static_cast<int>(left) : BM;
            return g;
        };
        if constexpr (MODE == MODE_SEP)
            epilogue_direct_sep<BNQ>(s, p.ep, p.y, tmem_base, accf0, acce0, p.num_tiles, limit,
                                     abort_flag, geo);
        else if constexpr (SC)
            epilogue_direct_pair_sc<BNQ>(s, p.ep, p.y, tmem_base, accf0, acce0, p.num_tiles,
                                         p.ktiles, p.sk, limit, abort_flag, geo, &p.sc);
        else
            epilogue_direct_pair<BNQ>(s, p.ep, p.y, tmem_base, accf0, acce0, p.num_tiles,
                                      p.ktiles, p.sk, limit, abort_flag, geo);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, C::TMEM_COLS);
    }
}

#include "qconv_ws.cuh"
#include "qconv_vs.cuh"
#include "qconv_gather.cuh"
#include "qconv_stempool.cuh"
#include "qconv_pw.cuh"
#include "qconv_cg2.cuh"
#include "qconv_dw.cuh"

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

CUtensorMapSwizzle swizzle_for_row(int row_bytes) {
    return row_bytes == 128 ? CU_TENSOR_MAP_SWIZZLE_128B
                            : (row_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                               : CU_TENSOR_MAP_SWIZZLE_32B);
}

// Activation im2col map: boxes of BM output pixels x `channels` channels.
bool encode_x_im2col(CUtensorMap* map, const ConvShape& s, const void* x, int channels) {
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
        upper, static_cast<cuuint32_t>(channels), BM, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
        swizzle_for_row(channels * 2), CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
        CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// Activation tiled map for halo boxes: `channels` x `cols` columns (Wo if 0) x `rows` rows
// of one image; with `step` > 1 the box takes every step-th column and row (it spans
// step * cols columns and step * rows rows).
bool encode_x_halo(CUtensorMap* map, const ConvShape& s, const void* x, int channels,
                   int rows, int cols = 0, int step = 1) {
    const cuuint64_t dims[4] = {static_cast<cuuint64_t>(s.Cin), static_cast<cuuint64_t>(s.W),
                                static_cast<cuuint64_t>(s.H), static_cast<cuuint64_t>(s.N)};
    const cuuint64_t strides[3] = {static_cast<cuuint64_t>(s.Cin) * 2,
                                   static_cast<cuuint64_t>(s.Cin) * 2 * s.W,
                                   static_cast<cuuint64_t>(s.Cin) * 2 * s.W * s.H};
    const cuuint32_t box[4] = {static_cast<cuuint32_t>(channels),
                               static_cast<cuuint32_t>((cols > 0 ? cols : s.Wo) * step),
                               static_cast<cuuint32_t>(rows * step), 1};
    const cuuint32_t estr[4] = {1, static_cast<cuuint32_t>(step), static_cast<cuuint32_t>(step),
                                1};
    const CUresult r = g_encode_tiled(
        map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(x), dims, strides, box, estr,
        CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle_for_row(channels * 2),
        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// Input of a 4-channel layer viewed as groups of G pixel pairs (16 G bytes):
// [N][H][W/(2G)][8 G], boxes of `boxg` groups x `rows` input rows of one image, no swizzle
// (dense rows in shared memory).
bool encode_x_pairs(CUtensorMap* map, const ConvShape& s, const void* x, int group, int boxg,
                    int rows) {
    const cuuint64_t WG = static_cast<cuuint64_t>(s.W / (2 * group));
    const cuuint64_t eb = 16ull * group;
    const cuuint64_t dims[4] = {8ull * group, WG, static_cast<cuuint64_t>(s.H),
                                static_cast<cuuint64_t>(s.N)};
    const cuuint64_t strides[3] = {eb, eb * WG, eb * WG * s.H};
    const cuuint32_t box[4] = {8u * group, static_cast<cuuint32_t>(boxg),
                               static_cast<cuuint32_t>(rows), 1};
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    const CUresult r = g_encode_tiled(
        map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(x), dims, strides, box, estr,
        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
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
                                      CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle_for_row(kappa * 2),
                                      CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                                      CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// The shared-memory opt-in is per device and kernel; set it once for each.
template <typename K>
cudaError_t set_smem_once(K kern, int bytes, std::atomic<unsigned long long>& done) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const unsigned long long bit = 1ull << (dev & 63);
    if (!(done.load() & bit)) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
        if (e != cudaSuccess) return e;
        done.fetch_or(bit);
    }
    return cudaSuccess;
}

template <int KAPPA, int BNQ, int MODE, bool SC = false>
cudaError_t launch_cfg(const CUtensorMap maps[6], const TcParams& prm, int grid,
                       cudaStream_t stream, const ScMaps* scm = nullptr) {
    using C = Cfg<KAPPA, BNQ, MODE>;
    if constexpr (!C::FITS || (SC && MODE != MODE_PAIR && MODE != MODE_QUAD)) {
        return cudaErrorInvalidValue;
    } else {
        auto kern = qconv_tc_kernel<KAPPA, BNQ, MODE, SC>;
        static std::atomic<unsigned long long> attr_done{0};
        cudaError_t e = set_smem_once(kern, C::SMEM_BYTES, attr_done);
        if (e != cudaSuccess) return e;
        ScMaps none;
        memset(&none, 0, sizeof(none));
        return launch_pdl(kern, dim3(grid), dim3(NUM_THREADS), C::SMEM_BYTES, stream, maps[0],
                          maps[1], maps[2], maps[3], maps[4], prm, scm != nullptr ? *scm : none);
    }
}

template <int KAPPA, int BNQ, int MODE>
constexpr bool cfg_fits() {
    return Cfg<KAPPA, BNQ, MODE>::FITS;
}

// Encoded tensor maps of recent calls, keyed by every value that goes into them, so a
// layer called repeatedly on the same buffers skips the host-side encodes.
struct MapKey {
    const void* ptr[6];
    int N, H, W, Cin, Cout, kh, kw, stride, pad, kappa, bnq, variant;
    bool operator==(const MapKey& o) const {
        for (int i = 0; i < 6; ++i)
            if (ptr[i] != o.ptr[i]) return false;
        return N == o.N && H == o.H && W == o.W && Cin == o.Cin && Cout == o.Cout &&
               kh == o.kh && kw == o.kw && stride == o.stride && pad == o.pad &&
               kappa == o.kappa && bnq == o.bnq && variant == o.variant;
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

bool cache_lookup(const MapKey& key, CUtensorMap* maps) {
    std::lock_guard<std::mutex> lk(g_map_mu);
    for (int i = 0; i < kMapCacheSize; ++i)
        if (g_map_cache[i].valid && g_map_cache[i].key == key) {
            for (int l = 0; l < 6; ++l) maps[l] = g_map_cache[i].maps[l];
            return true;
        }
    return false;
}

void cache_store(const MapKey& key, const CUtensorMap* maps) {
    std::lock_guard<std::mutex> lk(g_map_mu);
    MapEntry& e = g_map_cache[g_map_next];
    g_map_next = (g_map_next + 1) % kMapCacheSize;
    e.key = key;
    for (int l = 0; l < 6; ++l) e.maps[l] = maps[l];
    e.valid = true;
}

MapKey make_key(const ConvShape& s, const void* x, const void* const w[4], const void* out,
                int kappa, int bnq, int variant) {
    MapKey key;
    key.ptr[0] = x;
    for (int l = 0; l < 4; ++l) key.ptr[1 + l] = w[l];
    key.ptr[5] = out;
    key.N = s.N; key.H = s.H; key.W = s.W; key.Cin = s.Cin; key.Cout = s.Cout;
    key.kh = s.kh; key.kw = s.kw; key.stride = s.stride; key.pad = s.pad;
    key.kappa = kappa; key.bnq = bnq; key.variant = variant;
    return key;
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

int grid_for(const TcOptions& opt, int num_sms, int num_tiles) {
    int grid = opt.max_ctas > 0 ? opt.max_ctas : num_sms;
    if (grid > num_tiles) grid = num_tiles;
    return grid < 1 ? 1 : grid;
}

template <bool HALO, int KH, int NI, bool SEP>
cudaError_t launch_ws_kernel(const CUtensorMap& map, const WsParams& prm, int grid,
                             cudaStream_t stream) {
    auto kern = qconv_ws_kernel<HALO, KH, NI, SEP>;
    static std::atomic<unsigned long long> attr_done{0};
    cudaError_t e = set_smem_once(kern, WsCfg::SMEM_BYTES, attr_done);
    if (e != cudaSuccess) return e;
    return launch_pdl(kern, dim3(grid), dim3(WIDE_THREADS), WsCfg::SMEM_BYTES, stream, map, prm);
}

template <bool SEP>
cudaError_t launch_ws_form(const CUtensorMap& map, const WsParams& prm, int grid, bool halo,
                           bool k3x3, int ni, cudaStream_t stream) {
    if (ni == 2) {
        if (halo && k3x3) return launch_ws_kernel<true, 3, 2, SEP>(map, prm, grid, stream);
        if (halo) return launch_ws_kernel<true, 0, 2, SEP>(map, prm, grid, stream);
        return launch_ws_kernel<false, 0, 2, SEP>(map, prm, grid, stream);
    }
    if (halo && k3x3) return launch_ws_kernel<true, 3, ISSUERS, SEP>(map, prm, grid, stream);
    if (halo) return launch_ws_kernel<true, 0, ISSUERS, SEP>(map, prm, grid, stream);
    return launch_ws_kernel<false, 0, ISSUERS, SEP>(map, prm, grid, stream);
}

cudaError_t launch_ws(const ConvShape& s, const void* x, const void* const w[4],
                      const EpilogueArgs& ep, void* out, const TcOptions& opt, int num_sms,
                      cudaStream_t stream, char* err, size_t errlen) {
    WsParams prm;
    prm.s = s;
    prm.ep = ep;
    for (int l = 0; l < 4; ++l) prm.w[l] = static_cast<const __nv_bfloat16*>(w[l]);
    prm.y = out;
    prm.wait_limit_ns = opt.wait_limit_ns;
    prm.inject_stall = opt.inject_stall;
    prm.taps = s.kh * s.kw;
    const bool halo = ws_halo_ok(s) && opt.ws_halo != 0;
    prm.halo = halo ? 1 : 0;
    long long tiles;
    if (halo) {
        prm.R = BM / s.Wo;
        prm.tpi = (s.Ho + prm.R - 1) / prm.R;
        prm.kblocks = s.kw;
        prm.box_bytes = s.Wo * (prm.R + s.kh - 1) * WS_ROW_BYTES;
        tiles = static_cast<long long>(s.N) * prm.tpi;
    } else {
        prm.R = 0;
        prm.tpi = 0;
        prm.kblocks = prm.taps;
        prm.box_bytes = BM * WS_ROW_BYTES;
        tiles = (s.M + BM - 1) / BM;
    }
    if (tiles > 0x7fffffffLL) {
        snprintf(err, errlen, "too many tiles");
        return cudaErrorInvalidValue;
    }
    prm.num_tiles = static_cast<int>(tiles);
    prm.stage_bytes = (prm.box_bytes + 1023) & ~1023;
    const int ni = opt.ws_issuers == 2 || opt.ws_issuers == ISSUERS
                       ? opt.ws_issuers
                       : ws_issuers(prm.stage_bytes, prm.kblocks);
    int per = WsCfg::RING_BYTES / prm.stage_bytes / ni;
    if (per > WsCfg::NSTAGE / ni) per = WsCfg::NSTAGE / ni;
    if (per < 1) {
        snprintf(err, errlen, "weight-stationary pixel box of %d bytes does not fit %d issuers",
                 prm.box_bytes, ni);
        return cudaErrorInvalidValue;
    }
    prm.per = per;

    const MapKey key = make_key(s, x, w, out, 16, 16, halo ? 3 : 2);
    CUtensorMap maps[6];
    if (!cache_lookup(key, maps)) {
        const bool okx = halo ? encode_x_halo(&maps[0], s, x, 4 * 16, prm.R + s.kh - 1)
                              : encode_x_im2col(&maps[0], s, x, 4 * 16);
        if (!okx) {
            snprintf(err, errlen, "tensor-map encode failed for the activation tensor");
            return cudaErrorInvalidValue;
        }
        for (int l = 1; l < 6; ++l) maps[l] = maps[0];
        cache_store(key, maps);
    }
    const int grid = grid_for(opt, num_sms, prm.num_tiles);
    if (s.sep)
        set_kernel_name(halo ? "qconv_ws_kernel<halo,issuers=%d,sep>"
                             : "qconv_ws_kernel<im2col,issuers=%d,sep>",
                        ni);
    else
        set_kernel_name(halo ? "qconv_ws_kernel<halo,issuers=%d>"
                             : "qconv_ws_kernel<im2col,issuers=%d>",
                        ni);
    const bool k3x3 = s.kh == 3 && s.kw == 3;
    return s.sep ? launch_ws_form<true>(maps[0], prm, grid, halo, k3x3, ni, stream)
                 : launch_ws_form<false>(maps[0], prm, grid, halo, k3x3, ni, stream);
}

// Activation map of the vertical-tap kernel: boxes of 64 channels x P columns x 1 row x E
// images (one input row of E images, lane e P + c at shared-memory row e P + c).
bool encode_x_vs(CUtensorMap* map, const ConvShape& s, const void* x, int P, int E) {
    const cuuint64_t dims[4] = {static_cast<cuuint64_t>(s.Cin), static_cast<cuuint64_t>(s.W),
                                static_cast<cuuint64_t>(s.H), static_cast<cuuint64_t>(s.N)};
    const cuuint64_t strides[3] = {static_cast<cuuint64_t>(s.Cin) * 2,
                                   static_cast<cuuint64_t>(s.Cin) * 2 * s.W,
                                   static_cast<cuuint64_t>(s.Cin) * 2 * s.W * s.H};
    const cuuint32_t box[4] = {static_cast<cuuint32_t>(s.Cin), static_cast<cuuint32_t>(P), 1u,
                               static_cast<cuuint32_t>(E)};
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    const CUresult r = g_encode_tiled(
        map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(x), dims, strides, box, estr,
        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

template <int NBOX, bool SEP>
cudaError_t launch_vs_kernel(const CUtensorMap& map, const VsParams& prm, int grid,
                             cudaStream_t stream) {
    auto kern = qconv_vs_kernel<NBOX, SEP>;
    static std::atomic<unsigned long long> attr_done{0};
    cudaError_t e = set_smem_once(kern, VsCfg::SMEM_BYTES, attr_done);
    if (e != cudaSuccess) return e;
    return launch_pdl(kern, dim3(grid), dim3(VS_THREADS), VsCfg::SMEM_BYTES, stream, map, prm);
}

cudaError_t launch_vs(const ConvShape& s, const void* x, const void* const w[4],
                      const EpilogueArgs& ep, void* out, const TcOptions& opt, int num_sms,
                      cudaStream_t stream, char* err, size_t errlen) {
    VsParams prm;
    prm.s = s;
    prm.ep = ep;
    for (int l = 0; l < 4; ++l) prm.w[l] = static_cast<const __nv_bfloat16*>(w[l]);
    prm.y = out;
    prm.wait_limit_ns = opt.wait_limit_ns;
    prm.inject_stall = opt.inject_stall;
    int nbox = 0;
    if (!vs_ok(s) || !vs_layout(s.Wo, &nbox, &prm.E, &prm.P)) {
        snprintf(err, errlen,
                 "vertical-tap mode needs a 3x3 filter, stride 1, pad <= 2, Cin = Cout = 64 and "
                 "Wo + 2 <= %d or Wo dividing %d", BM, BM);
        return cudaErrorInvalidValue;
    }
    prm.box_bytes = prm.E * prm.P * 128;
    prm.row_bytes = (nbox * prm.box_bytes + 1023) & ~1023;
    prm.stage_bytes = (nbox == 1 ? 3 : 1) * prm.row_bytes;  // input rows per stage: 3 or 1
    prm.nst = VsCfg::RING_BYTES / prm.stage_bytes;
    if (prm.nst > VS_MAX_STAGES) prm.nst = VS_MAX_STAGES;
    if (prm.nst < 2) {
        snprintf(err, errlen, "vertical-tap stage of %d bytes does not fit", prm.stage_bytes);
        return cudaErrorInvalidValue;
    }
    const long long groups = (s.N + prm.E - 1) / prm.E;
    const int grid0 = opt.max_ctas > 0 ? opt.max_ctas : num_sms;
    prm.bh = opt.vs_rows >= 1 && opt.vs_rows <= VS_BH ? opt.vs_rows : vs_pick_bh(s, prm.E, grid0);
    prm.nbands = (s.Ho + prm.bh - 1) / prm.bh;
    const long long units = groups * prm.nbands;
    if (units > 0x7fffffffLL) {
        snprintf(err, errlen, "too many work units");
        return cudaErrorInvalidValue;
    }
    prm.num_units = static_cast<int>(units);

    const MapKey key = make_key(s, x, w, out, prm.P, prm.E, 12);
    CUtensorMap maps[6];
    if (!cache_lookup(key, maps)) {
        if (!encode_x_vs(&maps[0], s, x, prm.P, prm.E)) {
            snprintf(err, errlen, "tensor-map encode failed for the activation tensor");
            return cudaErrorInvalidValue;
        }
        for (int l = 1; l < 6; ++l) maps[l] = maps[0];
        cache_store(key, maps);
    }
    const int grid = grid_for(opt, num_sms, prm.num_units);
    set_kernel_name(s.sep ? "qconv_vs_kernel<boxes=%d,rows=%d,sep>"
                          : "qconv_vs_kernel<boxes=%d,rows=%d>",
                    nbox, prm.bh);
    if (nbox == 3)
        return s.sep ? launch_vs_kernel<3, true>(maps[0], prm, grid, stream)
                     : launch_vs_kernel<3, false>(maps[0], prm, grid, stream);
    return s.sep ? launch_vs_kernel<1, true>(maps[0], prm, grid, stream)
                 : launch_vs_kernel<1, false>(maps[0], prm, grid, stream);
}

cudaError_t launch_gather(const ConvShape& s, const void* x, const void* const w[4],
                          const EpilogueArgs& ep, void* out, const TcOptions& opt, int num_sms,
                          cudaStream_t stream, char* err, size_t errlen) {
    GatherParams prm;
    prm.s = s;
    prm.ep = ep;
    for (int l = 0; l < 4; ++l) prm.w[l] = static_cast<const __nv_bfloat16*>(w[l]);
    prm.y = out;
    prm.wait_limit_ns = opt.wait_limit_ns;
    prm.inject_stall = opt.inject_stall;
    prm.lead = s.pad & 1;
    prm.nsp = gather_nsp(s);
    prm.shift = (s.pad + prm.lead) / 2;
    const int W2 = s.W / 2;
    prm.group = W2 % 8 == 0 ? 8 : (W2 % 4 == 0 ? 4 : (W2 % 2 == 0 ? 2 : 1));
    prm.d0 = ((-prm.shift) % prm.group + prm.group) % prm.group;
    const int boxw = GA_TILE_W + prm.nsp - 1;  // pairs a tile reads per filter row
    prm.boxg = (prm.d0 + boxw + prm.group - 1) / prm.group;
    prm.box_bytes = prm.boxg * 16 * prm.group;
    prm.box_stride = prm.box_bytes;
    prm.stage_bytes = (s.kh * prm.box_stride + 1023) & ~1023;
    int per = GaCfg::RING_BYTES / prm.stage_bytes / ISSUERS;
    if (per > GaCfg::MAX_PER) per = GaCfg::MAX_PER;
    if (per < 1 || s.kh * prm.nsp > GA_MAX_UNITS || prm.boxg > 256 || s.kh > 256) {
        snprintf(err, errlen, "pixel-pair kernel: kh=%d kw=%d does not fit", s.kh, s.kw);
        return cudaErrorInvalidValue;
    }
    prm.per = per;
    prm.segs = (s.Wo + GA_TILE_W - 1) / GA_TILE_W;
    const long long rows = static_cast<long long>(s.N) * s.Ho;
    const long long tiles = rows * prm.segs;
    if (tiles > 0x7fffffffLL) {
        snprintf(err, errlen, "too many tiles");
        return cudaErrorInvalidValue;
    }
    prm.num_tiles = static_cast<int>(tiles);

    const MapKey key = make_key(s, x, w, out, 1, 16, 6);
    CUtensorMap maps[6];
    if (!cache_lookup(key, maps)) {
        if (!encode_x_pairs(&maps[0], s, x, prm.group, prm.boxg, s.kh)) {
            snprintf(err, errlen, "tensor-map encode failed for the activation tensor");
            return cudaErrorInvalidValue;
        }
        for (int l = 1; l < 6; ++l) maps[l] = maps[0];
        cache_store(key, maps);
    }
    const int grid = grid_for(opt, num_sms, prm.num_tiles);
    static std::atomic<unsigned long long> done_74{0}, done_any{0};
    set_kernel_name("qconv_pairs_kernel");
    if (s.kh == 7 && prm.nsp == 4) {  // the 7x7 stem
        auto kern = qconv_pairs_kernel<7, 4>;
        cudaError_t e = set_smem_once(kern, GaCfg::SMEM_BYTES, done_74);
        if (e != cudaSuccess) return e;
        return launch_pdl(kern, dim3(grid), dim3(WIDE_THREADS), GaCfg::SMEM_BYTES, stream,
                          maps[0], prm);
    } else {
        auto kern = qconv_pairs_kernel<0, 0>;
        cudaError_t e = set_smem_once(kern, GaCfg::SMEM_BYTES, done_any);
        if (e != cudaSuccess) return e;
        return launch_pdl(kern, dim3(grid), dim3(WIDE_THREADS), GaCfg::SMEM_BYTES, stream,
                          maps[0], prm);
    }
}

// Pointwise layer input: stride 1, [N H W][Cin] in boxes of 64 channels x `rows` pixels;
// stride 2, [N H / 2][2][W / 2][2][Cin] in boxes of 64 channels x 1 x Wo x 1 x `rows` (the
// sampled pixels of that many output rows).  128-byte swizzle.
bool encode_x_pw(CUtensorMap* map, const ConvShape& s, const void* x, int rows) {
    const cuuint64_t e = static_cast<cuuint64_t>(s.Cin) * 2;  // bytes per pixel
    const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    CUresult r;
    if (s.stride == 1) {
        const cuuint64_t dims[2] = {static_cast<cuuint64_t>(s.Cin),
                                    static_cast<cuuint64_t>(s.N) * s.H * s.W};
        const cuuint64_t strides[1] = {e};
        const cuuint32_t box[2] = {64, static_cast<cuuint32_t>(rows)};
        r = g_encode_tiled(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(x), dims,
                           strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                           CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    } else {
        const cuuint64_t dims[5] = {static_cast<cuuint64_t>(s.Cin), 2,
                                    static_cast<cuuint64_t>(s.W / 2), 2,
                                    static_cast<cuuint64_t>(s.N) * (s.H / 2)};
        const cuuint64_t strides[4] = {e, 2 * e, e * s.W, 2 * e * s.W};
        const cuuint32_t box[5] = {64, 1, static_cast<cuuint32_t>(s.Wo), 1,
                                   static_cast<cuuint32_t>(rows)};
        r = g_encode_tiled(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(x), dims,
                           strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                           CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                           CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    }
    return r == CUDA_SUCCESS;
}

template <int STRIDE, int ACT>
cudaError_t launch_pw_kernel(const CUtensorMap& map, const PwParams& prm, int grid,
                             cudaStream_t stream) {
    auto kern = qconv_pw_kernel<STRIDE, ACT>;
    static std::atomic<unsigned long long> attr_done{0};
    cudaError_t e = set_smem_once(kern, PwCfg::SMEM_BYTES, attr_done);
    if (e != cudaSuccess) return e;
    return launch_pdl(kern, dim3(grid), dim3(PW_THREADS), PwCfg::SMEM_BYTES, stream, map, prm);
}

cudaError_t launch_pw(const ConvShape& s, const void* x, const void* const w[4],
                      const EpilogueArgs& ep, void* out, const TcOptions& opt, int num_sms,
                      cudaStream_t stream, char* err, size_t errlen) {
    PwParams prm;
    prm.s = s;
    prm.ep = ep;
    for (int l = 0; l < 4; ++l) prm.w[l] = static_cast<const __nv_bfloat16*>(w[l]);
    prm.y = out;
    prm.wait_limit_ns = opt.wait_limit_ns;
    prm.inject_stall = opt.inject_stall;
    prm.kchunks = s.Cin / 64;
    prm.stages = PwCfg::max_stages(prm.kchunks);
    prm.mblocks = s.Cout / 128;
    prm.npix = s.M;
    // (no box extends past the tensor: tiles shrink for inputs smaller than one tile)
    if (s.stride == 1) {
        prm.rows_per_tile = 0;
        prm.tile_pix = s.M < PW_NPIX ? static_cast<int>(s.M) : PW_NPIX;
        prm.num_tiles = static_cast<int>((s.M + prm.tile_pix - 1) / prm.tile_pix);
    } else {
        const long long rows = static_cast<long long>(s.N) * s.Ho;
        prm.rows_per_tile = PW_NPIX / s.Wo;
        if (prm.rows_per_tile > rows) prm.rows_per_tile = static_cast<int>(rows);
        prm.tile_pix = prm.rows_per_tile * s.Wo;
        prm.num_tiles = static_cast<int>((rows + prm.rows_per_tile - 1) / prm.rows_per_tile);
    }
    if (prm.stages < 2 || s.M > 0x7fffffffLL) {
        snprintf(err, errlen, "pointwise kernel: Cin=%d does not fit", s.Cin);
        return cudaErrorInvalidValue;
    }
    const MapKey key = make_key(s, x, w, out, 64, 32, 8);
    CUtensorMap maps[6];
    if (!cache_lookup(key, maps)) {
        if (!encode_x_pw(&maps[0], s, x,
                         s.stride == 1 ? prm.tile_pix : prm.rows_per_tile)) {
            snprintf(err, errlen, "tensor-map encode failed for the activation tensor");
            return cudaErrorInvalidValue;
        }
        for (int l = 1; l < 6; ++l) maps[l] = maps[0];
        cache_store(key, maps);
    }
    // every CTA keeps one channel block: the grid is a multiple of the block count
    const long long work = static_cast<long long>(prm.mblocks) * prm.num_tiles;
    int grid = opt.max_ctas > 0 ? opt.max_ctas : num_sms;
    if (grid > work) grid = static_cast<int>(work);
    grid = grid / prm.mblocks * prm.mblocks;
    if (grid < prm.mblocks) grid = prm.mblocks;
    set_kernel_name(s.stride == 1 ? "qconv_pw_kernel<s1>" : "qconv_pw_kernel<s2>");
    const int act = s.act;
    if (s.stride == 1) {
        if (act == 1) return launch_pw_kernel<1, 1>(maps[0], prm, grid, stream);
        if (act == 2) return launch_pw_kernel<1, 2>(maps[0], prm, grid, stream);
        return launch_pw_kernel<1, 0>(maps[0], prm, grid, stream);
    }
    if (act == 1) return launch_pw_kernel<2, 1>(maps[0], prm, grid, stream);
    if (act == 2) return launch_pw_kernel<2, 2>(maps[0], prm, grid, stream);
    return launch_pw_kernel<2, 0>(maps[0], prm, grid, stream);
}

// fp32 RGB pixels [N][H][W][3] viewed as [N][H][3 W / 32][32]: boxes of `rows` whole rows
// (128-byte elements; W a multiple of 32).
bool encode_rgb_rows(CUtensorMap* map, const ConvShape& s, const float* rgb, int rows) {
    const cuuint64_t rb = 12ull * s.W;  // bytes per row
    const cuuint64_t dims[4] = {32, static_cast<cuuint64_t>(3 * s.W / 32),
                                static_cast<cuuint64_t>(s.H), static_cast<cuuint64_t>(s.N)};
    const cuuint64_t strides[3] = {128, rb, rb * s.H};
    const cuuint32_t box[4] = {32, static_cast<cuuint32_t>(3 * s.W / 32),
                               static_cast<cuuint32_t>(rows), 1};
    const cuuint32_t estr[4] = {1, 1, 1, 1};
    const CUresult r = g_encode_tiled(
        map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, const_cast<float*>(rgb), dims, strides, box,
        estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

// Sizes of the CTA-pair kernel for shape s with pixel staging stg (CG_PER_TAP, CG_HALO or
// CG_HALO2); false if the staging does not apply or its stage ring or the staged letters do
// not fit.
bool cg2_plan(const ConvShape& s, int stg, Cg2Params* prm) {
    if (!cg2_ok(s) || (stg == CG_HALO && !cg2_halo_ok(s)) ||
        (stg == CG_HALO2 && !cg2_halo2_ok(s)))
        return false;
    const bool halo = stg != CG_PER_TAP;
    prm->cpt = s.Cin / 64;
    prm->kchunks = s.kh * s.kw * prm->cpt;
    prm->letter_bytes = 32 * s.kh * s.kw * s.Qin * 2;
    long long tiles;
    if (stg == CG_HALO2) {
        // R output rows of Wp = Wo + 1 pixels per tile; four parity boxes of R + 1 rows of
        // Wp pixels per stage, each from a 1024-byte boundary.  A padding MMA row reads at
        // most Wp + 1 rows past the 128th row of box (0, 0) and Wp rows past that of box
        // (0, 1), both inside the following boxes; boxes (1, 0) and (1, 1) are read at
        // offsets of at most one row, within their (R + 1) Wp > 128 rows plus the next box.
        prm->Wp = s.Wo + 1;
        prm->R = BM / prm->Wp;
        prm->tpi = (s.Ho + prm->R - 1) / prm->R;
        const int box_rows = (prm->R + 1) * prm->Wp;
        prm->box_stride = (box_rows * 128 + 1023) / 1024 * 1024;
        prm->stage_bytes = 4 * prm->box_stride;
        prm->box_bytes = 4 * box_rows * 128;
        prm->nst = prm->cpt;
        tiles = static_cast<long long>(s.N) * prm->tpi;
    } else if (halo) {
        // R output rows of Wp = Wo + 2 pixels per tile; a stage holds the R + 2 input rows
        // of the box and every row an MMA of the last tap reads (128 + 2 Wp + 2)
        prm->Wp = s.Wo + 2;
        prm->R = BM / prm->Wp;
        prm->tpi = (s.Ho + prm->R - 1) / prm->R;
        const int box_rows = prm->R + 2;
        const int rows = box_rows * prm->Wp > BM + 2 * prm->Wp + 2 ? box_rows * prm->Wp
                                                                     : BM + 2 * prm->Wp + 2;
        prm->stage_bytes = (rows * 128 + 1023) / 1024 * 1024;
        prm->box_bytes = box_rows * prm->Wp * 128;
        prm->nst = prm->cpt;
        tiles = static_cast<long long>(s.N) * prm->tpi;
    } else {
        prm->stage_bytes = CgCfg::ACHUNK;
        prm->box_bytes = CgCfg::ACHUNK;
        prm->nst = prm->kchunks;
        tiles = (s.M + BM - 1) / BM;
    }
    const int ring = CgCfg::ring_bytes(prm->kchunks);
    const int ni = halo ? 1 : 2;  // MMA issuers (the kernel's NI)
    prm->per = ring / prm->stage_bytes / ni;
    if (prm->per > CgCfg::MAX_STAGES / ni) prm->per = CgCfg::MAX_STAGES / ni;
    // halo: at least two stages, so one lands while the other's MMAs run
    if (prm->per < (halo ? 2 : 1) || 4 * prm->letter_bytes > ring || tiles > 0x7ffffffeLL)
        return false;
    prm->num_tiles = static_cast<int>(tiles);
    prm->num_ptiles = static_cast<int>((tiles + 1) / 2);
    return true;
}

// The halo staging that fits shape s (CG_HALO or CG_HALO2), else CG_PER_TAP.
int cg2_halo_staging(const ConvShape& s) {
    Cg2Params prm = {};
    if (cg2_plan(s, CG_HALO, &prm)) return CG_HALO;
    if (cg2_plan(s, CG_HALO2, &prm)) return CG_HALO2;
    return CG_PER_TAP;
}

cudaError_t launch_cg2(const ConvShape& s, const void* x, const void* const w[4],
                       const EpilogueArgs& ep, void* out, const TcOptions& opt, int num_sms,
                       cudaStream_t stream, char* err, size_t errlen) {
    Cg2Params prm = {};
    const int stg = cg2_halo_staging(s);
    if (!cg2_plan(s, stg, &prm)) {
        snprintf(err, errlen, "CTA-pair kernel: Cin=%d Cout=%d %dx%d does not fit", s.Cin,
                 s.Cout, s.kh, s.kw);
        return cudaErrorInvalidValue;
    }
    prm.s = s;
    prm.ep = ep;
    for (int l = 0; l < 4; ++l) prm.w[l] = static_cast<const __nv_bfloat16*>(w[l]);
    prm.y = out;
    prm.wait_limit_ns = opt.wait_limit_ns;
    prm.inject_stall = opt.inject_stall;
    const MapKey key = make_key(s, x, w, out, 64, 32, 10 + stg);
    CUtensorMap maps[6];
    if (!cache_lookup(key, maps)) {
        const bool okx = stg == CG_HALO2 ? encode_x_halo(&maps[0], s, x, 64, prm.R + 1, prm.Wp, 2)
                         : stg == CG_HALO ? encode_x_halo(&maps[0], s, x, 64, prm.R + 2, prm.Wp)
                                          : encode_x_im2col(&maps[0], s, x, 64);
        if (!okx) {
            snprintf(err, errlen, "tensor map encoding failed for the activation tensor");
            return cudaErrorInvalidValue;
        }
        for (int l = 1; l < 6; ++l) maps[l] = maps[0];
        cache_store(key, maps);
    }
    int pairs = (opt.max_ctas > 0 ? opt.max_ctas : num_sms) / 2;
    if (pairs > prm.num_ptiles) pairs = prm.num_ptiles;
    if (pairs < 1) pairs = 1;
    set_kernel_name(stg == CG_HALO2  ? "qconv_cg2_kernel<halo2>"
                    : stg == CG_HALO ? "qconv_cg2_kernel<halo>"
                                     : "qconv_cg2_kernel");
    auto kern = stg == CG_HALO2  ? qconv_cg2_kernel<CG_HALO2, 1>
                : stg == CG_HALO ? qconv_cg2_kernel<CG_HALO, 1>
                                 : qconv_cg2_kernel<CG_PER_TAP, 2>;
    static std::atomic<unsigned long long> attr_done[3];
    cudaError_t e = set_smem_once(kern, CgCfg::SMEM_BYTES, attr_done[stg]);
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * pairs);
    cfg.blockDim = dim3(CG_THREADS);
    cfg.dynamicSmemBytes = CgCfg::SMEM_BYTES;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kern, maps[0], prm);
}

template <int ROWS, int NSP, int ACT, bool RGB>
cudaError_t launch_stem_pool_kernel(const CUtensorMap& map, const StemPoolParams& prm, int grid,
                                    cudaStream_t stream) {
    auto kern = qconv_stem_pool_kernel<ROWS, NSP, ACT, RGB>;
    static std::atomic<unsigned long long> attr_done{0};
    cudaError_t e = set_smem_once(kern, SpCfg::SMEM_BYTES, attr_done);
    if (e != cudaSuccess) return e;
    return launch_pdl(kern, dim3(grid), dim3(SP_THREADS), SpCfg::SMEM_BYTES, stream, map, prm);
}

// x: bf16 quaternion pixels [N][H][W][4], or (rgb) fp32 RGB pixels [N][H][W][3] mapped by
// Eq. 4 in the kernel's loader.
cudaError_t launch_stem_pool(const ConvShape& s, const void* x, const void* const w[4],
                             const EpilogueArgs& ep, void* out, const TcOptions& opt,
                             int num_sms, cudaStream_t stream, char* err, size_t errlen,
                             bool rgb = false) {
    StemPoolParams prm;
    prm.s = s;
    prm.ep = ep;
    for (int l = 0; l < 4; ++l) prm.w[l] = static_cast<const __nv_bfloat16*>(w[l]);
    prm.y = out;
    prm.wait_limit_ns = opt.wait_limit_ns;
    prm.inject_stall = opt.inject_stall;
    prm.lead = s.pad & 1;
    prm.nsp = gather_nsp(s);
    prm.shift = (s.pad + prm.lead) / 2;
    const int W2 = s.W / 2;
    prm.group = W2 % 8 == 0 ? 8 : (W2 % 4 == 0 ? 4 : (W2 % 2 == 0 ? 2 : 1));
    prm.d0 = ((-prm.shift) % prm.group + prm.group) % prm.group;
    prm.gx0 = (-prm.shift - prm.d0) / prm.group;  // exact: -shift - d0 is a multiple of G
    prm.nmma = (s.Wo + 15) / 16 * 16;
    const int boxw = prm.nmma + prm.nsp - 1;  // pairs the N rows read per input row
    const int boxg = (prm.d0 + boxw + prm.group - 1) / prm.group;
    prm.row_bytes = boxg * 16 * prm.group;
    prm.rows = s.kh + 2;
    prm.stage_bytes = (prm.rows * prm.row_bytes + 1023) & ~1023;
    prm.rgb = rgb ? static_cast<const float*>(x) : nullptr;
    prm.rgb_row_bytes = 12 * s.W;
    prm.rgb_stage_bytes = rgb ? (prm.rows * prm.rgb_row_bytes + 1023) & ~1023 : 0;
    int per = (SpCfg::RING_BYTES - SP_RGB_SLOTS * prm.rgb_stage_bytes) / prm.stage_bytes /
              SP_ISSUERS;
    if (per > SpCfg::MAX_PER) per = SpCfg::MAX_PER;
    prm.rgb_off = SpCfg::RING_OFF + SP_ISSUERS * per * prm.stage_bytes;
    if (!stem_pool_ok(s) || per < 1 || boxg > 256 || prm.rows > 256 ||
        (rgb && (s.W % 32 != 0 || 3 * s.W / 32 > 256))) {
        snprintf(err, errlen, "stem pooling kernel: kh=%d kw=%d W=%d does not fit", s.kh, s.kw,
                 s.W);
        return cudaErrorInvalidValue;
    }
    prm.per = per;
    prm.Hp = (s.Ho - 1) / 2 + 1;
    prm.Wp = (s.Wo - 1) / 2 + 1;
    prm.total_rows = static_cast<long long>(s.N) * prm.Hp;
    if (prm.total_rows > 0x7fffffffLL) {
        snprintf(err, errlen, "too many pooled rows");
        return cudaErrorInvalidValue;
    }
    const MapKey key = make_key(s, x, w, out, 1, 16, rgb ? 9 : 7);
    CUtensorMap maps[6];
    if (!cache_lookup(key, maps)) {
        const bool okx = rgb ? encode_rgb_rows(&maps[0], s, static_cast<const float*>(x), prm.rows)
                             : encode_x_pairs(&maps[0], s, x, prm.group, boxg, prm.rows);
        if (!okx) {
            snprintf(err, errlen, "tensor-map encode failed for the activation tensor");
            return cudaErrorInvalidValue;
        }
        for (int l = 1; l < 6; ++l) maps[l] = maps[0];
        cache_store(key, maps);
    }
    const int grid = grid_for(opt, num_sms, static_cast<int>(prm.total_rows));
    set_kernel_name(rgb ? "qconv_stem_pool_kernel<rgb>" : "qconv_stem_pool_kernel");
#define QUAN_SP_LAUNCH(R)                                                                    \
    if (prm.rows == 9 && prm.nsp == 4) { /* the 7x7 stem */                                  \
        if (s.act == 1) return launch_stem_pool_kernel<9, 4, 1, R>(maps[0], prm, grid, stream); \
        if (s.act == 2) return launch_stem_pool_kernel<9, 4, 2, R>(maps[0], prm, grid, stream); \
        return launch_stem_pool_kernel<9, 4, 0, R>(maps[0], prm, grid, stream);                \
    }                                                                                        \
    if (s.act == 1) return launch_stem_pool_kernel<0, 0, 1, R>(maps[0], prm, grid, stream);    \
    if (s.act == 2) return launch_stem_pool_kernel<0, 0, 2, R>(maps[0], prm, grid, stream);    \
    return launch_stem_pool_kernel<0, 0, 0, R>(maps[0], prm, grid, stream);
    if (rgb) {
        QUAN_SP_LAUNCH(true)
    }
    QUAN_SP_LAUNCH(false)
#undef QUAN_SP_LAUNCH
}

// ---------------------------------------------------------------- weight gradient
constexpr int DW_SMEM_MAX = 232448;  // dynamic shared memory a CTA may opt into

// Tiling of the tensor-core weight gradient (see qconv_dw.cuh); false if the shape has none.
bool dw_plan(const ConvShape& s, int num_sms, dwk::DwParams* p) {
    if (s.stride < 1 || s.stride > 2 || s.Cin % 64 != 0 || s.Cout % 64 != 0) return false;
    if (s.Cout > 256 && s.Cout % 256 != 0) return false;
    dwk::DwParams q = {};
    q.sep = s.sep ? 1 : 0;
    q.stride = s.stride;
    q.Ho = s.Ho; q.Wo = s.Wo; q.Qin = s.Qin; q.Qout = s.Qout;
    q.kh = s.kh; q.kw = s.kw; q.pad = s.pad; q.taps = s.kh * s.kw;
    q.nxc = s.Cin / 64;
    q.units = q.taps * q.nxc;
    q.npairs = (q.units + 1) / 2;
    q.ncols = s.Cout <= 256 ? s.Cout : 256;
    q.nyb = q.ncols / 64;
    int a_max = 512 / q.ncols;
    if (a_max > dwk::MAX_PAIRS) a_max = dwk::MAX_PAIRS;
    if (a_max > q.npairs) a_max = q.npairs;
    // the most unit pairs per CTA for which some pixel block fits; for those, the block
    // shape (Ht rows x Wbox columns, Wbox a multiple of 8 so a block is whole 1024-byte
    // swizzle atoms) with the least padding, preferring three or more pipeline stages
    bool found = false;
    for (int a_per = a_max; a_per >= 1 && !found; --a_per) {
        double best = 1e30;
        const int wcand[2] = {(s.Wo + 7) / 8 * 8, (s.Wo + 15) / 16 * 16};
        for (int wc = 0; wc < 2; ++wc) {
            const int Wbox = wcand[wc];
            if (Wbox * s.stride > 256) continue;  // the x box spans stride * Wbox columns
            for (int Ht = 1; Ht <= 8; ++Ht) {
                const int P = Wbox * Ht;
                if (P % 16 != 0 || P > 256 || Ht * s.stride > 256) continue;
                const long long stage =
                    static_cast<long long>(2 * a_per + q.nyb) * P * dwk::BOX_ROW;
                long long stages = (DW_SMEM_MAX - 1024 - dwk::BAR_BYTES -
                                    dwk::tail_bytes(P, s.stride)) /
                                   stage;
                if (stages > dwk::MAX_STAGES) stages = dwk::MAX_STAGES;
                if (stages < 2) continue;
                const int rb = (s.Ho + Ht - 1) / Ht;
                double score = static_cast<double>(P) * rb / (static_cast<double>(s.Wo) * s.Ho);
                if (stages < 3) score *= 1.15;
                if (P < 32) score *= 1.2;
                if (score < best) {
                    best = score;
                    q.a_per = a_per;
                    q.Wbox = Wbox; q.Ht = Ht; q.P = P; q.rblocks = rb;
                    q.stages = static_cast<int>(stages);
                    q.stage_bytes = static_cast<uint32_t>(stage);
                }
            }
        }
        found = best < 1e29;
    }
    if (!found) return false;
    q.pair_groups = (q.npairs + q.a_per - 1) / q.a_per;
    q.groups = q.pair_groups * (s.Cout / q.ncols);
    q.kblocks = static_cast<long long>(s.N) * q.rblocks;
    long long splits = num_sms / q.groups;
    if (splits < 1) splits = 1;
    if (splits > q.kblocks) splits = q.kblocks;
    q.splits = static_cast<int>(splits);
    if (static_cast<long long>(q.groups) * q.splits > 0x7fffffffLL) return false;
    uint32_t cols = 32;
    while (cols < static_cast<uint32_t>(q.a_per * q.ncols)) cols <<= 1;
    q.tmem_cols = cols;
    *p = q;
    return true;
}

// [N][H][W][C] bf16, boxes of 64 channels x Wbox columns x Ht rows of one image, SW128;
// with `step` > 1 the box traverses every step-th column and row (it spans step * Wbox
// columns and step * Ht rows, and the copy brings Wbox x Ht pixels).
bool encode_dw_map(CUtensorMap* map, const void* t, int C, int W, int H, int N, int Wbox,
                   int Ht, int step = 1) {
    const cuuint64_t dims[4] = {static_cast<cuuint64_t>(C), static_cast<cuuint64_t>(W),
                                static_cast<cuuint64_t>(H), static_cast<cuuint64_t>(N)};
    const cuuint64_t strides[3] = {static_cast<cuuint64_t>(C) * 2,
                                   static_cast<cuuint64_t>(C) * 2 * W,
                                   static_cast<cuuint64_t>(C) * 2 * W * H};
    const cuuint32_t box[4] = {64, static_cast<cuuint32_t>(Wbox * step),
                               static_cast<cuuint32_t>(Ht * step), 1};
    const cuuint32_t estr[4] = {1, static_cast<cuuint32_t>(step), static_cast<cuuint32_t>(step),
                                1};
    const CUresult r = g_encode_tiled(
        map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(t), dims, strides, box, estr,
        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

}  // namespace

size_t tc_split_workspace_bytes(int num_sms) {
    // a partial tile of the widest tile (bnq = 64: 4 x 64 fp32 columns x 128 rows) and a
    // flag per CTA of a full-width grid
    const size_t n = num_sms > 0 ? static_cast<size_t>(num_sms) : 0;
    return (n * 512 * 64 * sizeof(float) + n * 4 + 255) / 256 * 256;
}

bool tc_supported(const ConvShape& s, const void* x, const void* const w[4], const void* out,
                  const EpilogueArgs& ep) {
    auto al16 = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
    if ((s.Qin % 16 != 0 || s.Qout % 16 != 0) && (s.sep || !gather_ok(s))) return false;
    // TMA coordinates of the output (pixel index) are 32-bit
    if (s.M > 0x7fffffffLL) return false;
    if (!al16(x) || !al16(out) || !al16(w[0]) || !al16(w[1]) || !al16(w[2]) || !al16(w[3]))
        return false;
    // the epilogues read the residual and the per-channel vectors 16 bytes at a time
    if (ep.residual && !al16(ep.residual)) return false;
    if ((ep.bias && !al16(ep.bias)) || (ep.scale && !al16(ep.scale)) ||
        (ep.shift && !al16(ep.shift)))
        return false;
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
    if (s.sep && opt.mode != 0) {
        snprintf(err, errlen, "MMA-mode overrides apply to the full Hamilton form only");
        return cudaErrorInvalidValue;
    }
    if (!s.sep && gather_ok(s) && (opt.mode == 0 || opt.mode == 4))
        return launch_gather(s, x, w, ep, out, opt, num_sms, stream, err, errlen);
    if (opt.mode == 4) {
        snprintf(err, errlen,
                 "pixel-pair gather mode needs Cin = 4, Cout = 64, stride 2, even W and at "
                 "most %d K units", GA_MAX_UNITS);
        return cudaErrorInvalidValue;
    }
    if (pw_ok(s, ep) && (opt.mode == 0 || opt.mode == 5))
        return launch_pw(s, x, w, ep, out, opt, num_sms, stream, err, errlen);
    // The CTA-pair kernel: by default for stride-1 3x3 layers with 128 output channels,
    // whose halo stages feed 36 MMAs each; with per-tap stages (other shapes) only on
    // request, since four MMAs per stage leave the pixel loads' latency exposed and the
    // pair kernel below is faster there.
    // 3x3 stride-1 layers of 16 -> 16 quaternion channels: the vertical taps stacked along N,
    // by default where one box per input row serves (Wo + 2 lanes per image); with three
    // boxes per row (Wo dividing 128) the weight-stationary kernel below is faster
    int vs_nbox = 0, vs_e = 0, vs_p = 0;
    const bool vs_one_box = vs_ok(s) && vs_layout(s.Wo, &vs_nbox, &vs_e, &vs_p) && vs_nbox == 1;
    if (s.sep != 2 && vs_ok(s) && (opt.mode == 7 || (opt.mode == 0 && vs_one_box)))
        return launch_vs(s, x, w, ep, out, opt, num_sms, stream, err, errlen);
    if (opt.mode == 7) {
        snprintf(err, errlen,
                 "vertical-tap mode needs a 3x3 filter, stride 1, pad <= 2, Cin = Cout = 64 and "
                 "Wo + 2 <= %d or Wo dividing %d", BM, BM);
        return cudaErrorInvalidValue;
    }
    if (!s.sep && cg2_ok(s) &&
        (opt.mode == 6 || (opt.mode == 0 && cg2_halo_staging(s) != CG_PER_TAP)))
        return launch_cg2(s, x, w, ep, out, opt, num_sms, stream, err, errlen);
    if (opt.mode == 6) {
        snprintf(err, errlen,
                 "CTA-pair mode needs the full form, Cout = 128, Cin a multiple of 64 and "
                 "kh x kw x Cin <= %d", CG_MAX_K);
        return cudaErrorInvalidValue;
    }
    if (opt.mode == 5) {
        snprintf(err, errlen,
                 "pointwise mode needs a 1x1 filter, pad 0, stride 1 or 2 (even H and W, "
                 "Wo <= %d), Cin a multiple of 64 up to %d, Cout a multiple of 128 and no "
                 "residual", PW_NPIX, PW_MAX_CIN);
        return cudaErrorInvalidValue;
    }
    // Weight-stationary for 16 -> 16 quaternion channels (the whole expanded weight fits);
    // pair mode (N = 2 BNQ per MMA) otherwise, unless the tile is so narrow that even
    // pairs stay far below the tensor pipe's per-instruction cost.
    const bool ws_ok = s.Qin == 16 && s.Qout == 16 && s.kh * s.kw <= WS_MAX_TAPS;
    int kappa = pick_kappa(s.Qin, opt.kappa);
    const int bnq = pick_bnq(s.Qout, opt.bnq);
    int mode;
    if (s.sep == 2) mode = MODE_SEPT;
    else if (s.sep) mode = ws_ok ? MODE_WS : MODE_SEP;
    else if (opt.mode == 1) mode = MODE_QUAD;
    else if (opt.mode == 2) mode = MODE_PAIR;
    else if (opt.mode == 3) mode = MODE_WS;
    else mode = ws_ok ? MODE_WS : (bnq >= 32 ? MODE_PAIR : MODE_QUAD);
    if (mode == MODE_WS) {
        if (!ws_ok) {
            snprintf(err, errlen, "weight-stationary mode needs Cin = Cout = 64 and <= %d taps",
                     WS_MAX_TAPS);
            return cudaErrorInvalidValue;
        }
        return launch_ws(s, x, w, ep, out, opt, num_sms, stream, err, errlen);
    }
    if (kappa == 0 || bnq == 0) {
        snprintf(err, errlen, "requested tile (kappa=%d, bnq=%d) does not divide Qin=%d/Qout=%d",
                 opt.kappa, opt.bnq, s.Qin, s.Qout);
        return cudaErrorInvalidValue;
    }
    // Only two 6-slot stages of 64 x 64 letter blocks plus 64-channel pixel tiles fit in
    // shared memory; 32-channel K blocks give four.
    if (mode == MODE_PAIR && kappa == 64 && bnq == 64 && opt.kappa == 0) kappa = 32;
    {
        bool fits = true;
#define QUAN_FIT_CASE(K, B)                                                        \
    if (kappa == K && bnq == B)                                                    \
        fits = mode == MODE_PAIR ? cfg_fits<K, B, MODE_PAIR>()                     \
             : mode == MODE_SEP  ? cfg_fits<K, B, MODE_SEP>()                      \
             : mode == MODE_SEPT ? cfg_fits<K, B, MODE_SEPT>()                     \
                                 : cfg_fits<K, B, MODE_QUAD>();
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
    const MapKey key = make_key(s, x, w, out, kappa, bnq, 0);
    CUtensorMap maps[6];
    if (!cache_lookup(key, maps)) {
        if (!encode_x_im2col(&maps[0], s, x, kappa)) {
            snprintf(err, errlen, "cuTensorMapEncodeIm2col failed for the activation tensor");
            return cudaErrorInvalidValue;
        }
        for (int l = 0; l < 4; ++l)
            if (!encode_w(&maps[1 + l], s, w[l], kappa, bnq)) {
                snprintf(err, errlen, "cuTensorMapEncodeTiled failed for weight letter %d", l);
                return cudaErrorInvalidValue;
            }
        maps[5] = maps[0];
        cache_store(key, maps);
    }
    TcParams prm;
    prm.s = s;
    prm.ep = ep;
    prm.kchunks = s.Qin / kappa;
    prm.ktiles = s.kh * s.kw * prm.kchunks;
    prm.num_n_tiles = s.Qout / bnq;
    prm.y = out;
    const long long m_tiles = (s.M + BM - 1) / BM;
    const long long tiles = m_tiles * prm.num_n_tiles;
    if (tiles > 0x7fffffffLL) {
        snprintf(err, errlen, "too many tiles");
        return cudaErrorInvalidValue;
    }
    prm.num_tiles = static_cast<int>(tiles);
    prm.wait_limit_ns = opt.wait_limit_ns;
    prm.inject_stall = opt.inject_stall;
    const int grid = grid_for(opt, num_sms, prm.num_tiles);
    // K ranges split evenly over the CTAs when the tiles make between one and two waves
    // (the second one partial: at 196 tiles on 152 CTAs the whole-tile schedule runs two
    // full tile times where 1.3 would do) and the caller gave a workspace for the partial
    // tiles (full form only).  With more waves the contiguous ranges cost more, in the L2
    // reuse between neighbouring tiles the strided schedule keeps, than the last wave's
    // idle CTAs (measured: the backbone's 14 x 14 layers at 5.2 waves 6% slower, its 7 x 7
    // layers at 1.3 waves 13% faster)
    prm.sk.on = 0;
    prm.sk.partial = nullptr;
    prm.sk.flags = nullptr;
    const size_t slot_bytes = static_cast<size_t>(512) * bnq * sizeof(float);
    const size_t sk_need = static_cast<size_t>(grid) * slot_bytes + static_cast<size_t>(grid) * 4;
    if (opt.sk_ws != nullptr && opt.sk_ws_bytes >= sk_need &&
        (mode == MODE_PAIR || mode == MODE_QUAD) && prm.num_tiles > grid &&
        prm.num_tiles < 2 * grid) {
        prm.sk.on = 1;
        prm.sk.partial = static_cast<float*>(opt.sk_ws);
        prm.sk.flags = reinterpret_cast<unsigned*>(static_cast<char*>(opt.sk_ws) +
                                                   static_cast<size_t>(grid) * slot_bytes);
    }
    set_kernel_name(mode == MODE_PAIR   ? "qconv_tc_kernel<pair,kappa=%d,bnq=%d>"
                    : mode == MODE_SEP  ? "qconv_tc_kernel<sep,kappa=%d,bnq=%d>"
                    : mode == MODE_SEPT ? "qconv_tc_kernel<sep_t,kappa=%d,bnq=%d>"
                                        : "qconv_tc_kernel<quad,kappa=%d,bnq=%d>",
                    kappa, bnq);
    if (prm.sk.on) {  // the name records the split
        const size_t len = strlen(t_kernel_name);
        if (len > 0 && len + 10 < sizeof(t_kernel_name)) {
            t_kernel_name[len - 1] = '\0';
            strcat(t_kernel_name, ",splitk>");
        }
    }

#define QUAN_TC_CASE(K, B)                                                       \
    if (kappa == K && bnq == B)                                                  \
        return mode == MODE_PAIR   ? launch_cfg<K, B, MODE_PAIR>(maps, prm, grid, stream)  \
               : mode == MODE_SEP  ? launch_cfg<K, B, MODE_SEP>(maps, prm, grid, stream)   \
               : mode == MODE_SEPT ? launch_cfg<K, B, MODE_SEPT>(maps, prm, grid, stream)  \
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

// The convolution and a 1x1 shortcut on the same input in one QUAD/PAIR launch (the
// shortcut's N tiles after the convolution's, on the K blocks of the filter tap that reads
// x at (ho stride, wo stride)): the tile sizes, or false when the shapes do not allow it.
bool tc_shortcut_plan(const ConvShape& s, int qout_sc, const TcOptions& opt, int* kappa_out,
                      int* bnq_out, int* mode_out) {
    if (s.sep || s.Qin % 16 != 0 || s.Qout % 16 != 0 || qout_sc <= 0 || qout_sc % 16 != 0)
        return false;
    if (s.pad >= s.kh || s.pad >= s.kw) return false;
    // the 1x1 / stride shortcut without padding has the convolution's output size
    if ((s.H - 1) / s.stride + 1 != s.Ho || (s.W - 1) / s.stride + 1 != s.Wo) return false;
    int kappa = pick_kappa(s.Qin, opt.kappa);
    const int bnq = pick_bnq(s.Qout, opt.bnq);
    if (kappa == 0 || bnq == 0 || qout_sc % bnq != 0) return false;
    int mode;
    if (opt.mode == 1) mode = MODE_QUAD;
    else if (opt.mode == 2) mode = MODE_PAIR;
    else if (opt.mode == 0) mode = bnq >= 32 ? MODE_PAIR : MODE_QUAD;
    else return false;
    if (mode == MODE_PAIR && kappa == 64 && bnq == 64 && opt.kappa == 0) kappa = 32;
    bool fits = false;
#define QUAN_FIT_CASE(K, B)                                                          \
    if (kappa == K && bnq == B)                                                      \
        fits = mode == MODE_PAIR ? cfg_fits<K, B, MODE_PAIR>() : cfg_fits<K, B, MODE_QUAD>();
    QUAN_FIT_CASE(16, 16) QUAN_FIT_CASE(16, 32) QUAN_FIT_CASE(16, 64)
    QUAN_FIT_CASE(32, 16) QUAN_FIT_CASE(32, 32) QUAN_FIT_CASE(32, 64)
    QUAN_FIT_CASE(64, 16) QUAN_FIT_CASE(64, 32) QUAN_FIT_CASE(64, 64)
#undef QUAN_FIT_CASE
    if (!fits) return false;
    *kappa_out = kappa;
    *bnq_out = bnq;
    *mode_out = mode;
    return true;
}

bool tc_shortcut_supported(const ConvShape& s, const void* x, const void* const w[4],
                           const void* out, const EpilogueArgs& ep, const void* const wsc[4],
                           int qout_sc, const EpilogueArgs& ep_sc, const void* out_sc,
                           const TcOptions& opt) {
    int kappa, bnq, mode;
    if (!tc_shortcut_plan(s, qout_sc, opt, &kappa, &bnq, &mode)) return false;
    if (!tc_supported(s, x, w, out, ep)) return false;
    ConvShape s1 = s;  // the shortcut as a layer of its own, for the alignment checks
    s1.kh = s1.kw = 1;
    s1.pad = 0;
    s1.Qout = qout_sc;
    s1.Cout = 4 * qout_sc;
    EpilogueArgs e1 = ep_sc;
    e1.residual = nullptr;
    return ep_sc.residual == nullptr && tc_supported(s1, x, wsc, out_sc, e1);
}

cudaError_t launch_qconv_tc_shortcut(const ConvShape& s, const void* x, const void* const w[4],
                                     const EpilogueArgs& ep, void* out,
                                     const void* const wsc[4], int qout_sc, int act_sc,
                                     const EpilogueArgs& ep_sc, void* out_sc,
                                     const TcOptions& opt, int num_sms, cudaStream_t stream,
                                     char* err, size_t errlen) {
    if (!load_encoders()) {
        snprintf(err, errlen, "tensor-map encoders unavailable from the CUDA driver");
        return cudaErrorNotSupported;
    }
    int kappa, bnq, mode;
    if (!tc_shortcut_plan(s, qout_sc, opt, &kappa, &bnq, &mode)) {
        snprintf(err, errlen, "no fused shortcut form for this layer");
        return cudaErrorInvalidValue;
    }
    ConvShape s1 = s;  // the shortcut's 1x1 letters [Qout_sc][1][1][Qin]
    s1.kh = s1.kw = 1;
    s1.pad = 0;
    s1.Qout = qout_sc;
    s1.Cout = 4 * qout_sc;
    CUtensorMap maps[6];
    const MapKey key = make_key(s, x, w, out, kappa, bnq, 20);
    if (!cache_lookup(key, maps)) {
        if (!encode_x_im2col(&maps[0], s, x, kappa)) {
            snprintf(err, errlen, "cuTensorMapEncodeIm2col failed for the activation tensor");
            return cudaErrorInvalidValue;
        }
        for (int l = 0; l < 4; ++l)
            if (!encode_w(&maps[1 + l], s, w[l], kappa, bnq)) {
                snprintf(err, errlen, "cuTensorMapEncodeTiled failed for weight letter %d", l);
                return cudaErrorInvalidValue;
            }
        maps[5] = maps[0];
        cache_store(key, maps);
    }
    ScMaps scm;
    {
        CUtensorMap m2[6];
        const MapKey key2 = make_key(s1, x, wsc, out_sc, kappa, bnq, 21);
        if (!cache_lookup(key2, m2)) {
            for (int l = 0; l < 4; ++l)
                if (!encode_w(&m2[l], s1, wsc[l], kappa, bnq)) {
                    snprintf(err, errlen, "cuTensorMapEncodeTiled failed for shortcut letter %d",
                             l);
                    return cudaErrorInvalidValue;
                }
            m2[4] = m2[5] = m2[0];
            cache_store(key2, m2);
        }
        for (int l = 0; l < 4; ++l) scm.w[l] = m2[l];
    }
    TcParams prm;
    prm.s = s;
    prm.ep = ep;
    prm.kchunks = s.Qin / kappa;
    prm.ktiles = s.kh * s.kw * prm.kchunks;
    prm.sc.n_conv = s.Qout / bnq;
    prm.num_n_tiles = prm.sc.n_conv + qout_sc / bnq;
    prm.y = out;
    prm.sc.ktiles = prm.kchunks;
    prm.sc.dh = prm.sc.dw = s.pad;
    prm.sc.tap = s.pad * s.kw + s.pad;
    prm.sc.Qout = qout_sc;
    prm.sc.act = act_sc;
    prm.sc.y = out_sc;
    prm.sc.ep = ep_sc;
    prm.sc.ep.residual = nullptr;
    const long long tiles = (s.M + BM - 1) / BM * prm.num_n_tiles;
    if (tiles > 0x7fffffffLL) {
        snprintf(err, errlen, "too many tiles");
        return cudaErrorInvalidValue;
    }
    prm.num_tiles = static_cast<int>(tiles);
    prm.wait_limit_ns = opt.wait_limit_ns;
    prm.inject_stall = opt.inject_stall;
    prm.sk.on = 0;  // whole tiles: a split would cut shortcut and convolution tiles alike
    prm.sk.partial = nullptr;
    prm.sk.flags = nullptr;
    const int grid = grid_for(opt, num_sms, prm.num_tiles);
    set_kernel_name(mode == MODE_PAIR ? "qconv_tc_kernel<pair,kappa=%d,bnq=%d,shortcut>"
                                      : "qconv_tc_kernel<quad,kappa=%d,bnq=%d,shortcut>",
                    kappa, bnq);
#define QUAN_TC_CASE(K, B)                                                               \
    if (kappa == K && bnq == B)                                                          \
        return mode == MODE_PAIR                                                         \
                   ? launch_cfg<K, B, MODE_PAIR, true>(maps, prm, grid, stream, &scm)    \
                   : launch_cfg<K, B, MODE_QUAD, true>(maps, prm, grid, stream, &scm);
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

bool tc_stem_pool_supported(const ConvShape& s, const void* x, const void* const w[4],
                            const void* out, const EpilogueArgs& ep) {
    return stem_pool_ok(s) && tc_supported(s, x, w, out, ep);
}

cudaError_t launch_qconv_stem_pool(const ConvShape& s, const void* x, const void* const w[4],
                                   const EpilogueArgs& ep, void* out, const TcOptions& opt,
                                   int num_sms, cudaStream_t stream, char* err, size_t errlen) {
    if (!load_encoders()) {
        snprintf(err, errlen, "cuTensorMapEncodeTiled is not available");
        return cudaErrorInvalidValue;
    }
    return launch_stem_pool(s, x, w, ep, out, opt, num_sms, stream, err, errlen);
}

bool tc_stem_pool_rgb_supported(const ConvShape& s, const float* rgb, const void* const w[4],
                                const void* out, const EpilogueArgs& ep) {
    return stem_pool_ok(s) && s.W % 32 == 0 && 3 * s.W / 32 <= 256 &&
           tc_supported(s, rgb, w, out, ep);
}

cudaError_t launch_qconv_stem_pool_rgb(const ConvShape& s, const float* rgb,
                                       const void* const w[4], const EpilogueArgs& ep, void* out,
                                       const TcOptions& opt, int num_sms, cudaStream_t stream,
                                       char* err, size_t errlen) {
    if (!load_encoders()) {
        snprintf(err, errlen, "cuTensorMapEncodeTiled is not available");
        return cudaErrorInvalidValue;
    }
    return launch_stem_pool(s, rgb, w, ep, out, opt, num_sms, stream, err, errlen, true);
}

bool bwd_weight_tc_supported(const ConvShape& s, const void* x, const void* dy) {
    dwk::DwParams p;
    return dw_plan(s, 152, &p) && reinterpret_cast<uintptr_t>(x) % 16 == 0 &&
           reinterpret_cast<uintptr_t>(dy) % 16 == 0;
}

cudaError_t launch_bwd_weight_tc(const ConvShape& s, const void* x, const void* dy,
                                 float* const dw[4], int num_sms,
                                 unsigned long long wait_limit_ns, cudaStream_t stream,
                                 char* err, size_t errlen) {
    dwk::DwParams p;
    if (!dw_plan(s, num_sms, &p) || !bwd_weight_tc_supported(s, x, dy)) {
        snprintf(err, errlen, "no tensor-core weight-gradient tiling for this shape");
        return cudaErrorInvalidValue;
    }
    if (!load_encoders()) {
        snprintf(err, errlen, "cuTensorMapEncodeTiled is not available");
        return cudaErrorInvalidValue;
    }
    CUtensorMap mx, mdy;
    if (!encode_dw_map(&mx, x, s.Cin, s.W, s.H, s.N, p.Wbox, p.Ht, s.stride) ||
        !encode_dw_map(&mdy, dy, s.Cout, s.Wo, s.Ho, s.N, p.Wbox, p.Ht)) {
        snprintf(err, errlen, "tensor-map encode failed for the weight gradient");
        return cudaErrorInvalidValue;
    }
    const size_t bytes = static_cast<size_t>(s.Qout) * s.kh * s.kw * s.Qin * sizeof(float);
    for (int L = 0; L < 4; ++L) {
        cudaError_t e = cudaMemsetAsync(dw[L], 0, bytes, stream);
        if (e != cudaSuccess) return e;
    }
    p.wait_limit_ns = wait_limit_ns;
    p.dwr = dw[0];
    p.dwi = dw[1];
    p.dwj = dw[2];
    p.dwk = dw[3];
    const int smem = p.stages * static_cast<int>(p.stage_bytes) + dwk::BAR_BYTES +
                     dwk::tail_bytes(p.P, s.stride) + 1024;
    static std::atomic<unsigned long long> attr_done{0};
    cudaError_t e = set_smem_once(dwk::qconv_dw_kernel, DW_SMEM_MAX, attr_done);
    if (e != cudaSuccess) return e;
    set_kernel_name(p.sep ? "qconv_dw_kernel<pairs=%d,n=%d,sep>" : "qconv_dw_kernel<pairs=%d,n=%d>",
                    p.a_per, p.ncols);
    return launch_pdl(dwk::qconv_dw_kernel, dim3(static_cast<unsigned>(p.groups * p.splits)),
                      dim3(dwk::THREADS), static_cast<size_t>(smem), stream, mx, mdy, p);
}

const char* last_tc_kernel() { return t_kernel_name; }

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
