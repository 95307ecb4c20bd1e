// tc_common.cuh -- pieces shared by the tensor-core quaternion convolution kernels
// (qconv_tc.cu is the only translation unit that includes this file): constants, the
// device status word, descriptor helpers, bounded waits, the issuer bookkeeping and the
// register-only epilogues.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>

#include <cstdint>

#include "internal.h"
#include "ptx.cuh"

namespace quan {

// Device status word: bits set by kernels whose bounded waits ran out.
__device__ unsigned int g_status;

namespace tc {

constexpr int BM = 128;           // rows (output pixels) of the MMA tile
constexpr int NUM_THREADS = 384;  // 12 warps
constexpr int EPI_WARP0 = 4;      // warps 4..11: epilogue
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

// The same signs indexed by letter: bit (4 L + p) is set when letter L enters through input
// component p (output component L xor p) with a minus sign.
constexpr uint32_t letter_sign_table() {
    uint32_t t = 0;
    for (int L = 0; L < 4; ++L)
        for (int p = 0; p < 4; ++p) t |= ((NEG_MASK >> (4 * (L ^ p) + p)) & 1u) << (4 * L + p);
    return t;
}
constexpr uint32_t LETTER_SIGNS = letter_sign_table();

// The separable form of Eq. 7: output component m = sum over p of sign * (W_p conv x_p),
// bit (4 m + p) of SEP_NEG marking the negative terms,
//   y_r = +r -i -j -k,  y_i = +r +i +j -k,  y_j = +r -i +j +k,  y_k = +r +i -j +k.
// As a block weight it is row block m, column block p = sign * W_p; SEP_LETTER_SIGNS holds
// letter p's signs down its column, bit (4 p + m).
constexpr uint32_t SEP_NEG = (1u << 1) | (1u << 2) | (1u << 3)  // y_r: -i -j -k
                             | (1u << 7)                        // y_i: -k
                             | (1u << 9)                        // y_j: -i
                             | (1u << 14);                      // y_k: -j
constexpr uint32_t sep_letter_sign_table() {
    uint32_t t = 0;
    for (int p = 0; p < 4; ++p)
        for (int m = 0; m < 4; ++m) t |= ((SEP_NEG >> (4 * m + p)) & 1u) << (4 * p + m);
    return t;
}
constexpr uint32_t SEP_LETTER_SIGNS = sep_letter_sign_table();

// tcgen05 shared-memory matrix descriptors (K-major, swizzled operand tiles) are built
// as two 32-bit words: the low word holds the start address >> 4 (bits 0-13) and the
// leading byte offset (bits 16-29, unused for these layouts, set to 1); the high word
// holds the stride byte offset >> 4 (pitch of 8-row core-matrix groups), the
// descriptor version (bit 46) and the swizzle mode (bits 61-63).
__device__ __forceinline__ uint32_t desc_lo(uint32_t saddr) {
    return ((saddr & 0x3FFFFu) >> 4) | (1u << 16);
}

constexpr uint32_t desc_hi(uint32_t sbo_bytes, uint32_t layout) {
    return (sbo_bytes >> 4) | (1u << 14) | (layout << 29);
}

// swizzle mode of the descriptor for K-major rows of `row_bytes` (128, 64 or 32)
constexpr uint32_t desc_layout(int row_bytes) {
    return row_bytes == 128 ? 2u : (row_bytes == 64 ? 4u : 6u);
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
    if (act == 2) {
        // SiLU z / (1 + e^-z) with the fast exponential and division (a few ulp of fp32,
        // far below the bf16 output's rounding); z >= -80 keeps the divisor below 2^126,
        // where the fast division is exact enough (below that the value is ~0 anyway)
        return __fdividef(z, 1.0f + __expf(-fmaxf(z, -80.0f)));
    }
    return z;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    const __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<const uint32_t*>(&v);
}

__device__ __forceinline__ uint4 negate_bf16x8(uint4 v) {
    v.x ^= 0x80008000u;
    v.y ^= 0x80008000u;
    v.z ^= 0x80008000u;
    v.w ^= 0x80008000u;
    return v;
}

// Bounded wait: false once the CTA-wide abort flag is up or `limit` ns have passed (then
// the status bit is recorded and the abort flag raised).  Between checks the thread
// sleeps in the barrier wait (WAIT_SUSPEND_NS at most, woken early by the phase
// completing), so waiting roles leave the issue slots to the working ones.
constexpr uint32_t WAIT_SUSPEND_NS = 20000;

__device__ __forceinline__ bool wait_or_abort(uint32_t bar, uint32_t parity, uint64_t limit,
                                              volatile int* abort_flag, unsigned code) {
    if (mbar_try_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    while (true) {
        if (mbar_try_wait_sleep(bar, parity, WAIT_SUSPEND_NS)) return true;
        if (*abort_flag) return false;
        if (global_timer_ns() - t0 > limit) {
            atomicOr(&g_status, code);
            *abort_flag = 1;
            return false;
        }
    }
}

// Bounded wait for a sequence word in shared memory (written with st_release_shared) to
// reach `target` (wrap-safe comparison).  Same failure handling as wait_or_abort.
__device__ __forceinline__ bool flag_wait_or_abort(uint32_t addr, uint32_t target,
                                                   uint64_t limit, volatile int* abort_flag,
                                                   unsigned code) {
    if (static_cast<int>(ld_acquire_shared(addr) - target) >= 0) return true;
    const uint64_t t0 = global_timer_ns();
    while (true) {
        if (static_cast<int>(ld_acquire_shared(addr) - target) >= 0) return true;
        if (*abort_flag) return false;
        if (global_timer_ns() - t0 > limit) {
            atomicOr(&g_status, code);
            *abort_flag = 1;
            return false;
        }
        __nanosleep(32);
    }
}

// Wait for the most recent fill of each stage a producer armed, so that no copy still
// targets this CTA's shared memory when it exits after an abort.
__device__ __forceinline__ void drain_fills(uint32_t bar0, int stages, uint32_t filled,
                                            uint32_t parity, uint64_t limit) {
    for (int i = 0; i < stages; ++i) {
        if (!(filled & (1u << i))) continue;
        const uint64_t t0 = global_timer_ns();
        while (!mbar_try_wait(bar0 + 8u * i, (parity >> i) & 1u)) {
            if (global_timer_ns() - t0 > limit) {
                atomicOr(&g_status, STATUS_TIMEOUT_DRAIN);
                break;
            }
        }
    }
}

// Geometry of one output tile as the epilogue sees it.
struct EpiTile {
    long long m0;  // linear index of the pixel in TMEM lane 0
    int rows;      // valid lanes (pixels) of the tile
    int n_tile;    // quaternion output channel block
};

// Direct epilogue for 64-channel outputs (Qout = 16: one output-channel tile), used by the
// weight-stationary and pixel-pair kernels (16 warps: producer, 3 issuers, 12 epilogue).
// The tensor cores' operand reads keep the shared-memory pipe saturated, so this epilogue
// touches no shared memory.  Warps 4..15 form three groups of four (one warp per TMEM lane
// quadrant); group g takes the CTA's local tiles k with k % 3 == g, the tiles issuer g
// produced, so three tiles are in flight.  Per tile and per 32-channel half a warp
//   1. loads its 32 rows x 32 columns with one tcgen05.ld (once the second half is in
//      registers it releases the accumulator buffer, acce, 128 arrivals per tile);
//   2. transposes, within each group of 4 lanes, the 4 x 4 matrix of 8-channel chunks
//      (rows x chunks) with two shfl_xor stages, so lane i of lane group r holds
//      channels 32 half + 8i .. +7 of that group's 4 rows;
//   3. applies act(scale * (acc + bias) + shift + residual) (IQBN inference form of
//      Eq. 11-12) with its channels' vectors held in registers, rounds to bf16 and
//      writes 16 bytes per lane per row: every store instruction writes 64-byte halves of
//      8 whole output rows; the residual is read the same way.
constexpr int EPI_GROUPS = 3;
constexpr int WIDE_THREADS = 512;  // block size of the kernels using this epilogue
constexpr int EPI2_ACCE_COUNT = 128;  // the 4 warps of one group arrive once per tile

// Tiles of a CTA are issued round robin by NI threads (local tile k by issuer k % NI;
// NI = ISSUERS = 3, or 2 where three issuers would leave each with too few stages).
// mbarrier parity waits only tell a phase from its neighbours, so a waiter must never get
// two phases ahead of a barrier; that is guaranteed by letting every stage and
// accumulator buffer be used by one issuer only, whose program order then orders the
// uses:
//   - issuer i owns stages i * per .. i * per + per - 1; its n-th stage use (counting its
//     K blocks in order) is stage i * per + n % per in round n / per;
//   - issuer i owns accumulator buffers i and i + NI, alternating over its tiles;
//     a buffer's tiles all have the same parity, so one epilogue group drains it.
constexpr int ISSUERS = 3;
constexpr int ISSUER_ACC = 2 * ISSUERS;  // accumulator buffer barriers (64 columns each)

__device__ __forceinline__ void issuer_stage(int i, int n, int per, int& stage,
                                             uint32_t& phase) {
    stage = i * per + n % per;
    phase = static_cast<uint32_t>(n / per) & 1u;
}

// The same mapping walked one use at a time, without the division by `per` (an issuing
// thread's integer work between MMAs is idle tensor time): after n calls of next(),
// stage(i) and phase equal issuer_stage(i, n, ...).  One cursor serves every issuer whose
// use counts advance together.
struct StageCursor {
    int per, idx;
    uint32_t phase;
    __device__ __forceinline__ explicit StageCursor(int per_) : per(per_), idx(0), phase(0u) {}
    __device__ __forceinline__ int stage(int i) const { return i * per + idx; }
    __device__ __forceinline__ void next() {
        if (++idx == per) {
            idx = 0;
            phase ^= 1u;
        }
    }
};

template <int NI>
__device__ __forceinline__ void issuer_acc_n(int k, int& buf, uint32_t& use) {
    const int j = k / NI;
    buf = (k - j * NI) + NI * (j & 1);
    use = static_cast<uint32_t>(j >> 1) & 1u;
}

__device__ __forceinline__ void issuer_acc(int k, int& buf, uint32_t& use) {
    issuer_acc_n<ISSUERS>(k, buf, use);
}

// One transpose stage: lanes i and i ^ K exchange the chunks whose index differs from the
// lane in bit K (E[j] for bit_K(j) != bit_K(i), partner's E[j ^ K] in return).
template <int K, int NCH>
__device__ __forceinline__ void chunk_transpose_stage(float (&E)[NCH][8], int i) {
    const bool hi = (i & K) != 0;
#pragma unroll
    for (int j0 = 0; j0 < NCH; ++j0) {
        if (j0 & K) continue;
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const float send = hi ? E[j0][e] : E[j0 ^ K][e];
            const float recv = __shfl_xor_sync(0xffffffffu, send, K);
            if (hi)
                E[j0][e] = recv;
            else
                E[j0 ^ K][e] = recv;
        }
    }
}

// v[0..7] = p[c .. c + 7] (p 16-byte aligned, c a multiple of 4), or `fill` if p is null.
__device__ __forceinline__ void load8(const float* p, int c, float fill, float (&v)[8]) {
    if (p == nullptr) {
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = fill;
        return;
    }
    const float4 a = __ldg(reinterpret_cast<const float4*>(p + c));
    const float4 b = __ldg(reinterpret_cast<const float4*>(p + c + 4));
    v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
    v[4] = b.x; v[5] = b.y; v[6] = b.z; v[7] = b.w;
}

// Work units of a persistent CTA of the QUAD/PAIR kernel.  Without a split (sk = 0) a unit
// is a whole tile, the CTA taking tiles blockIdx.x + k gridDim.x.  With a split, the
// num_tiles x ktiles (tile, K block) iterations are cut into gridDim.x equal contiguous
// ranges, one per CTA (used only when num_tiles >= gridDim.x, so a range spans at least one
// tile and a tile is shared by at most two CTAs), so that every CTA does the same work
// whatever the tile count (the whole-tile schedule leaves most CTAs idle in a partial last
// wave).  A range then starts with the tail part of a tile (a HEAD unit: its accumulator
// goes to the CTA's partial slot in the caller's workspace and is flagged ready), runs
// whole tiles, and ends with the first part of a tile (a TAIL unit: the epilogue waits for
// the next CTA's flag, adds that CTA's partial and finishes the tile).  The head comes
// first in its CTA's run and the tail last in the other's, so the wait is normally over
// before it starts.
struct SplitK {
    int on;
    float* partial;      // workspace: one slot of 512 BNQ floats per CTA
    unsigned* flags;     // one flag per CTA: 1 while its partial is ready; the reader clears it
};
// A 1x1 shortcut fused into the convolution (the QUAD/PAIR kernel's SC form): its input is
// the convolution's filter tap (dh, dw) = (pad, pad) on the same input (x at (ho stride,
// wo stride)), so its N tiles n_conv .. num_n_tiles - 1 run the K blocks of that tap only,
// with their own letters, and write their own output tensor with their own epilogue.
struct ScParams {
    int n_conv;        // N tiles of the convolution; the rest are the shortcut's
    int ktiles;        // K blocks of a shortcut tile: Qin / KAPPA
    int tap, dh, dw;   // the convolution's filter tap that is the shortcut's input pixel
    int Qout;          // the shortcut's quaternion output channels
    int act;
    void* y;           // the shortcut's output [M][4 Qout]
    EpilogueArgs ep;   // its bias / IQBN scale and shift (no residual)
};
enum : int { UNIT_WHOLE = 0, UNIT_HEAD = 1, UNIT_TAIL = 2 };
struct Unit {
    int tile, k0, k1, kind;
};
struct UnitIter {
    int on, ktiles, num_tiles, tile;
    long long cur, hi;
    __device__ __forceinline__ UnitIter(int on_, int num_tiles_, int ktiles_)
        : on(on_), ktiles(ktiles_), num_tiles(num_tiles_), tile(static_cast<int>(blockIdx.x)) {
        const long long total = static_cast<long long>(num_tiles_) * ktiles_;
        cur = total * blockIdx.x / gridDim.x;
        hi = total * (blockIdx.x + 1) / gridDim.x;
    }
    __device__ __forceinline__ bool next(Unit& u) {
        if (!on) {
            if (tile >= num_tiles) return false;
            u.tile = tile;
            u.k0 = 0;
            u.k1 = ktiles;
            u.kind = UNIT_WHOLE;
            tile += static_cast<int>(gridDim.x);
            return true;
        }
        if (cur >= hi) return false;
        u.tile = static_cast<int>(cur / ktiles);
        u.k0 = static_cast<int>(cur - static_cast<long long>(u.tile) * ktiles);
        const long long left = hi - cur;
        u.k1 = left < ktiles - u.k0 ? u.k0 + static_cast<int>(left) : ktiles;
        u.kind = u.k0 > 0 ? UNIT_HEAD : (u.k1 < ktiles ? UNIT_TAIL : UNIT_WHOLE);
        cur += u.k1 - u.k0;
        return true;
    }
};

// Global-memory flag handshake between the CTAs sharing a tile (all CTAs of the grid are
// resident: one per SM), every wait bounded like the mbarrier waits.
__device__ __forceinline__ void st_release_gpu(unsigned* p, unsigned v) {
    asm volatile("st.release.gpu.global.u32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}
__device__ __forceinline__ unsigned ld_acquire_gpu(const unsigned* p) {
    unsigned v;
    asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}
__device__ __forceinline__ bool gflag_wait_or_abort(const unsigned* flag, uint64_t limit,
                                                    volatile int* abort_flag, unsigned code) {
    if (ld_acquire_gpu(flag) != 0u) return true;
    const uint64_t t0 = global_timer_ns();
    while (true) {
        __nanosleep(256);
        if (ld_acquire_gpu(flag) != 0u) return true;
        if (*abort_flag) return false;
        if (global_timer_ns() - t0 > limit) {
            atomicOr(&g_status, code);
            *abort_flag = 1;
            return false;
        }
    }
}

// Direct epilogue of the QUAD/PAIR kernel (warps 4..11, two per TMEM lane quadrant;
// warps 4..7 take output components r and i of every tile, warps 8..11 components j and k).
// Accumulator buffer b (of two, used round robin over the CTA's tiles) lives at TMEM
// columns [4 BNQ b, 4 BNQ (b+1)), component q at offset q BNQ.  A warp's share of a tile
// is NB = 2 BNQ / CH blocks of its 32 rows x CH = min(BNQ, 32) columns; for each block it
//   1. loads the block with one tcgen05.ld (after the last load of a tile it releases the
//      accumulator buffer: acce, 256 arrivals per tile);
//   2. transposes, within each group of NCH = CH / 8 lanes, the NCH x NCH matrix of
//      8-channel chunks (rows x chunks) with shfl_xor, so every lane holds one chunk of
//      NCH rows;
//   3. applies act(scale * (acc + bias) + shift + residual) (IQBN inference form of
//      Eq. 11-12; the affine step as fma(scale, acc, scale * bias + shift)), rounds to
//      bf16 and writes 16 bytes per lane per row: each store instruction covers CH * 2
//      contiguous bytes of 32 / NCH output rows.
// The blocks are software-pipelined: the TMEM load and the per-channel vectors of block
// b + 1 are requested before block b is processed, so their latency (hundreds of cycles
// each, with the tensor cores busy on the other buffer) overlaps the work on block b.
// No shared memory is touched (the tensor cores' operand reads keep that pipe busy); the
// per-channel vectors are read through the L1 cache, 16 bytes at a time.
template <int BNQ, typename Geo>
__device__ __forceinline__ void epilogue_direct_pair(const ConvShape& s, const EpilogueArgs& ep,
                                                     void* y, uint32_t tmem_base,
                                                     uint32_t accf0, uint32_t acce0,
                                                     int num_tiles, int ktiles, const SplitK& sk,
                                                     uint64_t limit,
                                                     volatile int* abort_flag, Geo geo) {
    constexpr int CH = BNQ < 32 ? BNQ : 32;  // columns per TMEM load
    constexpr int NCH = CH / 8;              // 8-channel chunks per load: 2 or 4
    constexpr int SLICES = BNQ / CH;
    constexpr int NB = 2 * SLICES;           // blocks per warp and tile
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int quad = warp & 3;                 // TMEM lane quadrant this warp may access
    const int half = (warp - EPI_WARP0) >> 2;  // output components 2 half, 2 half + 1
    const int ci = lane % NCH;                 // this lane's chunk after the transpose
    const int row0 = quad * 32 + NCH * (lane / NCH);  // its rows: row0 .. row0 + NCH - 1
    const long long Cout = s.Cout;
    const __nv_bfloat16* res = static_cast<const __nv_bfloat16*>(ep.residual);
    __nv_bfloat16* out = static_cast<__nv_bfloat16*>(y);
    // block b of this warp: component 2 half + b / SLICES, columns (b % SLICES) CH ..
    auto tmem_col = [&](int b) { return (2 * half + b / SLICES) * BNQ + (b % SLICES) * CH; };
    auto load_block = [&](uint32_t taddr, int b, uint32_t(&v)[CH]) {
        if constexpr (CH == 32)
            tmem_ld_32x32b_x32(taddr + tmem_col(b), v);
        else
            tmem_ld_32x32b_x16(taddr + tmem_col(b), v);
    };
    // the per-channel vectors of this lane's 8 channels of block b
    auto load_vectors = [&](int cb, float(&sc)[8], float(&sh)[8]) {
        float bi[8];
        load8(ep.scale, cb, 1.0f, sc);
        load8(ep.shift, cb, 0.0f, sh);
        load8(ep.bias, cb, 0.0f, bi);
#pragma unroll
        for (int e = 0; e < 8; ++e) sh[e] = fmaf(sc[e], bi[e], sh[e]);
    };
    // this thread's floats in a partial slot: block b, 4-float group j -> lanes contiguous
    const int ew = warp - EPI_WARP0;  // 0..7
    auto pslot = [&](const float* slot, int b, int j) {
        return reinterpret_cast<float4*>(const_cast<float*>(slot)) +
               ((ew * NB + b) * (CH / 4) + j) * 32 + lane;
    };
    int local = 0;
    UnitIter units(sk.on, num_tiles, ktiles);
    Unit unit;
    while (units.next(unit)) {
        const int tile = unit.tile;
        const int buf = local & 1;
        const uint32_t use = static_cast<uint32_t>(local >> 1) & 1u;
        ++local;
        bool ok = true;
        if (lane == 0)
            ok = wait_or_abort(accf0 + 8u * buf, use, limit, abort_flag, STATUS_TIMEOUT_EPILOGUE);
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        // leave together: a warp that gave up must not strand the others at a barrier
        if (named_bar_or(1, 256, !ok)) break;
        if (unit.kind == UNIT_TAIL) {
            // the rest of this tile's K blocks were done by the next CTA: wait for its partial
            bool ready = true;
            if (threadIdx.x == EPI_WARP0 * 32) {
                ready = gflag_wait_or_abort(sk.flags + blockIdx.x + 1, limit, abort_flag,
                                            STATUS_TIMEOUT_EPILOGUE);
                // cleared for the next call (whose writer runs only after this grid ends)
                if (ready) sk.flags[blockIdx.x + 1] = 0u;
            }
            if (named_bar_or(1, 256, !ready)) break;
        }
        tc_fence_after();
        const EpiTile g = geo(tile);
        const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                               static_cast<uint32_t>(buf * 4 * BNQ);
        const int c_tile = g.n_tile * BNQ + 8 * ci;  // + q Qout + slice offset: lane's channel
        uint32_t va[CH], vb[CH];
        float sca[8], sha[8], scb[8], shb[8];
        load_block(taddr, 0, va);
        load_vectors(c_tile + (2 * half) * s.Qout, sca, sha);
        tmem_ld_wait();
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            uint32_t(&v)[CH] = (b & 1) ? vb : va;
            uint32_t(&vn)[CH] = (b & 1) ? va : vb;
            float(&sc)[8] = (b & 1) ? scb : sca;
            float(&sh)[8] = (b & 1) ? shb : sha;
            float(&scn)[8] = (b & 1) ? sca : scb;
            float(&shn)[8] = (b & 1) ? sha : shb;
            const int q = 2 * half + b / SLICES;
            const int cb = c_tile + q * s.Qout + (b % SLICES) * CH;
            if (b + 1 < NB) {
                // next block in flight while this one is processed
                load_block(taddr, b + 1, vn);
                load_vectors(c_tile + (2 * half + (b + 1) / SLICES) * s.Qout +
                                 ((b + 1) % SLICES) * CH,
                             scn, shn);
            } else {
                // the tile's accumulator is in registers: hand the buffer back
                tc_fence_before();
                mbar_arrive_relaxed(acce0 + 8u * buf);
            }
            if (unit.kind == UNIT_HEAD) {
                // this CTA's share of the tile: the raw accumulator to the partial slot (L2)
                float* my_slot = sk.partial + static_cast<size_t>(blockIdx.x) * (512 * BNQ);
#pragma unroll
                for (int j = 0; j < CH / 4; ++j)
                    __stcg(pslot(my_slot, b, j),
                           make_float4(__uint_as_float(v[4 * j]), __uint_as_float(v[4 * j + 1]),
                                       __uint_as_float(v[4 * j + 2]), __uint_as_float(v[4 * j + 3])));
                if (b + 1 < NB) tmem_ld_wait();
                continue;
            }
            if (unit.kind == UNIT_TAIL) {
                // the next CTA's share, read from L2 (never from this SM's L1)
                const float* next_slot =
                    sk.partial + static_cast<size_t>(blockIdx.x + 1) * (512 * BNQ);
#pragma unroll
                for (int j = 0; j < CH / 4; ++j) {
                    const float4 q4 = __ldcg(pslot(next_slot, b, j));
                    v[4 * j] = __float_as_uint(__uint_as_float(v[4 * j]) + q4.x);
                    v[4 * j + 1] = __float_as_uint(__uint_as_float(v[4 * j + 1]) + q4.y);
                    v[4 * j + 2] = __float_as_uint(__uint_as_float(v[4 * j + 2]) + q4.z);
                    v[4 * j + 3] = __float_as_uint(__uint_as_float(v[4 * j + 3]) + q4.w);
                }
            }
            uint4 r4[NCH];
            if (res != nullptr) {
#pragma unroll
                for (int k = 0; k < NCH; ++k) {
                    r4[k] = make_uint4(0u, 0u, 0u, 0u);
                    if (row0 + k < g.rows)
                        r4[k] = ld_global_na(res + (g.m0 + row0 + k) * Cout + cb);
                }
            }
            float E[NCH][8];  // E[j][e]: channel 8 j + e of this lane's row
#pragma unroll
            for (int j = 0; j < NCH; ++j)
#pragma unroll
                for (int e = 0; e < 8; ++e) E[j][e] = __uint_as_float(v[8 * j + e]);
            if constexpr (NCH == 4) {
                chunk_transpose_stage<2, 4>(E, ci);
                chunk_transpose_stage<1, 4>(E, ci);
            } else {
                chunk_transpose_stage<1, 2>(E, ci);
            }
            // now E[k][e] = channel cb + e of row row0 + k
#pragma unroll
            for (int k = 0; k < NCH; ++k) {
                float rz[8];
                if (res != nullptr) {
                    const __nv_bfloat162* rh = reinterpret_cast<const __nv_bfloat162*>(&r4[k]);
#pragma unroll
                    for (int t = 0; t < 4; ++t) {
                        const float2 f = __bfloat1622float2(rh[t]);
                        rz[2 * t] = f.x;
                        rz[2 * t + 1] = f.y;
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < 8; ++e) rz[e] = 0.0f;
                }
                uint32_t w[4];
#pragma unroll
                for (int t = 0; t < 4; ++t) {
                    const float z0 = fmaf(sc[2 * t], E[k][2 * t], sh[2 * t]) + rz[2 * t];
                    const float z1 =
                        fmaf(sc[2 * t + 1], E[k][2 * t + 1], sh[2 * t + 1]) + rz[2 * t + 1];
                    w[t] = pack_bf16x2(activate(z0, s.act), activate(z1, s.act));
                }
                if (row0 + k < g.rows)
                    st_global_na(out + (g.m0 + row0 + k) * Cout + cb,
                                 make_uint4(w[0], w[1], w[2], w[3]));
            }
            if (b + 1 < NB) tmem_ld_wait();
        }
        if (unit.kind == UNIT_HEAD) {
            // every epilogue thread's partial stores are visible device-wide before the flag
            __threadfence();
            named_bar_sync(2, 256);
            if (threadIdx.x == EPI_WARP0 * 32) st_release_gpu(sk.flags + blockIdx.x, 1u);
        }
    }
}

// The same for the fused shortcut form of the QUAD/PAIR kernel (whole tiles): tiles from N
// tile sc->n_conv on are the shortcut's (ScParams), written with its own output, channel
// count, per-channel vectors and activation.
template <int BNQ, typename Geo>
__device__ __forceinline__ void epilogue_direct_pair_sc(const ConvShape& s, const EpilogueArgs& ep,
                                                     void* y, uint32_t tmem_base,
                                                     uint32_t accf0, uint32_t acce0,
                                                     int num_tiles, int ktiles, const SplitK& sk,
                                                     uint64_t limit,
                                                     volatile int* abort_flag, Geo geo,
                                                     const ScParams* sc) {
    constexpr int CH = BNQ < 32 ? BNQ : 32;  // columns per TMEM load
    constexpr int NCH = CH / 8;              // 8-channel chunks per load: 2 or 4
    constexpr int SLICES = BNQ / CH;
    constexpr int NB = 2 * SLICES;           // blocks per warp and tile
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int quad = warp & 3;                 // TMEM lane quadrant this warp may access
    const int half = (warp - EPI_WARP0) >> 2;  // output components 2 half, 2 half + 1
    const int ci = lane % NCH;                 // this lane's chunk after the transpose
    const int row0 = quad * 32 + NCH * (lane / NCH);  // its rows: row0 .. row0 + NCH - 1
    const long long Cout0 = s.Cout;
    const __nv_bfloat16* res0 = static_cast<const __nv_bfloat16*>(ep.residual);
    __nv_bfloat16* out0 = static_cast<__nv_bfloat16*>(y);
    // the tile's output parameters (the convolution's or the shortcut's)
    const EpilogueArgs* epp = &ep;
    // block b of this warp: component 2 half + b / SLICES, columns (b % SLICES) CH ..
    auto tmem_col = [&](int b) { return (2 * half + b / SLICES) * BNQ + (b % SLICES) * CH; };
    auto load_block = [&](uint32_t taddr, int b, uint32_t(&v)[CH]) {
        if constexpr (CH == 32)
            tmem_ld_32x32b_x32(taddr + tmem_col(b), v);
        else
            tmem_ld_32x32b_x16(taddr + tmem_col(b), v);
    };
    // the per-channel vectors of this lane's 8 channels of block b
    auto load_vectors = [&](int cb, float(&scv)[8], float(&sh)[8]) {
        const EpilogueArgs* e = &ep;
        e = epp;
        float bi[8];
        load8(e->scale, cb, 1.0f, scv);
        load8(e->shift, cb, 0.0f, sh);
        load8(e->bias, cb, 0.0f, bi);
#pragma unroll
        for (int e = 0; e < 8; ++e) sh[e] = fmaf(scv[e], bi[e], sh[e]);
    };
    int local = 0;
    UnitIter units(sk.on, num_tiles, ktiles);
    Unit unit;
    while (units.next(unit)) {
        const int tile = unit.tile;
        const int buf = local & 1;
        const uint32_t use = static_cast<uint32_t>(local >> 1) & 1u;
        ++local;
        bool ok = true;
        if (lane == 0)
            ok = wait_or_abort(accf0 + 8u * buf, use, limit, abort_flag, STATUS_TIMEOUT_EPILOGUE);
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        // leave together: a warp that gave up must not strand the others at a barrier
        if (named_bar_or(1, 256, !ok)) break;
        tc_fence_after();
        EpiTile g = geo(tile);
        long long Cout = Cout0;
        int Qout = s.Qout, act = s.act;
        const __nv_bfloat16* res = res0;
        __nv_bfloat16* out = out0;
        {
            // this tile's output: the convolution's or the fused shortcut's
            const bool sct = g.n_tile >= sc->n_conv;
            if (sct) {
                g.n_tile -= sc->n_conv;
                Qout = sc->Qout;
                act = sc->act;
                Cout = 4LL * Qout;
                epp = &sc->ep;
                res = nullptr;
                out = static_cast<__nv_bfloat16*>(sc->y);
            } else {
                epp = &ep;
            }
        }
        const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                               static_cast<uint32_t>(buf * 4 * BNQ);
        const int c_tile = g.n_tile * BNQ + 8 * ci;  // + q Qout + slice offset: lane's channel
        uint32_t va[CH], vb[CH];
        float sca[8], sha[8], scb[8], shb[8];
        load_block(taddr, 0, va);
        load_vectors(c_tile + (2 * half) * Qout, sca, sha);
        tmem_ld_wait();
#pragma unroll
        for (int b = 0; b < NB; ++b) {
            uint32_t(&v)[CH] = (b & 1) ? vb : va;
            uint32_t(&vn)[CH] = (b & 1) ? va : vb;
            float(&sc)[8] = (b & 1) ? scb : sca;
            float(&sh)[8] = (b & 1) ? shb : sha;
            float(&scn)[8] = (b & 1) ? sca : scb;
            float(&shn)[8] = (b & 1) ? sha : shb;
            const int q = 2 * half + b / SLICES;
            const int cb = c_tile + q * Qout + (b % SLICES) * CH;
            if (b + 1 < NB) {
                // next block in flight while this one is processed
                load_block(taddr, b + 1, vn);
                load_vectors(c_tile + (2 * half + (b + 1) / SLICES) * Qout +
                                 ((b + 1) % SLICES) * CH,
                             scn, shn);
            } else {
                // the tile's accumulator is in registers: hand the buffer back
                tc_fence_before();
                mbar_arrive_relaxed(acce0 + 8u * buf);
            }
            uint4 r4[NCH];
            if (res != nullptr) {
#pragma unroll
                for (int k = 0; k < NCH; ++k) {
                    r4[k] = make_uint4(0u, 0u, 0u, 0u);
                    if (row0 + k < g.rows)
                        r4[k] = ld_global_na(res + (g.m0 + row0 + k) * Cout + cb);
                }
            }
            float E[NCH][8];  // E[j][e]: channel 8 j + e of this lane's row
#pragma unroll
            for (int j = 0; j < NCH; ++j)
#pragma unroll
                for (int e = 0; e < 8; ++e) E[j][e] = __uint_as_float(v[8 * j + e]);
            if constexpr (NCH == 4) {
                chunk_transpose_stage<2, 4>(E, ci);
                chunk_transpose_stage<1, 4>(E, ci);
            } else {
                chunk_transpose_stage<1, 2>(E, ci);
            }
            // now E[k][e] = channel cb + e of row row0 + k
#pragma unroll
            for (int k = 0; k < NCH; ++k) {
                float rz[8];
                if (res != nullptr) {
                    const __nv_bfloat162* rh = reinterpret_cast<const __nv_bfloat162*>(&r4[k]);
#pragma unroll
                    for (int t = 0; t < 4; ++t) {
                        const float2 f = __bfloat1622float2(rh[t]);
                        rz[2 * t] = f.x;
                        rz[2 * t + 1] = f.y;
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < 8; ++e) rz[e] = 0.0f;
                }
                uint32_t w[4];
#pragma unroll
                for (int t = 0; t < 4; ++t) {
                    const float z0 = fmaf(sc[2 * t], E[k][2 * t], sh[2 * t]) + rz[2 * t];
                    const float z1 =
                        fmaf(sc[2 * t + 1], E[k][2 * t + 1], sh[2 * t + 1]) + rz[2 * t + 1];
                    w[t] = pack_bf16x2(activate(z0, act), activate(z1, act));
                }
                if (row0 + k < g.rows)
                    st_global_na(out + (g.m0 + row0 + k) * Cout + cb,
                                 make_uint4(w[0], w[1], w[2], w[3]));
            }
            if (b + 1 < NB) tmem_ld_wait();
        }
    }
}

// Epilogue of the separable form (Eq. 7, MODE_SEP of the QUAD/PAIR kernel).  The
// accumulator holds the four per-component convolutions D_p = W_p (*) X_p (component p at
// TMEM column offset p BNQ); output component m is the signed sum
//   y_r = D_r - D_i - D_j - D_k,  y_i = D_r + D_i + D_j - D_k,
//   y_j = D_r - D_i + D_j + D_k,  y_k = D_r + D_i - D_j + D_k,
// followed by the same act(scale * (y + bias) + shift).  Warps 4..7 take the first half of
// the tile's BNQ channels, warps 8..11 the second; every warp loads the four D_p of its 32
// rows for SS = min(BNQ / 2, 16) channels at a time, mixes them in registers and writes
// the four output components (a 2x2 chunk transpose across lane pairs when SS = 16, so a
// store instruction covers 32-byte pieces of 16 rows).  No shared memory; the per-channel
// vectors through L1.
template <int BNQ, typename Geo>
__device__ __forceinline__ void epilogue_direct_sep(const ConvShape& s, const EpilogueArgs& ep,
                                                    void* y, uint32_t tmem_base,
                                                    uint32_t accf0, uint32_t acce0,
                                                    int num_tiles, uint64_t limit,
                                                    volatile int* abort_flag, Geo geo) {
    constexpr int CS = BNQ / 2;             // channels per half (per warp group)
    constexpr int SS = CS < 16 ? CS : 16;   // channels per TMEM load
    constexpr int NSUB = CS / SS;
    constexpr int NCH = SS / 8;             // 8-channel chunks per load: 1 or 2
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int quad = warp & 3;
    const int half = (warp - EPI_WARP0) >> 2;
    const int ci = lane % NCH;
    const int row0 = quad * 32 + NCH * (lane / NCH);
    const long long Cout = s.Cout;
    __nv_bfloat16* out = static_cast<__nv_bfloat16*>(y);
    int local = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++local) {
        const int buf = local & 1;
        const uint32_t use = static_cast<uint32_t>(local >> 1) & 1u;
        bool ok = true;
        if (lane == 0)
            ok = wait_or_abort(accf0 + 8u * buf, use, limit, abort_flag, STATUS_TIMEOUT_EPILOGUE);
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        if (named_bar_or(1, 256, !ok)) break;
        tc_fence_after();
        const EpiTile g = geo(tile);
        const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                               static_cast<uint32_t>(buf * 4 * BNQ);
#pragma unroll
        for (int sub = 0; sub < NSUB; ++sub) {
            const int col0 = half * CS + sub * SS;  // column within a component block
            uint32_t d[4][SS];
#pragma unroll
            for (int p = 0; p < 4; ++p) {
                if constexpr (SS == 16)
                    tmem_ld_32x32b_x16(taddr + p * BNQ + col0, d[p]);
                else
                    tmem_ld_32x32b_x8(taddr + p * BNQ + col0, d[p]);
            }
            tmem_ld_wait();
            if (sub == NSUB - 1) {
                // the tile's accumulator is in registers: hand the buffer back
                tc_fence_before();
                mbar_arrive_relaxed(acce0 + 8u * buf);
            }
#pragma unroll
            for (int m = 0; m < 4; ++m) {
                float E[NCH][8];  // E[j][e]: channel col0 + 8 j + e of this lane's row
#pragma unroll
                for (int j = 0; j < NCH; ++j)
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        float z = 0.0f;
#pragma unroll
                        for (int p = 0; p < 4; ++p) {
                            const float dp = __uint_as_float(d[p][8 * j + e]);
                            z = ((SEP_NEG >> (4 * m + p)) & 1u) ? z - dp : z + dp;
                        }
                        E[j][e] = z;
                    }
                if constexpr (NCH == 2) chunk_transpose_stage<1, 2>(E, ci);
                // now E[k][e] = channel cb + e of row row0 + k
                const int cb = m * s.Qout + g.n_tile * BNQ + col0 + 8 * ci;
                float sc[8], sh[8];
                {
                    float bi[8];
                    load8(ep.scale, cb, 1.0f, sc);
                    load8(ep.shift, cb, 0.0f, sh);
                    load8(ep.bias, cb, 0.0f, bi);
#pragma unroll
                    for (int e = 0; e < 8; ++e) sh[e] = fmaf(sc[e], bi[e], sh[e]);
                }
#pragma unroll
                for (int k = 0; k < NCH; ++k) {
                    uint32_t w[4];
#pragma unroll
                    for (int t = 0; t < 4; ++t) {
                        const float z0 = fmaf(sc[2 * t], E[k][2 * t], sh[2 * t]);
                        const float z1 = fmaf(sc[2 * t + 1], E[k][2 * t + 1], sh[2 * t + 1]);
                        w[t] = pack_bf16x2(activate(z0, s.act), activate(z1, s.act));
                    }
                    if (row0 + k < g.rows)
                        st_global_na(out + (g.m0 + row0 + k) * Cout + cb,
                                     make_uint4(w[0], w[1], w[2], w[3]));
                }
            }
        }
    }
}

// NG epilogue groups, one per MMA issuer (warps 4 + 4 NG .. 15 take no part).
template <typename Geo, int NG = EPI_GROUPS>
__device__ __forceinline__ void epilogue_direct64(const ConvShape& s, const EpilogueArgs& ep,
                                                  void* y, uint32_t tmem_base, uint32_t accf0,
                                                  uint32_t acce0, int num_tiles, uint64_t limit,
                                                  volatile int* abort_flag, Geo geo) {
    static_assert(NG >= 1 && NG <= EPI_GROUPS, "each epilogue group drains one issuer's buffers");
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int quad = warp & 3;                // TMEM lane quadrant this warp may access
    const int grp = (warp - EPI_WARP0) >> 2;  // local tiles k with k % NG == grp
    if (grp >= NG) return;
    const int ci = lane & 3;                  // this lane's chunk after the transpose
    const int rg = lane >> 2;                 // group of 4 rows (4 lanes) within the warp
    // the chunks' per-channel vectors (channels 8 ci + 32 h + e), in registers
    float sc[2][8], sh[2][8];
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int e = 0; e < 8; ++e) {
            const int c = 32 * h + 8 * ci + e;
            const float b = ep.bias ? __ldg(ep.bias + c) : 0.0f;
            sc[h][e] = ep.scale ? __ldg(ep.scale + c) : 1.0f;
            sh[h][e] = fmaf(sc[h][e], b, ep.scale ? __ldg(ep.shift + c) : 0.0f);
        }
    const __nv_bfloat16* res = static_cast<const __nv_bfloat16*>(ep.residual);
    __nv_bfloat16* out = static_cast<__nv_bfloat16*>(y);
    int local = grp;
    for (int tile = blockIdx.x + grp * gridDim.x; tile < num_tiles;
         tile += NG * gridDim.x, local += NG) {
        int buf;
        uint32_t use;
        issuer_acc_n<NG>(local, buf, use);
        bool ok = true;
        if (lane == 0)
            ok = wait_or_abort(accf0 + 8u * buf, use, limit, abort_flag, STATUS_TIMEOUT_EPILOGUE);
        if (__shfl_sync(0xffffffffu, ok ? 1 : 0, 0) == 0) break;
        tc_fence_after();
        const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                               static_cast<uint32_t>(buf * 64);
        const EpiTile g = geo(tile);
        // this lane's rows after the transpose: quad*32 + 4 rg + k, k = 0..3
        const int row0 = quad * 32 + 4 * rg;
#pragma unroll
        for (int h = 0; h < 2; ++h) {
            uint32_t v[32];  // channel 32 h + c of this lane's row
            tmem_ld_32x32b_x32(taddr + 32 * h, v);
            tmem_ld_wait();
            if (h == 1) {
                // the accumulator is in registers: hand the buffer back to the MMA issuer
                tc_fence_before();
                mbar_arrive_relaxed(acce0 + 8u * buf);
            }
            const int c0 = 32 * h + 8 * ci;
            uint4 r4[4];
            if (res != nullptr) {
#pragma unroll
                for (int k = 0; k < 4; ++k) {
                    r4[k] = make_uint4(0u, 0u, 0u, 0u);
                    if (row0 + k < g.rows)
                        r4[k] = __ldg(
                            reinterpret_cast<const uint4*>(res + (g.m0 + row0 + k) * 64 + c0));
                }
            }
            float E[4][8];  // E[j][e]: channel 32 h + 8j + e of this lane's row
#pragma unroll
            for (int j = 0; j < 4; ++j)
#pragma unroll
                for (int e = 0; e < 8; ++e) E[j][e] = __uint_as_float(v[8 * j + e]);
            chunk_transpose_stage<2, 4>(E, ci);
            chunk_transpose_stage<1, 4>(E, ci);
            // now E[k][e] = channel c0 + e of row row0 + k
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                float rz[8];
                if (res != nullptr) {
                    const __nv_bfloat162* rh = reinterpret_cast<const __nv_bfloat162*>(&r4[k]);
#pragma unroll
                    for (int t = 0; t < 4; ++t) {
                        const float2 f = __bfloat1622float2(rh[t]);
                        rz[2 * t] = f.x;
                        rz[2 * t + 1] = f.y;
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < 8; ++e) rz[e] = 0.0f;
                }
                uint32_t w[4];
#pragma unroll
                for (int t = 0; t < 4; ++t) {
                    const float z0 = fmaf(sc[h][2 * t], E[k][2 * t], sh[h][2 * t]) + rz[2 * t];
                    const float z1 =
                        fmaf(sc[h][2 * t + 1], E[k][2 * t + 1], sh[h][2 * t + 1]) + rz[2 * t + 1];
                    w[t] = pack_bf16x2(activate(z0, s.act), activate(z1, s.act));
                }
                if (row0 + k < g.rows)
                    *reinterpret_cast<uint4*>(out + (g.m0 + row0 + k) * 64 + c0) =
                        make_uint4(w[0], w[1], w[2], w[3]);
            }
        }
    }
}

}  // namespace tc
}  // namespace quan
