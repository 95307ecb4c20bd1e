// tc_common.cuh -- pieces shared by the tensor-core quaternion convolution kernels
// (qconv_tc.cu is the only translation unit that includes this file): constants, the
// device status word, descriptor helpers, bounded waits and the 8-warp epilogue.
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
    if (act == 2) return z / (1.0f + __expf(-z));
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
    int sy, sz;    // TMA store coordinates after the channel one (2-D: sy = m0)
};

// Shared-memory resources of the epilogue: two staging blocks of 128 x BNQ bf16 (one per
// half; with WIDE, WBUFS blocks of 128 x 4 BNQ, one per tile parity when WBUFS = 2) and
// the per-channel vectors [2][4 BNQ] (16-byte aligned): the IQBN scale and the shift with
// the bias folded in.
template <int BNQ, bool WIDE = false, int WBUFS = 2>
struct EpiSmem {
    static_assert(WBUFS == 1 || WBUFS == 2, "one or two wide staging blocks");
    static constexpr int OUT_TILE = BM * BNQ * 2;
    static constexpr int STAGING_BYTES = WIDE ? WBUFS * 4 * OUT_TILE : 2 * OUT_TILE;
    static constexpr int PARAM_BYTES = 2 * 4 * BNQ * 4;
    static constexpr uint32_t OUT_ROW = BNQ * 2;
    static constexpr uint32_t OUT_SW_MASK = BNQ == 64 ? 7u : (BNQ == 32 ? 3u : 1u);
};

// The epilogue role (warps 4..11, two per TMEM lane quadrant; the first four warps
// handle output components r, i and the last four j, k).  For each tile of this CTA:
// wait for its accumulator buffer, apply act(scale*(acc+bias)+shift+residual) (IQBN
// inference form of Eq. 11-12), round to bf16, write a swizzled shared-memory block per
// component and store it with TMA (rows outside the tensor are clipped by the map).
// The affine step is evaluated as fma(scale, acc, scale*bias + shift): the folded shift
// is formed once per channel, and the two vectors are read as float4 broadcasts (the
// shared-memory pipe is shared with the tensor cores' operand reads, so the epilogue
// keeps its own shared-memory traffic small).
// With WIDE (4 BNQ = 64 channels = the whole output row, BNQ == Qout) all four
// components go into one 128-byte-row block and a single TMA store per tile; with
// WBUFS = 2 the block alternates between two buffers so the store overlaps the next
// tile, with WBUFS = 1 the next tile waits until the store has read the block.
// Accumulator buffer b (of NACC, used round robin) of a tile lives at TMEM columns
// [4 BNQ b, 4 BNQ (b+1)), component q at offset q BNQ.
template <int BNQ, bool STORE3D, typename Geo, bool WIDE = false, int WBUFS = 2, int NACC = 2>
__device__ __forceinline__ void epilogue_role(const ConvShape& s, const EpilogueArgs& ep,
                                              const CUtensorMap* tmap_y, uint32_t tmem_base,
                                              uint8_t* staging, float* prm_s,
                                              uint32_t accf0, uint32_t acce0, int num_tiles,
                                              uint64_t limit, volatile int* abort_flag,
                                              Geo geo) {
    using E = EpiSmem<BNQ, WIDE, WBUFS>;
    static_assert(!WIDE || BNQ == 16, "wide stores need 64-channel rows");
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int quad = warp & 3;                 // TMEM lane quadrant this warp may access
    const int half = (warp - EPI_WARP0) >> 2;  // output components 2*half, 2*half+1
    const int row = quad * 32 + lane;
    const bool leader = (warp == EPI_WARP0 + 4 * half) && lane == 0;
    const int etid = threadIdx.x - EPI_WARP0 * 32;  // 0..255
    const int Cout = s.Cout;
    const __nv_bfloat16* res = static_cast<const __nv_bfloat16*>(ep.residual);
    uint8_t* stg = staging + (WIDE ? 0 : half * E::OUT_TILE);
    uint32_t stg_addr = smem_u32(stg);
    int cached_n = -1;
    int local = 0;
    for (int tile = blockIdx.x; tile < num_tiles; tile += gridDim.x, ++local) {
        const int buf = local % NACC;
        const uint32_t use = static_cast<uint32_t>(local / NACC) & 1u;
        // one lane per warp polls the barrier (256 pollers would crowd the shared-memory
        // pipe that TMA and the barriers themselves use), then broadcasts the result
        bool ok = true;
        if (lane == 0)
            ok = wait_or_abort(accf0 + 8u * buf, use, limit, abort_flag, STATUS_TIMEOUT_EPILOGUE);
        ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
        // leave together: a warp that gave up must not strand the others at a barrier
        if (named_bar_or(1, 256, !ok)) break;
        tc_fence_after();
        const EpiTile g = geo(tile);
        if (g.n_tile != cached_n) {
            // per-channel vectors of this tile's 4 x BNQ channels -> shared memory
            named_bar_sync(1, 256);
            for (int i = etid; i < 4 * BNQ; i += 256) {
                const int c = (i / BNQ) * s.Qout + g.n_tile * BNQ + (i % BNQ);
                const float b = ep.bias ? __ldg(ep.bias + c) : 0.0f;
                const float sc = ep.scale ? __ldg(ep.scale + c) : 1.0f;
                const float sh = ep.scale ? __ldg(ep.shift + c) : 0.0f;
                prm_s[i] = sc;
                prm_s[4 * BNQ + i] = fmaf(sc, b, sh);
            }
            named_bar_sync(1, 256);
            cached_n = g.n_tile;
        }
        const long long m = g.m0 + row;
        const bool valid = row < g.rows;
        const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                               static_cast<uint32_t>(buf * 4 * BNQ);
        if constexpr (WIDE) {
            // block of this tile's parity (by tile count, not accumulator buffer); free once
            // the store of WBUFS tiles ago has read it
            stg = staging + (local % WBUFS) * 4 * E::OUT_TILE;
            stg_addr = smem_u32(stg);
            if (threadIdx.x == EPI_WARP0 * 32) bulk_wait_group_read<WBUFS - 1>();
            named_bar_sync(1, 256);
        }
#pragma unroll
        for (int qq = 0; qq < 2; ++qq) {
            const int q = 2 * half + qq;
            if constexpr (!WIDE) {
                // the staging block is free once the previous store has read it
                if (leader) bulk_wait_group_read<0>();
                named_bar_sync(2 + half, 128);
            }
            constexpr int CH = BNQ < 32 ? BNQ : 32;  // columns per TMEM load
#pragma unroll
            for (int j0 = 0; j0 < BNQ; j0 += CH) {
                uint32_t v[32];
                if constexpr (CH == 32) {
                    tmem_ld_32x32b_x32(taddr + q * BNQ + j0, v);
                } else {
                    uint32_t(&v16)[16] = *reinterpret_cast<uint32_t(*)[16]>(v);
                    tmem_ld_32x32b_x16(taddr + q * BNQ + j0, v16);
                }
                float rz[CH];
                if (res != nullptr && valid) {
                    const uint4* rp = reinterpret_cast<const uint4*>(
                        res + m * Cout + q * s.Qout + g.n_tile * BNQ + j0);
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
                const float4* ps4 = reinterpret_cast<const float4*>(prm_s + q * BNQ + j0);
                const float4* ph4 = reinterpret_cast<const float4*>(prm_s + 4 * BNQ + q * BNQ + j0);
#pragma unroll
                for (int u = 0; u < CH / 8; ++u) {
                    const float4 sa = ps4[2 * u], sb = ps4[2 * u + 1];
                    const float4 ha = ph4[2 * u], hb = ph4[2 * u + 1];
                    const float sc[8] = {sa.x, sa.y, sa.z, sa.w, sb.x, sb.y, sb.z, sb.w};
                    const float sh[8] = {ha.x, ha.y, ha.z, ha.w, hb.x, hb.y, hb.z, hb.w};
                    uint32_t w[4];
#pragma unroll
                    for (int t = 0; t < 4; ++t) {
                        const int e = 8 * u + 2 * t;
                        const float z0 = fmaf(sc[2 * t], __uint_as_float(v[e]), sh[2 * t]) + rz[e];
                        const float z1 =
                            fmaf(sc[2 * t + 1], __uint_as_float(v[e + 1]), sh[2 * t + 1]) + rz[e + 1];
                        w[t] = pack_bf16x2(activate(z0, s.act), activate(z1, s.act));
                    }
                    if constexpr (WIDE) {
                        // 128-byte row of all four components, 128-byte swizzle
                        const uint32_t chunk = static_cast<uint32_t>(q * (BNQ / 8) + j0 / 8 + u);
                        const uint32_t off = static_cast<uint32_t>(row) * 128 +
                                             ((chunk ^ (static_cast<uint32_t>(row) & 7u)) << 4);
                        *reinterpret_cast<uint4*>(stg + off) = make_uint4(w[0], w[1], w[2], w[3]);
                    } else {
                        // 16-byte chunk (j0/8 + u) of this row, swizzled like the TMA map
                        const uint32_t chunk = static_cast<uint32_t>(j0 / 8 + u);
                        const uint32_t off = static_cast<uint32_t>(row) * E::OUT_ROW +
                                             ((chunk ^ ((static_cast<uint32_t>(row) * E::OUT_ROW >>
                                                         7) & E::OUT_SW_MASK))
                                              << 4);
                        *reinterpret_cast<uint4*>(stg + off) = make_uint4(w[0], w[1], w[2], w[3]);
                    }
                }
            }
            if constexpr (!WIDE) {
                fence_proxy_async_smem();
                named_bar_sync(2 + half, 128);
                if (leader) {
                    const int c0 = q * s.Qout + g.n_tile * BNQ;
                    if constexpr (STORE3D)
                        tma_store_3d(tmap_y, stg_addr, c0, g.sy, g.sz);
                    else
                        tma_store_2d(tmap_y, stg_addr, c0, g.sy);
                    bulk_commit_group();
                }
            }
        }
        if constexpr (WIDE) {
            fence_proxy_async_smem();
            named_bar_sync(1, 256);
            if (threadIdx.x == EPI_WARP0 * 32) {
                if constexpr (STORE3D)
                    tma_store_3d(tmap_y, stg_addr, 0, g.sy, g.sz);
                else
                    tma_store_2d(tmap_y, stg_addr, 0, g.sy);
                bulk_commit_group();
            }
        }
        tc_fence_before();
        mbar_arrive(acce0 + 8u * buf);
    }
    if (leader || (WIDE && threadIdx.x == EPI_WARP0 * 32)) bulk_wait_group<0>();
}

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

// Tiles of a CTA are issued round robin by ISSUERS threads (local tile k by issuer
// k % ISSUERS).  mbarrier parity waits only tell a phase from its neighbours, so a waiter
// must never get two phases ahead of a barrier; that is guaranteed by letting every stage
// and accumulator buffer be used by one issuer only, whose program order then orders the
// uses:
//   - issuer i owns stages i * per .. i * per + per - 1; its n-th stage use (counting its
//     K blocks in order) is stage i * per + n % per in round n / per;
//   - issuer i owns accumulator buffers i and i + ISSUERS, alternating over its tiles;
//     a buffer's tiles all have the same parity, so one epilogue group drains it.
constexpr int ISSUERS = 3;
constexpr int ISSUER_ACC = 2 * ISSUERS;  // accumulator buffers in use

__device__ __forceinline__ void issuer_stage(int i, int n, int per, int& stage,
                                             uint32_t& phase) {
    stage = i * per + n % per;
    phase = static_cast<uint32_t>(n / per) & 1u;
}

__device__ __forceinline__ void issuer_acc(int k, int& buf, uint32_t& use) {
    const int j = k / ISSUERS;
    buf = (k - j * ISSUERS) + ISSUERS * (j & 1);
    use = static_cast<uint32_t>(j >> 1) & 1u;
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

template <typename Geo>
__device__ __forceinline__ void epilogue_direct64(const ConvShape& s, const EpilogueArgs& ep,
                                                  void* y, uint32_t tmem_base, uint32_t accf0,
                                                  uint32_t acce0, int num_tiles, uint64_t limit,
                                                  volatile int* abort_flag, Geo geo) {
    static_assert(EPI_GROUPS == ISSUERS, "each epilogue group drains one issuer's buffers");
    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const int quad = warp & 3;                // TMEM lane quadrant this warp may access
    const int grp = (warp - EPI_WARP0) >> 2;  // local tiles k with k % 3 == grp
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
         tile += EPI_GROUPS * gridDim.x, local += EPI_GROUPS) {
        int buf;
        uint32_t use;
        issuer_acc(local, buf, use);
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
                mbar_arrive(acce0 + 8u * buf);
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
