// qconv_ws.cuh -- weight-stationary tensor-core quaternion convolution (included by
// qconv_tc.cu inside its anonymous namespace).
//
// For layers with 16 quaternion channels in and out (64 real) the whole signed block
// weight of Eq. 6 fits in shared memory: 64 output rows x (taps x 64) K entries, 8 KB per
// tap.  Every CTA reads the compact letters once (taps x 2 KB, 1/4 of the block weight),
// expands them shared -> shared into the K-major 128-byte-swizzled layout, and from then
// on streams only pixels.  A pixel row of 64 channels holds all four input components,
// so one 16-wide K step of an MMA is one input component p, and an MMA of N = 64 covers
// all four output components.
//
// The separable form of Eq. 7 runs here too: its block weight has sign * W_p in every row
// block of column block p (ws_expand<.., true>), so the MMAs and the epilogue are those of
// the full form and the sign mix comes with the weight.
//
// Pixel staging, per tile of 128 output pixels:
//   halo     (stride 1, output width Wo a multiple of 8, at most 128): the tile is
//            R = 128 / Wo whole output rows of one image; for each horizontal filter
//            offset dw one tiled TMA box holds input rows r0 - pad .. r0 + R + kh - 2 at
//            columns dw - pad .. dw - pad + Wo - 1 (zero fill outside the image).  The
//            vertical offsets dh are descriptor offsets of dh * Wo rows into that box,
//            so kw boxes replace kh * kw.
//   per tap  otherwise: one im2col box of 128 pixels per filter tap.
//
// Roles (16 warps):
//   warp 0       TMA producer: the K blocks of each group of NI consecutive local tiles
//                interleaved (block 0 of each tile, then block 1, ...), each into the next
//                stage of the issuer that owns the tile.
//   warps 1..NI  MMA issuers taking the CTA's local tiles round robin, each waiting only
//                for its own stages and accumulator buffers (issuer_stage, issuer_acc_n in
//                tc_common.cuh; the tensor pipe keeps almost no queue and an issuing
//                thread's own waits and branches cost hundreds of cycles while its MMAs
//                are in flight).  Warp 1 owns TMEM.  NI = 3 hides those stalls best; NI = 2
//                gives each issuer half of the stage ring instead of a third, for pixel
//                boxes so large that three issuers would hold fewer stages than a tile
//                has K blocks (the third block's load then waits for the first block's
//                MMAs and its latency is exposed).
//   warps 2..15  expand the signed block weight once per CTA; then warps 4 .. 4 + 4 NI - 1
//                run the shared-memory-free direct epilogue (tc_common.cuh), one group of
//                four per issuer.

constexpr int WS_ROW_BYTES = 128;  // 64 channels x bf16: all four components of a pixel

struct WsParams {
    ConvShape s;
    EpilogueArgs ep;
    const __nv_bfloat16* w[4];  // compact letter tensors [16][kh][kw][16]
    void* y;                    // output [N][Ho][Wo][64]
    unsigned long long wait_limit_ns;
    int inject_stall;
    int taps;         // kh * kw
    int halo;         // row-block tiles with halo boxes
    int R;            // halo: output rows per tile
    int tpi;          // halo: tiles per image
    int kblocks;      // K blocks per tile: kw (halo) or taps
    int box_bytes;    // pixel box of one K block
    int stage_bytes;  // box rounded up to the 1024-byte swizzle period
    int per;          // stages owned by each issuer
    int num_tiles;
};

struct WsCfg {
    static constexpr int TAP_BYTES = 64 * WS_ROW_BYTES;  // expanded weight of one tap
    static constexpr int WSB_BYTES = WS_MAX_TAPS * TAP_BYTES;
    static constexpr int MAX_PER = 4;                // stages per issuer at most
    static constexpr int NSTAGE = ISSUERS * MAX_PER;  // stage barriers
    // full, empty, accf, acce, drain (one per issuer), wsready
    static constexpr int NUM_BARS = 2 * NSTAGE + 2 * ISSUER_ACC + ISSUERS + 1;
    static constexpr int TAIL_BYTES = WSB_BYTES + NUM_BARS * 8 + 16;
    static constexpr int SMEM_BYTES = 227 * 1024;
    static constexpr int RING_BYTES = ((SMEM_BYTES - 1024 - TAIL_BYTES) / 1024) * 1024;
    static constexpr int WSB_OFF = RING_BYTES;
    static constexpr int BAR_OFF = WSB_OFF + WSB_BYTES;
    static constexpr uint32_t DESC_HI = desc_hi(8 * WS_ROW_BYTES, desc_layout(WS_ROW_BYTES));
    static constexpr uint32_t TMEM_COLS = 512;  // ISSUER_ACC buffers of 64 columns
    static constexpr int EXP_WARPS = 14;  // warps 2..15 expand the weight
    static_assert(BAR_OFF + NUM_BARS * 8 + 16 + 1024 <= SMEM_BYTES, "WS shared memory");
    static_assert(4 * WS_MAX_TAPS * 32 <= 4 * EXP_WARPS * 32, "expansion in four rounds");
};

bool ws_halo_ok(const ConvShape& s) {
    if (s.stride != 1 || s.Wo % 8 != 0 || s.Wo > BM) return false;
    const int R = BM / s.Wo;
    const long long box = static_cast<long long>(s.Wo) * (R + s.kh - 1) * WS_ROW_BYTES;
    const long long stage = (box + 1023) & ~1023LL;
    return 2 * stage <= WsCfg::RING_BYTES;
}

// Issuers for a pixel stage of `stage_bytes` and `kblocks` K blocks per tile: three while
// that leaves each at least min(kblocks, 3) stages, else two.
int ws_issuers(int stage_bytes, int kblocks) {
    const int stages = WsCfg::RING_BYTES / stage_bytes;
    const int want = kblocks < 3 ? kblocks : 3;
    return stages / 3 >= want ? 3 : 2;
}

// Weight expansion by warps 2..15: for tap t, row n = (q, co) and K index k = (p, ci) the
// value is sign(q, p) * W_{q xor p}[co][t][ci], rows of 128 bytes, 128-byte swizzle.  Each
// 16-byte chunk of a compact letter L is read once from global memory (all of a thread's
// chunks in flight together) and written to its four places (p = 0..3, q = L xor p).
// TAPS > 0: the tap count known at compile time, so the chunk index splits with constant
// divisions (the expansion sits on every launch's critical path and is bound by its
// integer work); 0 = from the parameters.  SEP: the separable form of Eq. 7 instead, whose
// block weight has letter p in every row block of column block p (sign * W_p), so the
// same MMAs compute it with the sign mix folded into the weight.
template <int TAPS, bool SEP>
__device__ __forceinline__ void ws_expand(const WsParams& p, uint8_t* smem, int warp,
                                          int lane, uint32_t wsready_bar) {
    using C = WsCfg;
    const int et = (warp - 2) * 32 + lane;  // 0 .. 447
    constexpr int ET = C::EXP_WARPS * 32;
    const int taps = TAPS > 0 ? TAPS : p.taps;
    const int letter_chunks = taps * 32;  // 16-byte chunks of one letter (16 x taps x 16)
    const int total = 4 * letter_chunks;
    uint4 v[4];
#pragma unroll
    for (int r = 0; r < 4; ++r) {
        const int i = et + r * ET;
        if (i < total) {
            const int L = i / letter_chunks;
            v[r] = __ldg(reinterpret_cast<const uint4*>(p.w[L]) + (i - L * letter_chunks));
        }
    }
#pragma unroll
    for (int r = 0; r < 4; ++r) {
        const int i = et + r * ET;
        if (i >= total) continue;
        const int L = i / letter_chunks, off = i - L * letter_chunks;
        // chunk `off` of letter L holds W_L[co][t][ci0 .. ci0 + 7]
        const int co = off / (taps * 2), rem = off - co * (taps * 2);
        const int t = rem >> 1, half_ci = rem & 1;
        const uint32_t signs = ((SEP ? SEP_LETTER_SIGNS : LETTER_SIGNS) >> (4 * L)) & 15u;
        uint8_t* row = smem + C::WSB_OFF + t * C::TAP_BYTES + co * WS_ROW_BYTES;
        const int sw = co & 7;  // the row's 128-byte swizzle phase (q * 16 keeps it)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            // Hamilton: row block L xor j, column block j; separable: row block j, column L
            const int q = SEP ? j : L ^ j, ch = (SEP ? L : j) * 2 + half_ci;
            const uint4 u = ((signs >> j) & 1u) ? negate_bf16x8(v[r]) : v[r];
            *reinterpret_cast<uint4*>(row + q * 16 * WS_ROW_BYTES + ((ch ^ sw) << 4)) = u;
        }
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) mbar_arrive(wsready_bar);
}

// KH = 3: a 3x3 filter with halo staging, known at compile time, so the MMA issue loop is
// fully unrolled and the expansion's tap count is a constant; 0 = from the shape at run
// time.  NI: MMA issuers (2 or 3).  SEP: the separable block weight of Eq. 7.
template <bool HALO, int KH, int NI, bool SEP>
__global__ void __launch_bounds__(WIDE_THREADS, 1)
    qconv_ws_kernel(const __grid_constant__ CUtensorMap tmap_x, const WsParams p) {
    using C = WsCfg;
    static_assert(NI == 2 || NI == ISSUERS, "two or three issuers");
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::BAR_OFF);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::NUM_BARS);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (C::NSTAGE + s); };
    const uint32_t accf0 = bar0 + 8u * (2 * C::NSTAGE);
    const uint32_t acce0 = bar0 + 8u * (2 * C::NSTAGE + ISSUER_ACC);
    const uint32_t drain0 = bar0 + 8u * (2 * C::NSTAGE + 2 * ISSUER_ACC);
    const uint32_t wsready_bar = drain0 + 8u * NI;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const ConvShape& s = p.s;
    const uint64_t limit = p.wait_limit_ns;
    const int STAGES = NI * p.per;
    // this CTA's local tiles: blockIdx.x + k * gridDim.x, k < kt
    const int kt = (p.num_tiles - static_cast<int>(blockIdx.x) + static_cast<int>(gridDim.x) - 1) /
                   static_cast<int>(gridDim.x);

    griddep_launch_dependents();
    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            mbar_init(full_bar(i), 1);
            mbar_init(empty_bar(i), 1);
        }
        for (int b = 0; b < ISSUER_ACC; ++b) {
            mbar_init(accf0 + 8u * b, 1);
            mbar_init(acce0 + 8u * b, EPI2_ACCE_COUNT);
        }
        for (int i = 0; i < NI; ++i) mbar_init(drain0 + 8u * i, 1);
        mbar_init(wsready_bar, C::EXP_WARPS);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) tma_prefetch_desc(&tmap_x);
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
    // pixel rows of a tile: halo -> (image, first input row); per tap -> first pixel
    auto tile_base = [&](int tile, int& img, int& hbase, int& wbase) {
        if constexpr (HALO) {
            img = tile / p.tpi;
            const int r0 = (tile - img * p.tpi) * p.R;
            hbase = r0 - s.pad;
            wbase = -s.pad;
        } else {
            const long long m0 = static_cast<long long>(tile) * BM;
            img = static_cast<int>(m0 / hw);
            const int rem = static_cast<int>(m0 - static_cast<long long>(img) * hw);
            const int ho = rem / s.Wo, wo = rem - (rem / s.Wo) * s.Wo;
            wbase = wo * s.stride - s.pad;
            hbase = ho * s.stride - s.pad;
        }
    };

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint64_t pol_x = l2_policy_evict_normal();
            uint32_t filled = 0, fill_parity = 0;
            bool ok = true;
            StageCursor cur(p.per);
            for (int g0 = 0; ok && g0 < kt; g0 += NI) {
                const int ng = kt - g0 < NI ? kt - g0 : NI;
                int img[NI], hbase[NI], wbase[NI];
#pragma unroll
                for (int i = 0; i < NI; ++i)
                    if (i < ng)
                        tile_base(static_cast<int>(blockIdx.x) + (g0 + i) * static_cast<int>(gridDim.x),
                                  img[i], hbase[i], wbase[i]);
                for (int kb = 0; ok && kb < p.kblocks; ++kb, cur.next()) {
#pragma unroll
                    for (int i = 0; i < NI; ++i) {
                        if (i >= ng) break;
                        // K block kb of local tile g0 + i: use (g0 / NI) * kblocks + kb of
                        // issuer i, the same use count for every issuer of the group
                        const int stage = cur.stage(i);
                        const uint32_t phase = cur.phase;
                        if (!wait_or_abort(empty_bar(stage), phase ^ 1u, limit, abort_flag,
                                           STATUS_TIMEOUT_PRODUCER)) {
                            ok = false;
                            break;
                        }
                        const uint32_t fb = full_bar(stage);
                        mbar_arrive_expect_tx(fb, p.box_bytes);
                        filled |= 1u << stage;
                        fill_parity = (fill_parity & ~(1u << stage)) | (phase << stage);
                        const uint32_t dst = sbase + stage * p.stage_bytes;
                        if constexpr (HALO) {
                            // K block kb = horizontal filter offset dw
                            tma_load_4d(dst, &tmap_x, fb, 0, wbase[i] + kb, hbase[i], img[i], pol_x);
                        } else {
                            const int dh = kb / s.kw, dw = kb - (kb / s.kw) * s.kw;
                            tma_load_im2col_4d(dst, &tmap_x, fb, 0, wbase[i], hbase[i], img[i],
                                               static_cast<uint16_t>(dw),
                                               static_cast<uint16_t>(dh), pol_x);
                        }
                    }
                }
            }
            if (!ok || *abort_flag) drain_fills(full_bar(0), STAGES, filled, fill_parity, limit);
        }
    } else if (warp <= NI) {
        // ------------------------------------------------------------ MMA issuers
        if (warp >= 2) ws_expand<KH == 3 ? 9 : 0, SEP>(p, smem, warp, lane, wsready_bar);
        if (lane == 0) {
            constexpr uint32_t IDESC = make_idesc(BM, 64, 0);
            const int me = warp - 1;
            const uint32_t drain_bar = drain0 + 8u * me;
            bool ok = wait_or_abort(wsready_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
            int issued = 0;
            if (p.inject_stall && me == 0) {
                // Failure injection: wait on a barrier nothing arrives on.
                wait_or_abort(drain_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
                ok = false;
            }
            tc_fence_after();
            const uint32_t wsb_lo = desc_lo(sbase + C::WSB_OFF);
            const uint32_t row_lo = (s.Wo * WS_ROW_BYTES) >> 4;  // one output row of pixels
            const uint32_t b_row = (s.kw * C::TAP_BYTES) >> 4;    // one filter row of taps
            StageCursor cur(p.per);
            for (int k = me; ok && k < kt; k += NI) {
                int buf;
                uint32_t use;
                issuer_acc_n<NI>(k, buf, use);
                if (!wait_or_abort(acce0 + 8u * buf, use ^ 1u, limit, abort_flag,
                                   STATUS_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem_base + static_cast<uint32_t>(buf * 64);
                for (int kb = 0; kb < p.kblocks; ++kb) {
                    // use (k / NI) * kblocks + kb of this issuer
                    const int stage = cur.stage(me);
                    const uint32_t phase = cur.phase;
                    cur.next();
                    if (!wait_or_abort(full_bar(stage), phase, limit, abort_flag,
                                       STATUS_TIMEOUT_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a_lo0 = desc_lo(sbase + stage * p.stage_bytes);
                    if constexpr (HALO && KH > 0) {
                        const uint32_t b_lo0 = wsb_lo + ((kb * C::TAP_BYTES) >> 4);
#pragma unroll
                        for (int dh = 0; dh < KH; ++dh) {
#pragma unroll
                            for (int pc = 0; pc < 4; ++pc)
                                umma_f16_w(d, a_lo0 + dh * row_lo + pc * 2, C::DESC_HI,
                                           b_lo0 + dh * b_row + pc * 2, C::DESC_HI, IDESC,
                                           (kb | dh | pc) != 0 ? 1u : 0u);
                        }
                    } else if constexpr (HALO) {
                        for (int dh = 0; dh < s.kh; ++dh) {
                            const int tap = dh * s.kw + kb;
                            const uint32_t b_lo = wsb_lo + ((tap * C::TAP_BYTES) >> 4);
#pragma unroll
                            for (int pc = 0; pc < 4; ++pc)
                                umma_f16_w(d, a_lo0 + dh * row_lo + pc * 2, C::DESC_HI,
                                           b_lo + pc * 2, C::DESC_HI, IDESC,
                                           (kb | dh | pc) != 0 ? 1u : 0u);
                        }
                    } else {
                        const uint32_t b_lo = wsb_lo + ((kb * C::TAP_BYTES) >> 4);
#pragma unroll
                        for (int pc = 0; pc < 4; ++pc)
                            umma_f16_w(d, a_lo0 + pc * 2, C::DESC_HI, b_lo + pc * 2, C::DESC_HI,
                                       IDESC, (kb | pc) != 0 ? 1u : 0u);
                    }
                    ++issued;
                    umma_commit(empty_bar(stage));
                }
                if (!ok) break;
                umma_commit(accf0 + 8u * buf);
            }
            if (!ok && issued > 0) {
                // let this issuer's MMAs finish before TMEM is released
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
        ws_expand<KH == 3 ? 9 : 0, SEP>(p, smem, warp, lane, wsready_bar);
        // ------------------------------------------- epilogue (warps 4 .. 4 + 4 NI - 1)
        const int tpi = p.tpi, R = p.R, Ho = s.Ho, Wo = s.Wo;
        const long long M = s.M;
        auto geo = [tpi, R, Ho, Wo, M](int tile) {
            EpiTile g;
            g.n_tile = 0;
            if constexpr (HALO) {
                const int img = tile / tpi;
                const int r0 = (tile - img * tpi) * R;
                g.m0 = (static_cast<long long>(img) * Ho + r0) * Wo;
                const int nr = Ho - r0 < R ? Ho - r0 : R;
                g.rows = nr * Wo;
            } else {
                g.m0 = static_cast<long long>(tile) * BM;
                const long long left = M - g.m0;
                g.rows = left < BM ? static_cast<int>(left) : BM;
            }
            return g;
        };
        if (warp >= EPI_WARP0)
            epilogue_direct64<decltype(geo), NI>(s, p.ep, p.y, tmem_base, accf0, acce0,
                                                 p.num_tiles, limit, abort_flag, geo);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, C::TMEM_COLS);
    }
}
