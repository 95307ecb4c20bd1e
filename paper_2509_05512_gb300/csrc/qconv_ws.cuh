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
// Pixel staging, per tile of 128 output pixels:
//   halo     (stride 1, output width Wo a multiple of 8, at most 128): the tile is
//            R = 128 / Wo whole output rows of one image; for each horizontal filter
//            offset dw one tiled TMA box holds input rows r0 - pad .. r0 + R + kh - 2 at
//            columns dw - pad .. dw - pad + Wo - 1 (zero fill outside the image).  The
//            vertical offsets dh are descriptor offsets of dh * Wo rows into that box,
//            so kw boxes replace kh * kw.
//   per tap  otherwise: one im2col box of 128 pixels per filter tap.

constexpr int WS_ROW_BYTES = 128;  // 64 channels x bf16: all four components of a pixel

struct WsParams {
    ConvShape s;
    EpilogueArgs ep;
    const __nv_bfloat16* w[4];  // compact letter tensors [16][kh][kw][16]
    unsigned long long wait_limit_ns;
    int inject_stall;
    int taps;         // kh * kw
    int halo;         // row-block tiles with halo boxes
    int R;            // halo: output rows per tile
    int tpi;          // halo: tiles per image
    int kblocks;      // K blocks per tile: kw (halo) or taps
    int box_bytes;    // pixel box of one K block
    int stage_bytes;  // box rounded up to the 1024-byte swizzle period
    int stages;       // ring depth (<= MAX_STAGES)
    int num_tiles;
};

struct WsCfg {
    static constexpr int TAP_BYTES = 64 * WS_ROW_BYTES;  // expanded weight of one tap
    static constexpr int WSB_BYTES = WS_MAX_TAPS * TAP_BYTES;
    using E = EpiSmem<16, true>;
    // accumulator buffers in TMEM: enough that neither the MMAs' completion latency nor
    // the epilogue's turnaround stalls the MMA issue
    static constexpr int NACC = 4;
    static constexpr int NUM_BARS = 2 * MAX_STAGES + 2 * NACC + 2;  // full, empty, accf, acce, drain, wsready
    static constexpr int TAIL_BYTES =
        WSB_BYTES + E::STAGING_BYTES + E::PARAM_BYTES + NUM_BARS * 8 + 16;
    static constexpr int SMEM_BYTES = 227 * 1024;
    static constexpr int RING_BYTES = ((SMEM_BYTES - 1024 - TAIL_BYTES) / 1024) * 1024;
    static constexpr int WSB_OFF = RING_BYTES;
    static constexpr int STAGING_OFF = WSB_OFF + WSB_BYTES;
    static constexpr int PARAM_OFF = STAGING_OFF + E::STAGING_BYTES;
    static constexpr int BAR_OFF = PARAM_OFF + E::PARAM_BYTES;
    static_assert(PARAM_OFF % 16 == 0, "float4 reads of the epilogue vectors");
    static constexpr uint32_t DESC_HI = desc_hi(8 * WS_ROW_BYTES, desc_layout(WS_ROW_BYTES));
    static constexpr uint32_t TMEM_COLS = 64 * NACC;
    static constexpr int EXP_WARPS = 9;          // warps 2, 4..11 expand the weight
    static_assert(BAR_OFF + NUM_BARS * 8 + 16 + 1024 <= SMEM_BYTES, "WS shared memory");
};

bool ws_halo_ok(const ConvShape& s) {
    if (s.stride != 1 || s.Wo % 8 != 0 || s.Wo > BM) return false;
    const int R = BM / s.Wo;
    const long long box = static_cast<long long>(s.Wo) * (R + s.kh - 1) * WS_ROW_BYTES;
    const long long stage = (box + 1023) & ~1023LL;
    return 2 * stage <= WsCfg::RING_BYTES;
}

// KH > 0: the filter height, known at compile time (halo staging), so the MMA issue
// loop is fully unrolled; 0 = from the shape at run time.
template <bool HALO, int KH>
__global__ void __launch_bounds__(NUM_THREADS, 1)
    qconv_ws_kernel(const __grid_constant__ CUtensorMap tmap_x,
                    const __grid_constant__ CUtensorMap tmap_y, const WsParams p) {
    using C = WsCfg;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::BAR_OFF);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::NUM_BARS);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (MAX_STAGES + s); };
    const uint32_t accf0 = bar0 + 8u * (2 * MAX_STAGES);
    const uint32_t acce0 = bar0 + 8u * (2 * MAX_STAGES + C::NACC);
    const uint32_t drain_bar = bar0 + 8u * (2 * MAX_STAGES + 2 * C::NACC);
    const uint32_t wsready_bar = drain_bar + 8u;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const ConvShape& s = p.s;
    const uint64_t limit = p.wait_limit_ns;
    const int STAGES = p.stages;

    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            mbar_init(full_bar(i), 1);
            mbar_init(empty_bar(i), 1);
        }
        for (int b = 0; b < C::NACC; ++b) {
            mbar_init(accf0 + 8u * b, 1);
            mbar_init(acce0 + 8u * b, 8 * 32);
        }
        mbar_init(drain_bar, 1);
        mbar_init(wsready_bar, C::EXP_WARPS);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmap_x);
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

    if (warp == 0 || warp == 3) {
        // ------------------------------------------------------------ TMA producers
        // the two producer threads take alternate K blocks
        if (lane == 0) {
            const int role = warp == 0 ? 0 : 1;
            const uint64_t pol_x = l2_policy_evict_normal();
            int stage = 0;
            uint32_t phase = 0;
            uint32_t filled = 0, fill_parity = 0;
            bool ok = true;
            int kb_all = 0;
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
            // Cold pixels come from DRAM with a latency far above what the ring covers, so
            // the first producer asks L2 for this CTA's tiles PF tiles ahead of the ring.
            constexpr int PF = 2;
            auto prefetch_tile = [&](int tile) {
                if (role != 0 || tile >= p.num_tiles) return;
                int pimg, ph, pw;
                tile_base(tile, pimg, ph, pw);
                if constexpr (HALO)
                    tma_prefetch_l2_4d(&tmap_x, 0, pw + s.pad, ph, pimg);
                else
                    tma_prefetch_l2_im2col_4d(&tmap_x, 0, pw, ph, pimg,
                                              static_cast<uint16_t>(s.kw / 2),
                                              static_cast<uint16_t>(s.kh / 2));
            };
            for (int k = 0; k < PF; ++k) prefetch_tile(blockIdx.x + k * gridDim.x);
            for (int tile = blockIdx.x; ok && tile < p.num_tiles; tile += gridDim.x) {
                int img, hbase, wbase;
                tile_base(tile, img, hbase, wbase);
                prefetch_tile(tile + PF * gridDim.x);
                for (int kb = 0; kb < p.kblocks; ++kb, ++kb_all) {
                    if ((kb_all & 1) == role) {
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
                            tma_load_4d(dst, &tmap_x, fb, 0, wbase + kb, hbase, img, pol_x);
                        } else {
                            const int dh = kb / s.kw, dw = kb - (kb / s.kw) * s.kw;
                            tma_load_im2col_4d(dst, &tmap_x, fb, 0, wbase, hbase, img,
                                               static_cast<uint16_t>(dw),
                                               static_cast<uint16_t>(dh), pol_x);
                        }
                    }
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (!ok || *abort_flag) drain_fills(full_bar(0), STAGES, filled, fill_parity, limit);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t IDESC = make_idesc(BM, 64, 0);
            int stage = 0;
            uint32_t phase = 0;
            bool ok = wait_or_abort(wsready_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
            int issued = 0;
            if (p.inject_stall) {
                // Failure injection: wait on a barrier nothing arrives on.
                wait_or_abort(drain_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
                ok = false;
            }
            tc_fence_after();
            const uint32_t wsb_lo = desc_lo(sbase + C::WSB_OFF);
            int local = 0;
            const uint32_t row_lo = (s.Wo * WS_ROW_BYTES) >> 4;  // one output row of pixels
            for (int tile = blockIdx.x; ok && tile < p.num_tiles; tile += gridDim.x, ++local) {
                const int buf = local % C::NACC;
                const uint32_t use = static_cast<uint32_t>(local / C::NACC) & 1u;
                if (!wait_or_abort(acce0 + 8u * buf, use ^ 1u, limit, abort_flag,
                                   STATUS_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem_base + static_cast<uint32_t>(buf * 64);
                for (int kb = 0; kb < p.kblocks; ++kb) {
                    if (!wait_or_abort(full_bar(stage), phase, limit, abort_flag,
                                       STATUS_TIMEOUT_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a_lo0 = desc_lo(sbase + stage * p.stage_bytes);
                    if constexpr (HALO && KH > 0) {
                        const uint32_t b_lo0 = wsb_lo + ((kb * C::TAP_BYTES) >> 4);
                        const uint32_t b_row = (s.kw * C::TAP_BYTES) >> 4;
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
                            const uint32_t a_lo = a_lo0 + dh * row_lo;
                            const uint32_t b_lo = wsb_lo + ((tap * C::TAP_BYTES) >> 4);
#pragma unroll
                            for (int pc = 0; pc < 4; ++pc)
                                umma_f16_w(d, a_lo + pc * 2, C::DESC_HI, b_lo + pc * 2,
                                           C::DESC_HI, IDESC, (kb | dh | pc) != 0 ? 1u : 0u);
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
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (!ok) break;
                umma_commit(accf0 + 8u * buf);
            }
            if (!ok && issued > 0) {
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
        // ------------------------------------------------------------ weight expansion
        // warps 2 and 4..11 write the signed block weight: for tap t, row n = (q, co) and K
        // index k = (p, ci) the value is sign(q, p) * W_{q xor p}[co][t][ci], rows of 128
        // bytes, 128-byte swizzle.  Each 16-byte chunk of a compact letter L is read once
        // from global memory and written to its four places (p = 0..3, q = L xor p).
        const int et = warp == 2 ? lane : (warp - 3) * 32 + lane;  // 0 .. 287
        constexpr int ET = C::EXP_WARPS * 32;
        const int taps = p.taps;
        const int letter_chunks = taps * 32;  // 16-byte chunks of one letter (16 x taps x 16)
        for (int i = et; i < 4 * letter_chunks; i += ET) {
            const int L = i / letter_chunks, off = i - L * letter_chunks;
            const uint4 v = __ldg(reinterpret_cast<const uint4*>(p.w[L]) + off);
            // chunk `off` of letter L holds W_L[co][t][ci0 .. ci0 + 7]
            const int co = off / (taps * 2), rem = off - co * (taps * 2);
            const int t = rem >> 1, half_ci = rem & 1;
#pragma unroll
            for (int pc = 0; pc < 4; ++pc) {
                const int q = L ^ pc;
                const int n = q * 16 + co, ch = pc * 2 + half_ci;
                const uint4 u = ((NEG_MASK >> (4 * q + pc)) & 1u) ? negate_bf16x8(v) : v;
                *reinterpret_cast<uint4*>(smem + C::WSB_OFF + t * C::TAP_BYTES +
                                          n * WS_ROW_BYTES + ((ch ^ (n & 7)) << 4)) = u;
            }
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(wsready_bar);

        if (warp >= EPI_WARP0) {
            // -------------------------------------------------------- epilogue
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
                        g.sy = r0 * Wo;
                        g.sz = img;
                    } else {
                        g.m0 = static_cast<long long>(tile) * BM;
                        const long long left = M - g.m0;
                        g.rows = left < BM ? static_cast<int>(left) : BM;
                        g.sy = static_cast<int>(g.m0);
                        g.sz = 0;
                    }
                    return g;
                };
            epilogue_role<16, HALO, decltype(geo), true, 2, C::NACC>(
                s, p.ep, &tmap_y, tmem_base, smem + C::STAGING_OFF,
                reinterpret_cast<float*>(smem + C::PARAM_OFF), accf0, acce0, p.num_tiles, limit,
                abort_flag, geo);
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
