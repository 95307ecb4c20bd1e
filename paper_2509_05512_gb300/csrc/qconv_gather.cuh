// qconv_gather.cuh -- tensor-core quaternion convolution for layers with one quaternion
// input channel (the 4-channel stem of the backbone), included by qconv_tc.cu inside its
// anonymous namespace.
//
// With Q_in = 1 a pixel holds only 4 bf16 (8 bytes): too narrow for the tensor-map loads
// of the other kernels (a TMA row must be a multiple of 16 bytes) and far too narrow for
// a 16-wide K step per tap.  For stride-2 layers on inputs of even width, two horizontally
// adjacent pixels form an aligned 16-byte "pixel pair" [x_{2s}: r i j k | x_{2s+1}: r i j k],
// and the 7x7/2 filter window of an output pixel at column wo covers nsp = 4 consecutive
// pairs per filter row, starting at pair wo - (pad + lead) / 2 (lead = pad mod 2 is a
// filter column -1 whose weight is zero).  One 16-byte K unit is one (filter row, pair)
// and a pixel's im2col row is kh x nsp units (28 for the 7x7 stem: K = 224, 14 MMA K steps).
//
//   warps 12..15  gather: one thread per pixel row of the 128-pixel tile issues its
//                 units as 16-byte cp.async copies straight into the K-major 32-byte-
//                 swizzled A tile (pairs outside the image are zero-filled by the copy),
//                 through L1 so that the 4-7 fold reuse of input pairs between filter
//                 taps and neighbouring pixels stays on chip; a stage is handed to the
//                 MMA once the next one has been issued (one group of copies in flight
//                 behind the one being completed).
//   warp 1        TMEM owner and MMA issuer: 14 MMAs of M = 128, N = 64 per tile.
//   warps 0, 2..11  expand the signed block weight of Eq. 6 once per CTA:
//                 B[(q, co)][(ky, pair, e, p)] = sign(q, p) W_{q xor p}[co][ky][2 pair - lead + e]
//                 (zero outside the filter); then warps 4..11 run the wide epilogue.
// The zero-weight columns read real input pixels, which only matters for non-finite
// inputs (0 * inf); finite inputs give exactly the convolution of Eq. 5.

constexpr int GA_MAX_UNITS = 32;  // K <= 256
constexpr int GA_THREADS = 512;
constexpr int GA_GATHER_WARP0 = 12;

struct GatherParams {
    ConvShape s;
    EpilogueArgs ep;
    const __nv_bfloat16* x;
    const __nv_bfloat16* w[4];  // letter tensors [16][kh][kw][1]
    unsigned long long wait_limit_ns;
    int inject_stall;
    int nsp;          // pixel pairs per filter row
    int lead;         // pad mod 2: zero-weight filter column before the first pair
    int units;        // 16-byte K units per pixel row: kh * nsp rounded up to even
    int ksteps;       // units / 2
    int W2;           // W / 2 pairs per input row
    int stage_bytes;  // BM rows x units x 16 bytes
    int stages;
    int num_tiles;
};

struct GaCfg {
    static constexpr int CHUNK_A = BM * 32;  // one K step of the A tile: 128 rows x 32 bytes
    static constexpr int CHUNK_B = 64 * 32;  // one K step of the weight: 64 rows x 32 bytes
    static constexpr int B_BYTES = (GA_MAX_UNITS / 2) * CHUNK_B;
    using E = EpiSmem<16, true, 1>;
    static constexpr int NUM_BARS = 2 * MAX_STAGES + 6;  // full, empty, accf[2], acce[2], drain, bready
    static constexpr int TAIL_BYTES = B_BYTES + E::STAGING_BYTES + E::PARAM_BYTES +
                                      NUM_BARS * 8 + 16;
    static constexpr int SMEM_BYTES = 227 * 1024;
    static constexpr int RING_BYTES = ((SMEM_BYTES - 1024 - TAIL_BYTES) / 1024) * 1024;
    static constexpr int B_OFF = RING_BYTES;
    static constexpr int STAGING_OFF = B_OFF + B_BYTES;
    static constexpr int PARAM_OFF = STAGING_OFF + E::STAGING_BYTES;
    static constexpr int BAR_OFF = PARAM_OFF + E::PARAM_BYTES;
    static constexpr uint32_t DESC_HI = desc_hi(8 * 32, desc_layout(32));
    static constexpr uint32_t TMEM_COLS = 128;  // 2 buffers x 64 columns
    static constexpr int EXP_WARPS = 11;        // warps 0, 2..11
    static constexpr int GATHER_WARPS = 4;
    static_assert(BAR_OFF + NUM_BARS * 8 + 16 + 1024 <= SMEM_BYTES, "gather shared memory");
    static_assert(GA_GATHER_WARP0 + GATHER_WARPS == GA_THREADS / 32, "warp roles");
};

// Shapes the pixel-pair gather covers: one quaternion input channel, 16 quaternion
// output channels, stride 2, even input width, K within the weight region.
bool gather_ok(const ConvShape& s) {
    if (s.Qin != 1 || s.Qout != 16 || s.stride != 2 || (s.W & 1)) return false;
    const int lead = s.pad & 1;
    const int nsp = (s.kw + lead + 1) / 2;
    const long long units = static_cast<long long>(s.kh) * nsp;
    return units + (units & 1) <= GA_MAX_UNITS;
}

__global__ void __launch_bounds__(GA_THREADS, 1)
    qconv_gather_kernel(const __grid_constant__ CUtensorMap tmap_y, const GatherParams p) {
    using C = GaCfg;
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
    const uint32_t acce0 = bar0 + 8u * (2 * MAX_STAGES + 2);
    const uint32_t drain_bar = bar0 + 8u * (2 * MAX_STAGES + 4);
    const uint32_t bready_bar = bar0 + 8u * (2 * MAX_STAGES + 5);

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const ConvShape& s = p.s;
    const uint64_t limit = p.wait_limit_ns;
    const int STAGES = p.stages;

    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            mbar_init(full_bar(i), C::GATHER_WARPS);
            mbar_init(empty_bar(i), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(accf0 + 8u * b, 1);
            mbar_init(acce0 + 8u * b, 8 * 32);
        }
        mbar_init(drain_bar, 1);
        mbar_init(bready_bar, C::EXP_WARPS);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) tma_prefetch_desc(&tmap_y);
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), C::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp >= GA_GATHER_WARP0) {
        // ------------------------------------------------------------ pixel-pair gather
        const int m = (warp - GA_GATHER_WARP0) * 32 + lane;  // pixel row of the tile
        const int hw = s.Ho * s.Wo;
        const int s_shift = (s.pad + p.lead) / 2;
        // byte offset of (row m, unit u) in a stage: K step u / 2, 16-byte half u % 2,
        // 32-byte swizzle (the half flips on rows 4..7 of each 8-row group)
        const uint32_t row_off = static_cast<uint32_t>(m) * 32;
        const uint32_t sw = (static_cast<uint32_t>(m) >> 2) & 1u;
        const uint8_t* xb = reinterpret_cast<const uint8_t*>(p.x);
        int stage = 0, prev = -1;
        uint32_t phase = 0;
        bool aborted = false;
        for (int tile = blockIdx.x; tile < p.num_tiles; tile += gridDim.x) {
            // lane 0 waits for the stage and the warp follows it, so the warp stays
            // converged for the __syncwarp of the hand-off even when the wait gives up
            bool ok = true;
            if (lane == 0)
                ok = wait_or_abort(empty_bar(stage), phase ^ 1u, limit, abort_flag,
                                   STATUS_TIMEOUT_PRODUCER);
            if (__shfl_sync(0xffffffffu, ok ? 1 : 0, 0) == 0) {
                aborted = true;
                break;
            }
            const long long pix = static_cast<long long>(tile) * BM + m;
            const bool valid = pix < s.M;
            int img = 0, ho = 0, wo = 0;
            if (valid) {
                img = static_cast<int>(pix / hw);
                const int rem = static_cast<int>(pix - static_cast<long long>(img) * hw);
                ho = rem / s.Wo;
                wo = rem - ho * s.Wo;
            }
            const int iy0 = ho * 2 - s.pad;
            const int s0 = wo - s_shift;
            const uint32_t dst0 = sbase + stage * p.stage_bytes + row_off;
            int u = 0;
            for (int ky = 0; ky < s.kh; ++ky) {
                const int iy = iy0 + ky;
                const bool row_ok = valid && iy >= 0 && iy < s.H;
                const long long rbase = (static_cast<long long>(img) * s.H + iy) * p.W2;
                for (int j = 0; j < p.nsp; ++j, ++u) {
                    const int sp = s0 + j;
                    const bool ok = row_ok && sp >= 0 && sp < p.W2;
                    const uint8_t* src = ok ? xb + (rbase + sp) * 16 : xb;
                    const uint32_t dst = dst0 + (u >> 1) * C::CHUNK_A +
                                         ((static_cast<uint32_t>(u & 1) ^ sw) << 4);
                    cp_async_16_zfill(dst, src, ok ? 16u : 0u);
                }
            }
            for (; u < p.units; ++u) {
                const uint32_t dst = dst0 + (u >> 1) * C::CHUNK_A +
                                     ((static_cast<uint32_t>(u & 1) ^ sw) << 4);
                cp_async_16_zfill(dst, xb, 0u);
            }
            cp_async_commit();
            if (prev >= 0) {
                // the previous stage's copies have landed: publish it to the tensor cores
                cp_async_wait<1>();
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(full_bar(prev));
            }
            prev = stage;
            if (++stage == STAGES) {
                stage = 0;
                phase ^= 1u;
            }
        }
        cp_async_wait<0>();
        if (prev >= 0 && !aborted) {
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) mbar_arrive(full_bar(prev));
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t IDESC = make_idesc(BM, 64, 0);
            int stage = 0;
            uint32_t phase = 0;
            bool ok = wait_or_abort(bready_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
            int issued = 0;
            if (p.inject_stall) {
                // Failure injection: wait on a barrier nothing arrives on.
                wait_or_abort(drain_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
                ok = false;
            }
            tc_fence_after();
            const uint32_t b_lo0 = desc_lo(sbase + C::B_OFF);
            int local = 0;
            for (int tile = blockIdx.x; ok && tile < p.num_tiles; tile += gridDim.x, ++local) {
                const int buf = local & 1;
                const uint32_t use = static_cast<uint32_t>(local >> 1) & 1u;
                if (!wait_or_abort(acce0 + 8u * buf, use ^ 1u, limit, abort_flag,
                                   STATUS_TIMEOUT_MMA) ||
                    !wait_or_abort(full_bar(stage), phase, limit, abort_flag,
                                   STATUS_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem_base + static_cast<uint32_t>(buf * 64);
                const uint32_t a_lo0 = desc_lo(sbase + stage * p.stage_bytes);
                for (int c = 0; c < p.ksteps; ++c)
                    umma_f16_w(d, a_lo0 + ((c * C::CHUNK_A) >> 4), C::DESC_HI,
                               b_lo0 + ((c * C::CHUNK_B) >> 4), C::DESC_HI, IDESC,
                               c != 0 ? 1u : 0u);
                ++issued;
                umma_commit(empty_bar(stage));
                umma_commit(accf0 + 8u * buf);
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
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
        // warps 0, 2..11: one 16-byte K unit (filter row ky, pair j) of output row
        // n = (q, co) per item: 8 values, pixel e of the pair major, input component p minor.
        const int et = warp == 0 ? lane : (warp - 1) * 32 + lane;  // 0 .. 351
        constexpr int ET = C::EXP_WARPS * 32;
        const int taps = s.kh * s.kw;
        const int real_units = s.kh * p.nsp;
        for (int i = et; i < 64 * p.units; i += ET) {
            const int n = i / p.units, u = i - (i / p.units) * p.units;
            const int q = n >> 4, co = n & 15;
            const int ky = u / p.nsp, j = u - (u / p.nsp) * p.nsp;
            uint32_t packed[4];
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                const int kx = 2 * j - p.lead + e;
                const bool in = u < real_units && kx >= 0 && kx < s.kw;
                float v[4];
#pragma unroll
                for (int pc = 0; pc < 4; ++pc) {
                    float wv = 0.0f;
                    if (in) {
                        const int L = q ^ pc;
                        wv = __bfloat162float(p.w[L][co * taps + ky * s.kw + kx]);
                        if ((NEG_MASK >> (4 * q + pc)) & 1u) wv = -wv;
                    }
                    v[pc] = wv;
                }
                packed[2 * e] = pack_bf16x2(v[0], v[1]);
                packed[2 * e + 1] = pack_bf16x2(v[2], v[3]);
            }
            const uint32_t off = static_cast<uint32_t>(C::B_OFF + (u >> 1) * C::CHUNK_B + n * 32) +
                                 ((static_cast<uint32_t>(u & 1) ^ ((static_cast<uint32_t>(n) >> 2) & 1u))
                                  << 4);
            *reinterpret_cast<uint4*>(smem + off) =
                make_uint4(packed[0], packed[1], packed[2], packed[3]);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(bready_bar);

        if (warp >= EPI_WARP0) {
            // -------------------------------------------------------- epilogue
            const long long M = s.M;
            auto geo = [M](int tile) {
                EpiTile g;
                g.n_tile = 0;
                g.m0 = static_cast<long long>(tile) * BM;
                const long long left = M - g.m0;
                g.rows = left < BM ? static_cast<int>(left) : BM;
                g.sy = static_cast<int>(g.m0);
                g.sz = 0;
                return g;
            };
            epilogue_role<16, false, decltype(geo), true, 1>(
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
