// qconv_gather.cuh -- tensor-core quaternion convolution for layers with one quaternion
// input channel (the 4-channel stem of the backbone), included by qconv_tc.cu inside its
// anonymous namespace.
//
// With Q_in = 1 a pixel holds only 4 bf16 (8 bytes): too narrow for a 16-wide K step per
// tap and for the pixel-tile maps of the other kernels.  For stride-2 layers on inputs of
// even width, two horizontally adjacent pixels form an aligned 16-byte "pixel pair"
// [x_{2s}: r i j k | x_{2s+1}: r i j k], and in pair coordinates the horizontal stride is
// 1: output column wo reads pairs wo - shift + j, j = 0 .. nsp - 1, where
// shift = (pad + lead) / 2, lead = pad mod 2 is a leading filter column -1 of zero weight,
// and nsp (rounded up to even, 4 for the 7x7 stem) is the number of pairs per filter row.
//
// Tile = 128 consecutive output columns of one output row (one MMA of M = 128; columns
// past the row end are computed and never stored).  One 3-D TMA box per tile holds, for
// the kh consecutive input rows 2 ho - pad .. 2 ho - pad + kh - 1, the 128 + nsp - 1 pairs
// the tile reads, zero filled outside the image.  The box addresses the input in groups
// of G pairs (128-byte elements for W a multiple of 16), since the TMA unit's cost grows
// with the number of inner-dimension elements: 16-byte elements made a box 917 requests
// and its latency several microseconds.  The tile's first pair then sits d0 = (-shift)
// mod G pairs into the box.  The A operand of the K step
// (ky, pairs 2t, 2t + 1) is that box's row ky read as a K-major, non-swizzled matrix whose
// row m starts at pair m + 2t: 16-byte rows, 8-row groups 128 bytes apart (stride byte
// offset) and the second 8-element K half one pair (16 bytes) further on (leading byte
// offset) -- the overlapping rows of an im2col matrix come from the descriptor, so the
// pixels are read from global memory once per filter row and never copied on chip, and a
// tile costs one TMA instruction (the per-box issue cost of the TMA unit, not its bytes,
// limits boxes this narrow).
//
//   warp 0        TMA producer: one box per tile into a ring of stages.
//   warps 1..3    MMA issuers, one lane each, taking the CTA's tiles round robin: each
//                 waits for its tile's stage and accumulator buffer and issues the
//                 kh * nsp / 2 MMAs of M = 128, N = 64 (14 for the stem, K = 224) in one
//                 unrolled run.  The tensor pipe keeps almost no queue and the issuing
//                 thread's own waits and branches cost hundreds of cycles while its MMAs
//                 are in flight, so three issuers are needed to keep the pipe busy.  Each
//                 issuer owns its stages and two accumulator buffers (issuer_stage,
//                 issuer_acc in tc_common.cuh).  Warp 1 also owns TMEM.
//   warps 2..15   expand the signed block weight of Eq. 6 once per CTA:
//                 B[(q, co)][(ky, pair, e, p)] = sign(q, p) W_{q xor p}[co][ky][2 pair - lead + e]
//                 (zero outside the filter), K-major with a 32-byte swizzle; then warps
//                 4..15 run the direct epilogue (tc_common.cuh: no shared memory, coalesced
//                 global stores, columns past the end of the output row not stored).
// The zero-weight columns read real input pixels, which only matters for non-finite
// inputs (0 * inf); finite inputs give exactly the convolution of Eq. 5.

constexpr int GA_MAX_UNITS = 32;  // K <= 256
constexpr int GA_TILE_W = 128;    // output columns per tile

struct GatherParams {
    ConvShape s;
    EpilogueArgs ep;
    const __nv_bfloat16* w[4];  // letter tensors [16][kh][kw][1]
    void* y;                    // output [N][Ho][Wo][64]
    unsigned long long wait_limit_ns;
    int inject_stall;
    int nsp;          // pixel pairs per filter row (even)
    int lead;         // pad mod 2: zero-weight filter column before the first pair
    int shift;        // (pad + lead) / 2: first pair of output column 0 is -shift
    int group;        // G: pairs per TMA element (1, 2, 4 or 8)
    int d0;           // pairs from the box start to the tile's first pair
    int boxg;         // G-pair elements per filter row of the box
    int box_stride;   // bytes between filter rows in the box: boxg * 16 G
    int box_bytes;    // bytes of one filter row: boxg * 16 G
    int stage_bytes;
    int per;          // stages owned by each issuer
    int segs;         // tiles per output row
    int num_tiles;
};

struct GaCfg {
    static constexpr int CHUNK_B = 64 * 32;  // one K step of the weight: 64 rows x 32 bytes
    static constexpr int B_BYTES = (GA_MAX_UNITS / 2) * CHUNK_B;
    // the letter tensors during the weight expansion (4 x 16 x taps x 2 bytes, taps <= 64)
    static constexpr int SCRATCH_BYTES = 8 * 1024;
    static constexpr int MAX_PER = 4;                // stages per issuer at most
    static constexpr int NSTAGE = ISSUERS * MAX_PER;  // stage barriers
    // full, empty, accf, acce, drain (one per issuer), bready
    static constexpr int NUM_BARS = 2 * NSTAGE + 2 * ISSUER_ACC + ISSUERS + 1;
    static constexpr int TAIL_BYTES = B_BYTES + SCRATCH_BYTES + NUM_BARS * 8 + 16;
    static constexpr int SMEM_BYTES = 227 * 1024;
    static constexpr int RING_BYTES = ((SMEM_BYTES - 1024 - TAIL_BYTES) / 1024) * 1024;
    static constexpr int B_OFF = RING_BYTES;
    static constexpr int SCRATCH_OFF = B_OFF + B_BYTES;
    static constexpr int BAR_OFF = SCRATCH_OFF + SCRATCH_BYTES;
    // A: K-major, no swizzle, 8-row groups 128 bytes apart (the leading byte offset of
    // one pair, 16 bytes, is the low word's default); B: K-major rows of 32 bytes.
    static constexpr uint32_t A_DESC_HI = desc_hi(8 * 16, 0);
    static constexpr uint32_t B_DESC_HI = desc_hi(8 * 32, desc_layout(32));
    static constexpr uint32_t TMEM_COLS = 512;  // ISSUER_ACC buffers of 64 columns
    static constexpr int EXP_WARPS = 14;        // warps 2..15
    static_assert(BAR_OFF + NUM_BARS * 8 + 16 + 1024 <= SMEM_BYTES, "gather shared memory");
};

// nsp of a shape: pairs covering lead + kw filter columns, rounded up to even.
int gather_nsp(const ConvShape& s) {
    const int lead = s.pad & 1;
    const int nsp = (s.kw + lead + 1) / 2;
    return nsp + (nsp & 1);
}

// Weight expansion, run by warps 2..15 (EXP_WARPS): the signed block weight of Eq. 6 as
// K-major rows of 32-byte K steps with a 32-byte swizzle,
//   B[(q, co)][(ky, pair j, pixel e, component p)] = sign(q, p) W_{q xor p}[co][ky][2 j - lead + e]
// (zero outside the filter).  The four letter tensors are first copied to shared memory
// (a scratch area) with every thread's 16-byte loads in flight at once, then expanded
// shared -> shared.
__device__ __forceinline__ void expand_block_weight(const ConvShape& s, const GatherParams& p,
                                                    uint8_t* smem, int warp, int lane,
                                                    uint32_t bready_bar);

// Shapes the pixel-pair kernel covers: one quaternion input channel, 16 quaternion output
// channels, stride 2, even input width, K within the weight region.
bool gather_ok(const ConvShape& s) {
    if (s.Qin != 1 || s.Qout != 16 || s.stride != 2 || (s.W & 1)) return false;
    return static_cast<long long>(s.kh) * gather_nsp(s) <= GA_MAX_UNITS;
}


__device__ __forceinline__ void expand_block_weight(const ConvShape& s, const GatherParams& p,
                                                    uint8_t* smem, int warp, int lane,
                                                    uint32_t bready_bar) {
    using C = GaCfg;
    const int et = (warp - 2) * 32 + lane;  // 0 .. 447
    constexpr int ET = C::EXP_WARPS * 32;
    const int taps = s.kh * s.kw;
    // 1. letters [16][kh][kw][1] -> shared memory, 2 * taps 16-byte chunks per letter
    const int lchunks = 2 * taps, nchunks = 4 * lchunks;
    uint8_t* wl = smem + C::SCRATCH_OFF;
    {
        uint4 v[2];
#pragma unroll
        for (int r = 0; r < 2; ++r) {
            const int i = et + r * ET;
            if (i < nchunks) {
                const int L = i / lchunks;
                v[r] = __ldg(reinterpret_cast<const uint4*>(p.w[L]) + (i - L * lchunks));
            }
        }
#pragma unroll
        for (int r = 0; r < 2; ++r)
            if (et + r * ET < nchunks) reinterpret_cast<uint4*>(wl)[et + r * ET] = v[r];
        for (int i = et + 2 * ET; i < nchunks; i += ET) {
            const int L = i / lchunks;
            reinterpret_cast<uint4*>(wl)[i] =
                __ldg(reinterpret_cast<const uint4*>(p.w[L]) + (i - L * lchunks));
        }
    }
    named_bar_sync(5, ET);
    const __nv_bfloat16* wls = reinterpret_cast<const __nv_bfloat16*>(wl);
    // 2. one 16-byte K unit (filter row ky, pair j) of output row n = (q, co) per item:
    //    8 values, pixel e of the pair major, input component p minor
    const int units = s.kh * p.nsp;
    for (int i = et; i < 64 * units; i += ET) {
        const int n = i / units, u = i - (i / units) * units;
        const int q = n >> 4, co = n & 15;
        const int ky = u / p.nsp, j = u - (u / p.nsp) * p.nsp;
        uint32_t packed[4];
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int kx = 2 * j - p.lead + e;
            const bool in = kx >= 0 && kx < s.kw;
            float v[4];
#pragma unroll
            for (int pc = 0; pc < 4; ++pc) {
                float wv = 0.0f;
                if (in) {
                    const int L = q ^ pc;
                    wv = __bfloat162float(wls[(L * 16 + co) * taps + ky * s.kw + kx]);
                    if ((NEG_MASK >> (4 * q + pc)) & 1u) wv = -wv;
                }
                v[pc] = wv;
            }
            packed[2 * e] = pack_bf16x2(v[0], v[1]);
            packed[2 * e + 1] = pack_bf16x2(v[2], v[3]);
        }
        // K step u / 2, 16-byte half u % 2 of the 32-byte row, 32-byte swizzle
        const uint32_t off =
            static_cast<uint32_t>(C::B_OFF + (u >> 1) * C::CHUNK_B + n * 32) +
            ((static_cast<uint32_t>(u & 1) ^ ((static_cast<uint32_t>(n) >> 2) & 1u)) << 4);
        *reinterpret_cast<uint4*>(smem + off) =
            make_uint4(packed[0], packed[1], packed[2], packed[3]);
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) mbar_arrive(bready_bar);
}

// KH, NSP > 0: the filter height and pairs per filter row known at compile time, so the
// MMA issue loop is fully unrolled with constant descriptor offsets; 0 = from the
// parameters at run time.
template <int KH, int NSP>
__global__ void __launch_bounds__(WIDE_THREADS, 1)
    qconv_pairs_kernel(const __grid_constant__ CUtensorMap tmap_x, const GatherParams p) {
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
    auto empty_bar = [&](int s) { return bar0 + 8u * (C::NSTAGE + s); };
    const uint32_t accf0 = bar0 + 8u * (2 * C::NSTAGE);
    const uint32_t acce0 = bar0 + 8u * (2 * C::NSTAGE + ISSUER_ACC);
    const uint32_t drain0 = bar0 + 8u * (2 * C::NSTAGE + 2 * ISSUER_ACC);
    const uint32_t bready_bar = drain0 + 8u * ISSUERS;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const ConvShape& s = p.s;
    const uint64_t limit = p.wait_limit_ns;
    const int STAGES = ISSUERS * p.per;

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
        for (int i = 0; i < ISSUERS; ++i) mbar_init(drain0 + 8u * i, 1);
        mbar_init(bready_bar, C::EXP_WARPS);
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
    griddep_wait();  // the previous kernel's output (this layer's input) is complete

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint64_t pol_x = l2_policy_evict_normal();
            uint32_t filled = 0, fill_parity = 0;
            bool ok = true;
            const uint32_t tx = static_cast<uint32_t>(s.kh * p.box_bytes);
            StageCursor cur(p.per);  // advanced once per round of ISSUERS tiles
            int ki = 0;              // local tile k % ISSUERS
            for (int tile = blockIdx.x; tile < p.num_tiles; tile += gridDim.x) {
                const int row = tile / p.segs, seg = tile - (tile / p.segs) * p.segs;
                const int img = row / s.Ho, ho = row - (row / s.Ho) * s.Ho;
                // local tile k -> issuer k % ISSUERS, its (k / ISSUERS)-th stage use
                const int stage = cur.stage(ki);
                const uint32_t phase = cur.phase;
                if (++ki == ISSUERS) {
                    ki = 0;
                    cur.next();
                }
                if (!wait_or_abort(empty_bar(stage), phase ^ 1u, limit, abort_flag,
                                   STATUS_TIMEOUT_PRODUCER)) {
                    ok = false;
                    break;
                }
                const uint32_t fb = full_bar(stage);
                mbar_arrive_expect_tx(fb, tx);
                filled |= 1u << stage;
                fill_parity = (fill_parity & ~(1u << stage)) | (phase << stage);
                const uint32_t dst = sbase + stage * p.stage_bytes;
                tma_load_4d(dst, &tmap_x, fb, 0, (seg * GA_TILE_W - p.shift - p.d0) / p.group,
                            ho * 2 - s.pad, img, pol_x);
            }
            if (!ok || *abort_flag) drain_fills(full_bar(0), STAGES, filled, fill_parity, limit);
        }
    }
    if (warp >= 1 && warp <= ISSUERS) {
        // ------------------------------------------------------------ MMA issuers
        // (warps 2 and 3 first help with the weight expansion below)
        if (warp >= 2) expand_block_weight(s, p, smem, warp, lane, bready_bar);
        if (lane == 0) {
            constexpr uint32_t IDESC = make_idesc(BM, 64, 0);
            const int me = warp - 1;
            const uint32_t drain_bar = drain0 + 8u * me;
            bool ok = wait_or_abort(bready_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
            int issued = 0;
            if (p.inject_stall && me == 0) {
                // Failure injection: wait on a barrier nothing arrives on.
                wait_or_abort(drain_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
                ok = false;
            }
            tc_fence_after();
            const uint32_t b_lo0 = desc_lo(sbase + C::B_OFF);
            const int half = p.nsp / 2;
            // local tile k of this CTA is tile blockIdx.x + k * gridDim.x; this issuer's
            // tiles are k = me, me + ISSUERS, ...
            StageCursor cur(p.per);
            for (int k = me, tile = blockIdx.x + me * gridDim.x; ok && tile < p.num_tiles;
                 k += ISSUERS, tile += ISSUERS * gridDim.x) {
                int buf;
                uint32_t use;
                issuer_acc(k, buf, use);
                const int stage = cur.stage(me);  // this issuer's (k / ISSUERS)-th stage use
                const uint32_t phase = cur.phase;
                cur.next();
                if (!wait_or_abort(acce0 + 8u * buf, use ^ 1u, limit, abort_flag,
                                   STATUS_TIMEOUT_MMA) ||
                    !wait_or_abort(full_bar(stage), phase, limit, abort_flag,
                                   STATUS_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem_base + static_cast<uint32_t>(buf * 64);
                const uint32_t a_lo0 = desc_lo(sbase + stage * p.stage_bytes) + p.d0;
                const uint32_t box_lo = static_cast<uint32_t>(p.box_stride) >> 4;
                if constexpr (KH > 0) {
#pragma unroll
                    for (int ky = 0; ky < KH; ++ky)
#pragma unroll
                        for (int t = 0; t < NSP / 2; ++t) {
                            const int c = ky * (NSP / 2) + t;
                            umma_f16_w(d, a_lo0 + ky * box_lo + 2 * t, C::A_DESC_HI,
                                       b_lo0 + ((c * C::CHUNK_B) >> 4), C::B_DESC_HI, IDESC,
                                       c != 0 ? 1u : 0u);
                        }
                } else {
                    int c = 0;
                    for (int ky = 0; ky < s.kh; ++ky)
                        for (int t = 0; t < half; ++t, ++c)
                            umma_f16_w(d, a_lo0 + ky * box_lo + 2 * t, C::A_DESC_HI,
                                       b_lo0 + ((c * C::CHUNK_B) >> 4), C::B_DESC_HI, IDESC,
                                       c != 0 ? 1u : 0u);
                }
                ++issued;
                umma_commit(empty_bar(stage));
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
    } else if (warp >= EPI_WARP0) {
        expand_block_weight(s, p, smem, warp, lane, bready_bar);
        {
            // -------------------------------------------------------- epilogue
            const int segs = p.segs, Wo = s.Wo;
            auto geo = [segs, Wo](int tile) {
                EpiTile g;
                g.n_tile = 0;
                const int row = tile / segs, seg = tile - (tile / segs) * segs;
                g.m0 = static_cast<long long>(row) * Wo + seg * GA_TILE_W;
                const int left = Wo - seg * GA_TILE_W;
                g.rows = left < GA_TILE_W ? left : GA_TILE_W;
                return g;
            };
            epilogue_direct64<decltype(geo), EPI_GROUPS>(
                s, p.ep, p.y, tmem_base, accf0, acce0, p.num_tiles, limit, abort_flag, geo);
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
