// qconv_cg2.cuh -- weight-stationary quaternion convolution on CTA pairs (tcgen05
// cta_group::2) for 32 quaternion output channels (Cout = 128 real), the backbone's
// second stage.  Included by qconv_tc.cu inside its anonymous namespace.
//
// Why a pair.  An M = 128 MMA reads its A and B operands from shared memory at 128 bytes
// per clock, so with N = 64 (two output components of 32 channels, the pair decomposition
// of qconv_tc.cu) it costs the reads of 6 KB for 32 clocks of work; the whole signed block
// weight of Eq. 6 for 128 -> 128 real channels and 9 taps (288 KB) does not fit one CTA's
// shared memory, so N = 128 would have to re-expand letters on every tile.  A CTA pair
// runs M = 256 MMAs: each CTA holds the A operand of its own output pixels and HALF of
// the block weight (output components 0-1 in the even CTA, 2-3 in the odd one: at most
// 64 x 1152 bf16, 144 KB), expanded once per CTA and kept, and the tensor cores of the
// two SMs exchange the B halves.  One MMA is 256 x 128 x 16: per SM 4 KB of A and 2 KB of
// B for 64 clocks of work, so the operand reads leave room for the pixel stream.
//
//   A  pixels, K-major rows of 64 input channels (128 bytes, 128-byte swizzle), staged in
//      one of two ways:
//        halo  (stride 1, 3x3, Wp = Wo + 2 <= 128): a CTA tile is R = 128 / Wp output rows
//              of one image, and one TMA box per 64-channel chunk holds the R + 2 input rows
//              it reads at Wp columns -pad .. Wo + 1 - pad (zero fill outside the image),
//              row after row at a pitch of Wp pixels.  MMA row m = r Wp + c is output pixel
//              (r, c) (c >= Wo: padding, computed and not stored), and filter tap (dh, dw)
//              reads box row m + dh Wp + dw: every tap is the same box seen from another
//              start row.  The MMA applies the 128-byte swizzle to absolute shared-memory
//              addresses, as the TMA unit wrote it, so any 128-byte row offset is a valid
//              start (the descriptor's base-offset field stays 0).  One stage feeds
//              9 x 4 MMAs;
//        halo2 (stride 2, 3x3, Wp = Wo + 1 <= 128): the tile is R = 128 / Wp output rows
//              again, and a stage holds four boxes per 64-channel chunk, one per parity of
//              the input row and column (TMA element strides of 2): box (a, b) holds input
//              pixels (2 (h0 + i) - pad + a, 2 j - pad + b) for i = 0 .. R, j < Wp, at a row
//              pitch of Wp pixels.  Output pixel (r, c) reads input (2 r + dh - pad,
//              2 c + dw - pad), which is row (r + dh / 2) Wp + c + dw / 2 of box
//              (dh mod 2, dw mod 2), so tap (dh, dw) is again one box seen from a start row.
//              Each box starts on a 1024-byte boundary; a padding row past the end of a box
//              reads into the next box of the same stage (no box's MMAs reach past the
//              stage);
//        per tap  otherwise: one im2col box of 128 consecutive output pixels x 64 input
//              channels per (tap, chunk) stage (4 MMAs);
//   B  rows n = 32 q + co (real output channel c = q Qout + co = n), columns k = tap Cin +
//      p Qin + ci: B[n][k] = sign(q, p) W_{q xor p}[co][tap][ci]; the CTA of rank r keeps
//      rows 64 r .. 64 r + 63 as K-major 64-column chunks (128-byte swizzle);
//   D  TMEM of each CTA: its 128 MMA rows x the 128 output channels.
//
// The letters reach shared memory as four bulk copies (each letter tensor whole, into the
// space the pixel ring takes over afterwards) and are expanded shared -> shared: each
// 16-byte chunk of a letter is read once and written to its two places in this CTA's half
// (q = 2 r, 2 r + 1 with p = L xor q), with Eq. 5's sign.
//
// Roles.  Both CTAs: warp 0's lane 0 loads the letters, then the CTA's pixel boxes into a
// stage ring; warps 2..11 expand the CTA's B half; warps 4..11 are the direct epilogue of
// the CTA's 128 rows (tc_common.cuh's pair epilogue, with the per-channel vectors kept in
// registers, the residual read ahead of the accumulator, and the accumulator released to
// the even CTA).  Even CTA, per-tap staging: warps 1 and 2 (lane 0) issue the pair's MMAs
// for alternate pair tiles, each from its own share of the ring into its own two of four
// 128-column accumulators (a stage's four MMAs leave a single issuer's waits exposed);
// halo staging (either stride): warp 1 alone, through the whole ring (stages of 36 MMAs)
// and the four accumulators in order.  A stage is handed back to both producers and an accumulator to
// both epilogues by multicast commits.  Odd CTA: warp 1's lane 0 relays each of its landed
// stages to the even CTA's full barrier (a cluster-scope arrive), so the issuer waits on
// one barrier per stage.  Both CTAs allocate TMEM together (cta_group::2) and free it
// after a cluster barrier.  Every wait is bounded as in the other kernels.

constexpr int CG_THREADS = 384;
constexpr int CG_MAX_NI = 2;          // MMA issuers of the even CTA: 1 (halo) or 2 (per tap)
constexpr int CG_NACC = 4;            // accumulators of 128 columns
constexpr int CG_BUF_COLS = 128;
constexpr int CG_MAX_K = 1152;        // taps x Cin of the kept weight half (144 KB)
constexpr int CG_EXP_WARP0 = 2;       // warps 2..11 expand the B half
constexpr int CG_EXP_WARPS = 10;
constexpr int CG_EPI_THREADS = 256;   // warps 4..11
constexpr int CG_HALO_MAX_WP = 128;   // halo tiles: at least one padded output row per tile
// pixel staging of the kernel (its STG template argument)
constexpr int CG_PER_TAP = 0;
constexpr int CG_HALO = 1;            // stride 1: one box of R + 2 input rows per chunk
constexpr int CG_HALO2 = 2;           // stride 2: four parity boxes of R + 1 rows per chunk

struct Cg2Params {
    ConvShape s;
    EpilogueArgs ep;
    const __nv_bfloat16* w[4];  // letter tensors [32][kh][kw][Qin]
    void* y;                    // output [M][128]
    unsigned long long wait_limit_ns;
    int inject_stall;
    int kchunks;       // taps * Cin / 64: 64-column chunks of the kept weight half
    int cpt;           // Cin / 64: chunks per tap
    int nst;           // stages per tile: cpt (halo) or kchunks (per tap)
    int per;           // stages per issuer
    int stage_bytes;   // one stage of the pixel ring (a multiple of 1024)
    int box_bytes;     // bytes one stage's box delivers
    int letter_bytes;  // one letter tensor, 32 x taps x Qin bf16
    int num_tiles;     // CTA tiles
    int num_ptiles;    // pair tiles: two consecutive CTA tiles
    // halo staging
    int Wp;            // row pitch of a box, in pixels: Wo + 2 (stride 1) or Wo + 1 (stride 2)
    int R;             // output rows per tile: 128 / Wp
    int tpi;           // tiles per image: ceil(Ho / R)
    int box_stride;    // stride 2: bytes from one parity box of a stage to the next
};

struct CgCfg {
    static constexpr int BCHUNK = 64 * 128;   // 64 weight rows x 64 channels
    static constexpr int ACHUNK = 128 * 128;  // 128 pixels x 64 channels
    static constexpr int MAX_STAGES = 12;
    // full, empty (per stage), accf, acce (per accumulator), drain (per issuer), bready,
    // letters landed, letters read
    static constexpr int NUM_BARS = 2 * MAX_STAGES + 2 * CG_NACC + CG_MAX_NI + 3;
    static constexpr int SMEM_BYTES = 227 * 1024;
    static constexpr uint32_t DESC_HI = desc_hi(8 * 128, desc_layout(128));
    static constexpr uint32_t TMEM_COLS = 512;
    static_assert(NUM_BARS * 8 + 16 <= 1024, "pair barriers");
    // B half at 0 (kchunks x 8 KB), barriers in the next 1 KB, the stage ring after them
    __host__ __device__ static int ring_off(int kchunks) { return kchunks * BCHUNK + 1024; }
    static int ring_bytes(int kchunks) { return SMEM_BYTES - 1024 - ring_off(kchunks); }
};

// Shapes the kernel covers: the full form, 32 quaternion output channels, Cin a multiple of
// 64, taps x Cin <= 1152 (the four staged letters, 64 taps Cin bytes, then fit the ring).
bool cg2_ok(const ConvShape& s) {
    if (s.sep || s.Qout != 32 || s.Cin % 64 != 0) return false;
    return static_cast<long long>(s.kh) * s.kw * s.Cin <= CG_MAX_K;
}

// Halo staging: a 3x3 filter, stride 1 or 2, output rows narrow enough for one per tile.
bool cg2_halo_ok(const ConvShape& s) {
    return cg2_ok(s) && s.stride == 1 && s.kh == 3 && s.kw == 3 && s.Wo + 2 <= CG_HALO_MAX_WP;
}
bool cg2_halo2_ok(const ConvShape& s) {
    return cg2_ok(s) && s.stride == 2 && s.kh == 3 && s.kw == 3 && s.Wo + 1 <= CG_HALO_MAX_WP;
}

// This CTA's B half from the letters staged at `lsm` (letter L at L * letter_bytes, in the
// global layout [32][taps][Qin]): chunk i (16 bytes) of letter L holds
// W_L[co][tap][8 c8 .. 8 c8 + 7] with i = (co taps + tap) Qin / 8 + c8.  TAPS > 0: the tap
// count known at compile time and Qin / 8 a power of two (1 << cpr_log2), so the chunk
// index splits without run-time divisions.
template <int TAPS>
__device__ __forceinline__ void cg2_expand(const Cg2Params& p, uint32_t sbase, uint32_t lsm,
                                           uint32_t rank, int et, int cpr_log2) {
    constexpr int ET = CG_EXP_WARPS * 32;
    const ConvShape& s = p.s;
    const int Qin = s.Qin, taps = TAPS > 0 ? TAPS : s.kh * s.kw;
    const int cpr = Qin >> 3;  // chunks per (co, tap)
    const int per_letter = 32 * taps * cpr;
    const int total = 4 * per_letter;
    for (int i = et; i < total; i += ET) {
        int L, co, tap, c8;
        if constexpr (TAPS > 0) {
            const int j = i >> cpr_log2;  // (32 L + co) TAPS + tap
            c8 = i - (j << cpr_log2);
            const int lc = j / TAPS;
            tap = j - lc * TAPS;
            L = lc >> 5;
            co = lc & 31;
        } else {
            L = i / per_letter;
            const int off = i - L * per_letter;
            const int ct = off / cpr;
            c8 = off - ct * cpr;
            co = ct / taps;
            tap = ct - co * taps;
        }
        const uint4 v = lds_u4(lsm + static_cast<uint32_t>(i) * 16u);
#pragma unroll
        for (int b = 0; b < 2; ++b) {
            const int q = 2 * static_cast<int>(rank) + b, pc = L ^ q;
            const uint4 u = ((NEG_MASK >> (4 * q + pc)) & 1u) ? negate_bf16x8(v) : v;
            const int nl = 32 * b + co;
            const int k = tap * s.Cin + pc * Qin + 8 * c8;
            const int kc = k >> 6, uu = (k >> 3) & 7;
            sts_u4(sbase + static_cast<uint32_t>(kc * CgCfg::BCHUNK + nl * 128 +
                                                 ((uu ^ (nl & 7)) << 4)),
                   u);
        }
    }
}

// Bounded wait with cluster-scope acquire (arrivals from the peer CTA); otherwise as
// wait_or_abort.
__device__ __forceinline__ bool wait_cluster_or_abort(uint32_t bar, uint32_t parity,
                                                      uint64_t limit, volatile int* abort_flag,
                                                      unsigned code) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    while (true) {
        if (mbar_try_wait_sleep(bar, parity, WAIT_SUSPEND_NS) &&
            mbar_try_wait_cluster(bar, parity))
            return true;
        if (*abort_flag) return false;
        if (global_timer_ns() - t0 > limit) {
            atomicOr(&g_status, code);
            *abort_flag = 1;
            return false;
        }
    }
}

// One expansion warp: wait for the staged letters, expand this CTA's share, make the stores
// visible to the tensor cores, then tell the producer (the letters may be overwritten) and
// the even CTA's issuers (this part of the B half is ready).
template <int STG>
__device__ __forceinline__ void cg2_expand_warp(const Cg2Params& p, uint32_t sbase,
                                                uint32_t ring, uint32_t rank, int warp,
                                                int lane, uint32_t lbar, uint32_t lfree,
                                                uint32_t bready_bar, uint64_t limit,
                                                volatile int* abort_flag) {
    const int et = (warp - CG_EXP_WARP0) * 32 + lane;
    if (wait_or_abort(lbar, 0, limit, abort_flag, STATUS_TIMEOUT_EPILOGUE)) {
        if constexpr (STG != CG_PER_TAP)
            cg2_expand<9>(p, sbase, ring, rank, et, 31 - __clz(p.s.Qin >> 3));
        else
            cg2_expand<0>(p, sbase, ring, rank, et, 0);
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
        mbar_arrive(lfree);
        mbar_arrive_cluster(mapa_shared(bready_bar, 0));
    }
}

// Accumulator buffer and its use count for local pair tile k: with two issuers, issuer
// k mod 2 alternates between its own two buffers; with one, the four buffers in turn.
template <int NI>
__device__ __forceinline__ void cg2_acc(int k, int& buf, uint32_t& use) {
    if constexpr (NI == 1) {
        buf = k & 3;
        use = static_cast<uint32_t>(k >> 2) & 1u;
    } else {
        issuer_acc_n<NI>(k, buf, use);
    }
}

// STG: the pixel staging (CG_PER_TAP, CG_HALO or CG_HALO2).  NI: MMA issuers (one for
// halo staging, whose stages carry 36 MMAs each and are consumed in order from one ring;
// two for per-tap staging, whose four-MMA stages would leave a single issuer's waits
// exposed).
template <int STG, int NI>
__global__ void __launch_bounds__(CG_THREADS, 1)
    qconv_cg2_kernel(const __grid_constant__ CUtensorMap tmap_x, const Cg2Params p) {
    using C = CgCfg;
    constexpr bool HALO = STG != CG_PER_TAP;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);
    const int bar_off = p.kchunks * C::BCHUNK;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + bar_off);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::NUM_BARS);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int st) { return bar0 + 8u * st; };
    auto empty_bar = [&](int st) { return bar0 + 8u * (C::MAX_STAGES + st); };
    const uint32_t accf0 = bar0 + 8u * (2 * C::MAX_STAGES);
    const uint32_t acce0 = accf0 + 8u * CG_NACC;
    const uint32_t drain0 = acce0 + 8u * CG_NACC;
    const uint32_t bready_bar = drain0 + 8u * CG_MAX_NI;
    const uint32_t lbar = bready_bar + 8u;  // the four letter copies have landed
    const uint32_t lfree = lbar + 8u;       // every expansion warp has read the letters
    const uint32_t ring = sbase + static_cast<uint32_t>(C::ring_off(p.kchunks));

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const ConvShape& s = p.s;
    const uint64_t limit = p.wait_limit_ns;
    const uint32_t rank = cluster_ctarank();  // 0: the even CTA, which issues the MMAs
    const int STAGES = NI * p.per;
    const int pair = static_cast<int>(blockIdx.x) >> 1;
    const int npairs = static_cast<int>(gridDim.x) >> 1;
    // this pair's tiles: pair + k npairs, k < kt; the CTA's own tile is 2 (that) + rank
    const int kt = pair < p.num_ptiles ? (p.num_ptiles - pair + npairs - 1) / npairs : 0;

    griddep_launch_dependents();
    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            // even CTA: its own fill (expect_tx) and the odd CTA's relay; odd CTA: its fill
            mbar_init(full_bar(i), rank == 0 ? 2 : 1);
            mbar_init(empty_bar(i), 1);  // the even CTA's multicast commit
        }
        for (int b = 0; b < CG_NACC; ++b) {
            mbar_init(accf0 + 8u * b, 1);                   // multicast commit
            mbar_init(acce0 + 8u * b, 2 * CG_EPI_THREADS);  // both CTAs' epilogues (even CTA)
        }
        for (int i = 0; i < NI; ++i) mbar_init(drain0 + 8u * i, 1);
        mbar_init(bready_bar, 2 * CG_EXP_WARPS);  // both CTAs' expansions (even CTA)
        mbar_init(lbar, 1);
        mbar_init(lfree, CG_EXP_WARPS);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) tma_prefetch_desc(&tmap_x);
    if (warp == 1) {
        tmem_alloc_cg2(smem_u32(tmem_slot), C::TMEM_COLS);
        tmem_relinquish_cg2();
    }
    tc_fence_before();
    __syncthreads();
    // both CTAs' barriers exist before any cluster arrive or multicast commit reaches them
    cluster_sync_all();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    // The letters are staged and expanded before the dependency wait, overlapping the
    // previous kernel's last CTAs; every thread that touches activations (the pixel
    // producer, the epilogue) waits for that kernel before its first access.

    // CTA tile of local pair tile k
    auto cta_tile = [&](int k) { return 2 * (pair + k * npairs) + static_cast<int>(rank); };
    // image, first input row and first input column a tile reads (an odd CTA past the last
    // tile loads the last one and stores nothing)
    auto tile_origin = [&](int k, int& img, int& hbase, int& wbase) {
        if constexpr (HALO) {
            int t = cta_tile(k);
            if (t >= p.num_tiles) t = p.num_tiles - 1;
            img = t / p.tpi;
            hbase = (t - img * p.tpi) * p.R * s.stride - s.pad;
            wbase = -s.pad;
        } else {
            const int hw = s.Ho * s.Wo;
            const long long last = (s.M - 1) / BM * BM;
            long long m0 = static_cast<long long>(cta_tile(k)) * BM;
            if (m0 > last) m0 = last;
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
            // the letters into the ring's space; the pixels once the letters have been read
            mbar_arrive_expect_tx(lbar, 4u * static_cast<uint32_t>(p.letter_bytes));
            for (int l = 0; l < 4; ++l)
                bulk_load(ring + static_cast<uint32_t>(l * p.letter_bytes), p.w[l],
                          static_cast<uint32_t>(p.letter_bytes), lbar);
            bool ok = wait_or_abort(lfree, 0, limit, abort_flag, STATUS_TIMEOUT_PRODUCER);
            griddep_wait();  // the previous kernel's output (this layer's input) is complete
            StageCursor cur(p.per);
            for (int g0 = 0; ok && g0 < kt; g0 += NI) {
                const int ng = kt - g0 < NI ? kt - g0 : NI;
                int img[NI], hbase[NI], wbase[NI];
#pragma unroll
                for (int i = 0; i < NI; ++i)
                    if (i < ng) tile_origin(g0 + i, img[i], hbase[i], wbase[i]);
                int ch = 0, dh = 0, dw = 0;  // per tap: stage kc = (tap, ch), no divisions
                for (int kc = 0; ok && kc < p.nst; ++kc, cur.next()) {
                    if constexpr (HALO) {
                        ch = kc;
                    } else if (kc > 0 && ++ch == p.cpt) {
                        ch = 0;
                        if (++dw == s.kw) {
                            dw = 0;
                            ++dh;
                        }
                    }
#pragma unroll
                    for (int i = 0; i < NI; ++i) {
                        if (i >= ng) break;
                        const int stage = cur.stage(i);
                        const uint32_t phase = cur.phase;
                        if (!wait_cluster_or_abort(empty_bar(stage), phase ^ 1u, limit,
                                                   abort_flag, STATUS_TIMEOUT_PRODUCER)) {
                            ok = false;
                            break;
                        }
                        const uint32_t fb = full_bar(stage);
                        const uint32_t dst = ring + static_cast<uint32_t>(stage * p.stage_bytes);
                        mbar_arrive_expect_tx(fb, static_cast<uint32_t>(p.box_bytes));
                        filled |= 1u << stage;
                        fill_parity = (fill_parity & ~(1u << stage)) | (phase << stage);
                        if constexpr (STG == CG_HALO2) {
                            // the four parity boxes (row parity a, column parity b) at
                            // 2 a + b box strides
#pragma unroll
                            for (int ab = 0; ab < 4; ++ab)
                                tma_load_4d(dst + static_cast<uint32_t>(ab * p.box_stride),
                                            &tmap_x, fb, 64 * ch, wbase[i] + (ab & 1),
                                            hbase[i] + (ab >> 1), img[i], pol_x);
                        } else if constexpr (HALO) {
                            tma_load_4d(dst, &tmap_x, fb, 64 * ch, wbase[i], hbase[i], img[i],
                                        pol_x);
                        } else {
                            tma_load_im2col_4d(dst, &tmap_x, fb, 64 * ch, wbase[i], hbase[i],
                                               img[i], static_cast<uint16_t>(dw),
                                               static_cast<uint16_t>(dh), pol_x);
                        }
                    }
                }
            }
            if (!ok || *abort_flag) {
                drain_fills(full_bar(0), STAGES, filled, fill_parity, limit);
                drain_fills(lbar, 1, 1u, 0u, limit);  // the letter copies, if still landing
            }
        }
    } else if (warp <= CG_MAX_NI) {
        if (warp >= CG_EXP_WARP0)
            cg2_expand_warp<STG>(p, sbase, ring, rank, warp, lane, lbar, lfree, bready_bar,
                                 limit, abort_flag);
        if (rank == 0 && lane == 0 && warp <= NI) {
            // -------------------------------------------------- MMA issuers (even CTA)
            constexpr uint32_t IDESC = make_idesc(2 * BM, 128, 0);
            const int me = warp - 1;
            const uint32_t drain_bar = drain0 + 8u * me;
            bool ok = wait_cluster_or_abort(bready_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
            int issued = 0;
            if (p.inject_stall && me == 0) {
                // Failure injection: wait on a barrier nothing arrives on.
                wait_or_abort(drain_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
                ok = false;
            }
            tc_fence_after();
            const uint32_t b_lo0 = desc_lo(sbase);
            // halo: descriptor offset (16-byte units) of one box row of Wp pixels, and
            // (stride 2) of one parity box
            const uint32_t row1 = static_cast<uint32_t>(p.Wp * 8);
            const uint32_t box1 = static_cast<uint32_t>(p.box_stride >> 4);
            StageCursor cur(p.per);
            for (int k = me; ok && k < kt; k += NI) {
                int buf;
                uint32_t use;
                cg2_acc<NI>(k, buf, use);
                if (!wait_cluster_or_abort(acce0 + 8u * buf, use ^ 1u, limit, abort_flag,
                                           STATUS_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem_base + static_cast<uint32_t>(buf * CG_BUF_COLS);
                for (int kc = 0; kc < p.nst; ++kc) {
                    const int stage = cur.stage(me);
                    const uint32_t phase = cur.phase;
                    cur.next();
                    if (!wait_cluster_or_abort(full_bar(stage), phase, limit, abort_flag,
                                               STATUS_TIMEOUT_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a_lo =
                        desc_lo(ring + static_cast<uint32_t>(stage * p.stage_bytes));
                    if constexpr (HALO) {
                        // stage kc holds input channels 64 kc .. 64 kc + 63; tap (dh, dw)
                        // starts dh Wp + dw rows into the box (stride 1), or
                        // (dh / 2) Wp + dw / 2 rows into parity box (dh mod 2, dw mod 2)
                        // (stride 2), and uses weight chunk tap cpt + kc
#pragma unroll
                        for (int t = 0; t < 9; ++t) {
                            const int dh = t / 3, dw = t % 3;
                            uint32_t a_t;
                            if constexpr (STG == CG_HALO2)
                                a_t = a_lo + static_cast<uint32_t>(2 * (dh & 1) + (dw & 1)) * box1 +
                                      static_cast<uint32_t>(dh >> 1) * row1 +
                                      static_cast<uint32_t>((dw >> 1) * 8);
                            else
                                a_t = a_lo + static_cast<uint32_t>(dh) * row1 +
                                      static_cast<uint32_t>(dw * 8);
                            const uint32_t b_t =
                                b_lo0 + static_cast<uint32_t>(((t * p.cpt + kc) * C::BCHUNK) >> 4);
#pragma unroll
                            for (int kk = 0; kk < 4; ++kk)  // 16 channels: 32 bytes into a row
                                umma_f16_cg2(d, a_t + 2 * kk, C::DESC_HI, b_t + 2 * kk,
                                             C::DESC_HI, IDESC, (kc | t | kk) != 0 ? 1u : 0u);
                        }
                    } else {
                        const uint32_t b_lo =
                            b_lo0 + static_cast<uint32_t>((kc * C::BCHUNK) >> 4);
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk)
                            umma_f16_cg2(d, a_lo + 2 * kk, C::DESC_HI, b_lo + 2 * kk,
                                         C::DESC_HI, IDESC, (kc | kk) != 0 ? 1u : 0u);
                    }
                    ++issued;
                    umma_commit_cg2(empty_bar(stage), 3);  // both CTAs may refill the stage
                }
                if (!ok) break;
                umma_commit_cg2(accf0 + 8u * buf, 3);  // both CTAs' accumulators are ready
            }
            if (!ok && issued > 0) {
                // let this issuer's MMAs finish before TMEM is released
                umma_commit_cg2(drain_bar, 1);
                const uint64_t t0 = global_timer_ns();
                while (!mbar_try_wait(drain_bar, 0u)) {
                    if (global_timer_ns() - t0 > limit) {
                        atomicOr(&g_status, STATUS_TIMEOUT_DRAIN);
                        break;
                    }
                }
            }
        } else if (rank == 1 && warp == 1 && lane == 0) {
            // ---------------------------------- relay of the odd CTA's landed stages
            const uint32_t full_leader0 = mapa_shared(full_bar(0), 0);
            StageCursor cur(p.per);
            bool ok = true;
            for (int g0 = 0; ok && g0 < kt; g0 += NI) {
                const int ng = kt - g0 < NI ? kt - g0 : NI;
                for (int kc = 0; ok && kc < p.nst; ++kc, cur.next()) {
                    for (int i = 0; i < ng; ++i) {
                        const int stage = cur.stage(i);
                        if (!wait_or_abort(full_bar(stage), cur.phase, limit, abort_flag,
                                           STATUS_TIMEOUT_PRODUCER)) {
                            ok = false;
                            break;
                        }
                        mbar_arrive_cluster(full_leader0 + 8u * stage);
                    }
                }
            }
        }
    } else {
        cg2_expand_warp<STG>(p, sbase, ring, rank, warp, lane, lbar, lfree, bready_bar, limit,
                             abort_flag);
        griddep_wait();  // the residual complete, the output buffer no longer read
        if (warp >= EPI_WARP0) {
            // ------------------------------------------------------------ epilogue
            // (the pair epilogue of tc_common.cuh for 32 channels per component: warps 4..7
            // take components r and i, warps 8..11 j and k; the accumulator is released to
            // the even CTA, whose issuer refills it)
            constexpr int BNQ = 32, CH = 32, NCH = 4, NB = 2;
            const int quad = warp & 3;
            const int half = (warp - EPI_WARP0) >> 2;
            const int ci = lane % NCH;
            const int row0 = quad * 32 + NCH * (lane / NCH);
            const long long Cout = s.Cout;
            const __nv_bfloat16* res = static_cast<const __nv_bfloat16*>(p.ep.residual);
            __nv_bfloat16* out = static_cast<__nv_bfloat16*>(p.y);
            const uint32_t acce_leader0 = mapa_shared(acce0, 0);
            // the thread's MMA rows row0 + kq as output pixels of a tile: offset from the
            // tile's first pixel, row within the tile, and whether the row is an output
            int pix[NCH], prow[NCH];
            bool pval[NCH];
#pragma unroll
            for (int kq = 0; kq < NCH; ++kq) {
                const int m = row0 + kq;
                if constexpr (HALO) {
                    const int r = m / p.Wp, c = m - r * p.Wp;
                    pix[kq] = r * s.Wo + c;
                    prow[kq] = r;
                    pval[kq] = c < s.Wo && r < p.R;
                } else {
                    pix[kq] = m;
                    prow[kq] = m;
                    pval[kq] = true;
                }
            }
            // the per-channel vectors of the thread's two channel blocks (components
            // 2 half + b, channels 8 ci .. 8 ci + 7), for the whole run
            float sc[2][8], sh[2][8];
#pragma unroll
            for (int b = 0; b < NB; ++b) {
                const int cb = 8 * ci + (2 * half + b) * s.Qout;
                float bi[8];
                load8(p.ep.scale, cb, 1.0f, sc[b]);
                load8(p.ep.shift, cb, 0.0f, sh[b]);
                load8(p.ep.bias, cb, 0.0f, bi);
#pragma unroll
                for (int e = 0; e < 8; ++e) sh[b][e] = fmaf(sc[b][e], bi[e], sh[b][e]);
            }
            for (int k = 0; k < kt; ++k) {
                int buf;
                uint32_t use;
                cg2_acc<NI>(k, buf, use);
                // the tile's first output pixel and how many of its rows exist (known before
                // the accumulator is: the residual of block 0 is read while it is computed)
                const int t = cta_tile(k);
                long long base;
                int lim;
                if constexpr (HALO) {
                    const int img = t / p.tpi, h0 = (t - img * p.tpi) * p.R;
                    base = (static_cast<long long>(img) * s.Ho + h0) * s.Wo;
                    lim = t < p.num_tiles ? s.Ho - h0 : 0;
                } else {
                    base = static_cast<long long>(t) * BM;
                    const long long left = s.M - base;
                    lim = left <= 0 ? 0 : (left < BM ? static_cast<int>(left) : BM);
                }
                bool st[NCH];
#pragma unroll
                for (int kq = 0; kq < NCH; ++kq) st[kq] = pval[kq] && prow[kq] < lim;
                uint4 r4[NB][NCH];
                auto load_res = [&](int b) {
                    const int cb = 8 * ci + (2 * half + b) * s.Qout;
#pragma unroll
                    for (int kq = 0; kq < NCH; ++kq) {
                        r4[b][kq] = make_uint4(0u, 0u, 0u, 0u);
                        if (st[kq]) r4[b][kq] = ld_global_na(res + (base + pix[kq]) * Cout + cb);
                    }
                };
                if (res != nullptr) load_res(0);
                bool ok = true;
                if (lane == 0)
                    ok = wait_cluster_or_abort(accf0 + 8u * buf, use, limit, abort_flag,
                                               STATUS_TIMEOUT_EPILOGUE);
                ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
                if (named_bar_or(1, CG_EPI_THREADS, !ok)) break;
                tc_fence_after();
                const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                                       static_cast<uint32_t>(buf * CG_BUF_COLS);
                uint32_t va[CH], vb[CH];
                tmem_ld_32x32b_x32(taddr + (2 * half) * BNQ, va);
                tmem_ld_wait();
#pragma unroll
                for (int b = 0; b < NB; ++b) {
                    uint32_t(&v)[CH] = b ? vb : va;
                    const int q = 2 * half + b;
                    const int cb = 8 * ci + q * s.Qout;
                    if (b == 0) {
                        tmem_ld_32x32b_x32(taddr + (2 * half + 1) * BNQ, vb);
                        if (res != nullptr) load_res(1);
                    } else {
                        // the tile's accumulator is in registers: hand it back
                        tc_fence_before();
                        mbar_arrive_cluster_relaxed(acce_leader0 + 8u * buf);
                    }
                    float E[NCH][8];
#pragma unroll
                    for (int j = 0; j < NCH; ++j)
#pragma unroll
                        for (int e = 0; e < 8; ++e) E[j][e] = __uint_as_float(v[8 * j + e]);
                    chunk_transpose_stage<2, 4>(E, ci);
                    chunk_transpose_stage<1, 4>(E, ci);
#pragma unroll
                    for (int kq = 0; kq < NCH; ++kq) {
                        float rz[8];
                        if (res != nullptr) {
                            const __nv_bfloat162* rh =
                                reinterpret_cast<const __nv_bfloat162*>(&r4[b][kq]);
#pragma unroll
                            for (int t2 = 0; t2 < 4; ++t2) {
                                const float2 f = __bfloat1622float2(rh[t2]);
                                rz[2 * t2] = f.x;
                                rz[2 * t2 + 1] = f.y;
                            }
                        } else {
#pragma unroll
                            for (int e = 0; e < 8; ++e) rz[e] = 0.0f;
                        }
                        uint32_t wv[4];
#pragma unroll
                        for (int t2 = 0; t2 < 4; ++t2) {
                            const float z0 = fmaf(sc[b][2 * t2], E[kq][2 * t2], sh[b][2 * t2]) +
                                             rz[2 * t2];
                            const float z1 =
                                fmaf(sc[b][2 * t2 + 1], E[kq][2 * t2 + 1], sh[b][2 * t2 + 1]) +
                                rz[2 * t2 + 1];
                            wv[t2] = pack_bf16x2(activate(z0, s.act), activate(z1, s.act));
                        }
                        if (st[kq])
                            st_global_na(out + (base + pix[kq]) * Cout + cb,
                                         make_uint4(wv[0], wv[1], wv[2], wv[3]));
                    }
                    if (b == 0) tmem_ld_wait();
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    // the pair's MMAs into both CTAs' TMEM and both epilogues are done
    cluster_sync_all();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc_cg2(tmem_base, C::TMEM_COLS);
    }
}
