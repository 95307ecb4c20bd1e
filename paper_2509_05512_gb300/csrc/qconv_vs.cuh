// qconv_vs.cuh -- 3x3 stride-1 quaternion convolution with 16 quaternion channels in and out
// (64 real), the three vertical filter taps stacked along the MMA's N dimension.  Included
// by qconv_tc.cu inside its anonymous namespace.
//
// Why.  With 128 output pixels as an MMA's M rows and the 64 output channels as its N, one
// MMA of N = 64 reads 4 KB of pixels and 2 KB of weight from shared memory for 32 clocks of
// tensor work; at 128 bytes per clock those reads take 48 clocks, which caps such a kernel
// (qconv_ws.cuh) near 65% of the tensor peak.  Here one MMA multiplies 128 pixels of ONE
// INPUT ROW by the signed block weights (Eq. 6) of all three vertical taps dh of one
// horizontal tap dw: N = 192, 4 KB + 6 KB read for 96 clocks of work.  Its three 64-column
// results belong to three different output rows, since input row i meets filter row dh in
// output row i + pad - dh.  The accumulator therefore holds a band of up to four
// consecutive output rows side by side: output row j of the band (j = 0 .. 3) at TMEM
// columns 64 (3 - j) .. 64 (3 - j) + 63.  Input row t of the band (t = 0 .. r + 1, input
// row h0 - pad + t) adds to output rows t, t - 1, t - 2 through dh = 0, 1, 2, which are
// three adjacent column blocks in increasing dh order: one MMA whose B operand is the
// weight of taps (dh = 0, 1, 2; dw) stored one after the other.  Input rows at a band's
// edges meet fewer of its rows and use N = 64 or 128.  For a band of r = 4 rows a
// (dw, 16-channel) step costs 2 x 49 + 2 x 64 + 2 x 96 clocks for 4 x 3 x 32 clocks of
// work (92%).  The first MMA of an input row overwrites the output rows it is the first to
// reach (accumulate flag off) and adds to the others in a second MMA.
//
// Lanes (MMA rows).  A tile row of 128 lanes holds E images side by side, P lanes each:
// lane l = e P + c is image n0 + e, output column c (c >= Wo: padding, computed and not
// stored).  Two stagings of one input row of the E images:
//   one box    P = Wo + 2: a TMA box of the E images' input columns -pad .. P - 1 - pad; the
//              horizontal tap dw reads it from box row dw on (a 128-byte row offset of the A
//              descriptor: the tensor cores apply the 128-byte swizzle to absolute
//              shared-memory addresses, as the TMA unit wrote it), rows past the box being
//              padding lanes' garbage;
//   three boxes  P = Wo, 128 / Wo images (Wo dividing 128, when that fits more images): one
//              box per dw of the input columns dw - pad .. dw - pad + Wo - 1.
// Zero padding comes from the TMA unit's out-of-bounds fill; input rows outside the image
// are neither loaded nor multiplied.
//
// Work unit: a band of bh (<= 4) output rows of one group of E images; CTAs take units round
// robin.  A band of four rows stages all six input rows (rows outside the image as the TMA
// unit's zero boxes) and its MMA stream is unrolled at compile time, so the issuing thread
// does no integer work between MMAs (the tensor pipe queues almost nothing: a 75-instruction
// loop body between MMAs costs more than the MMAs); a partial band (the last of an image
// when bh does not divide Ho, or bh < 4) skips rows outside the image and is issued with
// run-time row parameters.  Roles (20 warps):
//   warps 0,2,3  TMA producers (lane 0 of each), through a ring of up to 12 stages of three
//                input rows (one box: each producer loads one of a stage's rows) or one
//                (three boxes: each loads one dw box), so the issuer waits once per 36 or
//                12 MMAs and the loads of a stage are issued by three threads at once;
//   warp 1       owns TMEM (two band buffers of 256 columns); lane 0 issues the MMAs, unit
//                after unit, into alternate buffers;
//   warps 4..19  expand the signed block weight once per CTA (72 KB, tap order (dw, dh)),
//                then drain the buffers: group g = (warp - 4) / 4 takes output row g of
//                each band, one warp per TMEM lane quadrant, in blocks of 16 columns (a 2 x 2
//                chunk transpose across lane pairs by shuffles, IQBN, activation, 16-byte
//                stores); the next block's TMEM load and residual are requested before a
//                block is processed, the first block's residual during the wait for the
//                accumulator, the next unit's residual lines are prefetched into L2, and the
//                per-channel vectors sit in shared memory (512 bytes, broadcast reads).
// Every wait is bounded; a wait that runs out sets a status bit and the CTA's abort flag,
// and the roles drain their copies and MMAs before TMEM is freed.

constexpr int VS_THREADS = 640;      // 20 warps
constexpr int VS_BH = 4;             // output rows per band buffer
constexpr int VS_BUF_COLS = VS_BH * 64;
constexpr int VS_MAX_STAGES = 12;
constexpr int VS_EPI_WARP0 = 4;      // warps 4..19: expansion, then the epilogue
constexpr int VS_EPI_THREADS = 512;
constexpr int VS_TAP_BYTES = 64 * 128;  // expanded weight of one tap: 64 rows x 64 channels
constexpr int VS_PRODUCERS = 3;      // TMA-issuing threads: lane 0 of warps 0, 2, 3

struct VsParams {
    ConvShape s;
    EpilogueArgs ep;
    const __nv_bfloat16* w[4];  // compact letter tensors [16][3][3][16]
    void* y;                    // output [N][Ho][Wo][64]
    unsigned long long wait_limit_ns;
    int inject_stall;
    int P;            // lanes per image
    int E;            // images per tile row
    int box_bytes;    // one box: E x P x 128
    int row_bytes;    // one input row's boxes (NBOX of them), rounded up to 1024
    int stage_bytes;  // rows per stage x row_bytes
    int nst;          // stages in the ring
    int bh;           // output rows per band (1 .. 4)
    int nbands;       // bands per image group: ceil(Ho / bh)
    int num_units;    // ceil(N / E) * nbands
};

struct VsCfg {
    static constexpr int SMEM_BYTES = 227 * 1024;
    static constexpr int RING_BYTES = 153 * 1024;  // ring of pixel stages at offset 0
    static constexpr int WSB_OFF = RING_BYTES;     // then the expanded weight (9 taps)
    static constexpr int WSB_BYTES = 9 * VS_TAP_BYTES;
    static constexpr int BAR_OFF = WSB_OFF + WSB_BYTES;
    // full, empty (per stage), accf, acce (per buffer), weight ready, drain
    static constexpr int NUM_BARS = 2 * VS_MAX_STAGES + 4 + 2;
    // the epilogue's per-channel vectors: scale[64], then scale * bias + shift[64] (fp32)
    static constexpr int VEC_OFF = BAR_OFF + 256;
    static constexpr uint32_t DESC_HI = desc_hi(8 * 128, desc_layout(128));
    static constexpr uint32_t TMEM_COLS = 2 * VS_BUF_COLS;
    static_assert(NUM_BARS * 8 + 16 <= 256, "VS barriers");
    static_assert(VEC_OFF + 512 + 1024 <= SMEM_BYTES, "VS shared memory");
};

// Lane layout of a shape's tile rows: false if neither staging fits 128 lanes.
bool vs_layout(int Wo, int* nbox, int* E, int* P) {
    const int e1 = Wo + 2 <= BM ? BM / (Wo + 2) : 0;
    const int e3 = (Wo <= BM && BM % Wo == 0) ? BM / Wo : 0;
    if (e3 > e1) {
        *nbox = 3; *E = e3; *P = Wo;
        return true;
    }
    if (e1 > 0) {
        *nbox = 1; *E = e1; *P = Wo + 2;
        return true;
    }
    return false;
}

bool vs_ok(const ConvShape& s) {
    int nbox, E, P;
    return s.Qin == 16 && s.Qout == 16 && s.kh == 3 && s.kw == 3 && s.stride == 1 &&
           s.pad <= 2 && vs_layout(s.Wo, &nbox, &E, &P);
}

// MMA clocks of one (dw, 16-channel) step over a band of r rows: N = 64 n costs about
// 49, 64, 96 clocks for n = 1, 2, 3 (operand reads vs. tensor work).
int vs_band_cost(int r) {
    static const int c[4] = {0, 49, 64, 96};
    int sum = 0;
    for (int t = 0; t <= r + 1; ++t) {
        const int lo = t - r + 1 > 0 ? t - r + 1 : 0, hi = t < 2 ? t : 2;
        sum += c[hi - lo + 1];
    }
    return sum;
}

// Band height with the least estimated time: waves of units x the band's MMA clocks.
int vs_pick_bh(const ConvShape& s, int E, int grid) {
    const long long groups = (s.N + E - 1) / E;
    int best = VS_BH;
    long long best_t = -1;
    for (int bh = VS_BH; bh >= 1; --bh) {
        const long long units = groups * ((s.Ho + bh - 1) / bh);
        const long long waves = (units + grid - 1) / grid;
        const long long t = waves * vs_band_cost(bh);
        if (best_t < 0 || t < best_t) {
            best_t = t;
            best = bh;
        }
    }
    return best;
}

// The signed block weight, once per CTA, by the 512 threads of warps 4..19: for tap (dh, dw),
// row n = 16 q + co and K index 16 p + ci the value is sign(q, p) W_{q xor p}[co][dh][dw][ci]
// (SEP: the separable form of Eq. 7, row block m, column block p = sign(m, p) W_p), stored
// as rows of 128 bytes with the 128-byte swizzle, tap (dh, dw) at (3 dw + dh) x 8 KB so that
// the three vertical taps of one dw are 192 consecutive rows.  Each 16-byte chunk of a
// letter is read once (all of a thread's chunks in flight together) and written to its four
// places.
template <bool SEP>
__device__ __forceinline__ void vs_expand(const VsParams& p, uint8_t* wsb, int et) {
    constexpr int LC = 9 * 32;  // 16-byte chunks of one letter: 16 co x 9 taps x 2 halves
    constexpr int TOTAL = 4 * LC;
    constexpr int ROUNDS = (TOTAL + VS_EPI_THREADS - 1) / VS_EPI_THREADS;
    uint4 v[ROUNDS];
#pragma unroll
    for (int r = 0; r < ROUNDS; ++r) {
        const int i = et + r * VS_EPI_THREADS;
        if (i < TOTAL) {
            const int L = i / LC;
            v[r] = __ldg(reinterpret_cast<const uint4*>(p.w[L]) + (i - L * LC));
        }
    }
#pragma unroll
    for (int r = 0; r < ROUNDS; ++r) {
        const int i = et + r * VS_EPI_THREADS;
        if (i >= TOTAL) continue;
        const int L = i / LC, off = i - L * LC;
        // chunk `off` of letter L holds W_L[co][t][ci0 .. ci0 + 7], t = 3 dh + dw
        const int co = off / 18, rem = off - co * 18;
        const int t = rem >> 1, half_ci = rem & 1;
        const int dh = t / 3, dw = t - 3 * dh;
        const uint32_t signs = ((SEP ? SEP_LETTER_SIGNS : LETTER_SIGNS) >> (4 * L)) & 15u;
        uint8_t* row = wsb + (3 * dw + dh) * VS_TAP_BYTES + co * 128;
        const int sw = co & 7;  // the row's swizzle phase (16 q rows further keeps it)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int q = SEP ? j : L ^ j, ch = (SEP ? L : j) * 2 + half_ci;
            const uint4 u = ((signs >> j) & 1u) ? negate_bf16x8(v[r]) : v[r];
            *reinterpret_cast<uint4*>(row + q * 16 * 128 + ((ch ^ sw) << 4)) = u;
        }
    }
}

// The 12 MMAs (+ 1: the first one split) of one input row: NB output rows met (N = 64 NB),
// of which the first NNEW (the lowest dh, the newest rows) are reached for the first time
// and overwritten by the first MMA.  d: TMEM column of the row met through the lowest dh;
// a0: the row's pixel box (A descriptor, low word); b0: the weight of tap (lowest dh, dw = 0).
template <int NBOX, int NB, int NNEW>
__device__ __forceinline__ void vs_row_mmas(uint32_t d, uint32_t a0, uint32_t b0) {
    constexpr uint32_t IDESC0 = make_idesc(BM, 0, 0);
    constexpr uint32_t ID = IDESC0 | ((8u * NB) << 17);
    constexpr uint32_t TAP_LO = VS_TAP_BYTES >> 4;
    constexpr uint32_t A_DW = NBOX == 1 ? (128 >> 4) : ((BM * 128) >> 4);
    constexpr uint32_t HI = VsCfg::DESC_HI;
    if constexpr (NNEW > 0) {
        umma_f16_w(d, a0, HI, b0, HI, IDESC0 | ((8u * NNEW) << 17), 0u);
        if constexpr (NNEW < NB)
            umma_f16_w(d + 64u * NNEW, a0, HI, b0 + NNEW * TAP_LO, HI,
                       IDESC0 | ((8u * (NB - NNEW)) << 17), 1u);
    } else {
        umma_f16_w(d, a0, HI, b0, HI, ID, 1u);
    }
#pragma unroll
    for (int dw = 0; dw < 3; ++dw)
#pragma unroll
        for (int kc = 0; kc < 4; ++kc) {
            if (dw == 0 && kc == 0) continue;
            umma_f16_w(d, a0 + dw * A_DW + kc * 2, HI, b0 + dw * 3 * TAP_LO + kc * 2, HI, ID, 1u);
        }
}

// Input row t of a full band (VS_BH output rows, every input row t = 0 .. VS_BH + 1 staged,
// rows outside the image as zero boxes): everything but the addresses is known at compile
// time, so the issuing thread does no integer work between MMAs.
template <int NBOX, int T>
__device__ __forceinline__ void vs_full_row(uint32_t dbuf, uint32_t a0, uint32_t wsb_lo) {
    constexpr int lo = T - VS_BH + 1 > 0 ? T - VS_BH + 1 : 0;
    constexpr int hi = T < 2 ? T : 2;
    constexpr int jtop = T - lo;
    constexpr int nnew = T <= VS_BH - 1 ? 1 : 0;
    vs_row_mmas<NBOX, hi - lo + 1, nnew>(dbuf + 64u * (VS_BH - 1 - jtop), a0,
                                         wsb_lo + lo * (VS_TAP_BYTES >> 4));
}

// The same for a row of a partial band (run-time row parameters).
template <int NBOX>
__device__ __forceinline__ void vs_any_row(uint32_t d, uint32_t a0, uint32_t b0, int nb,
                                           int nnew) {
    switch (nb * 4 + nnew) {
        case 4: vs_row_mmas<NBOX, 1, 0>(d, a0, b0); break;
        case 5: vs_row_mmas<NBOX, 1, 1>(d, a0, b0); break;
        case 8: vs_row_mmas<NBOX, 2, 0>(d, a0, b0); break;
        case 9: vs_row_mmas<NBOX, 2, 1>(d, a0, b0); break;
        case 10: vs_row_mmas<NBOX, 2, 2>(d, a0, b0); break;
        case 12: vs_row_mmas<NBOX, 3, 0>(d, a0, b0); break;
        case 13: vs_row_mmas<NBOX, 3, 1>(d, a0, b0); break;
        case 14: vs_row_mmas<NBOX, 3, 2>(d, a0, b0); break;
        default: vs_row_mmas<NBOX, 3, 3>(d, a0, b0); break;
    }
}

template <int NBOX, bool SEP>
__global__ void __launch_bounds__(VS_THREADS, 1)
    qconv_vs_kernel(const __grid_constant__ CUtensorMap tmap_x, const VsParams p) {
    using C = VsCfg;
    static_assert(NBOX == 1 || NBOX == 3, "one box per input row, or one per dw");
    constexpr int RPS = NBOX == 1 ? 3 : 1;  // input rows per stage
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::BAR_OFF);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::NUM_BARS);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int i) { return bar0 + 8u * i; };
    auto empty_bar = [&](int i) { return bar0 + 8u * (VS_MAX_STAGES + i); };
    const uint32_t accf0 = bar0 + 8u * (2 * VS_MAX_STAGES);
    const uint32_t acce0 = accf0 + 16u;
    const uint32_t wready_bar = acce0 + 16u;
    const uint32_t drain_bar = wready_bar + 8u;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const ConvShape& s = p.s;
    const uint64_t limit = p.wait_limit_ns;
    const int nst = p.nst;

    griddep_launch_dependents();
    if (threadIdx.x == 0) {
        for (int i = 0; i < nst; ++i) {
            mbar_init(full_bar(i), VS_PRODUCERS);
            mbar_init(empty_bar(i), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(accf0 + 8u * b, 1);
            mbar_init(acce0 + 8u * b, VS_EPI_THREADS);
        }
        mbar_init(wready_bar, VS_EPI_THREADS / 32);
        mbar_init(drain_bar, 1);
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
    // The block weight is expanded before the dependency wait, overlapping the previous
    // kernel's last CTAs; the producers and the epilogue wait for that kernel before their
    // first access to activations.

    // unit u: image group u / nbands, band u % nbands
    auto unit_geo = [&](int u, int& n0, int& h0, int& r) {
        const int g = u / p.nbands;
        const int band = u - g * p.nbands;
        n0 = g * p.E;
        h0 = band * p.bh;
        r = s.Ho - h0 < p.bh ? s.Ho - h0 : p.bh;
    };
    // input row t of a unit is staged (and multiplied) when its band is full (rows outside
    // the image then come as zero boxes) or when it lies inside the image
    auto row_staged = [&](int h0, int r, int t) {
        const int i = h0 - s.pad + t;
        return r == VS_BH || (i >= 0 && i < s.H);
    };
    const int pid = warp == 0 ? 0 : warp - 1;  // producer index (warps 0, 2, 3)

    if ((warp == 0 || warp == 2 || warp == 3) && lane == 0) {
        // ------------------------------------------------------------ TMA producers
        const uint64_t pol = l2_policy_evict_normal();
        uint32_t filled = 0, fill_parity = 0;
        int idx = 0;
        uint32_t phase = 0;
        bool ok = true;
        // three boxes: producer pid loads box dw = pid of every row; one box: producer pid loads
        // row pid of every stage (the TMA unit takes several threads' copies at once)
        const int x0 = (NBOX == 3 ? pid : 0) - s.pad;
        griddep_wait();  // the previous kernel's output (this layer's input) is complete
        for (int u = blockIdx.x; ok && u < p.num_units; u += gridDim.x) {
            int n0, h0, r;
            unit_geo(u, n0, h0, r);
            int q = 0;  // rows placed in the current stage
            for (int t = 0; t <= r + 1; ++t) {
                if (!row_staged(h0, r, t)) continue;
                if (q == 0) {
                    if (!wait_or_abort(empty_bar(idx), phase ^ 1u, limit, abort_flag,
                                       STATUS_TIMEOUT_PRODUCER)) {
                        ok = false;
                        break;
                    }
                    // rows of this stage: RPS, or fewer at the end of the unit
                    int nr = 1;
                    for (int t2 = t + 1; nr < RPS && t2 <= r + 1; ++t2)
                        if (row_staged(h0, r, t2)) ++nr;
                    const int mine = NBOX == 3 ? nr : (pid < nr ? 1 : 0);
                    mbar_arrive_expect_tx(full_bar(idx), mine * p.box_bytes);
                    filled |= 1u << idx;
                    fill_parity = (fill_parity & ~(1u << idx)) | (phase << idx);
                }
                if (NBOX == 3 || q == pid)
                    tma_load_4d(sbase + idx * p.stage_bytes + q * p.row_bytes +
                                    (NBOX == 3 ? pid * p.box_bytes : 0),
                                &tmap_x, full_bar(idx), 0, x0, h0 - s.pad + t, n0, pol);
                if (++q == RPS) {
                    q = 0;
                    if (++idx == nst) {
                        idx = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (ok && q != 0) {  // a partly filled last stage
                q = 0;
                if (++idx == nst) {
                    idx = 0;
                    phase ^= 1u;
                }
            }
        }
        if (!ok || *abort_flag) drain_fills(full_bar(0), nst, filled, fill_parity, limit);
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            bool ok = wait_or_abort(wready_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
            if (p.inject_stall) {
                // Failure injection: wait on a barrier nothing arrives on.
                wait_or_abort(drain_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
                ok = false;
            }
            tc_fence_after();
            const uint32_t wsb_lo = desc_lo(sbase + C::WSB_OFF);
            const uint32_t rb_lo = static_cast<uint32_t>(p.row_bytes) >> 4;
            int issued = 0, idx = 0;
            uint32_t phase = 0;
            auto take = [&](uint32_t& a) -> bool {
                if (!wait_or_abort(full_bar(idx), phase, limit, abort_flag, STATUS_TIMEOUT_MMA))
                    return false;
                tc_fence_after();
                a = desc_lo(sbase + idx * p.stage_bytes);
                return true;
            };
            auto give = [&]() {
                umma_commit(empty_bar(idx));
                ++issued;
                if (++idx == nst) {
                    idx = 0;
                    phase ^= 1u;
                }
            };
            int k = 0;
            for (int u = blockIdx.x; ok && u < p.num_units; u += gridDim.x, ++k) {
                const int buf = k & 1;
                const uint32_t use = static_cast<uint32_t>(k >> 1) & 1u;
                if (!wait_or_abort(acce0 + 8u * buf, use ^ 1u, limit, abort_flag,
                                   STATUS_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                int n0, h0, r;
                unit_geo(u, n0, h0, r);
                const uint32_t dbuf = tmem_base + static_cast<uint32_t>(buf * VS_BUF_COLS);
                uint32_t a;
                if (r == VS_BH) {
                    if constexpr (NBOX == 1) {
                        if (!take(a)) { ok = false; break; }
                        vs_full_row<NBOX, 0>(dbuf, a, wsb_lo);
                        vs_full_row<NBOX, 1>(dbuf, a + rb_lo, wsb_lo);
                        vs_full_row<NBOX, 2>(dbuf, a + 2 * rb_lo, wsb_lo);
                        give();
                        if (!take(a)) { ok = false; break; }
                        vs_full_row<NBOX, 3>(dbuf, a, wsb_lo);
                        vs_full_row<NBOX, 4>(dbuf, a + rb_lo, wsb_lo);
                        vs_full_row<NBOX, 5>(dbuf, a + 2 * rb_lo, wsb_lo);
                        give();
                    } else {
                        if (!take(a)) { ok = false; break; }
                        vs_full_row<NBOX, 0>(dbuf, a, wsb_lo);
                        give();
                        if (!take(a)) { ok = false; break; }
                        vs_full_row<NBOX, 1>(dbuf, a, wsb_lo);
                        give();
                        if (!take(a)) { ok = false; break; }
                        vs_full_row<NBOX, 2>(dbuf, a, wsb_lo);
                        give();
                        if (!take(a)) { ok = false; break; }
                        vs_full_row<NBOX, 3>(dbuf, a, wsb_lo);
                        give();
                        if (!take(a)) { ok = false; break; }
                        vs_full_row<NBOX, 4>(dbuf, a, wsb_lo);
                        give();
                        if (!take(a)) { ok = false; break; }
                        vs_full_row<NBOX, 5>(dbuf, a, wsb_lo);
                        give();
                    }
                } else {
                    // a partial band: rows outside the image are skipped, so the rows an
                    // input row reaches first are counted as the rows go (J)
                    int J = 0, q = 0;
                    for (int t = 0; t <= r + 1; ++t) {
                        if (!row_staged(h0, r, t)) continue;
                        const int lo = t - r + 1 > 0 ? t - r + 1 : 0;
                        const int hi = t < 2 ? t : 2;
                        const int jtop = t - lo, jbot = t - hi;
                        int nnew = jtop - (J > jbot ? J : jbot) + 1;
                        if (nnew < 0) nnew = 0;
                        if (jtop + 1 > J) J = jtop + 1;
                        if (q == 0 && !take(a)) {
                            ok = false;
                            break;
                        }
                        vs_any_row<NBOX>(dbuf + static_cast<uint32_t>(64 * (VS_BH - 1 - jtop)),
                                         a + q * rb_lo,
                                         wsb_lo + static_cast<uint32_t>(lo) * (VS_TAP_BYTES >> 4),
                                         hi - lo + 1, nnew);
                        if (++q == RPS) {
                            q = 0;
                            give();
                        }
                    }
                    if (!ok) break;
                    if (q != 0) give();
                }
                umma_commit(accf0 + 8u * buf);
            }
            if (!ok && issued > 0) {
                // let the MMAs finish before TMEM is released
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
    } else if (warp >= VS_EPI_WARP0) {
        const int et = threadIdx.x - VS_EPI_WARP0 * 32;
        vs_expand<SEP>(p, smem + C::WSB_OFF, et);
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) mbar_arrive(wready_bar);
        float* vec = reinterpret_cast<float*>(smem + C::VEC_OFF);
        if (et < 64) {
            const float sc = p.ep.scale ? __ldg(p.ep.scale + et) : 1.0f;
            const float b = p.ep.bias ? __ldg(p.ep.bias + et) : 0.0f;
            vec[et] = sc;
            vec[64 + et] = fmaf(sc, b, p.ep.scale ? __ldg(p.ep.shift + et) : 0.0f);
        }
        named_bar_sync(1, VS_EPI_THREADS);
        griddep_wait();  // the residual complete, the output buffer no longer read
        // ------------------------------------------------------------ epilogue
        // Per band row, four blocks of 16 columns; a block's 32 lanes x 2 chunks of 8 channels
        // are transposed across lane pairs, so lane 2 m + c holds chunk c of lanes row0 and
        // row0 + 1; the residual of block b + 1 is requested before block b is processed.
        const int quad = warp & 3;                   // TMEM lane quadrant of this warp
        const int j = (warp - VS_EPI_WARP0) >> 2;    // band row this group drains
        const int ci = lane & 1;                     // chunk of this lane after the transpose
        const int row0 = quad * 32 + 2 * (lane >> 1);  // its lanes row0, row0 + 1
        const int plane = s.Ho * s.Wo;
        // lane -> (image of the group, column), fixed for the whole run: poff = pixel offset
        // from the group's first image at the band row, img = image index (or a value that
        // fails every image check, for padding lanes)
        int img[2], poff[2];
#pragma unroll
        for (int kk = 0; kk < 2; ++kk) {
            const int l = row0 + kk;
            const int e = l / p.P, c = l - e * p.P;
            img[kk] = (c < s.Wo && e < p.E) ? e : 1 << 30;
            poff[kk] = e * plane + c;
        }
        const __nv_bfloat16* res = static_cast<const __nv_bfloat16*>(p.ep.residual);
        __nv_bfloat16* out = static_cast<__nv_bfloat16*>(p.y);
        // the residual of this warp's pixels of unit u (its 128-byte lines) into L2, one unit
        // ahead of its use, so the epilogue's residual loads do not wait for DRAM
        auto prefetch_res = [&](int u) {
            if (res == nullptr || ci != 0 || u >= p.num_units) return;
            int n0, h0, r;
            unit_geo(u, n0, h0, r);
            if (j >= r) return;
            const long long base = (static_cast<long long>(n0) * s.Ho + h0 + j) * s.Wo;
#pragma unroll
            for (int kk = 0; kk < 2; ++kk)
                if (n0 + img[kk] < s.N) prefetch_l2(res + (base + poff[kk]) * 64);
        };
        prefetch_res(blockIdx.x);
        int k = 0;
        for (int u = blockIdx.x; u < p.num_units; u += gridDim.x, ++k) {
            const int buf = k & 1;
            const uint32_t use = static_cast<uint32_t>(k >> 1) & 1u;
            prefetch_res(u + gridDim.x);
            int n0, h0, r;
            unit_geo(u, n0, h0, r);
            const bool mine = j < r;
            const long long base = (static_cast<long long>(n0) * s.Ho + h0 + j) * s.Wo;
            bool valid[2];
#pragma unroll
            for (int kk = 0; kk < 2; ++kk) valid[kk] = mine && n0 + img[kk] < s.N;
            auto load_res = [&](int b, uint4(&r4)[2]) {
#pragma unroll
                for (int kk = 0; kk < 2; ++kk) {
                    r4[kk] = make_uint4(0u, 0u, 0u, 0u);
                    if (res != nullptr && valid[kk])
                        r4[kk] = __ldg(reinterpret_cast<const uint4*>(
                            res + (base + poff[kk]) * 64 + 16 * b + 8 * ci));
                }
            };
            uint4 ra[2], rb[2];
            load_res(0, ra);  // in flight during the wait for the accumulator
            bool ok = true;
            if (lane == 0)
                ok = wait_or_abort(accf0 + 8u * buf, use, limit, abort_flag,
                                   STATUS_TIMEOUT_EPILOGUE);
            if (__shfl_sync(0xffffffffu, ok ? 1 : 0, 0) == 0) break;
            tc_fence_after();
            if (!mine) {
                mbar_arrive_relaxed(acce0 + 8u * buf);
                continue;
            }
            const uint32_t taddr = tmem_base + (static_cast<uint32_t>(quad * 32) << 16) +
                                   static_cast<uint32_t>(buf * VS_BUF_COLS + 64 * (VS_BH - 1 - j));
            uint32_t va[16], vb[16];  // TMEM blocks b (in use) and b + 1 (in flight)
            tmem_ld_32x32b_x16(taddr, va);
            tmem_ld_wait();
#pragma unroll
            for (int b = 0; b < 4; ++b) {
                uint4(&rc)[2] = (b & 1) ? rb : ra;
                uint4(&rn)[2] = (b & 1) ? ra : rb;
                uint32_t(&v)[16] = (b & 1) ? vb : va;
                uint32_t(&vn)[16] = (b & 1) ? va : vb;
                if (b + 1 < 4) {
                    tmem_ld_32x32b_x16(taddr + 16 * (b + 1), vn);
                    load_res(b + 1, rn);
                } else {
                    // the band row is in registers: hand the buffer back to the issuer
                    tc_fence_before();
                    mbar_arrive_relaxed(acce0 + 8u * buf);
                }
                float E[2][8];  // E[jj][e]: channel 16 b + 8 jj + e of this lane's row
#pragma unroll
                for (int jj = 0; jj < 2; ++jj)
#pragma unroll
                    for (int e = 0; e < 8; ++e) E[jj][e] = __uint_as_float(v[8 * jj + e]);
                chunk_transpose_stage<1, 2>(E, ci);
                // now E[kk][e] = channel c0 + e of lane row0 + kk
                const int c0 = 16 * b + 8 * ci;
                float sc[8], sh[8];
                {
                    const float4 s0 = *reinterpret_cast<const float4*>(vec + c0);
                    const float4 s1 = *reinterpret_cast<const float4*>(vec + c0 + 4);
                    const float4 h0v = *reinterpret_cast<const float4*>(vec + 64 + c0);
                    const float4 h1v = *reinterpret_cast<const float4*>(vec + 64 + c0 + 4);
                    sc[0] = s0.x; sc[1] = s0.y; sc[2] = s0.z; sc[3] = s0.w;
                    sc[4] = s1.x; sc[5] = s1.y; sc[6] = s1.z; sc[7] = s1.w;
                    sh[0] = h0v.x; sh[1] = h0v.y; sh[2] = h0v.z; sh[3] = h0v.w;
                    sh[4] = h1v.x; sh[5] = h1v.y; sh[6] = h1v.z; sh[7] = h1v.w;
                }
#pragma unroll
                for (int kk = 0; kk < 2; ++kk) {
                    const __nv_bfloat162* rh = reinterpret_cast<const __nv_bfloat162*>(&rc[kk]);
                    uint32_t w[4];
#pragma unroll
                    for (int t = 0; t < 4; ++t) {
                        const float2 f = __bfloat1622float2(rh[t]);
                        const float z0 = fmaf(sc[2 * t], E[kk][2 * t], sh[2 * t]) + f.x;
                        const float z1 = fmaf(sc[2 * t + 1], E[kk][2 * t + 1], sh[2 * t + 1]) + f.y;
                        w[t] = pack_bf16x2(activate(z0, s.act), activate(z1, s.act));
                    }
                    if (valid[kk])
                        *reinterpret_cast<uint4*>(out + (base + poff[kk]) * 64 + c0) =
                            make_uint4(w[0], w[1], w[2], w[3]);
                }
                if (b + 1 < 4) tmem_ld_wait();
            }
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
