// qconv_stempool.cuh -- the 4-channel stem convolution and the 3x3, stride-2, padding-1
// max pooling that follows it (component-wise pooling rule of Sec. III-D), in one kernel
// that writes only the pooled tensor.  Included by qconv_tc.cu inside its anonymous
// namespace (it uses the descriptor helpers, bounded waits and issuer bookkeeping of
// tc_common.cuh and the pixel-pair geometry of qconv_gather.cuh).
//
// Orientation.  The stem has one quaternion input channel and 64 real output channels, so
// with pixels as the MMA's M and channels as its N every MMA is N = 64, which on this part
// costs the shared-memory reads of an N = 128 one.  Here the roles are swapped: the MMA's
// M = 128 rows are the signed block weight of Eq. 6 stacked for TWO consecutive output
// rows, row R = 2 c + v holding real output channel c (= q Qout + co) for output row
// 2 i + v, and the MMA's N is the output row's pixels (Wo rounded up to 16).  A tile is one
// pooled row i: output rows 2 i and 2 i + 1 read input rows 4 i - pad .. 4 i - pad + kh + 1
// (kh + 2 rows; the filter of row v sits at box rows 2 v .. 2 v + kh - 1 and the weight is
// zero elsewhere), so K = (kh + 2) x (pixel pairs per filter row) x 8 and a tile costs
// (kh + 2) nsp / 2 MMAs of 128 x N x 16 (18 for the 7x7 stem: 128 x 112 x 16 each).
//
// Pixel pairs.  Two horizontally adjacent 4-channel pixels form a 16-byte pair; in pair
// coordinates the stride-2 filter has horizontal stride 1, and the B operand of a K step
// is one row of the TMA box read as a K-major, non-swizzled matrix whose row n starts at
// pair n + 2t (rows 16 bytes apart, 8-row groups 128 bytes apart, the second 8-element K
// half one pair further on): the overlapping rows of the im2col matrix come from the
// descriptor and the pixels are never copied on chip (same geometry as qconv_gather.cuh).
//
// Epilogue.  After tcgen05.ld (32 lanes x 32 bits) a thread holds ONE channel of ONE
// output row across consecutive pixels, so the horizontal 3-wide stride-2 max is plain
// register work; the vertical max pairs lane 2c' (row 2 i) with lane 2c' + 1 (row 2 i + 1)
// through one shuffle, and the previous tile's second row (2 i - 1) stays in registers:
// a CTA takes a contiguous band of pooled rows (plus, when the band starts inside an image,
// one priming tile whose second row it keeps and whose output it does not store).
// For ReLU and no activation the pooling is taken on the raw accumulators and the affine
// IQBN step and activation are applied once per pooled value: x -> act(fma(s, x, t) + 0)
// is non-decreasing for s >= 0 and rounding to bf16 is monotone, so that equals pooling
// the activated, rounded pixels; for a channel with s < 0 the expansion negates that
// channel's weights (the map is then non-decreasing in the negated accumulator, with |s|).
// SiLU is not monotone: there every pixel is activated before the max.
//
// RGB input (RGB = true): the Poincare mapping of Eq. 4 (Sec. III-A) is fused into the
// loader.  Warp 0's lane 0 loads the tile's kh + 2 rows of fp32 RGB pixels (one TMA box of
// whole rows) into a ring of SP_RGB_SLOTS staging slots, SP_RGB_SLOTS - 1 tiles ahead;
// warps 0 and 3 turn the rows a tile does not share with the previous one into the bf16
// quaternion pairs of the B stage (the MMAs read the shared rows from the previous stage), q = ((1 - n2), 2 r, 2 g, 2 b) / (1 + n2)
// with n2 = r^2 + g^2 + b^2 (the arithmetic of the stand-alone mapping kernel, so the
// result is bit-identical to mapping first), zero pairs outside the image (the
// convolution's zero padding of the quaternion input), and hand the stage to its issuer.
//
// Roles (20 warps, one CTA per SM, persistent over its band):
//   warp 0       TMA producer: one box of (kh + 2) input rows per tile into a ring of
//                stages (each of the two issuers owns half of the ring);
//   warps 1, 2   MMA issuers (one lane each), taking the band's tiles alternately; each
//                owns two 128-column TMEM accumulators (warp 1 also owns TMEM);
//   warps 2..19  expand the stacked block weight once per CTA;
//   warps 4..19  epilogue, four warps per TMEM lane quadrant (pooled columns 16 k ..
//                16 k + 15, output columns 32 k .. 32 k + 31), every warp on every tile in
//                order.  The epilogue's instruction count, not the MMAs, sets the pace of
//                this kernel, so its per-chunk work is kept to straight-line register code.
// Every wait is bounded (tc_common.cuh): a wait that runs out sets a status bit and the
// CTA-wide abort flag, the copies and MMAs in flight are drained, TMEM is freed and the
// kernel returns.

constexpr int SP_THREADS = 640;
constexpr int SP_ISSUERS = 2;
constexpr int SP_NACC = 2 * SP_ISSUERS;  // TMEM accumulator buffers
constexpr int SP_BUF_COLS = 128;         // columns per buffer: output rows of up to 128 pixels
constexpr int SP_MAX_UNITS = 36;         // 16-byte K units (pixel pairs) per A row: K <= 288
constexpr int SP_EXP_WARP0 = 2;          // warps 2..19 expand the block weight
constexpr int SP_EXP_WARPS = 18;
constexpr int SP_EPI_WARP0 = 4;          // warps 4..19: epilogue
constexpr int SP_EPI_THREADS = 512;
constexpr int SP_RGB_SLOTS = 3;          // RGB input: staging slots of kh + 2 RGB rows

struct StemPoolParams {
    ConvShape s;
    EpilogueArgs ep;
    const __nv_bfloat16* w[4];  // letter tensors [16][kh][kw][1]
    void* y;                    // pooled output [N][Hp][Wp][64]
    unsigned long long wait_limit_ns;
    int inject_stall;
    int nsp;          // pixel pairs per filter row (even)
    int lead;         // pad mod 2: zero-weight filter column before the first pair
    int shift;        // (pad + lead) / 2: first pair of output column 0 is -shift
    int group;        // G: pairs per TMA element
    int d0;           // pairs from the box start to output column 0's first pair
    int gx0;          // box start in G-pair elements: (-shift - d0) / G
    int row_bytes;    // bytes of one input row of the box
    int rows;         // input rows per tile: kh + 2
    int stage_bytes;
    int per;          // stages owned by each issuer
    int nmma;         // N of the MMA: Wo rounded up to 16
    int Hp, Wp;       // pooled output size
    long long total_rows;  // N * Hp pooled rows
    // RGB input only
    const float* rgb;     // [N][H][W][3] fp32
    int rgb_row_bytes;    // 12 W
    int rgb_stage_bytes;  // rows x 12 W, rounded up to 1 KB
    int rgb_off;          // offset of the staging slots (after the B ring)
};

struct SpCfg {
    static constexpr int CHUNK = 128 * 32;  // one K step of the weight: 128 rows x 32 bytes
    static constexpr int A_BYTES = (SP_MAX_UNITS / 2) * CHUNK;
    static constexpr int SCRATCH_BYTES = 8 * 1024;  // letters: 4 x 16 x taps x 2 bytes
    static constexpr int MAX_PER = 4;
    static constexpr int NSTAGE = SP_ISSUERS * MAX_PER;
    // full, empty (per stage), accf, acce (per buffer), drain (per issuer), bready,
    // RGB staging full and empty (per slot)
    static constexpr int NUM_BARS = 2 * NSTAGE + 2 * SP_NACC + SP_ISSUERS + 1 + 2 * SP_RGB_SLOTS;
    static constexpr int SMEM_BYTES = 227 * 1024;
    static constexpr int A_OFF = 0;
    static constexpr int SCRATCH_OFF = A_OFF + A_BYTES;
    static constexpr int BAR_OFF = SCRATCH_OFF + SCRATCH_BYTES;
    static constexpr int RING_OFF = BAR_OFF + 1024;  // barriers, TMEM slot, abort flag
    static constexpr int RING_BYTES = SMEM_BYTES - 1024 - RING_OFF;  // 1 KB alignment slack
    // A (weight): K-major rows of 32 bytes, 32-byte swizzle; B (pixels): K-major, no
    // swizzle, 8-row groups 128 bytes apart, leading byte offset 16 (the desc_lo default)
    static constexpr uint32_t A_DESC_HI = desc_hi(8 * 32, desc_layout(32));
    static constexpr uint32_t B_DESC_HI = desc_hi(8 * 16, 0);
    static constexpr uint32_t TMEM_COLS = 512;
    static_assert(NUM_BARS * 8 + 16 <= 1024, "stem-pool barriers");
    static_assert(SP_NACC * SP_BUF_COLS <= 512, "stem-pool TMEM");
};

// Shapes the kernel covers: one quaternion input channel, 16 quaternion output channels,
// stride 2, even input width, output rows of at most 128 pixels, K within the weight area.
bool stem_pool_ok(const ConvShape& s) {
    if (s.sep || s.Qin != 1 || s.Qout != 16 || s.stride != 2 || (s.W & 1)) return false;
    if (s.Wo > SP_BUF_COLS || s.kh > 64) return false;
    if (s.kh * s.kw * 4 * 16 * 2 > SpCfg::SCRATCH_BYTES) return false;
    return (s.kh + 2) * gather_nsp(s) <= SP_MAX_UNITS;
}

// The stacked block weight, K-major rows of 32-byte K steps with a 32-byte swizzle:
//   A[2 c + v][(r, pair j, pixel e, component p)]
//     = sign(q, p) W_{q xor p}[co][r - 2 v][2 j - lead + e]   (c = 16 q + co)
// (zero outside the filter), negated for a channel whose IQBN scale is negative when
// NEG_SCALE.  Run by warps 2..19; the letters go to shared memory first (every thread's
// 16-byte loads in flight at once), then shared -> shared.
template <bool NEG_SCALE>
__device__ __forceinline__ void sp_expand(const StemPoolParams& p, uint8_t* smem, int et,
                                          int lane, uint32_t bready_bar) {
    using C = SpCfg;
    constexpr int ET = SP_EXP_WARPS * 32;
    const ConvShape& s = p.s;
    const int taps = s.kh * s.kw;
    const int lchunks = 2 * taps, nchunks = 4 * lchunks;  // 16-byte chunks
    uint8_t* wl = smem + C::SCRATCH_OFF;
    for (int i = et; i < nchunks; i += ET) {
        const int L = i / lchunks;
        reinterpret_cast<uint4*>(wl)[i] =
            __ldg(reinterpret_cast<const uint4*>(p.w[L]) + (i - L * lchunks));
    }
    named_bar_sync(5, ET);
    const __nv_bfloat16* wls = reinterpret_cast<const __nv_bfloat16*>(wl);
    const int units = p.rows * p.nsp;
    // consecutive threads take consecutive rows R of one K unit (conflict-free with the
    // swizzle)
    for (int i = et; i < 128 * units; i += ET) {
        const int U = i >> 7, R = i & 127;
        const int c = R >> 1, v = R & 1;
        const int q = c >> 4, co = c & 15;
        const int r = U / p.nsp, j = U - (U / p.nsp) * p.nsp;
        const int ky = r - 2 * v;
        bool neg = false;
        if constexpr (NEG_SCALE) neg = p.ep.scale != nullptr && __ldg(p.ep.scale + c) < 0.0f;
        uint32_t packed[4];
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int kx = 2 * j - p.lead + e;
            const bool in = ky >= 0 && ky < s.kh && kx >= 0 && kx < s.kw;
            float vals[4];
#pragma unroll
            for (int pc = 0; pc < 4; ++pc) {
                float wv = 0.0f;
                if (in) {
                    wv = __bfloat162float(wls[((q ^ pc) * 16 + co) * taps + ky * s.kw + kx]);
                    if (((NEG_MASK >> (4 * q + pc)) & 1u) != static_cast<uint32_t>(neg)) wv = -wv;
                }
                vals[pc] = wv;
            }
            packed[2 * e] = pack_bf16x2(vals[0], vals[1]);
            packed[2 * e + 1] = pack_bf16x2(vals[2], vals[3]);
        }
        const uint32_t off =
            static_cast<uint32_t>(C::A_OFF + (U >> 1) * C::CHUNK + R * 32) +
            ((static_cast<uint32_t>(U & 1) ^ ((static_cast<uint32_t>(R) >> 2) & 1u)) << 4);
        *reinterpret_cast<uint4*>(smem + off) =
            make_uint4(packed[0], packed[1], packed[2], packed[3]);
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) mbar_arrive(bready_bar);
}

// One warp's 32-column chunk of a tile: output columns 2 j0 .. 2 j0 + 31 of this lane's
// (channel, output row 2 i + v) in acc, column 2 j0 - 1 in `carry` (already in the pooling
// domain), pooled columns j0 .. j0 + 15.  RAW (ReLU or no activation): the pooling domain
// is the accumulator itself, sign-adjusted by the expansion; otherwise the activated
// value.  Lane v stores the pooled columns j0 + 2 u + v; prev1 holds, at the same columns,
// the previous tile's second output row (2 i - 1) on entry and this tile's on return.
template <int ACT>
__device__ __forceinline__ void sp_chunk(const uint32_t (&acc)[32], float carry, int j0, int Wo,
                                         int Wp, bool rows_ok, bool v_ok, int v, float sc,
                                         float sh, bool store, float (&prev1)[8],
                                         __nv_bfloat16* op) {
    constexpr bool RAW = ACT != 2;
    float a[32];
#pragma unroll
    for (int k = 0; k < 32; ++k) {
        a[k] = __uint_as_float(acc[k]);
        if constexpr (!RAW) a[k] = activate(fmaf(sc, a[k], sh) + 0.0f, ACT);
    }
    const int lim = Wo - 2 * j0;
    if (lim < 32) {  // warp-uniform: the chunk runs past the output row
#pragma unroll
        for (int k = 0; k < 32; ++k)
            if (k >= lim) a[k] = -INFINITY;
    }
    float hm[16];  // horizontal 3-wide stride-2 max of this lane's row
#pragma unroll
    for (int t = 0; t < 16; ++t)
        hm[t] = fmax3(t == 0 ? carry : a[2 * t - 1], a[2 * t], a[2 * t + 1]);
    if (!rows_ok) {  // warp-uniform: output row 2 i + 1 is past the end (odd Ho)
#pragma unroll
        for (int t = 0; t < 16; ++t) hm[t] = v_ok ? hm[t] : -INFINITY;
    }
    float m[8];
#pragma unroll
    for (int u = 0; u < 8; ++u) {
        // lane v keeps column 2u + v of its row and receives the partner row's value there
        const float mine = v ? hm[2 * u + 1] : hm[2 * u];
        const float send = v ? hm[2 * u] : hm[2 * u + 1];
        const float recv = __shfl_xor_sync(0xffffffffu, send, 1);
        m[u] = fmax3(mine, recv, prev1[u]);
        prev1[u] = v ? mine : recv;  // output row 2 i + 1 at this lane's column
    }
    if (!store) return;  // warp-uniform (the priming tile)
#pragma unroll
    for (int u = 0; u < 8; ++u)
        if constexpr (RAW) m[u] = activate(fmaf(sc, m[u], sh) + 0.0f, ACT);
    if (j0 + 16 <= Wp) {  // warp-uniform
#pragma unroll
        for (int u = 0; u < 8; ++u) st_global_na_bf16(op + u * 128, __float2bfloat16_rn(m[u]));
    } else {
#pragma unroll
        for (int u = 0; u < 8; ++u)
            if (j0 + 2 * u + v < Wp) st_global_na_bf16(op + u * 128, __float2bfloat16_rn(m[u]));
    }
}

// Eq. 4 for one pixel pair (the arithmetic of poincare.cu): 8 bf16 = [q0: r i j k | q1].
__device__ __forceinline__ uint4 sp_poincare_pair(float2 a, float2 b, float2 c) {
    const float px[2][3] = {{a.x, a.y, b.x}, {b.y, c.x, c.y}};  // r0 g0 b0 | r1 g1 b1
    uint32_t w[4];
#pragma unroll
    for (int e = 0; e < 2; ++e) {
        const float rr = px[e][0], gg = px[e][1], bb = px[e][2];
        const float n2 = fmaf(rr, rr, fmaf(gg, gg, bb * bb));
        const float inv = __fdividef(1.0f, 1.0f + n2);
        const float two_inv = 2.0f * inv;
        w[2 * e] = pack_bf16x2((1.0f - n2) * inv, rr * two_inv);
        w[2 * e + 1] = pack_bf16x2(gg * two_inv, bb * two_inv);
    }
    return make_uint4(w[0], w[1], w[2], w[3]);
}

// Warps 0 and 3 (RGB input): rows r_begin .. rows - 1 of one tile's B stage, mapped from
// the tile's staging slot of RGB rows (rows 0 .. 3 of a tile that continues an image are
// rows 4 .. 7 of the previous tile: the MMAs read them from that tile's stage and they are
// not written again; r_begin is 4 then, else 0).  ct = 0 .. 63 this thread's index among the two warps, which takes the pairs ct
// and ct + 64 of each row; y0 = the tile's first input row; 32-bit shared addresses.  Under
// the MMAs' operand reads shared-memory accesses take hundreds of cycles, so all of a
// thread's loads (at most 2 pairs x MAXR rows) are issued before any pair is mapped.
template <int MAXR>
__device__ __forceinline__ void sp_convert_rgb(const StemPoolParams& p, uint32_t stage_sa,
                                               int r_begin, uint32_t slot_sa, int y0, int ct) {
    const ConvShape& s = p.s;
    const int gp = p.row_bytes / 16;  // pairs per box row
    const int pair0 = p.gx0 * p.group;
    const int W2 = s.W / 2;
    const uint32_t rb = static_cast<uint32_t>(p.row_bytes);
    const uint32_t rgb_rb = static_cast<uint32_t>(p.rgb_row_bytes);
    for (int r0 = r_begin; r0 < p.rows; r0 += MAXR) {
        float2 in[MAXR][2][3];
        bool live[MAXR][2];
#pragma unroll
        for (int a = 0; a < MAXR; ++a) {
            const int r = r0 + a, y = y0 + r;
            const bool row_in = r < p.rows && y >= 0 && y < s.H;
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                const int jb = ct + 64 * c, pi = pair0 + jb;
                live[a][c] = row_in && jb < gp && pi >= 0 && pi < W2;
                if (live[a][c]) {
                    const uint32_t src = slot_sa + r * rgb_rb + 24 * pi;
                    in[a][c][0] = lds_f2(src);
                    in[a][c][1] = lds_f2(src + 8);
                    in[a][c][2] = lds_f2(src + 16);
                }
            }
        }
#pragma unroll
        for (int a = 0; a < MAXR; ++a)
#pragma unroll
            for (int c = 0; c < 2; ++c) {
                const int r = r0 + a, jb = ct + 64 * c;
                if (r >= p.rows || jb >= gp) continue;
                sts_u4(stage_sa + r * rb + 16 * jb,
                       live[a][c] ? sp_poincare_pair(in[a][c][0], in[a][c][1], in[a][c][2])
                                  : make_uint4(0u, 0u, 0u, 0u));
            }
    }
}

// ROWS, NSP > 0: input rows per tile and pairs per filter row known at compile time (the
// MMA issue loop is then fully unrolled with constant descriptor offsets); 0 = run time.
template <int ROWS, int NSP, int ACT, bool RGB = false>
__global__ void __launch_bounds__(SP_THREADS, 1)
    qconv_stem_pool_kernel(const __grid_constant__ CUtensorMap tmap_x, const StemPoolParams p) {
    using C = SpCfg;
    constexpr bool RAW = ACT != 2;  // ReLU or none: pool the raw accumulators
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::BAR_OFF);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::NUM_BARS);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int st) { return bar0 + 8u * st; };
    auto empty_bar = [&](int st) { return bar0 + 8u * (C::NSTAGE + st); };
    const uint32_t accf0 = bar0 + 8u * (2 * C::NSTAGE);
    const uint32_t acce0 = accf0 + 8u * SP_NACC;
    const uint32_t drain0 = acce0 + 8u * SP_NACC;
    const uint32_t bready_bar = drain0 + 8u * SP_ISSUERS;
    const uint32_t rgbf0 = bready_bar + 8u;  // RGB staging slots: full, then empty
    const uint32_t rgbe0 = rgbf0 + 8u * SP_RGB_SLOTS;

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const ConvShape& s = p.s;
    const uint64_t limit = p.wait_limit_ns;
    const int STAGES = SP_ISSUERS * p.per;

    // this CTA's band of pooled rows [r0, r1), preceded by a priming tile (row r0 - 1)
    // when the band starts inside an image
    const long long r0 = static_cast<long long>(blockIdx.x) * p.total_rows / gridDim.x;
    const long long r1 = static_cast<long long>(blockIdx.x + 1) * p.total_rows / gridDim.x;
    const int prime = (r1 > r0 && r0 % p.Hp != 0) ? 1 : 0;
    const int ntiles = static_cast<int>(r1 - r0) + prime;
    const long long rfirst = r0 - prime;

    griddep_launch_dependents();
    if (threadIdx.x == 0) {
        for (int i = 0; i < STAGES; ++i) {
            mbar_init(full_bar(i), RGB ? 2 : 1);  // RGB: the two converter warps
            // RGB: a stage is also read by the next tile (the rows the two share)
            mbar_init(empty_bar(i), RGB ? 2 : 1);
        }
        for (int b = 0; b < SP_NACC; ++b) {
            mbar_init(accf0 + 8u * b, 1);
            mbar_init(acce0 + 8u * b, SP_EPI_THREADS);
        }
        for (int i = 0; i < SP_ISSUERS; ++i) mbar_init(drain0 + 8u * i, 1);
        mbar_init(bready_bar, SP_EXP_WARPS);
        for (int i = 0; i < SP_RGB_SLOTS; ++i) {
            mbar_init(rgbf0 + 8u * i, 1);
            mbar_init(rgbe0 + 8u * i, 2);
        }
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
    // kernel's last CTAs; the input loaders and the epilogue wait for that kernel before
    // their first access to activations.

    if (RGB && (warp == 0 || warp == 3)) {
        // ------------------------------------------------- RGB staging and conversion
        // (warp 3 first helps with the weight expansion)
        if (warp == 3) sp_expand<RAW>(p, smem, (warp - SP_EXP_WARP0) * 32 + lane, lane, bready_bar);
        griddep_wait();  // the previous kernel's output (this layer's input) is complete
        const int ct = (warp == 0 ? 0 : 32) + lane;
        const uint64_t pol_x = l2_policy_evict_first();
        const uint32_t tx = static_cast<uint32_t>(p.rows * p.rgb_row_bytes);
        uint32_t filled = 0, fill_parity = 0;
        int img = static_cast<int>(rfirst / p.Hp);
        int i = static_cast<int>(rfirst - static_cast<long long>(img) * p.Hp);
        int nimg = img, ni = i;  // the next tile to load
        auto load_next = [&](int k) -> bool {  // warp 0 lane 0: staging slot of tile k
            const int sl = k % SP_RGB_SLOTS;
            const uint32_t ph = static_cast<uint32_t>(k / SP_RGB_SLOTS) & 1u;
            if (!wait_or_abort(rgbe0 + 8u * sl, ph ^ 1u, limit, abort_flag,
                               STATUS_TIMEOUT_PRODUCER))
                return false;
            mbar_arrive_expect_tx(rgbf0 + 8u * sl, tx);
            filled |= 1u << sl;
            fill_parity = (fill_parity & ~(1u << sl)) | (ph << sl);
            tma_load_4d(sbase + p.rgb_off + sl * p.rgb_stage_bytes, &tmap_x, rgbf0 + 8u * sl, 0,
                        0, 4 * ni - s.pad, nimg, pol_x);
            if (++ni == p.Hp) {
                ni = 0;
                ++nimg;
            }
            return true;
        };
        bool ok = true;
        if (warp == 0 && lane == 0)
            for (int k = 0; ok && k < SP_RGB_SLOTS - 1 && k < ntiles; ++k) ok = load_next(k);
        StageCursor cur(p.per);
        int ki = 0, prev_stage = -1;
        for (int k = 0; k < ntiles; ++k) {
            const int stage = cur.stage(ki);
            const uint32_t phase = cur.phase;
            if (++ki == SP_ISSUERS) {
                ki = 0;
                cur.next();
            }
            // rows shared with the previous tile (same image): copied, not mapped again
            // (rows 4 .. rows - 1 of every stage are written, so the next tile's rows
            // 0 .. rows - 6, rows 4 .. rows - 2 here, are always in this tile's stage)
            const int r_begin = (prev_stage >= 0 && i != 0 && p.rows > 5) ? 4 : 0;
            const int sl = k % SP_RGB_SLOTS;
            if (warp == 0 && lane == 0 && ok && k + SP_RGB_SLOTS - 1 < ntiles)
                ok = load_next(k + SP_RGB_SLOTS - 1);
            if (lane == 0 && ok)
                ok = wait_or_abort(rgbf0 + 8u * sl,
                                   static_cast<uint32_t>(k / SP_RGB_SLOTS) & 1u, limit,
                                   abort_flag, STATUS_TIMEOUT_PRODUCER) &&
                     wait_or_abort(empty_bar(stage), phase ^ 1u, limit, abort_flag,
                                   STATUS_TIMEOUT_PRODUCER);
            ok = __shfl_sync(0xffffffffu, ok ? 1 : 0, 0) != 0;
            // both converter warps leave together; the barrier also orders the previous
            // tile's stage writes (of both warps) before this tile's copies from it
            if (named_bar_or(7, 64, !ok)) break;
            sp_convert_rgb<4>(p, sbase + C::RING_OFF + stage * p.stage_bytes, r_begin,
                              sbase + p.rgb_off + sl * p.rgb_stage_bytes, 4 * i - s.pad, ct);
            prev_stage = stage;
            fence_proxy_async_smem();
            __syncwarp();
            if (lane == 0) {
                mbar_arrive(full_bar(stage));
                mbar_arrive(rgbe0 + 8u * sl);
            }
            if (++i == p.Hp) {
                i = 0;
                ++img;
            }
        }
        if (warp == 0 && lane == 0 && (!ok || *abort_flag))
            drain_fills(rgbf0, SP_RGB_SLOTS, filled, fill_parity, limit);
    } else if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            griddep_wait();  // the previous kernel's output (this layer's input) is complete
            const uint64_t pol_x = l2_policy_evict_normal();
            uint32_t filled = 0, fill_parity = 0;
            bool ok = true;
            const uint32_t tx = static_cast<uint32_t>(p.rows * p.row_bytes);
            int img = static_cast<int>(rfirst / p.Hp);
            int i = static_cast<int>(rfirst - static_cast<long long>(img) * p.Hp);
            StageCursor cur(p.per);  // advanced once per round of SP_ISSUERS tiles
            int ki = 0;
            for (int k = 0; k < ntiles; ++k) {
                const int stage = cur.stage(ki);
                const uint32_t phase = cur.phase;
                if (++ki == SP_ISSUERS) {
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
                tma_load_4d(sbase + C::RING_OFF + stage * p.stage_bytes, &tmap_x, fb, 0, p.gx0,
                            4 * i - s.pad, img, pol_x);
                if (++i == p.Hp) {
                    i = 0;
                    ++img;
                }
            }
            if (!ok || *abort_flag) drain_fills(full_bar(0), STAGES, filled, fill_parity, limit);
        }
    } else if (warp <= SP_ISSUERS) {
        // ------------------------------------------------------------ MMA issuers
        // (warp 2 first helps with the weight expansion)
        if (warp >= SP_EXP_WARP0)
            sp_expand<RAW>(p, smem, (warp - SP_EXP_WARP0) * 32 + lane, lane, bready_bar);
        if (lane == 0) {
            const int me = warp - 1;
            const uint32_t drain_bar = drain0 + 8u * me;
            const uint32_t idesc = make_idesc(BM, p.nmma, 0);
            const int rows = ROWS > 0 ? ROWS : p.rows;
            const int half = (NSP > 0 ? NSP : p.nsp) / 2;
            bool ok = wait_or_abort(bready_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
            int issued = 0;
            if (p.inject_stall && me == 0) {
                // Failure injection: wait on a barrier nothing arrives on.
                wait_or_abort(drain_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
                ok = false;
            }
            tc_fence_after();
            const uint32_t a_lo0 = desc_lo(sbase + C::A_OFF);
            const uint32_t row_lo = static_cast<uint32_t>(p.row_bytes) >> 4;
            StageCursor cur(p.per);
            // RGB: tile k's rows 0..3 are rows 4..7 of tile k - 1's stage unless tile k
            // starts an image (the converters write rows 4..rows-1 of every stage); that
            // stage is the other issuer's (the same round, or the previous one)
            StageCursor prev_cur(p.per);
            const int other = 1 - me;
            for (int k = me; ok && k < ntiles; k += SP_ISSUERS) {
                int buf;
                uint32_t use;
                issuer_acc_n<SP_ISSUERS>(k, buf, use);
                const int stage = cur.stage(me);
                const uint32_t phase = cur.phase;
                cur.next();
                int prev_stage = -1, r_shared = 0;
                if constexpr (RGB) {
                    // tile k - 1 is the other issuer's: for me = 1 the same round, for me = 0
                    // the previous round (prev_cur lags by one round for issuer 0)
                    if (k >= 1) {
                        prev_stage = prev_cur.stage(other);
                        const long long rk = rfirst + k;
                        if (rk % p.Hp != 0 && p.rows > 5) r_shared = 4;
                    }
                    if (me == 1 || k >= 1) prev_cur.next();
                }
                if (!wait_or_abort(acce0 + 8u * buf, use ^ 1u, limit, abort_flag,
                                   STATUS_TIMEOUT_MMA) ||
                    !wait_or_abort(full_bar(stage), phase, limit, abort_flag,
                                   STATUS_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem_base + static_cast<uint32_t>(buf * SP_BUF_COLS);
                const uint32_t b_lo0 =
                    desc_lo(sbase + C::RING_OFF + stage * p.stage_bytes) + p.d0;
                // rows below r_shared (0..3): rows r + 4 of the previous tile's stage
                const uint32_t p_lo0 =
                    desc_lo(sbase + C::RING_OFF + (prev_stage < 0 ? 0 : prev_stage) *
                                                      p.stage_bytes) + p.d0 + 4 * row_lo;
                if constexpr (ROWS > 0) {
#pragma unroll
                    for (int r = 0; r < ROWS; ++r) {
                        const uint32_t rlo = (RGB && r < r_shared) ? p_lo0 + r * row_lo
                                                                   : b_lo0 + r * row_lo;
#pragma unroll
                        for (int t = 0; t < NSP / 2; ++t) {
                            const int u = r * (NSP / 2) + t;
                            umma_f16_w(d, a_lo0 + ((u * C::CHUNK) >> 4), C::A_DESC_HI,
                                       rlo + 2 * t, C::B_DESC_HI, idesc, u != 0 ? 1u : 0u);
                        }
                    }
                } else {
                    int u = 0;
                    for (int r = 0; r < rows; ++r) {
                        const uint32_t rlo = (RGB && r < r_shared) ? p_lo0 + r * row_lo
                                                                   : b_lo0 + r * row_lo;
                        for (int t = 0; t < half; ++t, ++u)
                            umma_f16_w(d, a_lo0 + ((u * C::CHUNK) >> 4), C::A_DESC_HI,
                                       rlo + 2 * t, C::B_DESC_HI, idesc, u != 0 ? 1u : 0u);
                    }
                }
                ++issued;
                umma_commit(empty_bar(stage));
                // RGB: the previous tile's stage is free once this tile's MMAs are done too
                if (RGB && prev_stage >= 0) umma_commit(empty_bar(prev_stage));
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
        sp_expand<RAW>(p, smem, (warp - SP_EXP_WARP0) * 32 + lane, lane, bready_bar);
        griddep_wait();  // the output buffer no longer read by earlier kernels
        if (warp >= SP_EPI_WARP0) {
            // -------------------------------------------------------- epilogue
            const int qd = warp & 3;                    // TMEM lane quadrant
            const int ch = (warp - SP_EPI_WARP0) >> 2;  // chunk: pooled columns 16 ch ..
            const int v = lane & 1;                     // output row 2 i + v
            const int c = 16 * qd + (lane >> 1);        // real output channel
            const int j0 = 16 * ch;
            const bool active = j0 < p.Wp;              // warp-uniform
            const float sc_raw = p.ep.scale ? __ldg(p.ep.scale + c) : 1.0f;
            const float bias = p.ep.bias ? __ldg(p.ep.bias + c) : 0.0f;
            const float sh = fmaf(sc_raw, bias, p.ep.shift ? __ldg(p.ep.shift + c) : 0.0f);
            // RAW: the expansion negated this channel's weights if its scale is negative
            const float sc = (RAW && sc_raw < 0.0f) ? -sc_raw : sc_raw;
            __nv_bfloat16* out = static_cast<__nv_bfloat16*>(p.y);
            float prev1[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) prev1[u] = -INFINITY;
            int img = static_cast<int>(rfirst / p.Hp);
            int i = static_cast<int>(rfirst - static_cast<long long>(img) * p.Hp);
            for (int k = 0; k < ntiles; ++k) {
                int buf;
                uint32_t use;
                issuer_acc_n<SP_ISSUERS>(k, buf, use);
                bool ok = true;
                if (lane == 0)
                    ok = wait_or_abort(accf0 + 8u * buf, use, limit, abort_flag,
                                       STATUS_TIMEOUT_EPILOGUE);
                if (__shfl_sync(0xffffffffu, ok ? 1 : 0, 0) == 0) break;
                tc_fence_after();
                const uint32_t taddr = tmem_base + (static_cast<uint32_t>(qd * 32) << 16) +
                                       static_cast<uint32_t>(buf * SP_BUF_COLS + 2 * j0);
                uint32_t acc[32];
                uint32_t cr = 0u;
                if (active) {
                    tmem_ld_32x32b_x32(taddr, acc);
                    if (ch > 0) cr = tmem_ld_32x32b_x1(taddr - 1);
                    tmem_ld_wait();
                }
                // the accumulator is in registers: hand the buffer back to its issuer
                tc_fence_before();
                mbar_arrive_relaxed(acce0 + 8u * buf);
                if (active) {
                    if (i == 0) {  // the first pooled row of an image: no row above
#pragma unroll
                        for (int u = 0; u < 8; ++u) prev1[u] = -INFINITY;
                    }
                    const bool rows_ok = 2 * i + 1 < s.Ho;
                    const bool v_ok = v == 0 || rows_ok;
                    float carry = -INFINITY;
                    if (ch > 0) {
                        carry = __uint_as_float(cr);
                        if constexpr (!RAW) carry = activate(fmaf(sc, carry, sh) + 0.0f, ACT);
                    }
                    __nv_bfloat16* op =
                        out + ((static_cast<long long>(img) * p.Hp + i) * p.Wp + j0 + v) * 64 + c;
                    sp_chunk<ACT>(acc, carry, j0, s.Wo, p.Wp, rows_ok, v_ok, v, sc, sh,
                                  k >= prime, prev1, op);
                }
                if (++i == p.Hp) {
                    i = 0;
                    ++img;
                }
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
