// qconv_dw.cuh -- weight gradient of the full-form quaternion convolution (Eq. 5) on the
// tensor cores, stride 1.  Included by qconv_tc.cu only.
//
// As a real contraction the forward convolution is y[px][m Qout + co] = sum over taps and
// real input channels of B[m][p] x[px + tap][p Qin + ci], with the signed block weight
// B[m][p] = sign(m, p) W_{m xor p} of Eq. 6.  Its real weight gradient for one tap is the
// plain product over output pixels
//     G_tap[c][d] = sum_px x[px + tap][c] dy[px][d]        (c: input, d: output channel),
// and each letter gathers its four signed blocks:
//     dW_L[co][tap][ci] = sum over (m, p) with m xor p = L of sign(m, p) G_tap[p Qin + ci][m Qout + co].
//
// Both MMA operands come straight from the NHWC tensors: a TMA box of 64 channels x P
// pixels (P = Ht rows x Wbox columns of one image) lands as P rows of 128 bytes, the
// MN-major SWIZZLE_128B layout (channels along M or N, pixels along K).  For a strided
// convolution the x box traverses every stride-th input pixel (the tensor map's element
// strides), so it lands in the same layout as the dy box of the output pixels it serves.  A holds two such
// boxes ("units": one tap's window of x, one 64-channel chunk) stacked to M = 128; B holds
// ncols / 64 boxes of dy, N = ncols.  A CTA owns a_per unit pairs (one TMEM accumulator of
// ncols fp32 columns each) and one ncols-wide group of output channels, for a contiguous
// range of pixel blocks (split K); its epilogue folds the 16 blocks into the letters and
// adds them to the fp32 outputs with atomics (zeroed before the launch).
// Separable form (Eq. 7, gradient Eq. 10): y_m = sum_p S[m][p] W_p conv x_p, so block
// (m, p) goes to letter p with Eq. 7's sign S[m][p] instead (the same 16 blocks: the
// product computes the 12 cross-component blocks the separable form does not use).

namespace dwk {

constexpr int THREADS = 256;  // warp 0 TMA producer, warp 1 MMA issuer, warp 2 TMEM owner,
constexpr int EPI_WARP0 = 4;  // warps 4-7 epilogue (TMEM lane quarters 0-3)
constexpr int MAX_PAIRS = 8;
constexpr int MAX_STAGES = 4;
constexpr int BOX_ROW = 128;  // bytes of one pixel's 64 channels
constexpr int BAR_BYTES = 256;
// Shared memory reserved past the barriers: the MMA reads of the last stage stay inside the
// CTA's allocation even for a descriptor whose two byte offsets were read the other way
// round (one pixel block plus 4 KB beyond the stage), and a strided x box (stride s) stays
// inside it even if the copy brought its s * s untraversed elements as well.
__host__ __device__ constexpr int tail_bytes(int P, int stride = 1) {
    return P * BOX_ROW + 4096 + (stride * stride - 1) * P * BOX_ROW;
}

struct DwParams {
    int Ho, Wo, Qin, Qout, kh, kw, pad, taps;
    int stride;              // the x boxes traverse every stride-th pixel (element strides)
    int Wbox, Ht, P;         // pixel block: Ht rows x Wbox columns = P pixels
    int rblocks;             // pixel blocks per image
    long long kblocks;       // N * rblocks
    int nxc, units, npairs;  // 64-channel chunks of x; units = taps * nxc; pairs of units
    int a_per, pair_groups;  // pairs per CTA; groups of pairs
    int ncols, nyb;          // output channels per CTA (N of each MMA); dy boxes per stage
    int groups, splits, stages;
    int sep;                 // 1: fold for the separable form
    uint32_t tmem_cols;
    uint32_t stage_bytes;
    unsigned long long wait_limit_ns;
    float* dwr;
    float* dwi;
    float* dwj;
    float* dwk;
};

// Shared-memory descriptor, low word, with a leading byte offset: for MN-major swizzled
// tiles it is the distance between successive 64-element (128-byte) groups along M or N.
__device__ __forceinline__ uint32_t desc_lo_lbo(uint32_t saddr, uint32_t lbo_bytes) {
    return ((saddr & 0x3FFFFu) >> 4) | ((lbo_bytes >> 4) << 16);
}

// kind::f16 instruction descriptor with both operands MN-major (transpose bits 15, 16).
__host__ __device__ constexpr uint32_t make_idesc_mn(int M, int N) {
    return make_idesc(M, N, 0) | (1u << 15) | (1u << 16);
}

__device__ __forceinline__ float* letter_ptr(const DwParams& p, int L) {
    return L == 0 ? p.dwr : (L == 1 ? p.dwi : (L == 2 ? p.dwj : p.dwk));
}

__global__ void __launch_bounds__(THREADS, 1)
    qconv_dw_kernel(const __grid_constant__ CUtensorMap tmap_x,
                    const __grid_constant__ CUtensorMap tmap_dy, const DwParams p) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + p.stages * p.stage_bytes);
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int s) { return bar0 + 8u * s; };
    auto empty_bar = [&](int s) { return bar0 + 8u * (MAX_STAGES + s); };
    const uint32_t done_bar = bar0 + 8u * (2 * MAX_STAGES);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * MAX_STAGES + 1);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const uint64_t limit = p.wait_limit_ns;
    // CTA -> (unit-pair group, output-channel group, K split); CTAs of one split are
    // adjacent in launch order, so they read the same pixel rows at about the same time
    const int g = static_cast<int>(blockIdx.x) % p.groups;
    const int split = static_cast<int>(blockIdx.x) / p.groups;
    const int pg = g % p.pair_groups, cg = g / p.pair_groups;
    const int pair0 = pg * p.a_per;
    const int npair = p.npairs - pair0 < p.a_per ? p.npairs - pair0 : p.a_per;
    const long long kb_begin = p.kblocks * split / p.splits;
    const long long kb_end = p.kblocks * (split + 1) / p.splits;
    const uint32_t box_bytes = static_cast<uint32_t>(p.P) * BOX_ROW;

    griddep_launch_dependents();
    if (threadIdx.x == 0) {
        for (int i = 0; i < p.stages; ++i) {
            mbar_init(full_bar(i), 1);
            mbar_init(empty_bar(i), 1);
        }
        mbar_init(done_bar, 1);
        *abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 0 && lane == 0) {
        tma_prefetch_desc(&tmap_x);
        tma_prefetch_desc(&tmap_dy);
    }
    if (warp == 2) {
        tmem_alloc(smem_u32(tmem_slot), p.tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;
    griddep_wait();  // x and dy complete, the zeroed outputs visible

    if (warp == 0) {
        // ---------------------------------------------------------------- TMA producer
        if (lane == 0) {
            const uint64_t pol = l2_policy_evict_normal();
            const uint32_t tx = static_cast<uint32_t>(2 * npair + p.nyb) * box_bytes;
            uint32_t filled = 0, fill_parity = 0;
            bool ok = true;
            int stage = 0;
            uint32_t phase = 0;
            for (long long kb = kb_begin; kb < kb_end; ++kb) {
                if (!wait_or_abort(empty_bar(stage), phase ^ 1u, limit, abort_flag,
                                   STATUS_TIMEOUT_PRODUCER)) {
                    ok = false;
                    break;
                }
                const int n = static_cast<int>(kb / p.rblocks);
                const int r0 = static_cast<int>(kb - static_cast<long long>(n) * p.rblocks) * p.Ht;
                const uint32_t fb = full_bar(stage);
                mbar_arrive_expect_tx(fb, tx);
                filled |= 1u << stage;
                fill_parity = (fill_parity & ~(1u << stage)) | (phase << stage);
                const uint32_t dst = sbase + stage * p.stage_bytes;
                for (int k = 0; k < 2 * npair; ++k) {
                    int u = 2 * pair0 + k;
                    if (u >= p.units) u = p.units - 1;  // odd unit count: repeat the last
                    const int tap = u / p.nxc, xc = u - tap * p.nxc;
                    const int dh = tap / p.kw, dw = tap - dh * p.kw;
                    tma_load_4d(dst + k * box_bytes, &tmap_x, fb, xc * 64, dw - p.pad,
                                r0 * p.stride - p.pad + dh, n, pol);
                }
                const uint32_t ydst = dst + 2 * p.a_per * box_bytes;
                for (int c = 0; c < p.nyb; ++c)
                    tma_load_4d(ydst + c * box_bytes, &tmap_dy, fb, cg * p.ncols + c * 64, 0, r0,
                                n, pol);
                if (++stage == p.stages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (!ok || *abort_flag)
                drain_fills(full_bar(0), p.stages, filled, fill_parity, limit);
        }
    } else if (warp == 1) {
        // ---------------------------------------------------------------- MMA issuer
        if (lane == 0) {
            const uint32_t idesc = make_idesc_mn(128, p.ncols);
            const uint32_t hi = desc_hi(1024, 2);  // 8-pixel groups 1024 bytes apart, SW128
            const uint32_t ksteps = static_cast<uint32_t>(p.P) / 16;
            int stage = 0;
            uint32_t phase = 0;
            bool first = true;
            for (long long kb = kb_begin; kb < kb_end; ++kb) {
                if (!wait_or_abort(full_bar(stage), phase, limit, abort_flag, STATUS_TIMEOUT_MMA))
                    break;
                tc_fence_after();
                const uint32_t a0 = sbase + stage * p.stage_bytes;
                const uint32_t b0 = a0 + 2 * p.a_per * box_bytes;
                for (uint32_t j = 0; j < ksteps; ++j) {
                    const uint32_t b_lo = desc_lo_lbo(b0 + j * 2048u, box_bytes);
                    for (int a = 0; a < npair; ++a) {
                        const uint32_t a_lo =
                            desc_lo_lbo(a0 + 2u * a * box_bytes + j * 2048u, box_bytes);
                        umma_f16_w(tmem_base + static_cast<uint32_t>(a * p.ncols), a_lo, hi, b_lo,
                                   hi, idesc, first ? 0u : 1u);
                    }
                    first = false;
                }
                umma_commit(empty_bar(stage));
                if (++stage == p.stages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            // arrives once every MMA issued above has completed (also after an abort, so
            // the teardown can wait for them before TMEM is released)
            umma_commit(done_bar);
        }
    } else if (warp >= EPI_WARP0) {
        // ---------------------------------------------------------------- epilogue
        const int q = warp - EPI_WARP0;  // TMEM lane quarter
        const bool ok = wait_or_abort(done_bar, 0, limit, abort_flag, STATUS_TIMEOUT_EPILOGUE);
        tc_fence_after();
        if (ok && !*abort_flag) {
            const int row = 32 * q + lane;  // x channel within the unit pair
            const long long wstride = static_cast<long long>(p.taps) * p.Qin;  // one co step
            for (int a = 0; a < npair; ++a) {
                const int u = 2 * (pair0 + a) + row / 64;
                const bool live = u < p.units;  // the repeated last unit is not written
                const int tap = (live ? u : 0) / p.nxc;
                const int c = ((live ? u : 0) - tap * p.nxc) * 64 + row % 64;
                const int pc = c / p.Qin, ci = c - pc * p.Qin;
                const long long row_off = static_cast<long long>(tap) * p.Qin + ci;
                for (int j0 = 0; j0 < p.ncols; j0 += 32) {
                    uint32_t v[32];
                    tmem_ld_32x32b_x32(
                        tmem_base + (static_cast<uint32_t>(32 * q) << 16) +
                            static_cast<uint32_t>(a * p.ncols + j0),
                        v);
                    tmem_ld_wait();
                    if (!live) continue;
                    // 16 columns never straddle two output components (Qout is a multiple
                    // of 16): letter, sign and base address are fixed per half
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const int d0 = cg * p.ncols + j0 + 16 * h;
                        const int m = d0 / p.Qout, co0 = d0 - m * p.Qout;
                        const bool neg = ((p.sep ? SEP_NEG : NEG_MASK) >> (4 * m + pc)) & 1u;
                        float* dst = letter_ptr(p, p.sep ? pc : (m ^ pc)) + co0 * wstride + row_off;
#pragma unroll
                        for (int jj = 0; jj < 16; ++jj) {
                            const float val = __uint_as_float(v[16 * h + jj]);
                            atomicAdd(dst + jj * wstride, neg ? -val : val);
                        }
                    }
                }
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 2) {
        // the issuer's last commit covers every MMA it issued: wait for it (bounded) so no
        // MMA still writes the accumulators when they are released
        if (lane == 0) {
            const uint64_t t0 = global_timer_ns();
            while (!mbar_try_wait(done_bar, 0u)) {
                if (global_timer_ns() - t0 > limit) {
                    atomicOr(&g_status, STATUS_TIMEOUT_DRAIN);
                    break;
                }
            }
        }
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, p.tmem_cols);
    }
}

}  // namespace dwk
