// qconv_pw.cuh -- pointwise (1x1, stride 1 or 2) quaternion convolution on the tensor
// cores, the bandwidth path for the memory-bound pointwise layers (the backbone's 1x1/2
// shortcuts) and the wide pointwise neck layer.  Included by qconv_tc.cu inside its
// anonymous namespace.
//
// Orientation.  A 1x1 layer reads each input pixel once and writes each output pixel once,
// so what matters is streaming pixels at HBM speed, not reusing them on chip.  The MMA's
// M = 128 rows are output channels and its N = 256 columns are pixels:
//   D[R][pix] = sum over k of A[R][k] * X[pix][k],
//   A[32 q + j][p Qin + ci] = sign(q, p) W_{q xor p}[32 b + j][ci]      (Eq. 6)
// for the CTA's block b of 32 quaternion output channels (rows R = 32 q + j, channel
// c = q Qout + 32 b + j, so a TMEM lane quadrant is one output component and a warp's 32
// lanes are 32 consecutive output channels).  The expanded block weight of the CTA's block
// (128 x Cin bf16, at most 128 KB) is built once in shared memory from the letters
// (16-byte loads, the sign as an XOR of the sign bits); pixels stream through a ring of
// stages of 256 pixels x 64 input channels (32 KB, 128-byte swizzle), one TMA box each:
//   stride 1: the input viewed as [N H W][Cin]: 256 consecutive pixels;
//   stride 2: the input viewed as [N H / 2][2][W / 2][2][Cin] (even H and W): a box with
//             both parity coordinates 0 holds rows of the sampled pixels, so a tile is R
//             whole output rows (R Wo <= 256 consecutive output pixels) and only the
//             sampled pixels leave HBM.
// The epilogue reads one channel of 64 pixels per thread (tcgen05.ld 32 lanes x 32 bits)
// and stores 2-byte values: a warp's store covers 64 contiguous bytes (32 channels of one
// pixel).  Every CTA keeps one channel block for its whole run (the grid is a multiple of
// the number of blocks), and the blocks of one pixel tile run on neighbouring CTAs, so a
// pixel tile read for one block is still in L2 for the others.
//
// Roles (20 warps, one CTA per SM, persistent):
//   warp 0       TMA producer (one lane);
//   warp 1       TMEM owner and MMA issuer (one lane): per tile Cin / 16 MMAs of
//                128 x 256 x 16 into one of two 256-column accumulators;
//   warps 2..19  expand the block weight once;
//   warps 4..19  epilogue: four warps per TMEM lane quadrant, 64 pixels each.
// Waits are bounded like every kernel here (tc_common.cuh).

constexpr int PW_THREADS = 640;
constexpr int PW_NPIX = 256;          // pixels per tile (the MMA's N)
constexpr int PW_MAX_CIN = 512;       // the expanded block weight: 128 x Cin bf16 <= 128 KB
constexpr int PW_EXP_WARP0 = 2;
constexpr int PW_EXP_WARPS = 18;
constexpr int PW_EPI_WARP0 = 4;
constexpr int PW_EPI_THREADS = 512;

struct PwParams {
    ConvShape s;
    EpilogueArgs ep;
    const __nv_bfloat16* w[4];  // letter tensors [Qout][1][1][Qin]
    void* y;                    // output [N][Ho][Wo][Cout]
    unsigned long long wait_limit_ns;
    int inject_stall;
    int kchunks;      // Cin / 64
    int stages;       // ring stages
    int mblocks;      // Cout / 128
    int tile_pix;     // output pixels per tile (256, or R Wo for stride 2)
    int rows_per_tile;  // stride 2: output rows per tile
    int num_tiles;    // pixel tiles
    long long npix;   // N Ho Wo
};

struct PwCfg {
    static constexpr int CHUNK = 128 * 128;                // one 64-channel K chunk of A
    static constexpr int A_BYTES = (PW_MAX_CIN / 64) * CHUNK;
    static constexpr int STAGE = PW_NPIX * 128;            // 256 pixels x 64 channels
    static constexpr int MAX_STAGES = 8;
    // full, empty (per stage), accf, acce (2 buffers), drain, bready
    static constexpr int NUM_BARS = 2 * MAX_STAGES + 4 + 1 + 1;
    static constexpr int SMEM_BYTES = 227 * 1024;
    static constexpr uint32_t DESC_HI = desc_hi(8 * 128, desc_layout(128));
    static constexpr uint32_t TMEM_COLS = 512;
    // A (the expanded weight, kchunks x 16 KB) sits at 0, the barriers in the next 1 KB,
    // the ring after them; a_bytes depends on Cin
    static int ring_off(int kchunks) { return kchunks * CHUNK + 1024; }
    static int max_stages(int kchunks) {
        const int n = (SMEM_BYTES - 1024 - ring_off(kchunks)) / STAGE;
        return n < MAX_STAGES ? n : MAX_STAGES;
    }
    static_assert(NUM_BARS * 8 + 16 <= 1024, "pointwise barriers");
};

// Shapes the kernel covers (the full Hamilton form, no residual).
bool pw_ok(const ConvShape& s, const EpilogueArgs& ep) {
    if (s.sep || ep.residual || s.kh != 1 || s.kw != 1 || s.pad != 0) return false;
    if (s.Cin % 64 != 0 || s.Cin > PW_MAX_CIN || s.Cout % 128 != 0) return false;
    if (s.stride == 1) return true;
    if (s.stride != 2 || (s.H & 1) || (s.W & 1) || s.Wo > PW_NPIX) return false;
    return true;
}

// A[R][k] for the CTA's channel block, K-major 64-channel chunks of 128 rows x 128 bytes
// with the 128-byte swizzle (16-byte unit u of row R at unit u ^ (R mod 8)).  One 16-byte
// unit per item: eight consecutive input channels of one component, one letter row.
__device__ __forceinline__ void pw_expand(const PwParams& p, uint8_t* smem, int mb, int et,
                                          int lane, uint32_t bready_bar) {
    constexpr int ET = PW_EXP_WARPS * 32;
    const int Qin = p.s.Qin;
    const int upr = p.s.Cin / 8;  // units per row
    for (int i = et; i < 128 * upr; i += ET) {
        const int R = i & 127, U = i >> 7;  // consecutive threads: consecutive rows
        const int q = R >> 5, j = R & 31;
        const int k = 8 * U, pc = k / Qin, ci = k - pc * Qin;
        uint4 v = __ldg(reinterpret_cast<const uint4*>(
            p.w[q ^ pc] + static_cast<long long>(32 * mb + j) * Qin + ci));
        if ((NEG_MASK >> (4 * q + pc)) & 1u) v = negate_bf16x8(v);
        const int kc = U >> 3, u = U & 7;
        const uint32_t off = static_cast<uint32_t>(kc * PwCfg::CHUNK + R * 128 +
                                                   ((u ^ (R & 7)) << 4));
        *reinterpret_cast<uint4*>(smem + off) = v;
    }
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) mbar_arrive(bready_bar);
}

template <int STRIDE, int ACT>
__global__ void __launch_bounds__(PW_THREADS, 1)
    qconv_pw_kernel(const __grid_constant__ CUtensorMap tmap_x, const PwParams p) {
    using C = PwCfg;
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const uint32_t sbase = smem_u32(smem);
    const int a_bytes = p.kchunks * C::CHUNK;
    uint64_t* bars = reinterpret_cast<uint64_t*>(smem + a_bytes);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + C::NUM_BARS);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    const uint32_t bar0 = smem_u32(bars);
    auto full_bar = [&](int st) { return bar0 + 8u * st; };
    auto empty_bar = [&](int st) { return bar0 + 8u * (C::MAX_STAGES + st); };
    const uint32_t accf0 = bar0 + 8u * (2 * C::MAX_STAGES);
    const uint32_t acce0 = accf0 + 16u;
    const uint32_t drain_bar = acce0 + 16u;
    const uint32_t bready_bar = drain_bar + 8u;
    const uint32_t ring = sbase + static_cast<uint32_t>(a_bytes + 1024);

    const int warp = threadIdx.x / 32, lane = threadIdx.x % 32;
    const ConvShape& s = p.s;
    const uint64_t limit = p.wait_limit_ns;
    // this CTA's channel block and its pixel tiles t = t0, t0 + tstep, ...
    const int mb = blockIdx.x % p.mblocks;
    const int t0 = blockIdx.x / p.mblocks, tstep = gridDim.x / p.mblocks;

    griddep_launch_dependents();
    if (threadIdx.x == 0) {
        for (int i = 0; i < p.stages; ++i) {
            mbar_init(full_bar(i), 1);
            mbar_init(empty_bar(i), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(accf0 + 8u * b, 1);
            mbar_init(acce0 + 8u * b, PW_EPI_THREADS);
        }
        mbar_init(drain_bar, 1);
        mbar_init(bready_bar, PW_EXP_WARPS);
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
    // kernel's last CTAs; the producer and the epilogue wait for that kernel before their
    // first access to activations.

    if (warp == 0) {
        // ------------------------------------------------------------ TMA producer
        if (lane == 0) {
            griddep_wait();  // the previous kernel's output (this layer's input) is complete
            const uint64_t pol = l2_policy_evict_normal();
            uint32_t filled = 0, fill_parity = 0;
            bool ok = true;
            int st = 0;
            uint32_t phase = 0;
            for (int t = t0; ok && t < p.num_tiles; t += tstep) {
                for (int kc = 0; kc < p.kchunks; ++kc) {
                    if (!wait_or_abort(empty_bar(st), phase ^ 1u, limit, abort_flag,
                                       STATUS_TIMEOUT_PRODUCER)) {
                        ok = false;
                        break;
                    }
                    const uint32_t fb = full_bar(st);
                    mbar_arrive_expect_tx(fb, static_cast<uint32_t>(128 * p.tile_pix));
                    filled |= 1u << st;
                    fill_parity = (fill_parity & ~(1u << st)) | (phase << st);
                    const uint32_t dst = ring + static_cast<uint32_t>(st * C::STAGE);
                    if constexpr (STRIDE == 1)
                        tma_load_2d(dst, &tmap_x, fb, 64 * kc, t * p.tile_pix, pol);
                    else
                        tma_load_5d(dst, &tmap_x, fb, 64 * kc, 0, 0, 0, t * p.rows_per_tile,
                                    pol);
                    if (++st == p.stages) {
                        st = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (!ok || *abort_flag) drain_fills(full_bar(0), p.stages, filled, fill_parity, limit);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            constexpr uint32_t IDESC = make_idesc(BM, PW_NPIX, 0);
            bool ok = wait_or_abort(bready_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
            int issued = 0;
            if (p.inject_stall) {
                // Failure injection: wait on a barrier nothing arrives on.
                wait_or_abort(drain_bar, 0, limit, abort_flag, STATUS_TIMEOUT_MMA);
                ok = false;
            }
            tc_fence_after();
            const uint32_t a_lo0 = desc_lo(sbase);
            int st = 0, local = 0;
            uint32_t phase = 0;
            for (int t = t0; ok && t < p.num_tiles; t += tstep, ++local) {
                const int buf = local & 1;
                const uint32_t use = static_cast<uint32_t>(local >> 1) & 1u;
                if (!wait_or_abort(acce0 + 8u * buf, use ^ 1u, limit, abort_flag,
                                   STATUS_TIMEOUT_MMA)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d = tmem_base + static_cast<uint32_t>(buf * PW_NPIX);
                for (int kc = 0; kc < p.kchunks; ++kc) {
                    if (!wait_or_abort(full_bar(st), phase, limit, abort_flag,
                                       STATUS_TIMEOUT_MMA)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t b_lo = desc_lo(ring + static_cast<uint32_t>(st * C::STAGE));
                    const uint32_t a_lo = a_lo0 + static_cast<uint32_t>((kc * C::CHUNK) >> 4);
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk)  // 16-channel steps: 32 bytes into the row
                        umma_f16_w(d, a_lo + 2 * kk, C::DESC_HI, b_lo + 2 * kk, C::DESC_HI,
                                   IDESC, (kc | kk) != 0 ? 1u : 0u);
                    ++issued;
                    umma_commit(empty_bar(st));
                    if (++st == p.stages) {
                        st = 0;
                        phase ^= 1u;
                    }
                }
                if (!ok) break;
                umma_commit(accf0 + 8u * buf);
            }
            if (!ok && issued > 0) {
                // let the issued MMAs finish before TMEM is released
                umma_commit(drain_bar);
                const uint64_t t1 = global_timer_ns();
                while (!mbar_try_wait(drain_bar, 0u)) {
                    if (global_timer_ns() - t1 > limit) {
                        atomicOr(&g_status, STATUS_TIMEOUT_DRAIN);
                        break;
                    }
                }
            }
        }
    } else {
        pw_expand(p, smem, mb, (warp - PW_EXP_WARP0) * 32 + lane, lane, bready_bar);
        griddep_wait();  // the output buffer no longer read by the previous kernel
        if (warp >= PW_EPI_WARP0) {
            // -------------------------------------------------------- epilogue
            const int qd = warp & 3;                     // TMEM lane quadrant: component
            const int part = (warp - PW_EPI_WARP0) >> 2;  // pixels 64 part .. 64 part + 63
            const int c = qd * s.Qout + 32 * mb + lane;  // real output channel
            const float sc = p.ep.scale ? __ldg(p.ep.scale + c) : 1.0f;
            const float bias = p.ep.bias ? __ldg(p.ep.bias + c) : 0.0f;
            const float sh = fmaf(sc, bias, p.ep.scale ? __ldg(p.ep.shift + c) : 0.0f);
            __nv_bfloat16* out = static_cast<__nv_bfloat16*>(p.y);
            const long long Cout = s.Cout;
            int local = 0;
            for (int t = t0; t < p.num_tiles; t += tstep, ++local) {
                const int buf = local & 1;
                const uint32_t use = static_cast<uint32_t>(local >> 1) & 1u;
                bool ok = true;
                if (lane == 0)
                    ok = wait_or_abort(accf0 + 8u * buf, use, limit, abort_flag,
                                       STATUS_TIMEOUT_EPILOGUE);
                if (__shfl_sync(0xffffffffu, ok ? 1 : 0, 0) == 0) break;
                tc_fence_after();
                const uint32_t taddr = tmem_base + (static_cast<uint32_t>(qd * 32) << 16) +
                                       static_cast<uint32_t>(buf * PW_NPIX + 64 * part);
                uint32_t v0[32], v1[32];
                tmem_ld_32x32b_x32(taddr, v0);
                tmem_ld_32x32b_x32(taddr + 32, v1);
                tmem_ld_wait();
                // the accumulator is in registers: hand the buffer back to the issuer
                tc_fence_before();
                mbar_arrive_relaxed(acce0 + 8u * buf);
                const long long pix0 = static_cast<long long>(t) * p.tile_pix;
                long long left = p.npix - pix0;
                if (left > p.tile_pix) left = p.tile_pix;
                const int n0 = 64 * part;  // this warp's first column
                __nv_bfloat16* op = out + (pix0 + n0) * Cout + c;
                if (n0 + 64 <= left) {  // warp-uniform: all 64 columns are pixels
#pragma unroll
                    for (int k = 0; k < 32; ++k) {
                        const float z = activate(fmaf(sc, __uint_as_float(v0[k]), sh), ACT);
                        st_global_na_bf16(op + k * Cout, __float2bfloat16_rn(z));
                    }
#pragma unroll
                    for (int k = 0; k < 32; ++k) {
                        const float z = activate(fmaf(sc, __uint_as_float(v1[k]), sh), ACT);
                        st_global_na_bf16(op + (32 + k) * Cout, __float2bfloat16_rn(z));
                    }
                } else {
#pragma unroll
                    for (int k = 0; k < 32; ++k)
                        if (n0 + k < left) {
                            const float z = activate(fmaf(sc, __uint_as_float(v0[k]), sh), ACT);
                            st_global_na_bf16(op + k * Cout, __float2bfloat16_rn(z));
                        }
#pragma unroll
                    for (int k = 0; k < 32; ++k)
                        if (n0 + 32 + k < left) {
                            const float z = activate(fmaf(sc, __uint_as_float(v1[k]), sh), ACT);
                            st_global_na_bf16(op + (32 + k) * Cout, __float2bfloat16_rn(z));
                        }
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
