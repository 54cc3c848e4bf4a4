// hcw_tc.cu -- tensor-core (tcgen05 + TMEM + TMA) kernels of the
// rotated-hypercube mixing layer, bf16 operands, fp32 accumulation.
//
// One persistent, warp-specialised kernel serves the three contractions of
// a layer (Sec. 3.1 wiring, Eq. (1) maps, chain-rule backward):
//
//   FWD  z_i  = x_i W_self^T + m_i x_{p(i)} W_nbr^T (+ bias), y = act(z) (+ x_i)
//   DX   dx_i = dz_i W_self + m_{p(i)} dz_{p(i)} W_nbr (+ dy_i)
//   DW   dW_self = sum_i dz_i^T x_i,  dW_nbr = sum_i m_i dz_i^T x_{p(i)}
//
// Partner tiles without a gather.  For the link distance k = 2^s, the token
// axis [B*n] is viewed as the 4-D tensor (d, lo = k, bit = 2, HI = B*n/(2k))
// (all strides multiples of 16 bytes).  One TMA box (64 features, lo_box, 1,
// hi_box) holds 128 (or 64) positions that share bit s; the box with the
// other bit value at the same (lo, HI) coordinates holds exactly their
// partners, row for row.  So a CTA owning 128 positions with bit s = beta
// computes
//      [x_beta | x_{1-beta}] . [W_self ; W_nbr]
// as ONE accumulation over K = 2d (self part, then partner part) into a
// single TMEM accumulator, and the causal rule (Sec. 3.1: only positions
// with bit s set receive) becomes "rows with bit 0 skip the partner part":
// 3d^2 instead of 4d^2 flops per token, no masked work.
//
// DX is the mirror image: position i takes dz_{p(i)} exactly when p(i)
// received from i (m_{p(i)} = 1), which for causal layers is bit s of i
// being 0.  Because p is an involution this is again a pure gather: every
// dx row is owned by one CTA, no atomics.
//
// DW contracts over tokens: A = dz^T and B = x^T (or the partner rows of x)
// are loaded as MN-major operands straight from the token-major activations;
// the token range is split so that the units fill the GPU, and the fp32
// partials are reduced in a fixed order by a separate kernel
// (deterministic).
//
// Roles (192 threads): warp 0 issues TMA loads into a STAGES-deep ring of
// shared-memory stages; warp 1 owns TMEM (2 x BN fp32 columns, a double
// buffered accumulator) and issues tcgen05.mma; warps 2..5 drain the
// accumulator through tcgen05.ld, apply the epilogue and store.  Every wait
// is bounded (hcw_ptx.cuh); a CTA that gives up records HCW_ERR_TIMEOUT,
// drains its in-flight copies and MMAs, frees TMEM and returns.
#include "hcw_internal.h"
#include "hcw_ptx.cuh"

namespace hcw {

namespace {

constexpr int kEpiWarps = 8;                       // two per TMEM lane quarter
constexpr int kThreads = 64 + 32 * kEpiWarps;      // producer, MMA, epilogue warps
constexpr int kBlockM = 128;
constexpr int kBlockK = 64;                        // bf16 elements per 128-byte row
constexpr int kABytes = kBlockM * kBlockK * 2;     // 16 KB
constexpr int kRingBytes = 192 * 1024;             // TMA stage ring
constexpr int kEpiBufBytes = 4096;                 // per epilogue warp: 32 rows x 128 B

__host__ __device__ constexpr int stage_bytes(int BN) { return kABytes + BN * kBlockK * 2; }
__host__ __device__ constexpr int num_stages(int BN) {
    return (kRingBytes / stage_bytes(BN)) > 8 ? 8 : (kRingBytes / stage_bytes(BN));
}

struct __align__(8) Barriers {
    uint64_t full[8];
    uint64_t empty[8];
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
};

template <int BN>
__host__ __device__ constexpr size_t smem_total() {
    return 1024 /* alignment slack */ + (size_t)num_stages(BN) * stage_bytes(BN) +
           (size_t)kEpiWarps * kEpiBufBytes + sizeof(Barriers);
}

// FWD/DX unit -> (row bit beta, row block t, column tile j, number of K steps)
struct RowUnit {
    int beta, t, j, steps;
};

__device__ __forceinline__ RowUnit decode_row_unit(const TcParams& p, int u) {
    RowUnit r;
    const int per_bit = p.n_rb * p.n_nt;
    int rem;
    if (u < p.n_full * per_bit) {
        const int g = u / per_bit;
        rem = u - g * per_bit;
        r.beta = g == 0 ? p.full_bit0 : p.full_bit1;
        r.steps = 2 * p.nK;
    } else {
        rem = u - p.n_full * per_bit;
        r.beta = p.half_bit;
        r.steps = p.nK;
    }
    r.t = rem / p.n_nt;
    r.j = rem - r.t * p.n_nt;
    return r;
}

// DW unit -> (which: 0 self / 1 partner, o tile, k tile, split, kb range)
struct WUnit {
    int which, ot, nt, split, kb0, kb1;
};

__device__ __forceinline__ WUnit decode_w_unit(const TcParams& p, int u) {
    WUnit w;
    const int tiles = p.n_ot * p.n_nt;
    const int units_self = p.splits_self * tiles;
    int rem;
    if (u < units_self) {
        w.which = 0;
        rem = u;
    } else {
        w.which = 1;
        rem = u - units_self;
    }
    w.split = rem / tiles;
    rem -= w.split * tiles;
    w.ot = rem / p.n_nt;
    w.nt = rem - w.ot * p.n_nt;
    const int nkb = w.which ? p.nkb_nbr : p.nkb_self;
    w.kb0 = w.split * p.kb_per_unit;
    w.kb1 = min(nkb, w.kb0 + p.kb_per_unit);
    return w;
}

// ---- epilogue staging ------------------------------------------------------
// Each epilogue warp owns 32 accumulator rows (one per lane, as tcgen05.ld
// delivers them) and moves them through a private 4 KB shared buffer so that
// global loads and stores are whole-line and coalesced.  Rows are 16-byte
// pieces XOR-swizzled by row so that both the row-wise accesses (a lane per
// row) and the line-wise accesses (lanes along a row) are conflict-free.
//   bf16 chunk: 32 rows x 32 values = 32 x 64 B, piece m of row r at word
//               16 r + 4 (m ^ ((r >> 1) & 3))
//   fp32 chunk: 32 rows x 32 values = 32 x 128 B, piece m of row r at word
//               32 r + 4 (m ^ (r & 7))
__device__ __forceinline__ uint32_t* bf16_piece(uint32_t* buf, int r, int m) {
    return buf + 16 * r + 4 * (m ^ ((r >> 1) & 3));
}
__device__ __forceinline__ uint32_t* f32_piece(uint32_t* buf, int r, int m) {
    return buf + 32 * r + 4 * (m ^ (r & 7));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
    __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    return *reinterpret_cast<uint32_t*>(&h);
}

__device__ __forceinline__ float2 unpack_bf16x2(uint32_t w) {
    __nv_bfloat162 h = *reinterpret_cast<__nv_bfloat162*>(&w);
    return __bfloat1622float2(h);
}

// Lane `lane` writes its row (32 bf16 given as 16 packed words) into the buffer.
__device__ __forceinline__ void stage_row_bf16(uint32_t* buf, int lane, const uint32_t (&w)[16]) {
#pragma unroll
    for (int m = 0; m < 4; ++m)
        *reinterpret_cast<uint4*>(bf16_piece(buf, lane, m)) =
            make_uint4(w[4 * m], w[4 * m + 1], w[4 * m + 2], w[4 * m + 3]);
}

__device__ __forceinline__ void read_row_bf16(const uint32_t* buf, int lane, uint32_t (&w)[16]) {
#pragma unroll
    for (int m = 0; m < 4; ++m) {
        uint4 u = *reinterpret_cast<const uint4*>(bf16_piece(const_cast<uint32_t*>(buf), lane, m));
        w[4 * m] = u.x;
        w[4 * m + 1] = u.y;
        w[4 * m + 2] = u.z;
        w[4 * m + 3] = u.w;
    }
}

// Line-wise mapping of a bf16 chunk: iteration it (0..3), lane -> row
// 8 it + lane / 4, piece lane % 4 (16 bytes of the row's 64).
__device__ __forceinline__ int line_row_bf16(int it, int lane) { return 8 * it + (lane >> 2); }

// Wait for this thread's tcgen05.ld and tie the destination registers to the
// wait so the compiler cannot read them earlier.
__device__ __forceinline__ void tmem_ld_wait_regs(uint32_t (&r)[32]) {
    asm volatile("tcgen05.wait::ld.sync.aligned;"
                 : "+r"(r[0]), "+r"(r[1]), "+r"(r[2]), "+r"(r[3]), "+r"(r[4]), "+r"(r[5]),
                   "+r"(r[6]), "+r"(r[7]), "+r"(r[8]), "+r"(r[9]), "+r"(r[10]), "+r"(r[11]),
                   "+r"(r[12]), "+r"(r[13]), "+r"(r[14]), "+r"(r[15]), "+r"(r[16]),
                   "+r"(r[17]), "+r"(r[18]), "+r"(r[19]), "+r"(r[20]), "+r"(r[21]),
                   "+r"(r[22]), "+r"(r[23]), "+r"(r[24]), "+r"(r[25]), "+r"(r[26]),
                   "+r"(r[27]), "+r"(r[28]), "+r"(r[29]), "+r"(r[30]), "+r"(r[31])
                 :
                 : "memory");
}

// Wait that only gives up on time (used to drain in-flight work after an
// abort, when the abort flag is already set).
__device__ __forceinline__ bool mbar_wait_drain(uint64_t* bar, uint32_t parity,
                                                uint64_t timeout_ns) {
    const uint64_t t0 = globaltimer_ns();
    while (!mbar_try_wait(bar, parity)) {
        if (globaltimer_ns() - t0 > timeout_ns) return false;
    }
    return true;
}

}  // namespace

// tmA : FWD x, DX dz: 4-D rows map, box (64, lo_box, 1, hi_box), 128 rows.
//       DW dz: same map shape with 64-token boxes.
// tmB0: FWD W_self [o][k] 2-D, box (64 k, BN o)   (K-major B)
//       DX  W_self [o][k] 2-D, box (64 k, 64 o)   (MN-major B, BN/64 boxes)
//       DW  x 4-D rows map with 64-token boxes    (MN-major B, BN/64 boxes)
// tmB1: FWD/DX W_nbr like tmB0; DW unused.
template <int MODE, int BN>
__global__ void __launch_bounds__(kThreads, 1)
    hcw_tc_kernel(const __grid_constant__ CUtensorMap tmA,
                  const __grid_constant__ CUtensorMap tmB0,
                  const __grid_constant__ CUtensorMap tmB1, const TcParams p) {
    constexpr int STAGES = num_stages(BN);
    constexpr int SB = stage_bytes(BN);
    constexpr int B_BYTES = BN * kBlockK * 2;
    constexpr uint32_t TMEM_COLS = 2 * BN;
    constexpr uint32_t IDESC = idesc_bf16_f32(kBlockM, BN, MODE == MODE_DW ? 1 : 0,
                                              MODE == MODE_FWD ? 0 : 1);

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint8_t* epi_smem = smem + (size_t)STAGES * SB;
    Barriers* bars =
        reinterpret_cast<Barriers*>(epi_smem + (size_t)kEpiWarps * kEpiBufBytes);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB0);
        if (MODE != MODE_DW) tma_prefetch_desc(&tmB1);
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&bars->full[s], 1);
            mbar_init(&bars->empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&bars->tfull[a], 1);
            mbar_init(&bars->tempty[a], kEpiWarps);
        }
        mbar_init(&bars->drain, 1);
        bars->abort = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc(&bars->tmem_base, TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = bars->tmem_base;
    volatile int* abort = &bars->abort;
    const uint64_t tmo = p.timeout_ns;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued_mask = 0, issued_phase = 0;
            bool ok = true;
            for (int u = blockIdx.x; u < p.n_units && ok; u += gridDim.x) {
                if (MODE != MODE_DW) {
                    const RowUnit r = decode_row_unit(p, u);
                    const int q0 = r.t * kBlockM;
                    const int lo0 = q0 % p.k, hi0 = q0 / p.k;
                    for (int ks = 0; ks < r.steps; ++ks) {
                        if (!mbar_wait(&bars->empty[stage], phase ^ 1, abort, tmo)) {
                            ok = false;
                            break;
                        }
                        uint8_t* sA = smem + (size_t)stage * SB;
                        uint8_t* sB = sA + kABytes;
                        mbar_arrive_expect_tx(&bars->full[stage], kABytes + B_BYTES);
                        issued_mask |= 1u << stage;
                        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
                        const int part = ks >= p.nK;
                        const int kk = part ? ks - p.nK : ks;
                        const int bitA = part ? 1 - r.beta : r.beta;
                        tma_load_4d(sA, &tmA, &bars->full[stage], kk * kBlockK, lo0, bitA, hi0);
                        const CUtensorMap* mb = part ? &tmB1 : &tmB0;
                        if (MODE == MODE_FWD) {
                            tma_load_2d(sB, mb, &bars->full[stage], kk * kBlockK, r.j * BN);
                        } else {
#pragma unroll
                            for (int jj = 0; jj < BN / 64; ++jj)
                                tma_load_2d(sB + jj * 8192, mb, &bars->full[stage],
                                            r.j * BN + jj * 64, kk * kBlockK);
                        }
                        if (++stage == STAGES) {
                            stage = 0;
                            phase ^= 1;
                        }
                    }
                } else {
                    const WUnit w = decode_w_unit(p, u);
                    for (int kb = w.kb0; kb < w.kb1; ++kb) {
                        if (!mbar_wait(&bars->empty[stage], phase ^ 1, abort, tmo)) {
                            ok = false;
                            break;
                        }
                        int bA, bB, qb;
                        if (w.which == 0) {
                            bA = kb >= p.qb;
                            qb = kb - bA * p.qb;
                            bB = bA;
                        } else if (p.causal) {
                            bA = 1;
                            bB = 0;
                            qb = kb;
                        } else {
                            bA = kb >= p.qb;
                            qb = kb - bA * p.qb;
                            bB = 1 - bA;
                        }
                        const int q0 = qb * 64;
                        const int lo0 = q0 % p.k, hi0 = q0 / p.k;
                        uint8_t* sA = smem + (size_t)stage * SB;
                        uint8_t* sB = sA + kABytes;
                        mbar_arrive_expect_tx(&bars->full[stage], kABytes + B_BYTES);
                        issued_mask |= 1u << stage;
                        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
                        tma_load_4d(sA, &tmA, &bars->full[stage], w.ot * kBlockM, lo0, bA, hi0);
                        tma_load_4d(sA + 8192, &tmA, &bars->full[stage], w.ot * kBlockM + 64, lo0,
                                    bA, hi0);
#pragma unroll
                        for (int jj = 0; jj < BN / 64; ++jj)
                            tma_load_4d(sB + jj * 8192, &tmB0, &bars->full[stage],
                                        w.nt * BN + jj * 64, lo0, bB, hi0);
                        if (++stage == STAGES) {
                            stage = 0;
                            phase ^= 1;
                        }
                    }
                }
            }
            if (!ok) {
                // let every copy this thread started land before the CTA exits
                for (int s = 0; s < STAGES; ++s)
                    if (issued_mask & (1u << s))
                        mbar_wait_drain(&bars->full[s], (issued_phase >> s) & 1u, tmo);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true, any = false;
            for (int u = blockIdx.x; u < p.n_units && ok; u += gridDim.x) {
                int steps;
                if (MODE != MODE_DW) {
                    steps = decode_row_unit(p, u).steps;
                } else {
                    const WUnit w = decode_w_unit(p, u);
                    steps = w.kb1 - w.kb0;
                }
                if (!mbar_wait(&bars->tempty[acc], acc_phase ^ 1, abort, tmo)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * BN);
                for (int ks = 0; ks < steps; ++ks) {
                    if (!mbar_wait(&bars->full[stage], phase, abort, tmo)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a_addr = smem_u32(smem + (size_t)stage * SB);
                    const uint32_t b_addr = a_addr + kABytes;
#pragma unroll
                    for (int kk = 0; kk < kBlockK / 16; ++kk) {
                        uint64_t adesc, bdesc;
                        if (MODE == MODE_DW)
                            adesc = smem_desc_sw128(a_addr + kk * 2048, 8192, 1024);
                        else
                            adesc = smem_desc_sw128(a_addr + kk * 32, 16, 1024);
                        if (MODE == MODE_FWD)
                            bdesc = smem_desc_sw128(b_addr + kk * 32, 16, 1024);
                        else
                            bdesc = smem_desc_sw128(b_addr + kk * 2048, 8192, 1024);
                        mma_bf16_f32(d_tmem, adesc, bdesc, IDESC, (ks | kk) != 0);
                    }
                    any = true;
                    mma_commit(&bars->empty[stage]);
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
                if (!ok) break;
                mma_commit(&bars->tfull[acc]);
                acc ^= 1;
                if (acc == 0) acc_phase ^= 1;
            }
            if (!ok && any) {
                // wait for the MMAs already issued before TMEM is released
                mma_commit(&bars->drain);
                mbar_wait_drain(&bars->drain, 0, tmo);
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue
        // Warp e (0..7) drains TMEM lane quarter warp % 4 (rows 32 q .. 32 q + 31
        // of the tile) and column half e / 4, in chunks of 32 columns.
        const int e = warp - 2;
        const int quarter = warp & 3;
        const int half = e >> 2;
        constexpr int NCH = BN / 64;                  // chunks per column half
        uint32_t* buf = reinterpret_cast<uint32_t*>(epi_smem + (size_t)e * kEpiBufBytes);
        int acc = 0;
        uint32_t acc_phase = 0;
        for (int u = blockIdx.x; u < p.n_units; u += gridDim.x) {
            // one lane waits, the warp follows its verdict (tcgen05.ld is warp-wide)
            int ok = 1;
            if (lane == 0) ok = mbar_wait(&bars->tfull[acc], acc_phase, abort, tmo);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) break;
            tc_fence_after();
            const uint32_t t_base = tmem_base + ((uint32_t)(quarter * 32) << 16) +
                                    (uint32_t)(acc * BN + half * (BN / 2));
            if (MODE != MODE_DW) {
                const RowUnit r = decode_row_unit(p, u);
                // tokens of this warp's 32 rows, as seen by the line-wise lanes
                // (row 8 it + lane / 4 for it = 0..3); -1 marks rows past the end
                long long tok_line[4];
#pragma unroll
                for (int it = 0; it < 4; ++it) {
                    const int q = r.t * kBlockM + quarter * 32 + line_row_bf16(it, lane);
                    tok_line[it] = q < p.Mh ? ((long long)(q >> p.s) << (p.s + 1)) +
                                                  ((long long)r.beta << p.s) + (q & (p.k - 1))
                                            : -1;
                }
                const int col_half = r.j * BN + half * (BN / 2);
                const bool has_res = (p.flags & 2u) != 0;
                const bool has_zp = MODE == MODE_DX && p.dz_out != nullptr;
                uint4 res_g[4], zp_g[4];
                auto load_lines = [&](const __nv_bfloat16* src, int c, uint4 (&g)[4]) {
#pragma unroll
                    for (int it = 0; it < 4; ++it) {
                        g[it] = make_uint4(0, 0, 0, 0);
                        if (tok_line[it] >= 0)
                            g[it] = __ldg(reinterpret_cast<const uint4*>(
                                src + tok_line[it] * p.d + col_half + c * 32 + 8 * (lane & 3)));
                    }
                };
                // line-wise registers -> per-row words (through the buffer)
                auto to_rows = [&](const uint4 (&g)[4], uint32_t (&w)[16]) {
#pragma unroll
                    for (int it = 0; it < 4; ++it)
                        *reinterpret_cast<uint4*>(
                            bf16_piece(buf, line_row_bf16(it, lane), lane & 3)) = g[it];
                    __syncwarp();
                    read_row_bf16(buf, lane, w);
                    __syncwarp();
                };
                // per-row words -> coalesced line stores (through the buffer)
                auto store_rows = [&](__nv_bfloat16* dst, int c, const uint32_t (&w)[16]) {
                    stage_row_bf16(buf, lane, w);
                    __syncwarp();
#pragma unroll
                    for (int it = 0; it < 4; ++it) {
                        const uint4 v = *reinterpret_cast<const uint4*>(
                            bf16_piece(buf, line_row_bf16(it, lane), lane & 3));
                        if (tok_line[it] >= 0)
                            *reinterpret_cast<uint4*>(dst + tok_line[it] * p.d + col_half +
                                                      c * 32 + 8 * (lane & 3)) = v;
                    }
                    __syncwarp();
                };
                if (has_res) load_lines(p.resid, 0, res_g);
                if (has_zp) load_lines(p.zprev, 0, zp_g);
#pragma unroll 1
                for (int c = 0; c < NCH; ++c) {
                    uint32_t raw[32];
                    tmem_ld_32x32b_x32(t_base + c * 32, raw);
                    tmem_ld_wait_regs(raw);
                    if (c == NCH - 1) {
                        // the accumulator is drained: hand it back to the MMA warp
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&bars->tempty[acc]);
                    }
                    uint32_t res_w[16], zp_w[16];
                    if (has_res) to_rows(res_g, res_w);
                    if (has_zp) to_rows(zp_g, zp_w);
                    if (c + 1 < NCH) {   // prefetch the next chunk's inputs
                        if (has_res) load_lines(p.resid, c + 1, res_g);
                        if (has_zp) load_lines(p.zprev, c + 1, zp_g);
                    }
                    float v[32];
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(raw[i]);
                    uint32_t w[16];
                    if (MODE == MODE_FWD) {
                        if (p.bias) {
                            const float4* b4 =
                                reinterpret_cast<const float4*>(p.bias + col_half + c * 32);
#pragma unroll
                            for (int i = 0; i < 8; ++i) {
                                const float4 bb = __ldg(b4 + i);
                                v[4 * i] += bb.x;
                                v[4 * i + 1] += bb.y;
                                v[4 * i + 2] += bb.z;
                                v[4 * i + 3] += bb.w;
                            }
                        }
                        if (p.zout) {
#pragma unroll
                            for (int i = 0; i < 16; ++i) w[i] = pack_bf16x2(v[2 * i], v[2 * i + 1]);
                            store_rows(p.zout, c, w);
                        }
                        if (p.flags & 4u) {
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] = v[i] > 0.f ? v[i] : 0.f;
                        }
                    }
                    if (has_res) {
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const float2 f = unpack_bf16x2(res_w[i]);
                            v[2 * i] += f.x;
                            v[2 * i + 1] += f.y;
                        }
                    }
#pragma unroll
                    for (int i = 0; i < 16; ++i) w[i] = pack_bf16x2(v[2 * i], v[2 * i + 1]);
                    if (p.out) store_rows(p.out, c, w);
                    if (has_zp) {
                        // fused ReLU gradient of the layer below: dz = g * (z > 0)
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const float2 zz = unpack_bf16x2(zp_w[i]);
                            const uint32_t lo = zz.x > 0.f ? (w[i] & 0xFFFFu) : 0u;
                            const uint32_t hi = zz.y > 0.f ? (w[i] & 0xFFFF0000u) : 0u;
                            w[i] = lo | hi;
                        }
                        store_rows(p.dz_out, c, w);
                    }
                }
            } else {
                const WUnit w = decode_w_unit(p, u);
                const int S = w.which ? p.splits_nbr : p.splits_self;
                float* dst_base;
                if (S == 1)
                    dst_base = w.which ? p.dw_nbr : p.dw_self;
                else
                    dst_base = p.dw_partial + ((size_t)w.which * p.splits_max + w.split) *
                                                  (size_t)p.d * p.d;
                const int o0 = w.ot * kBlockM + quarter * 32;
                const int col_half = w.nt * BN + half * (BN / 2);
#pragma unroll 1
                for (int c = 0; c < NCH; ++c) {
                    uint32_t raw[32];
                    tmem_ld_32x32b_x32(t_base + c * 32, raw);
                    tmem_ld_wait_regs(raw);
                    if (c == NCH - 1) {
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(&bars->tempty[acc]);
                    }
#pragma unroll
                    for (int m = 0; m < 8; ++m)
                        *reinterpret_cast<uint4*>(f32_piece(buf, lane, m)) =
                            make_uint4(raw[4 * m], raw[4 * m + 1], raw[4 * m + 2], raw[4 * m + 3]);
                    __syncwarp();
#pragma unroll
                    for (int it = 0; it < 8; ++it) {
                        const int rr = 4 * it + (lane >> 3);
                        const uint4 v =
                            *reinterpret_cast<const uint4*>(f32_piece(buf, rr, lane & 7));
                        if (o0 + rr < p.d)
                            *reinterpret_cast<uint4*>(dst_base + (size_t)(o0 + rr) * p.d +
                                                      col_half + c * 32 + 4 * (lane & 7)) = v;
                    }
                    __syncwarp();
                }
            }
            acc ^= 1;
            if (acc == 0) acc_phase ^= 1;
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(tmem_base, TMEM_COLS);
    }
}

template <int MODE, int BN>
static cudaError_t launch_one(const CUtensorMap& a, const CUtensorMap& b0, const CUtensorMap& b1,
                              const TcParams& p, int grid, cudaStream_t st) {
    constexpr size_t smem = smem_total<BN>();
    auto kern = hcw_tc_kernel<MODE, BN>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    kern<<<grid, kThreads, smem, st>>>(a, b0, b1, p);
    return cudaGetLastError();
}

cudaError_t launch_tc(int mode, int BN, const CUtensorMap& a, const CUtensorMap& b0,
                      const CUtensorMap& b1, const TcParams& p, int grid, cudaStream_t st) {
#define HCW_TC_CASE(M, N) \
    if (mode == M && BN == N) return launch_one<M, N>(a, b0, b1, p, grid, st);
    HCW_TC_CASE(MODE_FWD, 256)
    HCW_TC_CASE(MODE_FWD, 128)
    HCW_TC_CASE(MODE_FWD, 64)
    HCW_TC_CASE(MODE_DX, 256)
    HCW_TC_CASE(MODE_DX, 128)
    HCW_TC_CASE(MODE_DX, 64)
    HCW_TC_CASE(MODE_DW, 256)
    HCW_TC_CASE(MODE_DW, 128)
    HCW_TC_CASE(MODE_DW, 64)
#undef HCW_TC_CASE
    return cudaErrorInvalidValue;
}

size_t tc_smem_bytes(int BN) {
    return BN == 256 ? smem_total<256>() : BN == 128 ? smem_total<128>() : smem_total<64>();
}

int tc_stages(int BN) {
    return BN == 256 ? num_stages(256) : BN == 128 ? num_stages(128) : num_stages(64);
}

// ---------------------------------------------------------------- self-test
__global__ void wait_selftest_kernel(unsigned long long timeout_ns) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);
        abort_flag = 0;
        fence_mbar_init();
    }
    __syncthreads();
    // nothing ever arrives on `bar`: the bounded wait must give up and report
    if (threadIdx.x == 0) mbar_wait(&bar, 0, &abort_flag, timeout_ns);
    __syncthreads();
}

cudaError_t launch_wait_selftest(unsigned long long timeout_ns, cudaStream_t st) {
    wait_selftest_kernel<<<1, 32, 0, st>>>(timeout_ns);
    return cudaGetLastError();
}

cudaError_t error_word_read_clear(int* word) {
    const int zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(word, g_error_word, sizeof(int));
    if (e == cudaSuccess && *word) e = cudaMemcpyToSymbol(g_error_word, &zero, sizeof(int));
    return e;
}

}  // namespace hcw
