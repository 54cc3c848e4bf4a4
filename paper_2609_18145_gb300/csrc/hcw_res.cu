// hcw_res.cu -- resident stacked forward and input gradient of the
// rotated-hypercube mixing layer (Sec. 3.1 wiring, Eq. (1) maps, chain-rule
// backward) on pairs of SMs: bf16 operands, fp32 accumulation.
//
// Whole samples of n <= 256 positions fit in a pair's shared memory at
// d <= 512 (128 rows x 1 KB = 128 KB per CTA).  So a cluster of two CTAs
// takes 256 consecutive tokens and runs them through every layer of the
// launch without the activations leaving the chip between layers.  Per layer
// only the weights stream in (TMA, each CTA half of a column chunk); the
// epilogue writes the layer's output once (the saved activation that the
// backward pass reads) and puts it straight back into shared memory as the
// next layer's A operand.  Pairs never wait on one another.
//
// Partner rows without a gather.  The tile is K-major without swizzle, rows
// 16 bytes apart: 16-byte column chunk c of row r sits at c * 2048 + r * 16.
// In this layout the rows r - delta of all rows r form the same tile shifted
// by delta rows, i.e. one descriptor whose start moves by 16 delta bytes.  For
// the link distance delta = 2^sigma (in TMEM-lane space) the partner part of
// Eq. (1) is one MMA per K step over the shifted window, with a
// disable-output-lane vector that leaves only the receiving lanes.  Under the
// causal rule of Sec. 3.1 the lanes with bit sigma set receive from lane -
// delta; without it a second window at + delta serves the other lanes.  The
// disabled lanes read rows outside the tile (the ring before it and a guard
// after it keep those reads in bounds) and their results are discarded.  The
// price: the causal partner part is computed for all 128 lanes, of which 64
// keep it.  That is 4d^2 instead of 3d^2 flops per token, which the streaming
// kernel (hcw_tc.cu) avoids by grouping rows by bit.
//
// Rows to lanes.  For n <= 128, CTA r of the pair holds tokens r*128 ..
// r*128 + 127 of its tile (whole samples), and the partner of lane i is lane
// i ^ 2^s.  For n = 256 the same holds for s < 7.  A layer with s = 7 uses the
// other split (CTA = position bit 6; lane = bit 7, then bits 0..5), so that
// partners again share a CTA, at lane distance 64.  Between layers of
// different splits the rows go through global memory once, since the layer's
// output is stored there anyway: both CTAs meet on a barrier, then reload
// their new rows with TMA (64-token boxes, one 16-byte column chunk each).
//
// Input gradient.  This is the mirror image: a row gathers dz from its
// partner when the partner received from it.  The residual stream g (the
// gradient of a layer's output) stays in TMEM in fp32.  Layer l's MMAs
// accumulate onto g_l, so TMEM then holds g_{l-1} = g_l + dz_l W_self +
// (partner) dz_p W_nbr.  The epilogue forms dz_{l-1} = bf16(g_{l-1}) *
// mask_{l-1} as the next A operand and leaves g_{l-1} in place for the next
// layer's MMAs.  (The streaming kernels round g to bf16 at every layer; here
// it is rounded only where it leaves the chip.)
//
// Overlap.  For d >= 256 the N columns form two accumulators ("chunks"), each
// accumulated K block by K block (self product, then partner product of the
// block).  The epilogue of chunk 0 runs during chunk 1's MMAs and writes its
// columns into the A tile once those MMAs have passed the matching K blocks
// (the MMA thread commits when chunk 1 reaches the middle block).  The next
// layer's chunk 0 then runs its first half of the K blocks while chunk 1's
// epilogue runs.
//
// Roles (576 threads).
//   - Warp 0, lane 0: issues the TMA weight loads into a ring.  Both CTAs do
//     this, each loading its half of B; the copies complete on the leader's
//     barriers.
//   - Warp 1: owns TMEM; in the leader it issues the pair's MMAs.
//   - Warps 2..17: drain TMEM, four per lane quarter.
// Every wait is bounded.  A CTA that gives up records HCW_ERR_TIMEOUT, lets
// its in-flight copies and MMAs complete, and frees TMEM after a final
// cluster barrier.
#include <atomic>

#include "hcw.h"
#include "hcw_internal.h"
#include "hcw_ptx.cuh"

namespace hcw {

namespace {

constexpr int kRows = 128;                 // rows per CTA = TMEM lanes
constexpr int kEW = 16;                    // epilogue warps
constexpr int kThreads = 64 + 32 * kEW;    // 576
constexpr int kChunkBytes = kRows * 16;    // one 16-byte column chunk of the 128 rows
constexpr int kGuard = 1024;               // 64 rows x 16 bytes read past either end
constexpr int kSmemMax = 232448;

template <int D>
struct Geo {
    static constexpr int NCH = D >= 256 ? 2 : 1;       // accumulator chunks
    static constexpr int N = D / NCH;                   // MMA N (each CTA loads N/2 of B)
    static constexpr int WC = N / 4;                    // columns per epilogue warp per chunk
    static constexpr int SUB = WC / 32;                 // 32-column TMEM loads per chunk
    static constexpr int NK = D / 64;                   // 64-deep K blocks per part
    static constexpr int A_BYTES = (D / 8) * kChunkBytes;
    static constexpr int SB = (N / 2) * 64 * 2;         // one B stage (this CTA's half)
    static constexpr int BIAS_BYTES = 2 * D * 4;            // two layers' bias (forward)
    static constexpr int FIXED = 1024 /* alignment */ + A_BYTES + kGuard + BIAS_BYTES +
                                 256 /* barriers */;
    static constexpr int ST_RAW = (kSmemMax - FIXED) / SB;
    static constexpr int STAGES = ST_RAW > 8 ? 8 : ST_RAW;
    static constexpr size_t SMEM = (size_t)FIXED + (size_t)STAGES * SB;
    static constexpr uint32_t TMEM_COLS = D <= 128 ? 128 : (D <= 256 ? 256 : 512);
    static_assert(D % 128 == 0 && D <= 512, "resident widths");
    static_assert(WC % 32 == 0, "32-column TMEM loads");
    static_assert(STAGES >= 2 && STAGES * SB >= kGuard, "ring (also the guard before A)");
    static_assert(SMEM <= (size_t)kSmemMax, "shared memory budget");
};

struct __align__(8) ResBars {
    uint64_t full[8];
    uint64_t empty[8];
    uint64_t tfull[2];     // chunk h of a layer accumulated (both CTAs)
    uint64_t afree;        // chunk 1's MMAs have read the first half of the K blocks
    uint64_t aready[2];    // leader: both CTAs' A columns of chunk h written (2 x kEW arrivals)
    uint64_t xsync;        // both CTAs' outputs of a layer are in global memory
    uint64_t xload;        // the A tile of the next split has landed (TMA)
    uint64_t drain;
    uint32_t tmem_base;
    int abort;
};
static_assert(sizeof(ResBars) <= 256, "barrier block");

__host__ __device__ __forceinline__ bool alt_split(int s, int n) { return n == 256 && s == 7; }

// link distance of dimension s in TMEM-lane space: 2^sigma
__device__ __forceinline__ int lane_sigma(int s, int n) { return alt_split(s, n) ? 6 : s; }

// token held by TMEM lane `row` of CTA `rank` in pair tile `tile`
__device__ __forceinline__ int tok_of(int tile, int rank, int row, bool alt) {
    const int rho = alt ? (((row >> 6) << 7) | (rank << 6) | (row & 63)) : ((rank << 7) | row);
    return tile * 256 + rho;
}

// disable-output-lane words: bit j of word i set when bit sg of lane 32 i + j equals v
__device__ __forceinline__ void lane_mask(int sg, int v, uint32_t (&m)[4]) {
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        uint32_t w = 0;
        for (int j = 0; j < 32; ++j) w |= (uint32_t)((((i * 32 + j) >> sg) & 1) == v) << j;
        m[i] = w;
    }
}

__device__ __forceinline__ uint32_t and_mask_bf16x2(uint32_t w, uint32_t bits, int b) {
    const uint32_t keep = ((bits >> b) & 1u ? 0x0000FFFFu : 0u) |
                          ((bits >> (b + 1)) & 1u ? 0xFFFF0000u : 0u);
    return w & keep;
}

}  // namespace

template <int MODE, int D>
__global__ void __launch_bounds__(kThreads, 1) hcw_res_kernel(const __grid_constant__ ResLaunch L) {
    using G = Geo<D>;
    constexpr bool FWD = MODE == MODE_FWD;
    constexpr uint32_t IDESC = idesc_bf16_f32(2 * kRows, G::N, 0, FWD ? 0 : 1);
    constexpr int WPR = D / 32;   // ReLU mask words per row

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint8_t* ring = smem;
    uint8_t* A = smem + (size_t)G::STAGES * G::SB;
    float* bias_s = reinterpret_cast<float*>(A + G::A_BYTES + kGuard);   // [2][D]
    ResBars* bars = reinterpret_cast<ResBars*>(A + G::A_BYTES + kGuard + G::BIAS_BYTES);

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const int tile = (int)blockIdx.x >> 1;
    const bool causal = (L.flags & HCW_CAUSAL) != 0;
    const bool resid = (L.flags & HCW_RESIDUAL) != 0;
    const bool relu = (L.flags & HCW_ACT_RELU) != 0;

    if (threadIdx.x == 0) {
        for (int l = 0; l < L.n_layers; ++l) {
            tma_prefetch_desc(&L.wmap[l][0]);
            tma_prefetch_desc(&L.wmap[l][1]);
        }
        for (int s = 0; s < G::STAGES; ++s) {
            mbar_init(&bars->full[s], 1);
            mbar_init(&bars->empty[s], 1);
        }
        mbar_init(&bars->tfull[0], 1);
        mbar_init(&bars->tfull[1], 1);
        mbar_init(&bars->afree, 1);
        mbar_init(&bars->aready[0], 2 * kEW);
        mbar_init(&bars->aready[1], 2 * kEW);
        mbar_init(&bars->xsync, 2 * kEW);
        mbar_init(&bars->xload, 1);
        mbar_init(&bars->drain, 1);
        bars->abort = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc_pair(&bars->tmem_base, G::TMEM_COLS);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync_all();   // both CTAs' barriers exist before any cross-CTA access
    tc_fence_after();
    const uint32_t tmem_base = bars->tmem_base;
    volatile int* abort = &bars->abort;
    const uint64_t tmo = L.timeout_ns;

    if (warp == 0) {
        // ------------------------------------------------------------ producer (both CTAs)
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0, issued_mask = 0, issued_phase = 0;
            bool ok = true;
            for (int i = 0; i < L.n_layers && ok; ++i)
                for (int h = 0; h < G::NCH && ok; ++h)
                    for (int kb = 0; kb < G::NK && ok; ++kb) {
                        const int col = h * G::N + (int)rank * (G::N / 2);
                        for (int part = 0; part < 2; ++part) {
                            const CUtensorMap* m = &L.wmap[i][part];
                            if (!mbar_wait(&bars->empty[stage], phase ^ 1, abort, tmo)) {
                                ok = false;
                                break;
                            }
                            uint8_t* sB = ring + (size_t)stage * G::SB;
                            if (rank == 0) mbar_arrive_expect_tx(&bars->full[stage], 2 * G::SB);
                            issued_mask |= 1u << stage;
                            issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
                            const uint32_t fb = mapa_shared(&bars->full[stage], 0);
                            if (FWD)   // W[o][k]: 64 k x N/2 output rows, K-major
                                tma_load_2d_pair(sB, m, fb, kb * 64, col);
                            else       // W[o][k] read MN-major: 64 o rows x N/2 k columns
                                tma_load_3d_pair(sB, m, fb, 0, kb * 64, col / 64);
                            if (++stage == G::STAGES) {
                                stage = 0;
                                phase ^= 1;
                            }
                        }
                    }
            if (!ok && rank == 0) {
                // every copy of the pair completes on the leader's barriers: let them land
                for (int s = 0; s < G::STAGES; ++s)
                    if (issued_mask & (1u << s))
                        mbar_wait_drain(&bars->full[s], (issued_phase >> s) & 1u, tmo);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer (leader)
        if (lane == 0 && rank == 0) {
            int stage = 0;
            uint32_t phase = 0;
            bool ok = true, any = false;
            // the input gradient accumulates onto the residual stream g held in TMEM
            const bool init = !FWD && resid;
            const uint32_t a0 = smem_u32(A);
            for (int i = 0; i < L.n_layers && ok; ++i) {
                const int sg = lane_sigma(L.layer[i].s, L.n);
                const int delta = 1 << sg;
                // forward: receivers (bit sg set) take row - delta, and without the
                // causal rule the others take row + delta; the input gradient is the
                // mirror image (senders take the dz of row + delta first)
                uint32_t m1[4], m2[4];
                lane_mask(sg, FWD ? 0 : 1, m1);
                lane_mask(sg, FWD ? 1 : 0, m2);
                const int sh1 = FWD ? -delta : delta;
                const int sh2 = -sh1;
                const uint32_t par = (uint32_t)i & 1u;
                for (int h = 0; h < G::NCH && ok; ++h) {
                    const uint32_t d_tmem = tmem_base + (uint32_t)(h * G::N);
                    for (int kb = 0; kb < G::NK && ok; ++kb)
                        for (int part = 0; part < 2; ++part) {
                            if (h == 0 && part == 0 && (kb == 0 || (G::NCH == 2 && kb == G::NK / 2))) {
                                if (!mbar_wait_cluster(&bars->aready[kb == 0 ? 0 : 1], par, abort,
                                                       tmo)) {
                                    ok = false;
                                    break;
                                }
                                tc_fence_after();
                            }
                            if (!mbar_wait(&bars->full[stage], phase, abort, tmo)) {
                                ok = false;
                                break;
                            }
                            tc_fence_after();
                            const uint32_t b = smem_u32(ring + (size_t)stage * G::SB);
                            const uint32_t ab = a0 + (uint32_t)(kb * 8 * kChunkBytes);
                            auto bdesc = [&](int kk) {
                                return FWD ? smem_desc_sw128(b + kk * 32, 16, 1024)
                                           : smem_desc_sw128(b + kk * 2048, 8192, 1024);
                            };
                            auto adesc = [&](int kk, int shift) {
                                return smem_desc_rows16(
                                    ab + (uint32_t)(kk * 2 * kChunkBytes) + (uint32_t)(shift * 16),
                                    kChunkBytes);
                            };
                            // each stage's MMAs are one straight-line block: a branch
                            // between two tcgen05.mma of a stage halves the issue rate
                            if (part == 0) {
#pragma unroll
                                for (int kk = 0; kk < 4; ++kk)
                                    mma_bf16_f32_pair(d_tmem, adesc(kk, 0), bdesc(kk), IDESC,
                                                      (init || (kb | kk) != 0) ? 1u : 0u);
                            } else if (causal) {
#pragma unroll
                                for (int kk = 0; kk < 4; ++kk)
                                    mma_bf16_f32_pair_masked(d_tmem, adesc(kk, sh1), bdesc(kk),
                                                             IDESC, m1);
                            } else {
#pragma unroll
                                for (int kk = 0; kk < 4; ++kk) {
                                    mma_bf16_f32_pair_masked(d_tmem, adesc(kk, sh1), bdesc(kk),
                                                             IDESC, m1);
                                    mma_bf16_f32_pair_masked(d_tmem, adesc(kk, sh2), bdesc(kk),
                                                             IDESC, m2);
                                }
                            }
                            any = true;
                            mma_commit_pair(&bars->empty[stage], 3);
                            if (G::NCH == 2 && h == 1 && part == 1 && kb == G::NK / 2 - 1)
                                mma_commit_pair(&bars->afree, 3);
                            if (++stage == G::STAGES) {
                                stage = 0;
                                phase ^= 1;
                            }
                        }
                    if (!ok) break;
                    mma_commit_pair(&bars->tfull[h], 3);
                }
            }
            if (!ok && any) {
                // the pair's MMAs have completed before TMEM can be freed
                mma_commit_pair(&bars->drain, 1);
                mbar_wait_drain(&bars->drain, 0, tmo);
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue (both CTAs)
        // Warp e drains TMEM lane quarter warp % 4 (rows 32 q .. 32 q + 31) and,
        // of every chunk, the WC columns of slice e / 4.
        const int e = warp - 2;
        const int q = warp & 3;
        const int cs = e >> 2;
        const int row = q * 32 + lane;
        const int gw = e & 3;   // this warp within its group (the 4 warps of column slice cs)
        const uint32_t t_lane = tmem_base + ((uint32_t)(q * 32) << 16);
        const uint32_t aready_leader[2] = {mapa_shared(&bars->aready[0], 0),
                                           mapa_shared(&bars->aready[1], 0)};
        const uint32_t xs_own = mapa_shared(&bars->xsync, rank);
        const uint32_t xs_peer = mapa_shared(&bars->xsync, rank ^ 1u);
        uint32_t xs_phase = 0, xl_phase = 0;
        bool alive = true;

        auto col_of = [&](int h, int j) { return h * G::N + cs * G::WC + j * 32; };
        // 16-byte piece m (8 features) of the 32 columns at col, in this row of A
        auto apiece = [&](int col, int m) -> uint4* {
            return reinterpret_cast<uint4*>(A + (size_t)(col / 8 + m) * kChunkBytes + row * 16);
        };
        auto wait_all = [&](uint64_t* bar, uint32_t par) -> bool {
            const bool ok = mbar_wait(bar, par, abort, tmo);
            return __all_sync(0xffffffffu, ok) != 0;
        };
        auto wait_all_cluster = [&](uint64_t* bar, uint32_t par) -> bool {
            const bool ok = mbar_wait_cluster(bar, par, abort, tmo);
            return __all_sync(0xffffffffu, ok) != 0;
        };
        // this warp's A columns of chunk h (and its TMEM traffic) are done
        auto signal_ready = [&](int h) {
            fence_proxy_async_smem();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_remote(aready_leader[h]);
        };
        // The launch's input rows of the split `alt` into A (and, input gradient
        // with the residual, g into TMEM).
        auto load_input = [&](bool alt) {
            const int tok = tok_of(tile, (int)rank, row, alt);
#pragma unroll 1
            for (int h = 0; h < G::NCH; ++h)
#pragma unroll 1
                for (int j = 0; j < G::SUB; ++j) {
                    const int col = col_of(h, j);
                    if (FWD) {
                        const uint4* src = reinterpret_cast<const uint4*>(
                            static_cast<const __nv_bfloat16*>(L.in) + (size_t)tok * D + col);
                        uint4 v[4];
#pragma unroll
                        for (int m = 0; m < 4; ++m) v[m] = __ldg(src + m);
#pragma unroll
                        for (int m = 0; m < 4; ++m) *apiece(col, m) = v[m];
                    } else {
                        // g = the top layer's output gradient; dz = bf16(g) * mask
                        uint32_t g[32];
                        if (L.in_f32) {
                            const float4* src = reinterpret_cast<const float4*>(
                                static_cast<const float*>(L.in) + (size_t)tok * D + col);
#pragma unroll
                            for (int m = 0; m < 8; ++m) {
                                // written by the previous launch; this launch may
                                // overwrite it (split changes): no read-only cache
                                const float4 f = __ldcg(src + m);
                                g[4 * m] = __float_as_uint(f.x);
                                g[4 * m + 1] = __float_as_uint(f.y);
                                g[4 * m + 2] = __float_as_uint(f.z);
                                g[4 * m + 3] = __float_as_uint(f.w);
                            }
                        } else {
                            const uint4* src = reinterpret_cast<const uint4*>(
                                static_cast<const __nv_bfloat16*>(L.in) + (size_t)tok * D + col);
#pragma unroll
                            for (int m = 0; m < 4; ++m) {
                                const uint4 w = __ldg(src + m);
                                const uint32_t wv[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
                                for (int t = 0; t < 4; ++t) {
                                    const float2 f = unpack_bf16x2(wv[t]);
                                    g[8 * m + 2 * t] = __float_as_uint(f.x);
                                    g[8 * m + 2 * t + 1] = __float_as_uint(f.y);
                                }
                            }
                        }
                        if (resid) {
                            __syncwarp();
                            tmem_st_32x32b_x32(t_lane + (uint32_t)col, g);
                        }
                        const uint32_t bits =
                            L.in_mask ? __ldg(L.in_mask + (size_t)tok * WPR + col / 32) : ~0u;
                        uint32_t w[16];
#pragma unroll
                        for (int t = 0; t < 16; ++t)
                            w[t] = and_mask_bf16x2(
                                pack_bf16x2(__uint_as_float(g[2 * t]), __uint_as_float(g[2 * t + 1])),
                                bits, 2 * t);
                        uint4* dst = reinterpret_cast<uint4*>(L.in_dz + (size_t)tok * D + col);
#pragma unroll
                        for (int m = 0; m < 4; ++m) {
                            const uint4 v = make_uint4(w[4 * m], w[4 * m + 1], w[4 * m + 2], w[4 * m + 3]);
                            dst[m] = v;
                            *apiece(col, m) = v;
                        }
                    }
                }
            if (!FWD && resid) tmem_st_wait();
            signal_ready(0);
            if (G::NCH == 2) signal_ready(1);
        };

        load_input(alt_split(L.layer[0].s, L.n));

        for (int i = 0; i < L.n_layers && alive; ++i) {
            const ResLayer& ly = L.layer[i];
            const bool alt = alt_split(ly.s, L.n);
            const bool last = i == L.n_layers - 1;
            const bool alt_next = last ? alt : alt_split(L.layer[i + 1].s, L.n);
            const bool trans = !last && alt_next != alt;
            const bool to_a = !last && !trans;   // results go straight back into A
            const int tok = tok_of(tile, (int)rank, row, alt);
            const uint32_t par = (uint32_t)i & 1u;
            const int kind = ly.out_kind;
            // input gradient: the mask words of the layer below, fetched early
            uint32_t mw[G::NCH][G::SUB];
#pragma unroll
            for (int h = 0; h < G::NCH; ++h)
#pragma unroll
                for (int j = 0; j < G::SUB; ++j)
                    mw[h][j] = (!FWD && kind == RES_DZ && ly.mprev)
                                   ? __ldg(ly.mprev + (size_t)tok * WPR + col_of(h, j) / 32)
                                   : ~0u;
            // forward: this layer's bias into shared memory (buffer i & 1, last read
            // two layers back), one value a thread, visible after the barrier below
            float* bias_l = bias_s + (i & 1) * D;
            if (FWD) {
                const int t = e * 32 + lane;
                if (t < D) bias_l[t] = ly.bias ? __ldg(ly.bias + t) : 0.f;
                named_bar_sync(5, 32 * kEW);
            }
#pragma unroll 1
            for (int h = 0; h < G::NCH; ++h) {
                if (!wait_all(&bars->tfull[h], par)) {
                    alive = false;
                    break;
                }
                // chunk 0: A's first K blocks are free once chunk 1's MMAs have passed
                // them (the results go to A: as the next operand and to be stored)
                if (kind != RES_G && G::NCH == 2 && h == 0 && !wait_all(&bars->afree, par)) {
                    alive = false;
                    break;
                }
                tc_fence_after();
#pragma unroll 1
                for (int j = 0; j < G::SUB; ++j) {
                    const int col = col_of(h, j);
                    uint32_t raw[32];
                    __syncwarp();
                    tmem_ld_32x32b_x32(t_lane + (uint32_t)col, raw);
                    tmem_ld_wait_regs(raw);
                    float v[32];
#pragma unroll
                    for (int t = 0; t < 32; ++t) v[t] = __uint_as_float(raw[t]);
                    uint32_t w[16];
                    if (FWD) {
                        // z = acc + bias; mask bit (z > 0); act; + x (residual); bf16
                        const float4* b4 = reinterpret_cast<const float4*>(bias_l + col);
#pragma unroll
                        for (int m = 0; m < 8; ++m) {
                            const float4 bb = b4[m];
                            v[4 * m] += bb.x;
                            v[4 * m + 1] += bb.y;
                            v[4 * m + 2] += bb.z;
                            v[4 * m + 3] += bb.w;
                        }
                        if (ly.mout) {
                            uint32_t bits = 0;
#pragma unroll
                            for (int t = 0; t < 32; ++t) bits |= (v[t] > 0.f ? 1u : 0u) << t;
                            ly.mout[(size_t)tok * WPR + col / 32] = bits;
                        }
                        if (relu) {
#pragma unroll
                            for (int t = 0; t < 32; ++t) v[t] = v[t] > 0.f ? v[t] : 0.f;
                        }
                        if (resid) {
#pragma unroll
                            for (int m = 0; m < 4; ++m) {
                                const uint4 x4 = *apiece(col, m);
                                const uint32_t xw[4] = {x4.x, x4.y, x4.z, x4.w};
#pragma unroll
                                for (int t = 0; t < 4; ++t) {
                                    const float2 f = unpack_bf16x2(xw[t]);
                                    v[8 * m + 2 * t] += f.x;
                                    v[8 * m + 2 * t + 1] += f.y;
                                }
                            }
                        }
#pragma unroll
                        for (int t = 0; t < 16; ++t) w[t] = pack_bf16x2(v[2 * t], v[2 * t + 1]);
                    } else if (kind == RES_G) {
                        float4* dst = reinterpret_cast<float4*>(static_cast<float*>(ly.out) +
                                                                (size_t)tok * D + col);
#pragma unroll
                        for (int m = 0; m < 8; ++m)
                            dst[m] = make_float4(v[4 * m], v[4 * m + 1], v[4 * m + 2], v[4 * m + 3]);
                        continue;
                    } else {
                        // RES_DZ: dz_{l-1} = bf16(g) * mask_{l-1};  RES_DX: dx = bf16(g)
#pragma unroll
                        for (int t = 0; t < 16; ++t)
                            w[t] = and_mask_bf16x2(pack_bf16x2(v[2 * t], v[2 * t + 1]), mw[h][j],
                                                   2 * t);
                        if (trans && resid) {
                            float4* gs = reinterpret_cast<float4*>(L.gscratch + (size_t)tok * D + col);
#pragma unroll
                            for (int m = 0; m < 8; ++m)
                                gs[m] = make_float4(v[4 * m], v[4 * m + 1], v[4 * m + 2], v[4 * m + 3]);
                        }
                    }
#pragma unroll
                    for (int m = 0; m < 4; ++m)
                        *apiece(col, m) = make_uint4(w[4 * m], w[4 * m + 1], w[4 * m + 2], w[4 * m + 3]);
                }
                if (kind == RES_G) continue;
                if (to_a) signal_ready(h);
                // The group's 128 rows x WC columns are in A: store them to global
                // memory with row-contiguous pieces (lane = 8 rows x 4 chunks: per row
                // 64 contiguous bytes, per chunk 128 contiguous bytes of A).
                named_bar_sync(1 + cs, 128);
                {
                    constexpr int KCW = G::WC / 8;                   // chunks of the slice
                    constexpr int PIECES = kRows * KCW;              // 16-byte pieces
                    const int kc_base = col_of(h, 0) / 8;
                    __nv_bfloat16* ob = static_cast<__nv_bfloat16*>(ly.out);
#pragma unroll
                    for (int it = 0; it < PIECES / 128; ++it) {
                        const int blk = it * 4 + gw;                 // 32 pieces of this warp
                        const int r = (blk % (kRows / 8)) * 8 + (lane & 7);
                        const int kc = (blk / (kRows / 8)) * 4 + (lane >> 3);
                        const uint4 v4 = *reinterpret_cast<const uint4*>(
                            A + (size_t)(kc_base + kc) * kChunkBytes + r * 16);
                        const int tr = tok_of(tile, (int)rank, r, alt);
                        *reinterpret_cast<uint4*>(ob + (size_t)tr * D + (kc_base + kc) * 8) = v4;
                    }
                }
            }
            if (!alive) break;
            if (trans) {
                // every output of the pair is in global memory: meet, then reload the
                // rows of the next layer's split
                __threadfence();
                fence_proxy_async_global();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) {
                    mbar_arrive_remote(xs_own);
                    mbar_arrive_remote(xs_peer);
                }
                if (!wait_all_cluster(&bars->xsync, xs_phase)) {
                    alive = false;
                    break;
                }
                xs_phase ^= 1u;
                tc_fence_after();
                // the next split's rows: 64-token boxes of one 16-byte chunk each, all
                // completing on xload (one lane issues them)
                if (warp == 2 && lane == 0) {
                    mbar_arrive_expect_tx(&bars->xload, (uint32_t)G::A_BYTES);
                    for (int kc = 0; kc < D / 8; ++kc)
                        for (int half = 0; half < 2; ++half) {
                            const int t0 = alt_next ? tile * 256 + half * 128 + (int)rank * 64
                                                    : tile * 256 + (int)rank * kRows + half * 64;
                            tma_load_3d(A + (size_t)kc * kChunkBytes + half * 1024, &L.imap[i],
                                        &bars->xload, 0, t0, kc);
                        }
                }
                if (!FWD && resid) {
                    // g of the rows this lane now holds, into TMEM
                    const int tok2 = tok_of(tile, (int)rank, row, alt_next);
#pragma unroll 1
                    for (int h = 0; h < G::NCH; ++h)
#pragma unroll 1
                        for (int j = 0; j < G::SUB; ++j) {
                            const int col = col_of(h, j);
                            const float4* gs =
                                reinterpret_cast<const float4*>(L.gscratch + (size_t)tok2 * D + col);
                            uint32_t g[32];
#pragma unroll
                            for (int m = 0; m < 8; ++m) {
                                const float4 f = __ldcg(gs + m);
                                g[4 * m] = __float_as_uint(f.x);
                                g[4 * m + 1] = __float_as_uint(f.y);
                                g[4 * m + 2] = __float_as_uint(f.z);
                                g[4 * m + 3] = __float_as_uint(f.w);
                            }
                            __syncwarp();
                            tmem_st_32x32b_x32(t_lane + (uint32_t)col, g);
                        }
                    tmem_st_wait();
                }
                if (!wait_all(&bars->xload, xl_phase)) {
                    alive = false;
                    break;
                }
                xl_phase ^= 1u;
                signal_ready(0);
                if (G::NCH == 2) signal_ready(1);
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    cluster_sync_all();   // neither CTA frees the pair's TMEM while the other uses it
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc_pair(tmem_base, Geo<D>::TMEM_COLS);
    }
}

namespace {

template <int MODE, int D>
cudaError_t launch_res_t(const ResLaunch& L, cudaStream_t st) {
    constexpr size_t smem = Geo<D>::SMEM;
    auto kern = hcw_res_kernel<MODE, D>;
    // the shared-memory opt-in is a per-device function attribute: set it once per device
    static std::atomic<uint64_t> configured[4] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    const uint64_t bit = 1ull << (dev & 63);
    std::atomic<uint64_t>& word = configured[(dev >> 6) & 3];
    if (dev >= 256 || !(word.load(std::memory_order_acquire) & bit)) {
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        if (dev < 256) word.fetch_or(bit, std::memory_order_acq_rel);
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(L.tokens / kRows));
    cfg.blockDim = dim3((unsigned)kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, L);
}

}  // namespace

bool res_supported(int d, int n, long long tokens) {
    return (d == 128 || d == 256 || d == 512) && n >= 2 && n <= 256 && tokens > 0 &&
           tokens % 256 == 0;
}

cudaError_t launch_res(int mode, const ResLaunch& L, cudaStream_t st) {
    if (!res_supported(L.d, L.n, L.tokens) || L.n_layers < 1 || L.n_layers > kMaxStackLayers)
        return cudaErrorInvalidValue;
    if (mode == MODE_FWD) {
        if (L.d == 512) return launch_res_t<MODE_FWD, 512>(L, st);
        if (L.d == 256) return launch_res_t<MODE_FWD, 256>(L, st);
        return launch_res_t<MODE_FWD, 128>(L, st);
    }
    if (mode == MODE_DX) {
        if (L.d == 512) return launch_res_t<MODE_DX, 512>(L, st);
        if (L.d == 256) return launch_res_t<MODE_DX, 256>(L, st);
        return launch_res_t<MODE_DX, 128>(L, st);
    }
    return cudaErrorInvalidValue;
}

cudaError_t res_error_word_read_clear(int* word) {
    const int zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(word, g_error_word, sizeof(int));
    if (e == cudaSuccess && *word) e = cudaMemcpyToSymbol(g_error_word, &zero, sizeof(int));
    return e;
}

}  // namespace hcw
