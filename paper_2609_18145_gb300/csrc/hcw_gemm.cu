// hcw_gemm.cu -- the plain GEMMs of the character-LM block around the stack
// (the FFN with hidden h, the output head, and their gradients): bf16
// operands, fp32 accumulation.
//
//   C[M][N] = op(A) op(B)      A: [M][K] row-major, or [K][M] (ta)
//                              B: [K][N] row-major, or [N][K] (tb)
//
// An operand whose contraction index K runs along its rows in memory is
// "K-major" (A without ta, B with tb: activations [T][K] and weights [N][K]);
// the others are "MN-major" (token-major activations contracted over the
// tokens, as in the weight gradients, and weights used untransposed).  Both
// are read by TMA straight from their row-major layout: a K-major operand as
// 64-element rows (128-byte swizzle), an MN-major one as blocks of 64 rows of
// 64 columns, which is the layout tcgen05 reads as an MN-major operand.
//
// A cluster of two CTAs (one per SM) computes 256 x 256 output tiles with
// tcgen05.mma.cta_group::2: CTA r of the pair loads rows 128 r .. 128 r + 127
// of the tile's A and columns 128 r .. 128 r + 127 of its B, so each SM takes
// in 32 KB per 64-deep K step for 2 M multiply-adds.  In each CTA a producer
// thread fills a ring of six stages, the leader's MMA thread issues the pair's
// MMAs into a double-buffered TMEM accumulator (each CTA holds its 128 rows),
// and eight warps drain the CTA's 128 x 256 fp32 results.  Tiles are handed
// out round robin; a GEMM with few tiles and a long K (the weight gradients,
// K = the tokens) splits K, each split writing its fp32 partial sums, which a
// second kernel adds in split order (deterministic).
//
// The epilogue either stores fp32 C, or applies the FFN's elementwise step
// and stores bf16: relu(C + bias[col]) (the hidden activations), or C where
// the stored activation aux[row][col] > 0 (the pre-activation gradient).
//
// Every wait is bounded: a CTA that gives up records HCW_ERR_TIMEOUT in the
// error word, lets its copies and MMAs in flight finish, frees TMEM and
// returns.  Shapes TMA cannot read (a K-major row not a multiple of 16 bytes,
// an MN-major one not a multiple of 64 elements) go to a plain tiled kernel.
#include "hcw.h"
#include "hcw_internal.h"
#include "hcw_ptx.cuh"

#include <mutex>
#include <utility>

namespace hcw {

namespace {

constexpr int kGM = 128;                    // tile rows per CTA (256 per pair)
constexpr int kGN = 256;                    // tile columns (128 of B per CTA)
constexpr int kGK = 64;                     // K step: one 128-byte row of bf16
constexpr int kGStages = 5;
constexpr int kGABytes = kGM * kGK * 2;     // 16 KB
constexpr int kGBBytes = kGN / 2 * kGK * 2; // 16 KB
constexpr int kGStage = kGABytes + kGBBytes;
constexpr int kGEpiWarps = 8;               // two per TMEM lane quarter, 128 columns each
constexpr int kGThreads = 64 + 32 * kGEpiWarps;
constexpr uint32_t kGTmemCols = 2 * kGN;
constexpr int kGPatch = 4096;               // a 32-row x 128-byte output patch
constexpr int kGStaging = kGEpiWarps * 2 * kGPatch;   // two patches per epilogue warp
constexpr unsigned long long kGemmTimeoutNs = 2000000000ull;

struct __align__(8) GemmBars {
    uint64_t full[kGStages];    // leader: both CTAs' copies of a stage landed
    uint64_t empty[kGStages];   // each CTA: the pair's MMAs have read the stage
    uint64_t tfull[2];          // each CTA: an accumulator is complete
    uint64_t tempty[2];         // leader: both CTAs have drained an accumulator
    uint64_t drain;
    uint64_t aux[kGEpiWarps];   // each epilogue warp: its aux patch landed
    uint32_t tmem_base;
    int abort;
};

constexpr size_t kGSmem = 1024 + (size_t)kGStages * kGStage + kGStaging + sizeof(GemmBars);
static_assert(kGSmem <= 232448, "shared memory budget");

struct GemmArgs {
    CUtensorMap mA, mB;
    CUtensorMap mOut;           // output patches: fp32 (N, M, splits) box (32, 32, 1), or
                                // bf16 (N, M) box (64, 32); 128-byte swizzle
    CUtensorMap mAux;           // EPI_RELU_GRAD: aux (N, M) bf16, box (64, 32)
    int tma_out;                // the patches go out (and aux comes in) by TMA
    float* C;                   // EPI_F32: [M][N], or the split partials [splits][M][N]
    __nv_bfloat16* out;         // EPI_BIAS_RELU / EPI_RELU_GRAD: [M][N] bf16
    const float* bias;          // EPI_BIAS_RELU: [N]
    const __nv_bfloat16* aux;   // EPI_RELU_GRAD: [M][N]
    float* colsum;              // EPI_RELU_GRAD: [N] += column sums of the bf16 output, or null
    int M, N, K;
    int mt, nt;                 // tile counts (256-row tiles, 256-column tiles)
    int splits, kps;            // K splits and K steps per split
    // batched (both operands MN-major, EPI_F32): `splits` counts independent
    // products instead of K splits; mA / mB carry the batch as a 4th dimension
    // and each unit takes the whole K range of product s into C[s]
    int batched;
    uint32_t stage_tx;          // bytes one CTA's two copies of a stage land
    int vec;                    // rows of the output start 16-byte aligned
    unsigned long long timeout_ns;
};

template <bool A_MN, bool B_MN, int EPI>
__global__ void __launch_bounds__(kGThreads, 1) gemm_pair_kernel(const __grid_constant__ GemmArgs a) {
    constexpr uint32_t IDESC = idesc_bf16_f32(2 * kGM, kGN, A_MN ? 1 : 0, B_MN ? 1 : 0);
    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint8_t* staging = smem + (size_t)kGStages * kGStage;
    GemmBars* bars = reinterpret_cast<GemmBars*>(staging + kGStaging);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const int pair = (int)blockIdx.x >> 1, n_pairs = (int)gridDim.x >> 1;
    const int tiles = a.mt * a.nt;
    const int n_units = tiles * a.splits;
    const int nkb = (a.K + kGK - 1) / kGK;
    const uint64_t tmo = a.timeout_ns;

    if (threadIdx.x == 0) {
        tma_prefetch_desc(&a.mA);
        tma_prefetch_desc(&a.mB);
        for (int s = 0; s < kGStages; ++s) {
            mbar_init(&bars->full[s], 1);
            mbar_init(&bars->empty[s], 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(&bars->tfull[i], 1);
            mbar_init(&bars->tempty[i], 2 * kGEpiWarps);
        }
        mbar_init(&bars->drain, 1);
        for (int i = 0; i < kGEpiWarps; ++i) mbar_init(&bars->aux[i], 1);
        bars->abort = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc_pair(&bars->tmem_base, kGTmemCols);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync_all();   // both CTAs' barriers exist before any cross-CTA arrive
    tc_fence_after();
    // the prologue above touched no global memory: it overlaps the end of the
    // kernel before this one when launched as a programmatic dependent
    pdl_wait();
    pdl_trigger();
    const uint32_t tmem_base = bars->tmem_base;
    volatile int* abort = &bars->abort;
    // unit u -> (split, tile row, tile column), tile columns fastest: the pairs
    // running together share their A rows (and B, the weights, is small)
    auto unit_k = [&](int u, int& kb0, int& kb1) {
        const int s = u / tiles;
        kb0 = a.batched ? 0 : s * a.kps;
        kb1 = a.batched ? nkb : (kb0 + a.kps < nkb ? kb0 + a.kps : nkb);
    };

    if (warp == 0) {
        // ------------------------------------------------------------ producer (both CTAs)
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0, issued_mask = 0, issued_phase = 0;
            bool ok = true;
            for (int u = pair; u < n_units && ok; u += n_pairs) {
                const int rem = u % tiles, mi = rem / a.nt, ni = rem - mi * a.nt;
                int kb0, kb1;
                unit_k(u, kb0, kb1);
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!mbar_wait(&bars->empty[stage], phase ^ 1, abort, tmo)) {
                        ok = false;
                        break;
                    }
                    uint8_t* sA = smem + (size_t)stage * kGStage;
                    uint8_t* sB = sA + kGABytes;
                    if (rank == 0) mbar_arrive_expect_tx(&bars->full[stage], 2 * a.stage_tx);
                    issued_mask |= 1u << stage;
                    issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
                    const uint32_t fb = mapa_shared(&bars->full[stage], 0);
                    // this CTA's 128 rows of A and 128 columns of B: two 64-wide
                    // blocks of an MN-major operand, or 128 rows of a K-major one
                    const int a_row = 2 * mi * kGM + (int)rank * kGM;
                    const int b_row = ni * kGN + (int)rank * (kGN / 2);
                    if (A_MN && B_MN && a.batched) {
                        const int bi = u / tiles;   // the product
                        tma_load_4d_pair(sA, &a.mA, fb, 0, kb * kGK, a_row / 64, bi);
                        tma_load_4d_pair(sB, &a.mB, fb, 0, kb * kGK, b_row / 64, bi);
                    } else {
                        if (A_MN)
                            tma_load_3d_pair(sA, &a.mA, fb, 0, kb * kGK, a_row / 64);
                        else
                            tma_load_2d_pair(sA, &a.mA, fb, kb * kGK, a_row);
                        if (B_MN)
                            tma_load_3d_pair(sB, &a.mB, fb, 0, kb * kGK, b_row / 64);
                        else
                            tma_load_2d_pair(sB, &a.mB, fb, kb * kGK, b_row);
                    }
                    if (++stage == kGStages) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
            }
            if (!ok && rank == 0)
                // every copy of the pair completes on the leader's barriers
                for (int s = 0; s < kGStages; ++s)
                    if (issued_mask & (1u << s))
                        mbar_wait_drain(&bars->full[s], (issued_phase >> s) & 1u, tmo);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer (leader)
        if (lane == 0 && rank == 0) {
            int stage = 0, acc = 0;
            uint32_t phase = 0, acc_phase = 0;
            bool ok = true, any = false;
            for (int u = pair; u < n_units && ok; u += n_pairs) {
                int kb0, kb1;
                unit_k(u, kb0, kb1);
                if (!mbar_wait(&bars->tempty[acc], acc_phase ^ 1, abort, tmo)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * kGN);
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!mbar_wait(&bars->full[stage], phase, abort, tmo)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = smem_u32(smem + (size_t)stage * kGStage);
                    const uint32_t sb = sa + kGABytes;
#pragma unroll
                    for (int kk = 0; kk < kGK / 16; ++kk) {
                        const uint64_t ad = A_MN ? smem_desc_sw128(sa + kk * 2048, 8192, 1024)
                                                 : smem_desc_sw128(sa + kk * 32, 16, 1024);
                        const uint64_t bd = B_MN ? smem_desc_sw128(sb + kk * 2048, 8192, 1024)
                                                 : smem_desc_sw128(sb + kk * 32, 16, 1024);
                        mma_bf16_f32_pair(d_tmem, ad, bd, IDESC,
                                          (kb != kb0 || kk != 0) ? 1u : 0u);
                    }
                    any = true;
                    mma_commit_pair(&bars->empty[stage], 3);
                    if (++stage == kGStages) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
                if (!ok) break;
                mma_commit_pair(&bars->tfull[acc], 3);
                acc ^= 1;
                if (acc == 0) acc_phase ^= 1;
            }
            if (any) {
                // the pair's MMAs have completed before TMEM can be freed
                mma_commit_pair(&bars->drain, 1);
                mbar_wait_drain(&bars->drain, 0, tmo);
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue (both CTAs)
        // warp e drains TMEM lane quarter warp % 4 (rows 32 q .. 32 q + 31 of
        // this CTA's 128) and columns [128 (e / 4), 128 (e / 4) + 128)
        const int e = warp - 2;
        const int quarter = warp & 3, chalf = e >> 2;
        int acc = 0, nbuf = 0;
        uint32_t acc_phase = 0, aux_phase = 0;
        bool aux_pending = false;
        auto patch_buf = [&](int b) { return staging + (size_t)(2 * e + b) * kGPatch; };
        // 16-byte chunk m of row r of a 128-byte-swizzled patch
        auto patch_chunk = [](uint8_t* buf, int r, int m) {
            return reinterpret_cast<uint4*>(buf + r * 128 + ((m ^ (r & 7)) << 4));
        };
        for (int u = pair; u < n_units; u += n_pairs) {
            const int s = u / tiles, rem = u % tiles, mi = rem / a.nt, ni = rem - mi * a.nt;
            const int row0 = 2 * mi * kGM + (int)rank * kGM + quarter * 32;   // the warp's rows
            const int row = row0 + lane;
            const int colw = ni * kGN + chalf * 128;                          // and columns
            // EPI_RELU_GRAD: the aux patches of the tile's two 64-column halves go
            // into the warp's two buffers before the accumulator is ready (the
            // stores of the tile before have read them by then); the second half
            // is stored only if the first is, so half hh lands in buffer nbuf ^ hh
            int n_aux = 0;
            if (EPI == EPI_RELU_GRAD && a.tma_out) {
                n_aux = (row0 < a.M && colw < a.N) + (row0 < a.M && colw + 64 < a.N);
                if (lane == 0 && n_aux > 0) {
                    bulk_wait_read<0>();
                    mbar_arrive_expect_tx(&bars->aux[e], (uint32_t)(n_aux * kGPatch));
                    tma_load_2d(patch_buf(nbuf), &a.mAux, &bars->aux[e], colw, row0);
                    if (n_aux > 1)
                        tma_load_2d(patch_buf(nbuf ^ 1), &a.mAux, &bars->aux[e], colw + 64, row0);
                    aux_pending = true;
                }
            }
            const bool okw = mbar_wait(&bars->tfull[acc], acc_phase, abort, tmo);
            if (!__all_sync(0xffffffffu, okw)) break;
            tc_fence_after();
            const uint32_t tbase = tmem_base + ((uint32_t)(quarter * 32) << 16) +
                                   (uint32_t)(acc * kGN + chalf * 128);
            const uint32_t tempty_leader = mapa_shared(&bars->tempty[acc], 0);
            if (a.tma_out) {
                // Patches of 32 rows x 128 bytes through shared memory (128-byte
                // swizzle), stored by TMA.  A warp alternates two patch buffers and
                // fills one only for a store it issues, so the store that last read
                // a buffer is always the second most recent (bulk_wait_read<1>).
                bool okp = true;
                if (EPI == EPI_F32) {
#pragma unroll 1
                    for (int c = 0; c < 4; ++c) {
                        const bool st = row0 < a.M && colw + c * 32 < a.N;   // warp-uniform
                        uint32_t raw[32];
                        if (st) {
                            __syncwarp();
                            tmem_ld_32x32b_x32(tbase + (uint32_t)(c * 32), raw);
                            tmem_ld_wait_regs(raw);
                        }
                        if (c == 3) {
                            tc_fence_before();
                            __syncwarp();
                            if (lane == 0) mbar_arrive_remote_tmem(tempty_leader);
                        }
                        if (!st) continue;
                        uint8_t* buf = patch_buf(nbuf);
                        nbuf ^= 1;
                        if (lane == 0) bulk_wait_read<1>();   // its store of two patches ago has read it
                        __syncwarp();
#pragma unroll
                        for (int m = 0; m < 8; ++m)
                            *patch_chunk(buf, lane, m) =
                                make_uint4(raw[4 * m], raw[4 * m + 1], raw[4 * m + 2], raw[4 * m + 3]);
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            tma_store_3d(&a.mOut, buf, colw + c * 32, row0, s);
                            bulk_commit();
                        }
                    }
                } else {
#pragma unroll 1
                    for (int hh = 0; hh < 2; ++hh) {
                        const int c0 = colw + hh * 64;
                        if (!(row0 < a.M && c0 < a.N)) {   // warp-uniform: nothing to store
                            if (hh == 1) {
                                tc_fence_before();
                                __syncwarp();
                                if (lane == 0) mbar_arrive_remote_tmem(tempty_leader);
                            }
                            continue;
                        }
                        uint8_t* buf = patch_buf(nbuf);
                        nbuf ^= 1;
                        if (lane == 0 && EPI != EPI_RELU_GRAD) bulk_wait_read<1>();
                        uint32_t r0[32], r1[32];
                        __syncwarp();
                        tmem_ld_32x32b_x32(tbase + (uint32_t)(hh * 64), r0);
                        tmem_ld_32x32b_x32(tbase + (uint32_t)(hh * 64 + 32), r1);
                        tmem_ld_wait_regs(r0);
                        tmem_ld_wait_regs(r1);
                        if (hh == 1) {
                            tc_fence_before();
                            __syncwarp();
                            if (lane == 0) mbar_arrive_remote_tmem(tempty_leader);
                        }
                        if (EPI == EPI_RELU_GRAD && hh == 0) {
                            // both halves' aux patches (one barrier phase per tile)
                            const bool okx = mbar_wait(&bars->aux[e], aux_phase, abort, tmo);
                            if (!__all_sync(0xffffffffu, okx)) {
                                okp = false;
                                break;
                            }
                            aux_phase ^= 1;
                            aux_pending = false;
                        }
                        __syncwarp();
#pragma unroll
                        for (int m = 0; m < 8; ++m) {
                            float v[8];
#pragma unroll
                            for (int j = 0; j < 8; ++j)
                                v[j] = __uint_as_float(m < 4 ? r0[8 * m + j] : r1[8 * (m - 4) + j]);
                            if (EPI == EPI_BIAS_RELU) {
                                const float4* b4 = reinterpret_cast<const float4*>(a.bias + c0 + 8 * m);
                                float4 b0 = make_float4(0.f, 0.f, 0.f, 0.f), b1 = b0;
                                if (c0 + 8 * m < a.N) {   // N % 8 == 0: all eight or none
                                    b0 = __ldg(b4);
                                    b1 = __ldg(b4 + 1);
                                }
                                const float bb[8] = {b0.x, b0.y, b0.z, b0.w, b1.x, b1.y, b1.z, b1.w};
#pragma unroll
                                for (int j = 0; j < 8; ++j) {
                                    const float x = v[j] + bb[j];
                                    v[j] = x > 0.f ? x : 0.f;
                                }
                            } else {
                                const uint4 q = *patch_chunk(buf, lane, m);
                                const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
                                for (int j = 0; j < 4; ++j) {
                                    const float2 am = unpack_bf16x2(w[j]);
                                    v[2 * j] = am.x > 0.f ? v[2 * j] : 0.f;
                                    v[2 * j + 1] = am.y > 0.f ? v[2 * j + 1] : 0.f;
                                }
                            }
                            *patch_chunk(buf, lane, m) =
                                make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]),
                                           pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
                        }
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            tma_store_2d(&a.mOut, buf, c0, row0);
                            bulk_commit();
                        }
                        if (EPI == EPI_RELU_GRAD && a.colsum) {
                            // lane l adds up columns c0 + 2l, c0 + 2l + 1 of the patch's
                            // 32 rows (the stored bf16 values; rows past M hold 0)
                            const int m = lane >> 2, wd = lane & 3;
                            float s0 = 0.f, s1 = 0.f;
#pragma unroll 8
                            for (int r = 0; r < 32; ++r) {
                                const float2 f = unpack_bf16x2(*reinterpret_cast<const uint32_t*>(
                                    buf + r * 128 + ((m ^ (r & 7)) << 4) + 4 * wd));
                                s0 += f.x;
                                s1 += f.y;
                            }
                            const int col = c0 + 2 * lane;
                            if (col < a.N) {
                                atomicAdd(a.colsum + col, s0);
                                atomicAdd(a.colsum + col + 1, s1);
                            }
                        }
                    }
                }
                if (!okp) break;
                acc ^= 1;
                if (acc == 0) acc_phase ^= 1;
                continue;
            }
#pragma unroll 1
            for (int c = 0; c < 4; ++c) {
                uint32_t raw[32];
                __syncwarp();
                tmem_ld_32x32b_x32(tmem_base + ((uint32_t)(quarter * 32) << 16) +
                                       (uint32_t)(acc * kGN + chalf * 128 + c * 32),
                                   raw);
                tmem_ld_wait_regs(raw);
                if (c == 3) {
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive_remote_tmem(tempty_leader);
                }
                const int col0 = ni * kGN + chalf * 128 + c * 32;
                if (row >= a.M || col0 >= a.N) continue;
                const bool full = a.vec && col0 + 32 <= a.N;
                if (EPI == EPI_F32) {
                    float* dst = a.C + (size_t)s * a.M * a.N + (size_t)row * a.N + col0;
                    if (full) {
#pragma unroll
                        for (int m = 0; m < 8; ++m)
                            reinterpret_cast<float4*>(dst)[m] = make_float4(
                                __uint_as_float(raw[4 * m]), __uint_as_float(raw[4 * m + 1]),
                                __uint_as_float(raw[4 * m + 2]), __uint_as_float(raw[4 * m + 3]));
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            if (col0 + i < a.N) dst[i] = __uint_as_float(raw[i]);
                    }
                } else {
                    __nv_bfloat16* dst = a.out + (size_t)row * a.N + col0;
                    if (full) {
                        float v[32];
                        if (EPI == EPI_BIAS_RELU) {
                            const float4* b4 = reinterpret_cast<const float4*>(a.bias + col0);
#pragma unroll
                            for (int m = 0; m < 8; ++m) {
                                const float4 b = __ldg(b4 + m);
                                v[4 * m] = __uint_as_float(raw[4 * m]) + b.x;
                                v[4 * m + 1] = __uint_as_float(raw[4 * m + 1]) + b.y;
                                v[4 * m + 2] = __uint_as_float(raw[4 * m + 2]) + b.z;
                                v[4 * m + 3] = __uint_as_float(raw[4 * m + 3]) + b.w;
                            }
#pragma unroll
                            for (int i = 0; i < 32; ++i) v[i] = v[i] > 0.f ? v[i] : 0.f;
                        } else {
                            const uint4* m4 =
                                reinterpret_cast<const uint4*>(a.aux + (size_t)row * a.N + col0);
#pragma unroll
                            for (int m = 0; m < 4; ++m) {
                                const uint4 q = __ldg(m4 + m);
                                const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
                                for (int j = 0; j < 4; ++j) {
                                    const float2 am = unpack_bf16x2(w[j]);
                                    const int i = 8 * m + 2 * j;
                                    v[i] = am.x > 0.f ? __uint_as_float(raw[i]) : 0.f;
                                    v[i + 1] = am.y > 0.f ? __uint_as_float(raw[i + 1]) : 0.f;
                                }
                            }
                        }
#pragma unroll
                        for (int m = 0; m < 4; ++m)
                            reinterpret_cast<uint4*>(dst)[m] = make_uint4(
                                pack_bf16x2(v[8 * m], v[8 * m + 1]),
                                pack_bf16x2(v[8 * m + 2], v[8 * m + 3]),
                                pack_bf16x2(v[8 * m + 4], v[8 * m + 5]),
                                pack_bf16x2(v[8 * m + 6], v[8 * m + 7]));
                        if (EPI == EPI_RELU_GRAD && a.colsum) {
#pragma unroll
                            for (int i = 0; i < 32; ++i)
                                atomicAdd(a.colsum + col0 + i,
                                          __bfloat162float(__float2bfloat16_rn(v[i])));
                        }
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i) {
                            if (col0 + i >= a.N) continue;
                            float x = __uint_as_float(raw[i]);
                            if (EPI == EPI_BIAS_RELU) {
                                x += a.bias[col0 + i];
                                x = x > 0.f ? x : 0.f;
                            } else {
                                const float am =
                                    __bfloat162float(a.aux[(size_t)row * a.N + col0 + i]);
                                x = am > 0.f ? x : 0.f;
                            }
                            dst[i] = __float2bfloat16_rn(x);
                            if (EPI == EPI_RELU_GRAD && a.colsum)
                                atomicAdd(a.colsum + col0 + i, __bfloat162float(dst[i]));
                        }
                    }
                }
            }
            acc ^= 1;
            if (acc == 0) acc_phase ^= 1;
        }
        // an aux patch still on its way lands, and every store of this warp has
        // read its buffer, before the CTA exits
        if (aux_pending && lane == 0) mbar_wait_drain(&bars->aux[e], aux_phase, tmo);
        if (lane == 0) bulk_wait<0>();
        __syncwarp();
    }

    tc_fence_before();
    __syncthreads();
    cluster_sync_all();   // neither CTA frees the pair's TMEM while the other uses it
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc_pair(tmem_base, kGTmemCols);
    }
}

// C[i] = sum over the splits s, in order, of part[s][i]; four at a time
__global__ void gemm_split_reduce_kernel(const float* part, int splits, size_t count, float* C,
                                         bool vec) {
    pdl_wait();   // until the kernel before it in the stream has finished
    pdl_trigger();
    const size_t n4 = vec ? count / 4 : 0;
    for (size_t i = blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < n4;
         i += (size_t)gridDim.x * blockDim.x) {
        float4 acc = reinterpret_cast<const float4*>(part)[i];
        for (int s = 1; s < splits; ++s) {
            const float4 v = reinterpret_cast<const float4*>(part + (size_t)s * count)[i];
            acc.x += v.x;
            acc.y += v.y;
            acc.z += v.z;
            acc.w += v.w;
        }
        reinterpret_cast<float4*>(C)[i] = acc;
    }
    for (size_t i = n4 * 4 + blockIdx.x * (size_t)blockDim.x + threadIdx.x; i < count;
         i += (size_t)gridDim.x * blockDim.x) {
        float acc = part[i];
        for (int s = 1; s < splits; ++s) acc += part[(size_t)s * count + i];
        C[i] = acc;
    }
}

// The plain path: 64 x 64 output tiles, 256 threads, 4 x 4 outputs each, K in
// steps of 16 staged through shared memory.  Any shape and alignment; the
// same epilogues as the tensor-core kernel (e.epi).
__global__ void __launch_bounds__(256) gemm_simt_kernel(int M, int N, int K,
                                                         const __nv_bfloat16* A, bool ta,
                                                         const __nv_bfloat16* B, bool tb,
                                                         float* C, GemmEpi e) {
    pdl_wait();   // until the kernel before it in the stream has finished
    pdl_trigger();
    __shared__ float As[16][65];
    __shared__ float Bs[16][65];
    const int tm = blockIdx.y * 64, tn = blockIdx.x * 64;
    const int tx = threadIdx.x & 15, ty = threadIdx.x >> 4;
    float acc[4][4] = {};
    for (int k0 = 0; k0 < K; k0 += 16) {
        for (int i = threadIdx.x; i < 16 * 64; i += 256) {
            const int kk = i / 64, mm = i % 64;
            const int gm = tm + mm, gn = tn + mm, gk = k0 + kk;
            float av = 0.f, bv = 0.f;
            if (gm < M && gk < K)
                av = __bfloat162float(ta ? A[(size_t)gk * M + gm] : A[(size_t)gm * K + gk]);
            if (gn < N && gk < K)
                bv = __bfloat162float(tb ? B[(size_t)gn * K + gk] : B[(size_t)gk * N + gn]);
            As[kk][mm] = av;
            Bs[kk][mm] = bv;
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < 16; ++kk)
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] += As[kk][ty * 4 + i] * Bs[kk][tx * 4 + j];
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int gm = tm + ty * 4 + i, gn = tn + tx * 4 + j;
            if (gm >= M || gn >= N) continue;
            const size_t o = (size_t)gm * N + gn;
            if (e.kind == EPI_F32) {
                C[o] = acc[i][j];
            } else if (e.kind == EPI_BIAS_RELU) {
                const float x = acc[i][j] + e.bias[gn];
                e.out[o] = __float2bfloat16_rn(x > 0.f ? x : 0.f);
            } else {
                e.out[o] = __float2bfloat16_rn(__bfloat162float(e.aux[o]) > 0.f ? acc[i][j] : 0.f);
                if (e.colsum) atomicAdd(e.colsum + gn, __bfloat162float(e.out[o]));
            }
        }
}

typedef CUresult (*GemmEncodeFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                 const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                 const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                 CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

GemmEncodeFn gemm_encode_fn() {
    static GemmEncodeFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<GemmEncodeFn>(p);
    });
    return fn;
}

// A K-major operand [rows][K] bf16 as 64-element rows: box (64, box_rows).
bool map_kmajor(CUtensorMap* m, const void* base, int rows, int K, int box_rows) {
    GemmEncodeFn enc = gemm_encode_fn();
    if (!enc) return false;
    cuuint64_t dims[2] = {(cuuint64_t)K, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)K * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    cuuint32_t estr[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
               estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// An MN-major operand, the row-major [K][cols] matrix, as (64 columns, K rows,
// cols / 64 blocks): box (64, 64, nblk) lands nblk blocks of 64 rows x 64
// columns one after the other.
bool map_mnmajor(CUtensorMap* m, const void* base, int K, int cols, int nblk) {
    GemmEncodeFn enc = gemm_encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {64, (cuuint64_t)K, (cuuint64_t)(cols / 64)};
    cuuint64_t strides[2] = {(cuuint64_t)cols * 2, 128};
    cuuint32_t box[3] = {64, 64, (cuuint32_t)nblk};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
               estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// A batch of MN-major operands, product b at base + b * batch_bytes, each the
// row-major [K][cols] matrix: (64 columns, K rows, cols / 64 blocks, batch),
// box (64, 64, nblk, 1).
bool map_mnmajor_batched(CUtensorMap* m, const void* base, int K, int cols, int nblk, int batch,
                         size_t batch_bytes) {
    GemmEncodeFn enc = gemm_encode_fn();
    if (!enc || batch_bytes % 16) return false;
    cuuint64_t dims[4] = {64, (cuuint64_t)K, (cuuint64_t)(cols / 64), (cuuint64_t)batch};
    cuuint64_t strides[3] = {(cuuint64_t)cols * 2, 128, (cuuint64_t)batch_bytes};
    cuuint32_t box[4] = {64, 64, (cuuint32_t)nblk, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box,
               estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// fp32 output [splits][M][N] as (N, M, splits), box (32, 32, 1): 32 x 32
// patches clipped at each split's M rows; 128-byte swizzle.
bool map_out_f32(CUtensorMap* m, void* base, int M, int N, int splits) {
    GemmEncodeFn enc = gemm_encode_fn();
    if (!enc || (reinterpret_cast<uintptr_t>(base) & 15) || N % 4) return false;
    cuuint64_t dims[3] = {(cuuint64_t)N, (cuuint64_t)M, (cuuint64_t)splits};
    cuuint64_t strides[2] = {(cuuint64_t)N * 4, (cuuint64_t)M * N * 4};
    cuuint32_t box[3] = {32, 32, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 3, base, dims, strides, box, estr,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// bf16 [M][N] as (N, M), box (64, 32): 32-row x 64-column patches; 128-byte
// swizzle.
bool map_patch_bf16(CUtensorMap* m, const void* base, int M, int N) {
    GemmEncodeFn enc = gemm_encode_fn();
    if (!enc || (reinterpret_cast<uintptr_t>(base) & 15) || N % 8) return false;
    cuuint64_t dims[2] = {(cuuint64_t)N, (cuuint64_t)M};
    cuuint64_t strides[1] = {(cuuint64_t)N * 2};
    cuuint32_t box[2] = {64, 32};
    cuuint32_t estr[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides, box,
               estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int gemm_sms() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1)
        return 148;
    return n;
}

template <bool A_MN, bool B_MN, int EPI>
cudaError_t launch_gemm_pair(const GemmArgs& a, int grid, cudaStream_t st) {
    auto kern = gemm_pair_kernel<A_MN, B_MN, EPI>;
    static std::once_flag once[64];
    static cudaError_t set_err[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::call_once(once[dev], [&] {
        set_err[dev] = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                            (int)kGSmem);
    });
    if (set_err[dev] != cudaSuccess) return set_err[dev];
    // clusters of two CTAs (the grid is even)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3((unsigned)kGThreads);
    cfg.dynamicSmemBytes = kGSmem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kern, a);
}

// The instantiated (layout, epilogue) combinations: every layout for fp32
// output; the bias + ReLU epilogue on two K-major operands (activations times
// transposed weights); the ReLU-gradient epilogue on a K-major A and an
// MN-major B (a gradient times untransposed weights).
cudaError_t launch_gemm_any(bool a_mn, bool b_mn, int epi, const GemmArgs& a, int grid,
                            cudaStream_t st) {
    if (epi == EPI_F32)
        return a_mn ? (b_mn ? launch_gemm_pair<true, true, EPI_F32>(a, grid, st)
                            : launch_gemm_pair<true, false, EPI_F32>(a, grid, st))
                    : (b_mn ? launch_gemm_pair<false, true, EPI_F32>(a, grid, st)
                            : launch_gemm_pair<false, false, EPI_F32>(a, grid, st));
    if (epi == EPI_BIAS_RELU && !a_mn && !b_mn)
        return launch_gemm_pair<false, false, EPI_BIAS_RELU>(a, grid, st);
    if (epi == EPI_RELU_GRAD && !a_mn && b_mn)
        return launch_gemm_pair<false, true, EPI_RELU_GRAD>(a, grid, st);
    return cudaErrorNotSupported;
}

bool epi_has_kernel(bool a_mn, bool b_mn, int epi) {
    return epi == EPI_F32 || (epi == EPI_BIAS_RELU && !a_mn && !b_mn) ||
           (epi == EPI_RELU_GRAD && !a_mn && b_mn);
}

}  // namespace

namespace {

// K splits for an M x N x K product on `sms` SMs (sms / 2 pairs): the count
// that minimises the estimated time, waves of units x K steps per unit (about
// 0.35 us each) plus writing and re-reading the fp32 partials (about 6 TB/s),
// with each split at least four K steps long and the partials within
// `ws_bytes`.
int choose_splits(int M, int N, int K, int sms, size_t ws_bytes) {
    const long long tiles = (long long)((M + 2 * kGM - 1) / (2 * kGM)) * ((N + kGN - 1) / kGN);
    sms /= 2;   // pairs
    const int nkb = (K + kGK - 1) / kGK;
    const double part_us = (double)M * N * 8.0 / 6.0e6;   // one split's partials, us
    int best = 1;
    double best_t = (double)((tiles + sms - 1) / sms) * nkb * 0.35;
    for (int s = 2; s <= 64 && s * 4 <= nkb; ++s) {
        if ((size_t)s * M * N * sizeof(float) > ws_bytes) break;
        const int kps = (nkb + s - 1) / s;
        const int real = (nkb + kps - 1) / kps;
        const double t = (double)((tiles * real + sms - 1) / sms) * kps * 0.35 + real * part_us;
        if (t < best_t) {
            best_t = t;
            best = real;
        }
    }
    return best;
}

}  // namespace

cudaError_t gemm_bf16(int M, int N, int K, const void* A, bool ta, const void* B, bool tb,
                      float* C, const GemmEpi& epi, float* split_ws, size_t split_ws_bytes,
                      cudaStream_t st, int* launches) {
    *launches = 0;
    if (M <= 0 || N <= 0 || K <= 0 || !A || !B) return cudaErrorInvalidValue;
    bool bad;
    switch (epi.kind) {
        case EPI_F32: bad = !C; break;
        case EPI_BIAS_RELU: bad = !epi.out || !epi.bias; break;
        case EPI_RELU_GRAD: bad = !epi.out || !epi.aux; break;
        default: bad = true;
    }
    if (bad) return cudaErrorInvalidValue;
    const bool a_mn = ta, b_mn = !tb;
    const auto aligned = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
    // what TMA can read: 16-byte row strides, MN-major operands in whole
    // 64-column blocks
    const bool tc = aligned(A) && aligned(B) && (a_mn ? M % 64 == 0 : K % 8 == 0) &&
                    (b_mn ? N % 64 == 0 : K % 8 == 0) && epi_has_kernel(a_mn, b_mn, epi.kind) &&
                    gemm_encode_fn() != nullptr;
    if (!tc) {
        dim3 grid((unsigned)((N + 63) / 64), (unsigned)((M + 63) / 64));
        const cudaError_t e = launch_pdl(gemm_simt_kernel, grid, dim3(256), 0, st, M, N, K,
                                         static_cast<const __nv_bfloat16*>(A), ta,
                                         static_cast<const __nv_bfloat16*>(B), tb, C, epi);
        if (e == cudaSuccess) *launches = 1;
        return e;
    }
    // boxes no larger than the operand (the rows / blocks a smaller box leaves
    // in shared memory only reach output rows and columns that are not stored)
    const int a_box = a_mn ? (M / 64 < kGM / 64 ? M / 64 : kGM / 64) : (M < kGM ? M : kGM);
    const int b_box = b_mn ? (N / 64 < kGN / 128 ? N / 64 : kGN / 128) : (N < kGN / 2 ? N : kGN / 2);
    GemmArgs a;
    memset(&a, 0, sizeof(a));
    if (!(a_mn ? map_mnmajor(&a.mA, A, K, M, a_box) : map_kmajor(&a.mA, A, M, K, a_box)) ||
        !(b_mn ? map_mnmajor(&a.mB, B, K, N, b_box) : map_kmajor(&a.mB, B, N, K, b_box)))
        return cudaErrorInvalidValue;
    a.stage_tx = (uint32_t)(kGK * 2) * (uint32_t)((a_mn ? 64 * a_box : a_box) +
                                                  (b_mn ? 64 * b_box : b_box));
    a.M = M;
    a.N = N;
    a.K = K;
    a.mt = (M + 2 * kGM - 1) / (2 * kGM);
    a.nt = (N + kGN - 1) / kGN;
    const int nkb = (K + kGK - 1) / kGK;
    const int sms = gemm_sms();
    const int splits =
        split_ws && epi.kind == EPI_F32 ? choose_splits(M, N, K, sms, split_ws_bytes) : 1;
    a.kps = (nkb + splits - 1) / splits;
    a.splits = (nkb + a.kps - 1) / a.kps;   // no empty split
    if (epi.kind == EPI_F32) {
        a.C = a.splits > 1 ? split_ws : C;
        a.vec = (N % 4 == 0) && aligned(a.C);
        a.tma_out = map_out_f32(&a.mOut, a.C, M, N, a.splits);
    } else {
        a.out = epi.out;
        a.bias = epi.bias;
        a.aux = epi.aux;
        a.colsum = epi.kind == EPI_RELU_GRAD ? epi.colsum : nullptr;
        a.vec = (N % 8 == 0) && aligned(epi.out) &&
                (epi.kind == EPI_BIAS_RELU ? aligned(epi.bias) : aligned(epi.aux));
        a.tma_out = a.vec && map_patch_bf16(&a.mOut, epi.out, M, N) &&
                    (epi.kind != EPI_RELU_GRAD || map_patch_bf16(&a.mAux, epi.aux, M, N));
    }
    a.timeout_ns = kGemmTimeoutNs;
    const int units = a.mt * a.nt * a.splits;
    const int pairs = units < sms / 2 ? units : sms / 2;
    cudaError_t e = launch_gemm_any(a_mn, b_mn, epi.kind, a, 2 * (pairs > 0 ? pairs : 1), st);
    if (e != cudaSuccess) return e;
    *launches = 1;
    if (a.splits > 1) {
        const size_t count = (size_t)M * N;
        const size_t want = (count / 4 + 255) / 256;
        const unsigned g = (unsigned)(want < (size_t)sms * 8 ? (want ? want : 1) : (size_t)sms * 8);
        e = launch_pdl(gemm_split_reduce_kernel, dim3(g), dim3(256), 0, st,
                       static_cast<const float*>(split_ws), a.splits, count, C,
                       aligned(C) && aligned(split_ws));
        if (e == cudaSuccess) *launches = 2;
    }
    return e;
}

cudaError_t gemm_bf16_f32(int M, int N, int K, const void* A, bool ta, const void* B, bool tb,
                          float* C, float* split_ws, size_t split_ws_bytes, cudaStream_t st,
                          int* launches) {
    GemmEpi epi;
    epi.kind = EPI_F32;
    epi.bias = nullptr;
    epi.aux = nullptr;
    epi.out = nullptr;
    epi.colsum = nullptr;
    return gemm_bf16(M, N, K, A, ta, B, tb, C, epi, split_ws, split_ws_bytes, st, launches);
}

cudaError_t gemm_bf16_f32_batched(int M, int N, int K, const void* A, size_t a_batch_bytes,
                                  const void* B, size_t b_batch_bytes, float* C, int batch,
                                  cudaStream_t st, int* launches) {
    *launches = 0;
    if (M <= 0 || N <= 0 || K <= 0 || batch <= 0 || !A || !B || !C) return cudaErrorInvalidValue;
    const auto aligned = [](const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; };
    const bool tc = aligned(A) && aligned(B) && aligned(C) && M % 64 == 0 && N % 64 == 0 &&
                    a_batch_bytes % 16 == 0 && b_batch_bytes % 16 == 0 &&
                    gemm_encode_fn() != nullptr;
    if (!tc) {
        // shapes TMA cannot read: one product after another
        for (int b = 0; b < batch; ++b) {
            int nl = 0;
            const cudaError_t e =
                gemm_bf16_f32(M, N, K, static_cast<const uint8_t*>(A) + b * a_batch_bytes, true,
                              static_cast<const uint8_t*>(B) + b * b_batch_bytes, false,
                              C + (size_t)b * M * N, nullptr, 0, st, &nl);
            if (e != cudaSuccess) return e;
            *launches += nl;
        }
        return cudaSuccess;
    }
    const int a_box = M / 64 < kGM / 64 ? M / 64 : kGM / 64;
    const int b_box = N / 64 < kGN / 128 ? N / 64 : kGN / 128;
    GemmArgs a;
    memset(&a, 0, sizeof(a));
    if (!map_mnmajor_batched(&a.mA, A, K, M, a_box, batch, a_batch_bytes) ||
        !map_mnmajor_batched(&a.mB, B, K, N, b_box, batch, b_batch_bytes))
        return cudaErrorInvalidValue;
    a.stage_tx = (uint32_t)(kGK * 2) * (uint32_t)(64 * a_box + 64 * b_box);
    a.M = M;
    a.N = N;
    a.K = K;
    a.mt = (M + 2 * kGM - 1) / (2 * kGM);
    a.nt = (N + kGN - 1) / kGN;
    a.batched = 1;
    a.splits = batch;
    a.kps = (K + kGK - 1) / kGK;
    a.C = C;
    a.vec = N % 4 == 0;
    a.tma_out = map_out_f32(&a.mOut, C, M, N, batch);
    a.timeout_ns = kGemmTimeoutNs;
    const int sms = gemm_sms();
    const int units = a.mt * a.nt * batch;
    const int pairs = units < sms / 2 ? units : sms / 2;
    const cudaError_t e = launch_gemm_any(true, true, EPI_F32, a, 2 * pairs, st);
    if (e == cudaSuccess) *launches = 1;
    return e;
}

cudaError_t gemm_error_word_read_clear(int* word) {
    const int zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(word, g_error_word, sizeof(int));
    if (e == cudaSuccess && *word) e = cudaMemcpyToSymbol(g_error_word, &zero, sizeof(int));
    return e;
}

}  // namespace hcw

extern "C" {

size_t hcw_gemm_workspace_bytes(int M, int N, int K) {
    if (M < 1 || N < 1 || K < 1) return 0;
    const size_t unlimited = (size_t)64 * M * N * sizeof(float);
    const int s = hcw::choose_splits(M, N, K, hcw::gemm_sms(), unlimited);
    return s > 1 ? (size_t)s * M * N * sizeof(float) : 0;
}

int hcw_gemm_bf16(int M, int N, int K, const void* A, int ta, const void* B, int tb, float* C,
                  void* workspace, size_t ws_bytes, void* stream) {
    if (M < 1 || N < 1 || K < 1 || !A || !B || !C || (ta != 0 && ta != 1) ||
        (tb != 0 && tb != 1))
        return HCW_ERR_INVALID_ARG;
    if (workspace && (reinterpret_cast<uintptr_t>(workspace) & 15)) return HCW_ERR_ALIGNMENT;
    const auto span = [](const void* p, size_t bytes) {
        return std::make_pair(reinterpret_cast<uintptr_t>(p),
                              reinterpret_cast<uintptr_t>(p) + bytes);
    };
    const auto overlap = [](std::pair<uintptr_t, uintptr_t> x, std::pair<uintptr_t, uintptr_t> y) {
        return x.first < y.second && y.first < x.second;
    };
    const auto c = span(C, (size_t)M * N * sizeof(float));
    if (overlap(c, span(A, (size_t)M * K * 2)) || overlap(c, span(B, (size_t)K * N * 2)) ||
        (workspace && ws_bytes && overlap(c, span(workspace, ws_bytes))))
        return HCW_ERR_ALIASING;
    int launches = 0;
    const cudaError_t e = hcw::gemm_bf16_f32(M, N, K, A, ta != 0, B, tb != 0, C,
                                             static_cast<float*>(workspace),
                                             workspace ? ws_bytes : 0, (cudaStream_t)stream,
                                             &launches);
    return hcw::count_launch(e, launches);
}

int hcw_gemm_bf16_batched(int M, int N, int K, const void* A, long long a_stride, const void* B,
                          long long b_stride, float* C, int batch, void* stream) {
    if (M < 1 || N < 1 || K < 1 || batch < 1 || a_stride < 0 || b_stride < 0 || !A || !B || !C)
        return HCW_ERR_INVALID_ARG;
    const auto span = [](const void* p, size_t bytes) {
        return std::make_pair(reinterpret_cast<uintptr_t>(p),
                              reinterpret_cast<uintptr_t>(p) + bytes);
    };
    const auto overlap = [](std::pair<uintptr_t, uintptr_t> x, std::pair<uintptr_t, uintptr_t> y) {
        return x.first < y.second && y.first < x.second;
    };
    const size_t nb = (size_t)batch - 1;
    const auto c = span(C, (size_t)batch * M * N * sizeof(float));
    if (overlap(c, span(A, (nb * (size_t)a_stride + (size_t)K * M) * 2)) ||
        overlap(c, span(B, (nb * (size_t)b_stride + (size_t)K * N) * 2)))
        return HCW_ERR_ALIASING;
    int launches = 0;
    const cudaError_t e = hcw::gemm_bf16_f32_batched(M, N, K, A, (size_t)a_stride * 2, B,
                                                     (size_t)b_stride * 2, C, batch,
                                                     (cudaStream_t)stream, &launches);
    return hcw::count_launch(e, launches);
}

}  // extern "C"
