// hcw_decode.cu -- one-token decode of a causal stack (Sec. 6, "Deployability":
// the decode path runs one token at a time, and a sparse layer needs only the
// last k inputs it links to, so its cache does not grow).
//
// B sequences advance together by one position t.  Layer l with link distance
// k_l (2^s for the hypercube link along dimension s, k for a shift layer) keeps
// a ring of k_l + 1 slots; the input of position p sits in slot p mod (k_l + 1).
// Position t receives at layer l when bit s of t is set (hypercube link) or
// t >= k (shift); its partner is position t - k_l, in slot (t + 1) mod
// (k_l + 1), which is never the slot t's own input goes to.  So layer l's
// epilogue writes its output straight into layer l + 1's ring, and nothing is
// read and overwritten within one step.
//
// The sequences never interact inside a layer (Eq. (1) mixes position t with
// one earlier position of the same sequence), so one position of the whole
// stack splits into independent blocks of 16 rows.  A thread-block cluster of
// C CTAs (C <= 16) runs one row block through all L layers; CTA q of the
// cluster owns output columns [q OC, (q + 1) OC), OC = d / C.  Per layer:
//   - a producer thread streams the CTA's weight rows (OC rows of W_nbr, then
//     of W_self, in K chunks) into a ring of shared-memory stages, and the
//     partner rows (16 x d, inputs of earlier positions) into a partner
//     buffer, running ahead of the layers.  Each moves as ONE TMA copy, a
//     3-D box (64 features, rows, K tiles) with the 128-byte swizzle that lands
//     as consecutive 64-feature tiles; one tensor map over the whole cache
//     serves every ring slot;
//   - eight MMA warps contract the partner part first (it does not depend on
//     the previous layer), then the self part once the layer input is
//     complete: [16 x d] x [d x OC] twice, fp32 accumulation;
//   - the epilogue (bias, ReLU, residual, bf16) writes the CTA's 16 x OC slice
//     to the next layer's ring slot in global memory and pushes it into every
//     cluster CTA's input buffer of the next layer with asynchronous remote
//     stores (distributed shared memory) that count their bytes on that CTA's
//     "input ready" mbarrier: the layer input is complete when all 16 x d x 2
//     bytes have landed, with no fence or barrier between the CTAs.
// No layer boundary goes through global memory or a grid-wide barrier.
//
// Two contractions (decode_kernel<TC>, chosen with hcw_set_decode_kernel):
//   - TC = false (the default): eight warps share the K range with the
//     warp-level bf16 MMA (m16n8k16) and add their 16 x 8 blocks into the
//     CTA's row sums;
//   - TC = true: one thread issues tcgen05.mma.  A tile holds 16 rows, below
//     the 64-row minimum, so the MMA runs with M = 64 on the 16 rows (its
//     other 48 rows read whatever follows in shared memory; only D's rows
//     0..15, TMEM lanes 0..15, are used) and N = OC.  The operands are already
//     in the MMA's K-major 128-byte-swizzled layout.  Warp 7 issues, warp 0
//     drains D into the row sums, and a layer's partner part is contracted
//     into the other of two accumulators while the layer before is drained.
// A layer is a chain (input in, contraction, epilogue, pushes out).  Issuing
// a layer's 32 partner-part MMAs (N = OC = 32 at d = 512, K = 16) only after
// its input arrived costs 0.75 us a layer, so one thread's tcgen05.mma run
// about 45 cycles each in sequence, where the eight warps' MMAs run side by
// side; the commit, the TMEM drain and a proxy fence (the remote stores are
// generic writes that the MMA reads through the async proxy) add to the chain.
// So the tensor-core version is the slower of the two here.
#include "hcw_internal.h"
#include "hcw_ptx.cuh"

namespace hcw {

namespace {

constexpr int kRows = 16;          // rows of a row block
constexpr int kMmaWarps = 8;       // warps 0..7: MMA + epilogue (TC: warp 7 issues, warps
                                   // 0..6 run the epilogue); warp 8: producer
constexpr int kThreads = (kMmaWarps + 1) * 32;
// TC: accumulators a layer's K tiles alternate over, for each layer parity (64
// columns each); four in turn measured no faster than one
constexpr int kNAcc = 1;
constexpr uint32_t kTmemCols = 2 * kNAcc * 64 < 32 ? 32 : 2 * kNAcc * 64;
constexpr int kMaxStages = 8;

struct DecodeArgs {
    CUtensorMap mWs, mWn;   // [L d][d] bf16, box (64 features, OC rows, kc / 64 tiles)
    CUtensorMap mCache;     // the rings as [rows][d] bf16, box (64, 16, d / 64)
    CUtensorMap mX;         // x_t [B][d] bf16, box (64, 16, d / 64)
    int prow[kMaxDecodeLayers];                 // cache row of the partner slot, or -1
    __nv_bfloat16* out[kMaxDecodeLayers];       // [B][d] next layer's ring slot, or y_t
    const float* bias;     // [L][d] or null
    __nv_bfloat16* ring0;  // layer 0's ring slot of position t
    DecodeGeo g;
    int L, B;
    unsigned flags;
    unsigned long long timeout_ns;
};

// barrier slots
enum : int {
    B_FULL = 0,                       // [kMaxStages] stage filled (tx bytes)
    B_EMPTY = kMaxStages,             // [kMaxStages] stage consumed (8 MMA warps, or a commit)
    B_XS_READY = 2 * kMaxStages,      // [2] layer input complete (tx bytes from every cluster CTA)
    B_X0 = 2 * kMaxStages + 2,        // x_t rows loaded
    B_XP_FULL = 2 * kMaxStages + 3,   // [2] partner rows loaded
    B_XP_FREE = 2 * kMaxStages + 5,   // [2] partner buffer consumed (8 MMA warps, or a commit)
    B_DFULL = 2 * kMaxStages + 7,     // TC: [2] a layer's accumulator complete (commit)
    B_TFREE = 2 * kMaxStages + 9,     // TC: [2] a layer's accumulator drained by warp 0
    B_DRAIN = 2 * kMaxStages + 11,    // TC: the issuer's last MMAs completed
    B_COUNT = 2 * kMaxStages + 12
};

// Shared memory (1024-byte aligned): Xs[2] (layer inputs) and Xp[2] (partner
// rows), each d / 64 tiles of 16 rows x 128 bytes; stages[S], each kc / 64
// tiles of OC rows x 128 bytes; all bf16 in the 128-byte swizzle (16-byte
// chunk c of row r at chunk c ^ (r & 7)).  Then red[2][16][OC] fp32 (the
// partial sums of alternate layers), the mbarriers and the abort word.
struct Smem {
    uint8_t* base;
    const DecodeGeo& g;
    __device__ Smem(uint8_t* b, const DecodeGeo& geo) : base(b), g(geo) {}
    __device__ uint8_t* xs(int buf) const { return base + (size_t)buf * kRows * g.d * 2; }
    __device__ uint8_t* xpart(int buf) const { return base + (size_t)(2 + buf) * kRows * g.d * 2; }
    __device__ uint8_t* stage(int s) const {
        return base + (size_t)4 * kRows * g.d * 2 + (size_t)s * g.oc * g.kc * 2;
    }
    __device__ float* red(int buf) const {
        return reinterpret_cast<float*>(stage(g.stages)) + buf * kRows * g.oc;
    }
    __device__ uint64_t* bars() const {
        return reinterpret_cast<uint64_t*>(red(2));
    }
    __device__ int* abort_word() const { return reinterpret_cast<int*>(bars() + B_COUNT); }
    __device__ uint32_t* tmem_slot() const {
        return reinterpret_cast<uint32_t*>(abort_word() + 1);
    }
};

// byte offset of the 16-byte chunk holding features [8 c, 8 c + 8) of row r
// in a swizzled buffer of 64-feature tiles, tile_bytes apart
__device__ __forceinline__ uint32_t sw_off(int r, int col, uint32_t tile_bytes) {
    const int ch = (col >> 3) & 7;
    return (uint32_t)(col >> 6) * tile_bytes + r * 128 + ((ch ^ (r & 7)) << 4);
}

__device__ __forceinline__ void ldmatrix_x4(uint32_t addr, uint32_t& r0, uint32_t& r1,
                                            uint32_t& r2, uint32_t& r3) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
                 : "r"(addr));
}
__device__ __forceinline__ void ldmatrix_x2(uint32_t addr, uint32_t& r0, uint32_t& r1) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x2.shared.b16 {%0, %1}, [%2];"
                 : "=r"(r0), "=r"(r1)
                 : "r"(addr));
}

// D (16 x 8, fp32) += A (16 x 16 bf16, row-major) * B (16 x 8 bf16, column-major)
__device__ __forceinline__ void mma_16816(float* c, const uint32_t* a, uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, "
        "{%4, %5, %6, %7}, {%8, %9}, {%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// 16 bytes into the shared memory of a cluster CTA; the bytes complete on that
// CTA's mbarrier (both given by shared::cluster addresses in the same CTA)
__device__ __forceinline__ void st_async_v4(uint32_t addr, uint4 v, uint32_t bar) {
    asm volatile(
        "st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.b32 [%0], {%1, %2, %3, %4}, "
        "[%5];" ::"r"(addr),
        "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w), "r"(bar)
        : "memory");
}

// K chunk c of a part: [c kc, min(d, (c + 1) kc))
__device__ __forceinline__ int chunk_len(const DecodeGeo& g, int c) {
    const int k0 = c * g.kc;
    return g.d - k0 < g.kc ? g.d - k0 : g.kc;
}

// The end of a layer for one epilogue thread (8 columns of one row, v =
// the row sums plus bias): ReLU, residual, bf16; the result goes into every
// cluster CTA's next-layer input (remote stores counted on its input barrier)
// and, for a valid row, to the layer's output in global memory.
__device__ __forceinline__ void decode_epilogue(const DecodeArgs& a, const Smem& sm, float (&v)[8],
                                                uint4 xin, int l, int xb, int q, int row0,
                                                int vr, int pr, int pc8, uint32_t poff) {
    const DecodeGeo& g = a.g;
    const int d = g.d, col0 = q * g.oc;
    if (a.flags & 4u) {
#pragma unroll
        for (int e = 0; e < 8; ++e) v[e] = v[e] > 0.f ? v[e] : 0.f;
    }
    if (a.flags & 2u) {
        const uint32_t w[4] = {xin.x, xin.y, xin.z, xin.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 f = unpack_bf16x2(w[e]);
            v[2 * e] += f.x;
            v[2 * e + 1] += f.y;
        }
    }
    uint4 pk;
    pk.x = pack_bf16x2(v[0], v[1]);
    pk.y = pack_bf16x2(v[2], v[3]);
    pk.z = pack_bf16x2(v[4], v[5]);
    pk.w = pack_bf16x2(v[6], v[7]);
    if (l + 1 < a.L) {
        const uint8_t* dst = sm.xs(xb ^ 1) + poff;
        const uint64_t* rb = &sm.bars()[B_XS_READY + (xb ^ 1)];
        for (int cr = 0; cr < g.csize; ++cr)
            st_async_v4(mapa_shared(dst, cr), pk, mapa_shared(rb, cr));
    }
    if (pr < vr) {
        if (l == 0)   // position t's layer-0 input into layer 0's ring
            *reinterpret_cast<uint4*>(a.ring0 + (size_t)(row0 + pr) * d + col0 + pc8) = xin;
        *reinterpret_cast<uint4*>(a.out[l] + (size_t)(row0 + pr) * d + col0 + pc8) = pk;
    }
}

// The MMA and epilogue warps of decode_kernel<true>: warp 7 issues the
// tcgen05 MMAs, warp 0 drains each layer's accumulator into the row sums, and
// warps 0..6 run the epilogue (bias, ReLU, residual, bf16, pushes).
__device__ __forceinline__ void decode_tc_body(const DecodeArgs& a, const Smem& sm, int warp,
                                            int lane, int q, int row0, int vr) {
    const DecodeGeo& g = a.g;
    uint64_t* bars = sm.bars();
    const int d = g.d, oc = g.oc, col0 = q * oc, nch = g.nchunks;
    const uint32_t xtile = kRows * 128, wtile = (uint32_t)oc * 128;
    volatile int* abort = sm.abort_word();
    const uint32_t IDESC = idesc_bf16_f32(64, oc, 0, 0);
    const uint32_t tmem_base = *reinterpret_cast<volatile uint32_t*>(sm.tmem_slot());
    const int packs = kRows * oc / 8;   // epilogue: a thread per 8 columns of a row
    const int pr = threadIdx.x / (oc / 8), pc8 = (threadIdx.x % (oc / 8)) * 8;
    const uint32_t poff = sw_off(pr, col0 + pc8, xtile);
    bool ok = true;
    if (warp == kMmaWarps - 1) {
        if (lane == 0) {
            // ---------------------------------------------- MMA issuer
            uint32_t it = 0;
            int xp_uses[2] = {0, 0};
            for (int l = 0; l < a.L && ok; ++l) {
                const int xb = l & 1, ab = l & 1;
                const bool recv = a.prow[l] >= 0;
                // the accumulator of this parity has been drained (layer l - 2)
                if (l >= 2)
                    ok = mbar_wait(&bars[B_TFREE + ab], ((l - 2) >> 1) & 1, abort, a.timeout_ns);
                if (!ok) break;
                tc_fence_after();
                // K tile j of the layer goes to accumulator j mod kNAcc: consecutive
                // MMAs do not wait on each other's result
                int tix = 0;
                for (int part = recv ? 1 : 0; part >= 0 && ok; --part) {
                    uint32_t X;
                    if (part) {
                        ok = mbar_wait(&bars[B_XP_FULL + xb], xp_uses[xb]++ & 1, abort,
                                       a.timeout_ns);
                        X = smem_u32(sm.xpart(xb));
                    } else {
                        ok = l == 0 ? mbar_wait(&bars[B_X0], 0, abort, a.timeout_ns)
                                    : mbar_wait_cluster(&bars[B_XS_READY + xb], ((l - 1) >> 1) & 1,
                                                        abort, a.timeout_ns);
                        X = smem_u32(sm.xs(xb));
                        // the input came by remote stores (generic proxy); the MMAs
                        // read it through the async proxy
                        if (ok) fence_proxy_async_smem();
                    }
                    if (!ok) break;
                    tc_fence_after();
                    for (int c = 0; c < nch && ok; ++c, ++it) {
                        const int s = (int)(it % (uint32_t)g.stages);
                        ok = mbar_wait(&bars[B_FULL + s], (it / g.stages) & 1, abort, a.timeout_ns);
                        if (!ok) break;
                        tc_fence_after();
                        const uint32_t W = smem_u32(sm.stage(s));
                        const int tiles = chunk_len(g, c) / 64, t0 = c * g.kc / 64;
                        for (int t = 0; t < tiles; ++t, ++tix) {
                            const uint32_t d_tmem =
                                tmem_base + (uint32_t)((ab * kNAcc + tix % kNAcc) * 64);
#pragma unroll
                            for (int kk = 0; kk < 4; ++kk) {
                                const uint64_t ad = smem_desc_sw128(
                                    X + (uint32_t)(t0 + t) * xtile + kk * 32, 16, 1024);
                                const uint64_t bd =
                                    smem_desc_sw128(W + (uint32_t)t * wtile + kk * 32, 16, 1024);
                                mma_bf16_f32(d_tmem, ad, bd, IDESC,
                                             (tix < kNAcc && kk == 0) ? 0u : 1u);
                            }
                        }
                        mma_commit(&bars[B_EMPTY + s]);
                    }
                    if (ok && part) mma_commit(&bars[B_XP_FREE + xb]);
                }
                if (ok) mma_commit(&bars[B_DFULL + ab]);
            }
            if (!ok) *abort = 1;
            // the MMAs have completed before the CTA frees TMEM at the end
            if (it > 0) {
                mma_commit(&bars[B_DRAIN]);
                mbar_wait_drain(&bars[B_DRAIN], 0, a.timeout_ns);
            }
        }
        __syncwarp();
        return;
    }
    for (int l = 0; l < a.L; ++l) {
        const int xb = l & 1, ab = l & 1;
        // the next layer's input arrives as 16 x d x 2 bytes from the cluster
        if (threadIdx.x == 0 && l + 1 < a.L)
            mbar_arrive_expect_tx(&bars[B_XS_READY + (xb ^ 1)], (uint32_t)kRows * d * 2);
        // this thread's bias values, loaded while the layer runs
        float4 bv0 = make_float4(0.f, 0.f, 0.f, 0.f), bv1 = bv0;
        if (a.bias && (int)threadIdx.x < packs) {
            const float4* bl = reinterpret_cast<const float4*>(a.bias + (size_t)l * d + col0 + pc8);
            bv0 = __ldg(bl);
            bv1 = __ldg(bl + 1);
        }
        float* red = sm.red(xb);
        if (warp == 0) {
            // D rows 0..15 (TMEM lanes 0..15) into this layer's row sums
            bool r = ok && mbar_wait(&bars[B_DFULL + ab], (l >> 1) & 1, abort, a.timeout_ns);
            ok = __all_sync(0xffffffffu, r);
            if (ok) {
                tc_fence_after();
                // the accumulators the layer's K tiles went to, added in order
                const int ntiles = (a.prow[l] >= 0 ? 2 : 1) * (d / 64);
                const int nacc = ntiles < kNAcc ? ntiles : kNAcc;
                for (int c0 = 0; c0 < oc; c0 += 32) {
                    float sum[32];
#pragma unroll
                    for (int e = 0; e < 32; ++e) sum[e] = 0.f;
                    for (int ac = 0; ac < nacc; ++ac) {
                        uint32_t raw[32];
                        tmem_ld_32x32b_x32(
                            tmem_base + (uint32_t)((ab * kNAcc + ac) * 64 + c0), raw);
                        tmem_ld_wait_regs(raw);
#pragma unroll
                        for (int e = 0; e < 32; ++e) sum[e] += __uint_as_float(raw[e]);
                    }
                    const int nc = oc - c0 < 32 ? oc - c0 : 32;
                    if (lane < kRows) {
#pragma unroll
                        for (int e = 0; e < 32; ++e)
                            if (e < nc) red[lane * oc + c0 + e] = sum[e];
                    }
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(&bars[B_TFREE + ab]);
            }
        }
        // the layer input (the residual) is complete here: every thread takes
        // the barrier's acquire before it reads it
        {
            bool r = ok && (l == 0 ? mbar_wait(&bars[B_X0], 0, abort, a.timeout_ns)
                                   : mbar_wait_cluster(&bars[B_XS_READY + xb], ((l - 1) >> 1) & 1,
                                                       abort, a.timeout_ns));
            ok = __all_sync(0xffffffffu, r);
        }
        // every thread past this point has finished the previous layer's
        // epilogue, so the other row-sum buffer is free again
        named_bar_sync(1, (kMmaWarps - 1) * 32);
        if (ok && (int)threadIdx.x < packs) {
            const uint4 xin = *reinterpret_cast<const uint4*>(sm.xs(xb) + poff);
            const float* rr = red + pr * oc + pc8;
            const float bvals[8] = {bv0.x, bv0.y, bv0.z, bv0.w, bv1.x, bv1.y, bv1.z, bv1.w};
            float v[8];
#pragma unroll
            for (int e = 0; e < 8; ++e) v[e] = rr[e] + bvals[e];
            decode_epilogue(a, sm, v, xin, l, xb, q, row0, vr, pr, pc8, poff);
        }
    }
}

template <bool TC>
__global__ void __launch_bounds__(kThreads, 1) decode_kernel(const __grid_constant__ DecodeArgs a) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t* base = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    const DecodeGeo& g = a.g;
    const Smem sm(base, g);
    uint64_t* bars = sm.bars();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int q = (int)cluster_ctarank();
    const int row0 = (int)(blockIdx.x / g.csize) * kRows;   // this cluster's row block
    const int vr = a.B - row0 < kRows ? a.B - row0 : kRows;   // valid rows
    const int d = g.d, oc = g.oc, col0 = q * oc;
    const int nch = g.nchunks;
    const uint32_t xtile = kRows * 128, wtile = (uint32_t)oc * 128;
    volatile int* abort = sm.abort_word();

    for (int i = threadIdx.x; i < 2 * kRows * oc; i += kThreads) sm.red(0)[i] = 0.f;
    if (threadIdx.x == 0) {
        *abort = 0;
        for (int s = 0; s < g.stages; ++s) {
            mbar_init(&bars[B_FULL + s], 1);
            mbar_init(&bars[B_EMPTY + s], TC ? 1 : kMmaWarps);
        }
        mbar_init(&bars[B_XS_READY + 0], 1);
        mbar_init(&bars[B_XS_READY + 1], 1);
        mbar_init(&bars[B_X0], 1);
        for (int b = 0; b < 2; ++b) {
            mbar_init(&bars[B_XP_FULL + b], 1);
            mbar_init(&bars[B_XP_FREE + b], TC ? 1 : kMmaWarps);
            mbar_init(&bars[B_DFULL + b], 1);
            mbar_init(&bars[B_TFREE + b], 1);
        }
        mbar_init(&bars[B_DRAIN], 1);
        fence_mbar_init();
    }
    if (TC && warp == 0) {
        tmem_alloc(sm.tmem_slot(), kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync_all();   // barriers initialised in every CTA of the cluster
    tc_fence_after();

    if (warp == kMmaWarps) {
        // ---------------------------------------------------------- producer
        if (lane == 0) {
            tma_prefetch_desc(&a.mWs);
            tma_prefetch_desc(&a.mWn);
            tma_prefetch_desc(&a.mCache);
            uint32_t it = 0;            // weight chunks issued
            int xp_fills[2] = {0, 0};   // partner-buffer fills issued
            bool ok = true;
            mbar_arrive_expect_tx(&bars[B_X0], (uint32_t)kRows * d * 2);
            tma_load_3d(sm.xs(0), &a.mX, &bars[B_X0], 0, row0, 0);
            for (int l = 0; l < a.L && ok; ++l) {
                const int prow = a.prow[l];
                if (prow >= 0) {
                    const int b = l & 1, u = xp_fills[b];
                    if (u > 0)
                        ok = mbar_wait(&bars[B_XP_FREE + b], (u - 1) & 1, abort, a.timeout_ns);
                    if (!ok || *abort) {
                        ok = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&bars[B_XP_FULL + b], (uint32_t)kRows * d * 2);
                    tma_load_3d(sm.xpart(b), &a.mCache, &bars[B_XP_FULL + b], 0, prow + row0, 0);
                    xp_fills[b] = u + 1;
                }
                // weight chunks: the partner part (if any), then the self part
                for (int part = prow >= 0 ? 1 : 0; part >= 0 && ok; --part) {
                    const CUtensorMap* mW = part ? &a.mWn : &a.mWs;
                    for (int c = 0; c < nch; ++c) {
                        const int s = (int)(it % (uint32_t)g.stages);
                        const int klen = chunk_len(g, c);
                        if (it >= (uint32_t)g.stages)
                            ok = mbar_wait(&bars[B_EMPTY + s], ((it / g.stages) - 1) & 1, abort,
                                           a.timeout_ns);
                        if (!ok || *abort) {
                            ok = false;
                            break;
                        }
                        // a ragged last chunk is the box's first klen / 64 tiles; the
                        // rest fall past d and arrive as zeros (counted in full)
                        mbar_arrive_expect_tx(&bars[B_FULL + s], (uint32_t)oc * g.kc * 2);
                        tma_load_3d(sm.stage(s), mW, &bars[B_FULL + s], 0, l * d + col0,
                                    c * g.kc / 64);
                        ++it;
                    }
                }
            }
            // after an abort: let every copy this CTA issued land before it exits
            if (!ok) {
                mbar_wait_drain(&bars[B_X0], 0, a.timeout_ns);
                for (uint32_t j = it > (uint32_t)g.stages ? it - g.stages : 0; j < it; ++j)
                    mbar_wait_drain(&bars[B_FULL + j % g.stages], (j / g.stages) & 1,
                                    a.timeout_ns);
                for (int b = 0; b < 2; ++b)
                    if (xp_fills[b] > 0)
                        mbar_wait_drain(&bars[B_XP_FULL + b], (xp_fills[b] - 1) & 1,
                                        a.timeout_ns);
            }
        }
        __syncwarp();
    } else if (TC) {
        decode_tc_body(a, sm, warp, lane, q, row0, vr);
    } else {
        // ---------------------------------------------------- MMA + epilogue
        const int nb_count = oc / 8;               // n8 blocks: 2, 4 or 8
        const int ksplit = kMmaWarps / nb_count;   // warps sharing an n8 block
        const int nb = warp % nb_count, kh = warp / nb_count;
        const int gr = lane >> 2, gc = (lane & 3) * 2;
        // ldmatrix lanes: A rows lane & 15, feature chunk + (lane >> 4); B
        // (weight) rows nb 8 + (lane & 7), feature chunk + ((lane >> 3) & 1)
        const int ar = lane & 15, ahi = lane >> 4;
        const int br = nb * 8 + (lane & 7), bhi = (lane >> 3) & 1;
        uint32_t it = 0;
        int xp_uses[2] = {0, 0};
        bool ok = true;
        // every lane waits (each gets the acquire); the outcome is made
        // warp-uniform so that the aligned MMAs never run divergent
        auto wait = [&](uint64_t* bar, uint32_t parity, bool cluster) {
            bool r = ok && (cluster ? mbar_wait_cluster(bar, parity, abort, a.timeout_ns)
                                    : mbar_wait(bar, parity, abort, a.timeout_ns));
            ok = __all_sync(0xffffffffu, r);
        };
        const int packs = kRows * oc / 8;   // epilogue: a thread per 8 columns of a row
        const int pr = threadIdx.x / (oc / 8), pc8 = (threadIdx.x % (oc / 8)) * 8;
        const uint32_t poff = sw_off(pr, col0 + pc8, xtile);
        for (int l = 0; l < a.L; ++l) {
            const int xb = l & 1;
            const bool recv = a.prow[l] >= 0;
            // the next layer's input arrives as 16 x d x 2 bytes from the cluster
            if (threadIdx.x == 0 && l + 1 < a.L)
                mbar_arrive_expect_tx(&bars[B_XS_READY + (xb ^ 1)], (uint32_t)kRows * d * 2);
            // this thread's bias values, loaded while the layer runs
            float4 bv0 = make_float4(0.f, 0.f, 0.f, 0.f), bv1 = bv0;
            if (a.bias && (int)threadIdx.x < packs) {
                const float4* bl =
                    reinterpret_cast<const float4*>(a.bias + (size_t)l * d + col0 + pc8);
                bv0 = __ldg(bl);
                bv1 = __ldg(bl + 1);
            }
            // four independent accumulators: consecutive MMAs do not wait on each other
            float acc[4][4];
#pragma unroll
            for (int u = 0; u < 4; ++u)
#pragma unroll
                for (int e = 0; e < 4; ++e) acc[u][e] = 0.f;
            for (int part = recv ? 1 : 0; part >= 0; --part) {
                uint32_t X;
                if (part) {
                    wait(&bars[B_XP_FULL + xb], xp_uses[xb]++ & 1, false);
                    X = smem_u32(sm.xpart(xb));
                } else {
                    if (l == 0)
                        wait(&bars[B_X0], 0, false);
                    else
                        wait(&bars[B_XS_READY + xb], ((l - 1) >> 1) & 1, true);
                    X = smem_u32(sm.xs(xb));
                }
                for (int c = 0; c < nch; ++c, ++it) {
                    const int s = (int)(it % (uint32_t)g.stages);
                    wait(&bars[B_FULL + s], (it / g.stages) & 1, false);
                    if (ok) {
                        const uint32_t W = smem_u32(sm.stage(s));
                        const int ks_n = chunk_len(g, c) / 16;
                        const int kc0 = c * g.kc;
                        int ks = kh;
                        for (; ks + 3 * ksplit < ks_n; ks += 4 * ksplit) {
                            uint32_t af[4][4], bf[4][2];
#pragma unroll
                            for (int u = 0; u < 4; ++u) {
                                const int kl = (ks + u * ksplit) * 16;
                                ldmatrix_x4(X + sw_off(ar, kc0 + kl + ahi * 8, xtile), af[u][0],
                                            af[u][1], af[u][2], af[u][3]);
                                ldmatrix_x2(W + sw_off(br, kl + bhi * 8, wtile), bf[u][0],
                                            bf[u][1]);
                            }
#pragma unroll
                            for (int u = 0; u < 4; ++u) mma_16816(acc[u], af[u], bf[u][0], bf[u][1]);
                        }
                        for (; ks < ks_n; ks += ksplit) {
                            const int kl = ks * 16;
                            uint32_t af[4], b0, b1;
                            ldmatrix_x4(X + sw_off(ar, kc0 + kl + ahi * 8, xtile), af[0], af[1],
                                        af[2], af[3]);
                            ldmatrix_x2(W + sw_off(br, kl + bhi * 8, wtile), b0, b1);
                            mma_16816(acc[0], af, b0, b1);
                        }
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&bars[B_EMPTY + s]);
                }
                if (part && lane == 0) mbar_arrive(&bars[B_XP_FREE + xb]);
            }
            // this warp's partial 16 x 8 block into the CTA's sums of this layer
            float* red = sm.red(xb);
            const int cb = nb * 8 + gc;
            atomicAdd(&red[gr * oc + cb], acc[0][0] + acc[1][0] + acc[2][0] + acc[3][0]);
            atomicAdd(&red[gr * oc + cb + 1], acc[0][1] + acc[1][1] + acc[2][1] + acc[3][1]);
            atomicAdd(&red[(gr + 8) * oc + cb], acc[0][2] + acc[1][2] + acc[2][2] + acc[3][2]);
            atomicAdd(&red[(gr + 8) * oc + cb + 1], acc[0][3] + acc[1][3] + acc[2][3] + acc[3][3]);
            // every thread past this point has finished the previous layer's
            // epilogue, so the other partial-sum buffer is free again
            named_bar_sync(1, kMmaWarps * 32);
            if ((int)threadIdx.x < packs) {
                const uint4 xin = *reinterpret_cast<const uint4*>(sm.xs(xb) + poff);
                float* rr = red + pr * oc + pc8;
                const float bvals[8] = {bv0.x, bv0.y, bv0.z, bv0.w, bv1.x, bv1.y, bv1.z, bv1.w};
                float v[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    v[e] = rr[e] + bvals[e];
                    rr[e] = 0.f;
                }
                decode_epilogue(a, sm, v, xin, l, xb, q, row0, vr, pr, pc8, poff);
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync_all();   // no CTA leaves while a peer may still write its shared memory
    if (TC && warp == 0) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc(*sm.tmem_slot(), kTmemCols);
    }
}

}  // namespace

bool decode_geometry(int d, DecodeGeo* g) {
    if (d < 64 || d % 64 != 0 || d > 1024) return false;
    int oc = 16;
    while (d / oc > 16) oc *= 2;   // C = d / OC CTAs, at most 16; OC in {16, 32, 64}
    g->d = d;
    g->oc = oc;
    g->csize = d / oc;
    g->kc = oc == 64 ? 128 : 256;
    if (g->kc > d) g->kc = d;
    g->nchunks = (d + g->kc - 1) / g->kc;
    const size_t fixed =
        1024 + (size_t)4 * kRows * d * 2 + (size_t)2 * kRows * oc * 4 + B_COUNT * 8 + 16;
    const size_t stage = (size_t)oc * g->kc * 2;
    const size_t budget = 226 * 1024;
    const int s = (int)((budget - fixed) / stage);
    g->stages = s > kMaxStages ? kMaxStages : s;
    return g->stages >= 2;
}

size_t decode_smem_bytes(const DecodeGeo& g) {
    return 1024 + (size_t)4 * kRows * g.d * 2 + (size_t)g.stages * g.oc * g.kc * 2 +
           (size_t)2 * kRows * g.oc * 4 + B_COUNT * 8 + 16;
}

cudaError_t launch_decode(const DecodeLaunch& p, cudaStream_t st) {
    if (p.L < 1 || p.L > kMaxDecodeLayers) return cudaErrorInvalidValue;
    DecodeArgs a;
    a.mWs = p.mWs;
    a.mWn = p.mWn;
    a.mCache = p.mCache;
    a.mX = p.mX;
    for (int l = 0; l < p.L; ++l) {
        a.prow[l] = p.prow[l];
        a.out[l] = p.out[l];
    }
    a.bias = p.bias;
    a.ring0 = p.ring0;
    a.g = p.g;
    a.L = p.L;
    a.B = p.B;
    a.flags = p.flags;
    a.timeout_ns = p.timeout_ns;
    const size_t smem = decode_smem_bytes(p.g);
    auto kern = p.tc ? decode_kernel<true> : decode_kernel<false>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e == cudaSuccess && p.g.csize > 8)
        e = cudaFuncSetAttribute(kern, cudaFuncAttributeNonPortableClusterSizeAllowed, 1);
    if (e != cudaSuccess) return e;
    const int blocks = (p.B + kRows - 1) / kRows;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(blocks * p.g.csize));
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = (unsigned)p.g.csize;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int clusters = 0;
    e = cudaOccupancyMaxActiveClusters(&clusters, kern, &cfg);
    if (e != cudaSuccess) return e;
    if (clusters < 1) return cudaErrorInvalidConfiguration;
    return cudaLaunchKernelEx(&cfg, kern, a);
}

cudaError_t decode_error_word_read_clear(int* word) {
    const int zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(word, g_error_word, sizeof(int));
    if (e == cudaSuccess && *word) e = cudaMemcpyToSymbol(g_error_word, &zero, sizeof(int));
    return e;
}

}  // namespace hcw
