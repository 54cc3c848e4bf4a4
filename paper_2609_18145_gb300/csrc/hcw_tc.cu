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
// are loaded as MN-major operands straight from the token-major activations.
// A launch over up to 16 layers gives every (layer, part, output tile) one
// unit over the whole token range; a single layer splits the token range so
// that its units fill the GPU and a separate kernel reduces the fp32
// partials in a fixed order.  Both are deterministic.
//
// Roles: warp 0 issues TMA loads into a ring of shared-memory stages; warp 1
// owns TMEM (2 x BN fp32 columns, a double-buffered accumulator) and issues
// tcgen05.mma; the other warps drain the accumulator through tcgen05.ld:
// sixteen of them for tiles of 128 or 256 columns (four per TMEM lane
// quarter, each a 32-row patch of BN/4 columns), eight for narrower tiles.
// The epilogue is latency-bound (TMEM loads, residual loads, store
// completion), so the warps per scheduler matter more than the work per
// warp.  All epilogue I/O goes through TMA: each epilogue warp has one 4 KB
// buffer; the residual rows of its patch are TMA-loaded into it before the
// accumulator is ready, each lane overwrites its own row in place with the
// result, and a TMA store writes the patch back.  Every
// wait is bounded (hcw_ptx.cuh); a CTA that gives up records
// HCW_ERR_TIMEOUT, drains its in-flight copies and MMAs, frees TMEM and
// returns.
#include <atomic>
#include <type_traits>

#include "hcw_internal.h"
#include "hcw_ptx.cuh"

namespace hcw {

namespace {

constexpr int kMaxEpiWarps = 16;
constexpr int kUnitQ = 8;                          // claimed units in flight per CTA
constexpr int kDwHelpers = 4;                      // DW: epilogue warps that also release stages
constexpr int kBlockM = 128;
constexpr int kBlockK = 64;                        // bf16 elements per 128-byte row
constexpr int kABytes = kBlockM * kBlockK * 2;     // 16 KB
constexpr int kRingBytes = 144 * 1024;             // TMA stage ring
constexpr int kRingBytesDwf = 192 * 1024;          // MODE_DWF: no epilogue buffers
constexpr int kEpiBufBytes = 4096;                 // one epilogue patch: 32 rows x <= 128 B

// epilogue warps (a multiple of 4: one group per TMEM lane quarter), threads,
// and columns of the patch each epilogue warp drains
__host__ __device__ constexpr int epi_warps(int BN) { return BN >= 128 ? 16 : 8; }
__host__ __device__ constexpr int cta_threads(int BN) { return 64 + 32 * epi_warps(BN); }
__host__ __device__ constexpr int warp_cols(int BN) { return BN / (epi_warps(BN) / 4); }

__host__ __device__ constexpr int stage_bytes(int BN) { return kABytes + BN * kBlockK * 2; }
__host__ __device__ constexpr int num_stages(int BN, int MODE = MODE_FWD) {
    // MODE_DWF takes its stages in pairs (the bit-0 and bit-1 rows of a block):
    // an even count
    return MODE == MODE_DWF
               ? ((kRingBytesDwf / stage_bytes(BN)) > 8 ? 8 : (kRingBytesDwf / stage_bytes(BN))) & ~1
               : ((kRingBytes / stage_bytes(BN)) > 8 ? 8 : (kRingBytes / stage_bytes(BN)));
}

struct __align__(8) Barriers {
    uint64_t full[8];
    uint64_t empty[8];
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint64_t drain;
    uint64_t epi_load[kMaxEpiWarps];              // residual patch landed in a warp's buffer
    uint32_t tmem_base;
    int abort;
    int dep_unit;   // the producer has seen the inputs of this CTA's units up to this ordinal
    int unit_q[kUnitQ];   // dynamic scheduling: unit claimed for ordinal o, in slot o % kUnitQ
    int q_pub;            // highest ordinal published in unit_q
    int q_read;           // slot reads so far (the MMA thread and every epilogue warp)
    // stacked row launches: epilogue warps whose stores of the unit in slot o %
    // kUnitQ have completed, per published output (0: the counters' output,
    // 1: the input gradient's g); the last one publishes the CTA's rows
    int pub_done[2][kUnitQ];
};

// epilogue patch buffers (MODE_DWF stores from registers)
template <int MODE, int BN>
__host__ __device__ constexpr size_t epi_smem_bytes() {
    return MODE == MODE_DWF ? 0 : (size_t)epi_warps(BN) * kEpiBufBytes;
}

// Stages of the pair variant of the row kernels: this CTA's A and half of B,
// as many as the shared memory left by the epilogue buffers holds (at most 8;
// five at BN = 256, six at BN = 128).
constexpr size_t kSmemBudget = 232448;
__host__ __device__ constexpr int pair_row_stage_bytes(int BN) { return kABytes + BN * kBlockK; }
__host__ __device__ constexpr int tc_pair_stages(int BN) {
    return (int)((kSmemBudget - 1024 - (size_t)epi_warps(BN) * kEpiBufBytes - sizeof(Barriers)) /
                 pair_row_stage_bytes(BN)) > 8
               ? 8
               : (int)((kSmemBudget - 1024 - (size_t)epi_warps(BN) * kEpiBufBytes -
                        sizeof(Barriers)) /
                       pair_row_stage_bytes(BN));
}

template <int MODE, int BN, bool PAIR = false>
__host__ __device__ constexpr size_t smem_total() {
    return 1024 /* alignment slack */ +
           (PAIR ? (size_t)tc_pair_stages(BN) * pair_row_stage_bytes(BN)
                 : (size_t)num_stages(BN, MODE) * stage_bytes(BN)) +
           epi_smem_bytes<MODE, BN>() + sizeof(Barriers);
}

// FWD/DX unit -> (row bit beta, row block t, column tile j, number of K steps)
struct RowUnit {
    int beta, t, j, steps;
};

__device__ __forceinline__ RowUnit decode_row_unit(const TcParams& p, int u, bool stacked,
                                                   bool mirror = false, bool shift = false) {
    RowUnit r;
    const int per_bit = p.n_rb * p.n_nt;
    int g, rem;
    if (!stacked) {
        // one layer: the long (two-part) units first, then the short ones
        g = u / per_bit;
        rem = u - g * per_bit;
        r.t = rem / p.n_nt;
        r.j = rem - r.t * p.n_nt;
    } else {
        // a run of layers: row block by row block, so that the next layer's
        // first blocks find their inputs early
        r.t = u / (2 * p.n_nt);
        rem = u - r.t * 2 * p.n_nt;
        g = rem / p.n_nt;
        r.j = rem - g * p.n_nt;
    }
    if (shift) {
        // a shift layer of Eq. (1) in a stacked launch: every row takes both
        // parts (the rows before k read zeros); g picks one of the row block's
        // two 128-token runs
        r.beta = g;
        r.steps = 2 * p.nK;
        return r;
    }
    if (g < p.n_full) {
        r.beta = g == 0 ? p.full_bit0 : p.full_bit1;
        r.steps = 2 * p.nK;
    } else {
        r.beta = p.half_bit;
        r.steps = p.nK;
    }
    // input-gradient units of a fused launch (parameters set for the forward):
    // under the causal rule the rows that take both parts are the other bit value
    if (mirror && p.n_full == 1) r.beta ^= 1;
    return r;
}

// The 128-token chunks holding the rows of a row unit that starts at
// compressed row q0 (for link distance k = 2^s) and their partners.
__device__ __forceinline__ void row_unit_chunks(int q0, int s, int k, int& ca, int& cb) {
    const int tok_a = ((q0 >> s) << (s + 1)) + (q0 & (k - 1));
    ca = tok_a >> 7;
    cb = k >= 128 ? ((tok_a + k) >> 7) : ca + 1;
}

// Bounded waits for the inputs of a shift-layer unit of a stacked launch: its
// own 128 tokens [tok0, tok0 + 128) (positions pos0 .. pos0 + 127 of one
// sample of n) and its partner rows at offset `off` (-k forward, +k input
// gradient), clipped to the sample -- rows outside it load as zeros and are
// nobody's output.  At most three 128-token chunks.
__device__ bool wait_shift_chunks(const int* ctr, int n_chunks, int tokens, int d, int tok0,
                                  int pos0, int n, int off, volatile int* abort,
                                  uint64_t timeout_ns);

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

// Weight-gradient unit u of a launch.  One layer: decode_w_unit.  A run of
// independent layers: every layer's self-part units first (the long ones),
// then the partner-part units, layer-major inside each group.
__device__ __forceinline__ WUnit decode_w_any(const TcParams& p, int u, bool stacked,
                                              int n_layers, int& layer) {
    if (!stacked) {
        layer = 0;
        return decode_w_unit(p, u);
    }
    const int tiles = p.n_ot * p.n_nt;
    const int self_pl = tiles * p.splits_self;
    const int nbr_pl = tiles * p.splits_nbr;
    int local;
    if (u < n_layers * self_pl) {
        layer = u / self_pl;
        local = u - layer * self_pl;
    } else {
        const int v = u - n_layers * self_pl;
        layer = v / nbr_pl;
        local = self_pl + (v - layer * nbr_pl);
    }
    return decode_w_unit(p, local);
}

// 16-byte piece m of patch row r in an epilogue buffer, in the layout of the
// TMA box that fills / drains it: 128-byte rows with the 128-byte swizzle
// (piece m ^ (r & 7)), or 64-byte rows with the 64-byte swizzle
// (piece m ^ ((r >> 1) & 3)).  Either way the lanes of a warp, one row
// each, touch distinct banks.
template <int ROW_BYTES>
__device__ __forceinline__ uint4* patch_piece(uint8_t* buf, int r, int m) {
    if (ROW_BYTES == 128) return reinterpret_cast<uint4*>(buf + r * 128 + ((m ^ (r & 7)) << 4));
    return reinterpret_cast<uint4*>(buf + r * 64 + ((m ^ ((r >> 1) & 3)) << 4));
}

__device__ __forceinline__ int ld_acquire_gpu(const int* p) {
    int v;
    asm volatile("ld.acquire.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

__device__ __forceinline__ int ld_acquire_cta_shared(const int* p) {
    int v;
    asm volatile("ld.acquire.cta.shared::cta.b32 %0, [%1];" : "=r"(v) : "r"(smem_u32(p)) : "memory");
    return v;
}

__device__ __forceinline__ void st_release_cta_shared(int* p, int v) {
    asm volatile("st.release.cta.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(p)), "r"(v) : "memory");
}

// Bounded wait until *ctr >= target (a counter other CTAs raise), with
// acquire semantics; records a timeout like mbar_wait.
__device__ __forceinline__ bool wait_counter(const int* ctr, int target, volatile int* abort,
                                             uint64_t timeout_ns) {
    if (ld_acquire_gpu(ctr) >= target) return true;
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t it = 1;; ++it) {
        __nanosleep(64);
        if (ld_acquire_gpu(ctr) >= target) return true;
        if ((it & 15u) == 0) {
            if (*abort) return false;
            if (globaltimer_ns() - t0 > timeout_ns) {
                atomicExch(&g_error_word, kErrTimeout);
                *abort = 1;
                return false;
            }
        }
    }
}

__device__ __forceinline__ int ld_relaxed_gpu(const int* p) {
    int v;
    asm volatile("ld.relaxed.gpu.global.b32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
    return v;
}

// Adds v to *p with release semantics: every write this thread made visible
// before it (here: TMA stores that have completed, after a proxy fence) is
// seen by whoever acquires the new value.
__device__ __forceinline__ void red_release_gpu_add(int* p, int v) {
    asm volatile("red.release.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

__device__ __forceinline__ void fence_acq_rel_gpu() {
    asm volatile("fence.acq_rel.gpu;" ::: "memory");
}

__device__ __forceinline__ void red_relaxed_gpu_add(int* p, int v) {
    asm volatile("red.relaxed.gpu.global.add.s32 [%0], %1;" ::"l"(p), "r"(v) : "memory");
}

// Two fp32 values in one 64-bit register pair, and the packed fp32 arithmetic
// of the FP32 pipe (each instruction rounds both lanes like its scalar form).
__device__ __forceinline__ uint64_t f32x2_pack(float a, float b) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(a), "f"(b));
    return r;
}
__device__ __forceinline__ float2 f32x2_unpack(uint64_t r) {
    float a, b;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(r));
    return make_float2(a, b);
}
__device__ __forceinline__ uint64_t f32x2_add(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("add.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ uint64_t f32x2_mul(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}
__device__ __forceinline__ uint64_t f32x2_fma(uint64_t a, uint64_t b, uint64_t c) {
    uint64_t r;
    asm("fma.rn.f32x2 %0, %1, %2, %3;" : "=l"(r) : "l"(a), "l"(b), "l"(c));
    return r;
}
__device__ __forceinline__ float mul_sat_f32(float a, float b) {
    float r;
    asm("mul.rn.sat.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
    return r;
}
// (2^100, 2^100) as a packed pair
constexpr uint64_t kF32x2Pow100 = 0x7180000071800000ull;
// bf16 pair -> fp32 pair (exact: the bf16 bits are the high half of each float)
__device__ __forceinline__ uint64_t bf16x2_to_f32x2(uint32_t w) {
    return f32x2_pack(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
}

// 32 ReLU mask bits (bit c = column c) -> the AND-masks of 16 bf16 column
// pairs: pair q keeps its low half iff bit 2q is set, its high half iff bit
// 2q + 1 is.  t[k] = mw << (7 - k) puts bits k, k + 8, k + 16, k + 24 at the
// sign positions of its four bytes; prmt in sign-replicate mode (selector
// nibble 8 | byte) turns a selected byte into 0xFF or 0x00 by its sign bit, so
// each pair's mask is one prmt of t[2i] and t[2i + 1] (the pair's two bits sit
// in the same byte b = q / 4 of both).
struct PairMasks {
    uint32_t t[8];
    __device__ __forceinline__ explicit PairMasks(uint32_t mw) {
#pragma unroll
        for (int k = 0; k < 8; ++k) t[k] = mw << (7 - k);
    }
    __device__ __forceinline__ uint32_t operator()(int q) const {
        const int i = q & 3, b = q >> 2;
        const uint32_t sel = (uint32_t)(8 | b) | (uint32_t)(8 | b) << 4 |
                             (uint32_t)(12 | b) << 8 | (uint32_t)(12 | b) << 12;
        uint32_t r;
        asm("prmt.b32 %0, %1, %2, %3;" : "=r"(r) : "r"(t[2 * i]), "r"(t[2 * i + 1]), "r"(sel));
        return r;
    }
};

// Adds v to the shared int *p with acquire-release semantics at CTA scope and
// returns the previous value.
__device__ __forceinline__ int atom_add_acq_rel_cta_shared(int* p, int v) {
    int old;
    asm volatile("atom.acq_rel.cta.shared::cta.add.s32 %0, [%1], %2;"
                 : "=r"(old)
                 : "r"(smem_u32(p)), "r"(v)
                 : "memory");
    return old;
}

// Bounded wait until both counters reach their targets (n of them: 1 or 2),
// with acquire semantics.  The first look reads both at once (relaxed) and,
// when both are complete, acquires with one fence; otherwise each is waited
// for in turn like wait_counter.
__device__ __forceinline__ bool wait_counters2(const int* c0, int t0, const int* c1, int t1, int n,
                                               volatile int* abort, uint64_t timeout_ns) {
    const int v0 = ld_relaxed_gpu(c0);
    const int v1 = n > 1 ? ld_relaxed_gpu(c1) : t1;
    if (v0 >= t0 && v1 >= t1) {
        fence_acq_rel_gpu();
        return true;
    }
    return wait_counter(c0, t0, abort, timeout_ns) &&
           (n < 2 || wait_counter(c1, t1, abort, timeout_ns));
}

__device__ bool wait_shift_chunks(const int* ctr, int n_chunks, int tokens, int d, int tok0,
                                  int pos0, int n, int off, volatile int* abort,
                                  uint64_t timeout_ns) {
    int c[3];
    int nc = 0;
    c[nc++] = tok0 >> 7;
    const int a = max(pos0 + off, 0), b = min(pos0 + off + 127, n - 1);
    if (a <= b) {
        const int base = tok0 - pos0;   // the sample's first token
        const int ca = (base + a) >> 7, cb = (base + b) >> 7;
        if (ca != c[0]) c[nc++] = ca;
        if (cb != ca && cb != c[0]) c[nc++] = cb;
    }
    for (int i = 0; i < nc; ++i) {
        if (c[i] >= n_chunks) continue;   // rows past the end: nothing to wait for
        if (!wait_counter(ctr + c[i], min(128, tokens - (c[i] << 7)) * d, abort, timeout_ns))
            return false;
    }
    return true;
}

// Warp-wide bounded wait until every one of the n_chunks completion counters
// ctr[c] shows its 128-token chunk complete (min(128, tokens - 128 c) * d
// elements).  Each lane polls every 32nd counter; the lanes acquire what they
// observed (a fence after the relaxed loads) and meet in a warp barrier before
// any of them goes on.  Records a timeout like mbar_wait.
__device__ bool wait_chunks_warp(const int* ctr, int n_chunks, int tokens, int d,
                                 volatile int* abort, uint64_t timeout_ns) {
    const int lane = threadIdx.x & 31;
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t it = 0;; ++it) {
        bool mine = true;
        for (int c0 = 0; c0 < n_chunks; c0 += 128) {
            int v[4], need[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int c = c0 + lane + 32 * j;
                need[j] = c < n_chunks ? min(128, tokens - (c << 7)) * d : 0;
                v[j] = c < n_chunks ? ld_relaxed_gpu(ctr + c) : 0;
            }
#pragma unroll
            for (int j = 0; j < 4; ++j) mine = mine && v[j] >= need[j];
        }
        if (__all_sync(0xffffffffu, mine)) {
            fence_acq_rel_gpu();
            __syncwarp();
            return true;
        }
        __nanosleep(200);
        int give_up = 0;
        if (lane == 0 && (it & 15u) == 15u) {
            if (*abort) {
                give_up = 1;
            } else if (globaltimer_ns() - t0 > timeout_ns) {
                atomicExch(&g_error_word, kErrTimeout);
                *abort = 1;
                give_up = 1;
            }
        }
        if (__shfl_sync(0xffffffffu, give_up, 0)) return false;
    }
}

// Bounded wait until the shared counter *p >= target (acquire); records a
// timeout like mbar_wait.
template <bool CLUSTER = false>
__device__ __forceinline__ bool wait_shared_geq(const int* p, int target, volatile int* abort,
                                                uint64_t timeout_ns) {
    auto load = [&]() { return CLUSTER ? ld_acquire_cluster_local(p) : ld_acquire_cta_shared(p); };
    if (load() >= target) return true;
    const uint64_t t0 = globaltimer_ns();
    for (uint32_t it = 1;; ++it) {
        if (load() >= target) return true;
        if ((it & 63u) == 0) {
            if (*abort) return false;
            if (globaltimer_ns() - t0 > timeout_ns) {
                atomicExch(&g_error_word, kErrTimeout);
                *abort = 1;
                return false;
            }
        }
    }
}

}  // namespace

// Maps of layer l (L.maps[l][i]):
//   0 tmA : FWD x, DX dz: 4-D rows map, box (64, lo_box, 1, hi_box) = 128 rows.
//           DW dz: 5-D (64, lo, bit, HI, d/64), box of 64 rows x 2 blocks (M = 128).
//   1 tmB0: FWD W_self [o][k] 2-D, box (64 k, BN o)   (K-major B)
//           DX  W_self [o][k] 3-D (64, o, d/64), box (64, 64, BN/64): the
//               MN-major B, BN/64 blocks of 64 columns in one copy
//           DW  x rows 5-D (64, lo, bit, HI, d/64), box (64, 64 rows, BN/64)
//   2 tmB1: FWD/DX W_nbr like tmB0; DW unused.
//   3 tmE0: FWD x / DX dy rows (residual patches, loaded); DW dW partials [2*S*d][d] fp32
//   4 tmE1: FWD y / DX dx rows (patches stored);           DW dW_self [d][d] fp32
//   5 tmE2: DX dz rows of the layer below (stored);        DW dW_nbr  [d][d] fp32
// Patch maps have 32-row boxes whose inner extent is one patch row.
//
// A stacked forward launch (NL > 1) covers L.n_layers consecutive layers;
// unit u belongs to layer u / units_per_layer and the units are ordered
// layer by layer and, within a layer, row block by row block.  The input
// rows of a unit of layer l > 0 are outputs of layer l - 1: before loading
// them the producer waits until the completion counters of the 128-token
// chunks they lie in show every element written (each epilogue warp adds the
// elements of a patch once its TMA stores have landed).  All earlier units
// of the launch have smaller indices and each CTA takes its units in order,
// so the lowest unfinished unit can always proceed.
template <int MODE, int BN, int NL, bool PAIR>
__global__ void __launch_bounds__(cta_threads(BN), 1)
    hcw_tc_kernel(const __grid_constant__ TcLaunch<NL> L) {
    // PAIR (stacked forward / input gradient): clusters of two CTAs, 256-row
    // tiles with tcgen05.mma.cta_group::2; each CTA loads its own 128 rows and
    // half of the weight tile, the leader issues the MMAs (see hcw_dwp_kernel)
    static_assert(!PAIR || ((MODE == MODE_FWD || MODE == MODE_DX || MODE == MODE_FDX) && NL > 1),
                  "pair modes");
    static_assert(MODE != MODE_FDX || PAIR, "the fused launch runs on pairs");
    constexpr int STAGES = PAIR ? tc_pair_stages(BN) : num_stages(BN, MODE);
    constexpr bool DWF = MODE == MODE_DWF;
    static_assert(!DWF || STAGES % 2 == 0, "pairs of stages");
    constexpr int B_BYTES = BN * kBlockK * 2;
    constexpr int B_LOAD = PAIR ? B_BYTES / 2 : B_BYTES;    // B bytes this CTA loads per stage
    constexpr int SB = kABytes + B_LOAD;
    constexpr uint32_t TMEM_COLS = 2 * BN;
    constexpr uint32_t IDESC = idesc_bf16_f32(PAIR ? 2 * kBlockM : kBlockM, BN,
                                              (MODE == MODE_DW || DWF) ? 1 : 0,
                                              MODE == MODE_FWD ? 0 : 1);
    // the fused launch's forward units: B (the weights) K-major
    constexpr uint32_t IDESC_FWD = idesc_bf16_f32(PAIR ? 2 * kBlockM : kBlockM, BN, 0, 0);
    // whether layer l of the launch is a forward layer, and (fused launch) the
    // first input-gradient layer
    auto is_fwd = [&](int l) {
        return MODE == MODE_FWD || (MODE == MODE_FDX && l < L.n_fwd);
    };
    const int first_dx = MODE == MODE_FDX ? L.n_fwd : 0;
    constexpr int EW = epi_warps(BN);
    constexpr int WCOLS = warp_cols(BN);               // columns per epilogue warp
    static_assert(EW <= kMaxEpiWarps && WCOLS % 32 == 0 && WCOLS <= 64, "epilogue split");
    constexpr bool STACKED = NL > 1;
    const TcParams& p = L.p;
    const int upl = p.n_units;                          // units per layer
    const int n_units = upl * L.n_layers;

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    uint8_t* epi_smem = smem + (size_t)STAGES * SB;               // 1024-aligned
    Barriers* bars = reinterpret_cast<Barriers*>(epi_smem + (DWF ? 0 : (size_t)EW * kEpiBufBytes));

    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        // the first layer's tensor maps; the last epilogue warp prefetches the
        // others while the first units load (a 32-layer launch's 192 maps in
        // this thread took ~3.5 us of the prologue, and one layer's at a time
        // in the producer lengthened every layer step)
        for (int i = 0; i < kTcMaps; ++i) tma_prefetch_desc(&L.maps[0][i]);
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&bars->full[s], 1);
            // DW: the MMA commit and the helper warps (which read the dz tiles for
            // the bias gradient) both release a stage
            mbar_init(&bars->empty[s], (MODE == MODE_DW || DWF) ? 1 + kDwHelpers : 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&bars->tfull[a], 1);
            mbar_init(&bars->tempty[a], PAIR ? 2 * EW : EW);
        }
        for (int e = 0; e < EW; ++e) mbar_init(&bars->epi_load[e], 1);
        mbar_init(&bars->drain, 1);
        bars->abort = 0;
        bars->dep_unit = -1;
        bars->q_pub = -1;
        bars->q_read = 0;
        for (int i = 0; i < 2 * kUnitQ; ++i) (&bars->pub_done[0][0])[i] = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        if (PAIR) {
            tmem_alloc_pair(&bars->tmem_base, TMEM_COLS);
            tmem_relinquish_pair();
        } else {
            tmem_alloc(&bars->tmem_base, TMEM_COLS);
            tmem_relinquish();
        }
    }
    tc_fence_before();
    __syncthreads();
    if (PAIR) cluster_sync_all();   // both CTAs' barriers exist before any cross-CTA access
    tc_fence_after();
    const uint32_t rank = PAIR ? cluster_ctarank() : 0;
    const uint32_t tmem_base = bars->tmem_base;
    volatile int* abort = &bars->abort;
    const uint64_t tmo = p.timeout_ns;
    // the weight-gradient launch behind the fused one may take the SMs this
    // launch's CTAs leave at its end; it waits for its operands on the
    // completion counters (every CTA of this launch is resident by then)
    if (MODE == MODE_FDX) pdl_trigger();
    // Stacked launches hand out units dynamically, in increasing order, from a
    // global counter: CTAs that draw short units take more of them, so no CTA
    // runs far behind the others and stalls the next layer's units.  The
    // producer claims a unit and publishes it in a shared slot; the MMA thread
    // and the epilogue warps read it by ordinal.  Otherwise CTA b takes units
    // b, b + grid, b + 2 grid, ...
    const bool dyn = STACKED && L.sched != nullptr;
    auto consume_unit = [&](int ord) -> int {   // -1: no more units, -2: aborted
        if (!dyn) {
            const int u = (int)blockIdx.x + ord * (int)gridDim.x;
            return u < n_units ? u : -1;
        }
        if (!wait_shared_geq<PAIR>(&bars->q_pub, ord, abort, tmo)) return -2;
        const int u = *reinterpret_cast<volatile int*>(&bars->unit_q[ord % kUnitQ]);
        __threadfence_block();
        atomicAdd(&bars->q_read, 1);
        return u;
    };

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued_mask = 0, issued_phase = 0;
            bool ok = true;
            for (int ordinal = 0; ok; ++ordinal) {
                int u;
                if (PAIR && rank == 1) {
                    // the pair's units come from the leader, through this CTA's slots
                    u = consume_unit(ordinal);
                    if (u == -2) {
                        ok = false;
                        break;
                    }
                } else if (dyn) {
                    // a pair outside the tail pairs leaves once the last layer's
                    // units are being handed out (a unit it still draws by a race
                    // it runs: any CTA may run any unit)
                    if (L.tail_pairs > 0 && ((int)blockIdx.x >> (PAIR ? 1 : 0)) >= L.tail_pairs &&
                        ld_relaxed_gpu(L.sched) >= (L.n_layers - 1) * upl)
                        u = n_units;
                    else
                        u = atomicAdd(L.sched, 1);
                    if (u >= n_units) u = -1;
                    // the slot's previous unit has been read by every consumer
                    if (ordinal >= kUnitQ &&
                        !wait_shared_geq(&bars->q_read, (ordinal - kUnitQ + 1) * (EW + 1), abort,
                                         tmo)) {
                        ok = false;
                        break;
                    }
                    if (PAIR) {
                        // ... and in the other CTA of the pair
                        const uint32_t peer_read = mapa_shared(&bars->q_read, 1);
                        const int need = (ordinal - kUnitQ + 1) * (EW + 1);
                        bool okp = true;
                        if (ordinal >= kUnitQ && ld_acquire_cluster_remote(peer_read) < need) {
                            const uint64_t t0 = globaltimer_ns();
                            while (ld_acquire_cluster_remote(peer_read) < need) {
                                if (*abort || globaltimer_ns() - t0 > tmo) {
                                    if (!*abort) atomicExch(&g_error_word, kErrTimeout);
                                    *abort = 1;
                                    okp = false;
                                    break;
                                }
                            }
                        }
                        if (!okp) {
                            ok = false;
                            break;
                        }
                        st_remote(mapa_shared(&bars->unit_q[ordinal % kUnitQ], 1), u);
                        st_release_cluster_remote(mapa_shared(&bars->q_pub, 1), ordinal);
                    }
                    bars->unit_q[ordinal % kUnitQ] = u;
                    st_release_cta_shared(&bars->q_pub, ordinal);
                } else {
                    u = (int)blockIdx.x + ordinal * (int)gridDim.x;
                    if (u >= n_units) u = -1;
                }
                if (u < 0) break;
                int l = STACKED ? u / upl : 0;
                const int ul = STACKED ? u - l * upl : u;
                WUnit w{};
                if (MODE == MODE_DW) w = decode_w_any(p, u, STACKED, L.n_layers, l);
                const TcLayer& ly = L.layer[l];
                const CUtensorMap* mA = &L.maps[l][0];
                if (DWF) {
                    // unit (layer, output-row tile ot, column tile nt): for every block of
                    // 64 compressed rows, its bit-0 rows then its bit-1 rows (a pair of
                    // stages), dz and the layer input each in one copy
                    const int ot = ul / p.n_nt, nt = ul - ot * p.n_nt;
                    const CUtensorMap* mX = &L.maps[l][1];
                    st_release_cta_shared(&bars->dep_unit, ordinal);
                    for (int pq = 0; pq < p.qb && ok; ++pq) {
                        const int q0 = pq * 64;
                        const int lo0 = q0 & (ly.k - 1), hi0 = q0 >> ly.s;
                        for (int bit = 0; bit < 2; ++bit) {
                            if (!mbar_wait(&bars->empty[stage], phase ^ 1, abort, tmo)) {
                                ok = false;
                                break;
                            }
                            uint8_t* sA = smem + (size_t)stage * SB;
                            uint8_t* sB = sA + kABytes;
                            mbar_arrive_expect_tx(&bars->full[stage], kABytes + B_BYTES);
                            issued_mask |= 1u << stage;
                            issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
                            tma_load_5d(sA, mA, &bars->full[stage], 0, lo0, bit, hi0,
                                        ot * (kBlockM / 64));
                            tma_load_5d(sB, mX, &bars->full[stage], 0, lo0, bit, hi0,
                                        nt * (BN / 64));
                            if (++stage == STAGES) {
                                stage = 0;
                                phase ^= 1;
                            }
                        }
                    }
                } else if (MODE != MODE_DW) {
                    const bool ufwd = is_fwd(l);
                    // a shift layer (stacked launches): map 0 views the input as
                    // (features, position, sample, 1); the unit's 128 tokens are
                    // positions pos0 .. pos0 + 127 of sample smp, their partners
                    // pos0 + soff .. (zeros outside the sample)
                    const bool shl = STACKED && ly.shift > 0;
                    RowUnit r = decode_row_unit(p, ul, STACKED, !ufwd && MODE == MODE_FDX, shl);
                    if (PAIR) r.t = 2 * r.t + (int)rank;   // this CTA's half of the 256 rows
                    const int q0 = r.t * kBlockM;
                    const int lo0 = q0 & (ly.k - 1), hi0 = q0 >> ly.s;
                    const int tok0 = (hi0 << (ly.s + 1)) + (r.beta << ly.s) + lo0;
                    const int smp = shl ? tok0 / p.seq_n : 0;
                    const int pos0 = shl ? tok0 - smp * p.seq_n : 0;
                    const int soff = ufwd ? -ly.shift : ly.shift;
                    if (STACKED && (l > 0 || (MODE == MODE_DX && L.top_dy != nullptr))) {
                        // the unit's rows and their partners: two 128-token chunks,
                        // written by the layer before (or by this launch's prologue)
                        const int* ctr = l > 0 ? L.counters + (size_t)(l - 1) * L.n_chunks
                                               : L.in_counters;
                        if (shl) {
                            ok = wait_shift_chunks(ctr, L.n_chunks, L.tokens, p.d, tok0, pos0,
                                                   p.seq_n, soff, abort, tmo);
                        } else {
                            int cs[2];
                            row_unit_chunks(q0, ly.s, ly.k, cs[0], cs[1]);
                            // chunks past the end (ragged tail) have nothing to wait for
                            const int nc = (cs[0] < L.n_chunks) + (cs[1] < L.n_chunks);
                            if (cs[0] >= L.n_chunks) cs[0] = cs[1];
                            if (nc > 0)
                                ok = wait_counters2(ctr + cs[0],
                                                    min(128, L.tokens - (cs[0] << 7)) * p.d,
                                                    ctr + cs[1],
                                                    min(128, L.tokens - (cs[1] << 7)) * p.d, nc,
                                                    abort, tmo);
                        }
                        if (!ok) break;
                        fence_proxy_async_global();
                    }
                    st_release_cta_shared(&bars->dep_unit, ordinal);
                    for (int ks = 0; ks < r.steps; ++ks) {
                        if (!mbar_wait(&bars->empty[stage], phase ^ 1, abort, tmo)) {
                            ok = false;
                            break;
                        }
                        uint8_t* sA = smem + (size_t)stage * SB;
                        uint8_t* sB = sA + kABytes;
                        issued_mask |= 1u << stage;
                        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
                        const int part = ks >= p.nK;
                        const int kk = part ? ks - p.nK : ks;
                        // partner part: the rows of the other bit value, or (pair_rows)
                        // the same rows of the row-aligned partner tensor (map 5)
                        const bool same = part && ly.pair_rows;
                        const CUtensorMap* mAk = same ? &L.maps[l][5] : mA;
                        const CUtensorMap* mb = &L.maps[l][part ? 2 : 1];
                        // A box coordinates after the feature block: (lo, bit, HI) of
                        // the hypercube view, or (position, sample, 0) of a shift layer
                        int c1 = lo0, c2 = part && !same ? 1 - r.beta : r.beta, c3 = hi0;
                        if (shl) {
                            c1 = part ? pos0 + soff : pos0;
                            c2 = smp;
                            c3 = 0;
                        }
                        if (PAIR) {
                            // both CTAs' copies complete on the leader's barrier
                            if (rank == 0) mbar_arrive_expect_tx(&bars->full[stage], 2 * SB);
                            const uint32_t fb = mapa_shared(&bars->full[stage], 0);
                            tma_load_4d_pair(sA, mAk, fb, kk * kBlockK, c1, c2, c3);
                            if (ufwd)
                                tma_load_2d_pair(sB, mb, fb, kk * kBlockK,
                                                 r.j * BN + (int)rank * (BN / 2));
                            else
                                tma_load_3d_pair(sB, mb, fb, 0, kk * kBlockK,
                                                 r.j * (BN / 64) + (int)rank * (BN / 128));
                        } else {
                            mbar_arrive_expect_tx(&bars->full[stage], kABytes + B_BYTES);
                            tma_load_4d(sA, mAk, &bars->full[stage], kk * kBlockK, c1, c2, c3);
                            if (ufwd)
                                tma_load_2d(sB, mb, &bars->full[stage], kk * kBlockK, r.j * BN);
                            else   // BN / 64 blocks of 64 W columns x 64 rows, one copy
                                tma_load_3d(sB, mb, &bars->full[stage], 0, kk * kBlockK,
                                            r.j * (BN / 64));
                        }
                        if (++stage == STAGES) {
                            stage = 0;
                            phase ^= 1;
                        }
                    }
                } else {
                    st_release_cta_shared(&bars->dep_unit, ordinal);
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
                        const int lo0 = q0 & (ly.k - 1), hi0 = q0 >> ly.s;
                        uint8_t* sA = smem + (size_t)stage * SB;
                        uint8_t* sB = sA + kABytes;
                        mbar_arrive_expect_tx(&bars->full[stage], kABytes + B_BYTES);
                        issued_mask |= 1u << stage;
                        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
                        // 64 positions x (2 | BN / 64) blocks of 64 features, one copy each
                        tma_load_5d(sA, mA, &bars->full[stage], 0, lo0, bA, hi0,
                                    w.ot * (kBlockM / 64));
                        tma_load_5d(sB, &L.maps[l][1], &bars->full[stage], 0, lo0, bB, hi0,
                                    w.nt * (BN / 64));
                        if (++stage == STAGES) {
                            stage = 0;
                            phase ^= 1;
                        }
                    }
                }
            }
            if (!ok && (!PAIR || rank == 0)) {
                // let every copy this thread started land before the CTA exits (a
                // pair's copies all complete on the leader's barriers)
                for (int s = 0; s < STAGES; ++s)
                    if (issued_mask & (1u << s))
                        mbar_wait_drain(&bars->full[s], (issued_phase >> s) & 1u, tmo);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        // (a pair's MMAs are issued by its leader alone)
        if (lane == 0 && (!PAIR || rank == 0)) {
            int stage = 0;
            uint32_t phase = 0;
            int acc = 0;
            uint32_t acc_phase = 0;
            bool ok = true, any = false;
            for (int ord = 0; ok; ++ord) {
                const int u = consume_unit(ord);
                if (u == -2) {
                    ok = false;
                    break;
                }
                if (u < 0) break;
                const int ul = STACKED ? u % upl : u;
                if (DWF) {
                    // self-part accumulator at TMEM column 0, partner part at BN
                    if (!mbar_wait(&bars->tempty[0], acc_phase ^ 1, abort, tmo)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t d_self = tmem_base, d_nbr = tmem_base + BN;
                    for (int pq = 0; pq < p.qb && ok; ++pq) {
                        // stage (bit-0 rows) and stage + 1 (bit-1 rows): STAGES is even
                        if (!mbar_wait(&bars->full[stage], phase, abort, tmo) ||
                            !mbar_wait(&bars->full[stage + 1], phase, abort, tmo)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t a0 = smem_u32(smem + (size_t)stage * SB), x0 = a0 + kABytes;
                        const uint32_t a1 = a0 + SB, x1 = a1 + kABytes;
                        auto dsc = [](uint32_t base, int kk) {
                            return smem_desc_sw128(base + kk * 2048, 8192, 1024);
                        };
#pragma unroll
                        for (int kk = 0; kk < kBlockK / 16; ++kk)
                            mma_bf16_f32(d_self, dsc(a0, kk), dsc(x0, kk), IDESC, (pq | kk) != 0);
#pragma unroll
                        for (int kk = 0; kk < kBlockK / 16; ++kk)
                            mma_bf16_f32(d_self, dsc(a1, kk), dsc(x1, kk), IDESC, 1);
                        // bit-1 rows receive from their bit-0 partners (causal); both
                        // directions without the causal rule
#pragma unroll
                        for (int kk = 0; kk < kBlockK / 16; ++kk)
                            mma_bf16_f32(d_nbr, dsc(a1, kk), dsc(x0, kk), IDESC, (pq | kk) != 0);
                        if (!p.causal) {
#pragma unroll
                            for (int kk = 0; kk < kBlockK / 16; ++kk)
                                mma_bf16_f32(d_nbr, dsc(a0, kk), dsc(x1, kk), IDESC, 1);
                        }
                        any = true;
                        mma_commit(&bars->empty[stage]);
                        mma_commit(&bars->empty[stage + 1]);
                        stage += 2;
                        if (stage == STAGES) {
                            stage = 0;
                            phase ^= 1;
                        }
                    }
                    if (!ok) break;
                    mma_commit(&bars->tfull[0]);
                    acc_phase ^= 1;
                    continue;
                }
                int steps;
                // the B operand: K-major (forward: W rows) or MN-major (input
                // gradient: W columns); a fused launch picks it per unit
                uint32_t idesc = IDESC, b_step = MODE == MODE_FWD ? 32 : 2048,
                         b_lbo = MODE == MODE_FWD ? 16 : 8192;
                if (MODE == MODE_FDX && is_fwd(u / upl)) {
                    idesc = IDESC_FWD;
                    b_step = 32;
                    b_lbo = 16;
                }
                if (MODE != MODE_DW) {
                    steps = decode_row_unit(p, ul, STACKED, false,
                                            STACKED && L.layer[u / upl].shift > 0)
                                .steps;
                } else {
                    int lw;
                    const WUnit w = decode_w_any(p, u, STACKED, L.n_layers, lw);
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
                        if (MODE == MODE_DW)
                            bdesc = smem_desc_sw128(b_addr + kk * 2048, 8192, 1024);
                        else
                            bdesc = smem_desc_sw128(b_addr + kk * b_step, b_lbo, 1024);
                        if (PAIR)
                            mma_bf16_f32_pair(d_tmem, adesc, bdesc, idesc, (ks | kk) != 0);
                        else
                            mma_bf16_f32(d_tmem, adesc, bdesc, idesc, (ks | kk) != 0);
                    }
                    any = true;
                    if (PAIR)
                        mma_commit_pair(&bars->empty[stage], 3);   // both CTAs' stage
                    else
                        mma_commit(&bars->empty[stage]);
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
                if (!ok) break;
                if (PAIR)
                    mma_commit_pair(&bars->tfull[acc], 3);
                else
                    mma_commit(&bars->tfull[acc]);
                acc ^= 1;
                if (acc == 0) acc_phase ^= 1;
            }
            if (!ok && any) {
                // wait for the MMAs already issued before TMEM is released
                if (PAIR)
                    mma_commit_pair(&bars->drain, 1);
                else
                    mma_commit(&bars->drain);
                mbar_wait_drain(&bars->drain, 0, tmo);
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue
        // Warp e drains TMEM lane quarter warp % 4 (rows 32 q .. 32 q + 31 of the
        // tile) and column slice e / 4 (WCOLS columns): one patch per tile.
        const int e = warp - 2;
        const int quarter = warp & 3;
        const int cslice = e >> 2;
        uint8_t* buf = epi_smem + (size_t)e * kEpiBufBytes;
        if (STACKED && e == EW - 1)
            for (int i = kTcMaps + lane; i < L.n_layers * kTcMaps; i += 32)
                tma_prefetch_desc(&L.maps[i / kTcMaps][i % kTcMaps]);
        uint32_t ld_phase = 0;
        int hstage = 0;          // DW helper warps: ring position, as the MMA thread's
        uint32_t hphase = 0;
        int acc = 0;
        uint32_t acc_phase = 0;
        bool alive = true;
        int ordinal = 0;
        // every lane observes the barrier; the warp proceeds only if all did
        // (tcgen05.ld and the patch accesses are warp-wide)
        auto wait_bar = [&](uint64_t* bar, uint32_t parity) -> bool {
            const bool ok = mbar_wait(bar, parity, abort, tmo);
            return __all_sync(0xffffffffu, ok) != 0;
        };
        auto wait_acc = [&]() -> bool {
            const bool ok = wait_bar(&bars->tfull[acc], acc_phase);
            if (ok) tc_fence_after();
            return ok;
        };
        auto load_acc = [&](uint32_t col, uint32_t (&raw)[32]) {
            __syncwarp();   // tcgen05.ld is .sync.aligned: the whole warp, converged
            tmem_ld_32x32b_x32(tmem_base + ((uint32_t)(quarter * 32) << 16) +
                                   (uint32_t)(acc * BN + cslice * WCOLS) + col,
                               raw);
            tmem_ld_wait_regs(raw);
        };
        auto release_acc = [&]() {
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                if (PAIR)
                    mbar_arrive_remote_tmem(mapa_shared(&bars->tempty[acc], 0));   // the leader's
                else
                    mbar_arrive(&bars->tempty[acc]);
            }
        };
        // make this warp's shared-memory writes visible to TMA, then store
        auto publish = [&]() {
            fence_proxy_async_smem();
            __syncwarp();
        };
        // the producer has checked this unit's inputs (lane 0 waits, bounded)
        auto wait_inputs = [&](int ord) -> bool {
            int ok = 1;
            if (lane == 0) {
                const uint64_t t0 = globaltimer_ns();
                while (ld_acquire_cta_shared(&bars->dep_unit) < ord) {
                    if (*abort || globaltimer_ns() - t0 > tmo) {
                        ok = 0;
                        break;
                    }
                }
                if (ok) fence_proxy_async_global();
            }
            return __shfl_sync(0xffffffffu, ok, 0) != 0;
        };
        // Helper warps (e < kDwHelpers) of the weight-gradient modes follow the
        // MMA thread through a unit's `steps` stages and release each one; with
        // do_cs (a unit that covers every token of its output-row tile) they
        // also add up the dz tile's columns on the way: dbias of rows o_base ..
        // o_base + 127.  Thread t sums the 16-byte piece c of box t / 64 (64 dz
        // rows each) over the tile rows r = t % 8 (mod 8), then the eight row
        // phases are added with shuffles: a fixed order.
        auto helper_pass = [&](int steps, bool do_cs, float* colsum, int o_base) -> bool {
            const int t = e * 32 + lane;
            const int box = t >> 6, c = (t >> 3) & 7, tp = t & 7;
            float cs[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) cs[i] = 0.f;
            for (int ks = 0; ks < steps; ++ks) {
                if (!wait_bar(&bars->full[hstage], hphase)) return false;
                if (do_cs) {
                    const uint8_t* sA = smem + (size_t)hstage * SB + box * 8192;
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const int r = tp + 8 * i;
                        const uint4 q = *reinterpret_cast<const uint4*>(sA + r * 128 + ((c ^ tp) << 4));
                        const uint32_t wv[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
                        for (int j = 0; j < 4; ++j) {
                            const float2 f = unpack_bf16x2(wv[j]);
                            cs[2 * j] += f.x;
                            cs[2 * j + 1] += f.y;
                        }
                    }
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(&bars->empty[hstage]);
                if (++hstage == STAGES) {
                    hstage = 0;
                    hphase ^= 1;
                }
            }
            if (do_cs) {
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    cs[i] += __shfl_xor_sync(0xffffffffu, cs[i], 1);
                    cs[i] += __shfl_xor_sync(0xffffffffu, cs[i], 2);
                    cs[i] += __shfl_xor_sync(0xffffffffu, cs[i], 4);
                }
                const int o0 = o_base + box * 64 + c * 8;
                if (tp == 0 && o0 < p.d) {
                    float4* dst = reinterpret_cast<float4*>(colsum + o0);
                    dst[0] = make_float4(cs[0], cs[1], cs[2], cs[3]);
                    dst[1] = make_float4(cs[4], cs[5], cs[6], cs[7]);
                }
            }
            return true;
        };
        if (MODE == MODE_DX && STACKED && L.top_dy != nullptr) {
            // The top layer's dz = dy * mask (or dy) for this CTA's 128-token
            // chunks (b, b + grid, ...).  The chunk's 16-byte pieces are spread
            // over the epilogue warps, eight loads in flight per lane; each warp
            // then counts the elements it wrote in the chunk's counter (a release
            // after a proxy fence: the readers are TMA copies).
            const int gpr = p.d / 8;                        // 16-byte pieces per row
            constexpr int kU = 8;
            for (int c = (int)blockIdx.x; c < L.n_chunks; c += (int)gridDim.x) {
                const int rows = min(128, L.tokens - (c << 7));
                const int n = rows * gpr;                   // pieces in the chunk
                const size_t base = ((size_t)c << 7) * (size_t)gpr;
                const uint4* src = reinterpret_cast<const uint4*>(L.top_dy) + base;
                uint4* dst = reinterpret_cast<uint4*>(L.top_dz) + base;
                const uint32_t* mrow = L.top_mask ? L.top_mask + ((size_t)c << 7) * (p.d >> 5)
                                                  : nullptr;
                int mine = 0;
                for (int i0 = e * 32 + lane; i0 < n; i0 += kU * EW * 32) {
                    uint4 v[kU];
                    uint32_t mw[kU];
#pragma unroll
                    for (int j = 0; j < kU; ++j) {
                        const int i = i0 + j * EW * 32;
                        if (i < n) {
                            v[j] = src[i];
                            // piece i covers columns 8 (i % gpr) .. + 7 of row i / gpr
                            mw[j] = mrow ? mrow[(i / gpr) * (p.d >> 5) + ((i % gpr) >> 2)] : ~0u;
                        }
                    }
#pragma unroll
                    for (int j = 0; j < kU; ++j) {
                        const int i = i0 + j * EW * 32;
                        if (i < n) {
                            const uint32_t bits = (mw[j] >> (((i % gpr) & 3) * 8)) & 0xFFu;
                            uint32_t w[4] = {v[j].x, v[j].y, v[j].z, v[j].w};
#pragma unroll
                            for (int q = 0; q < 4; ++q)
                                w[q] &= ((bits >> (2 * q)) & 1u ? 0x0000FFFFu : 0u) |
                                        ((bits >> (2 * q + 1)) & 1u ? 0xFFFF0000u : 0u);
                            dst[i] = make_uint4(w[0], w[1], w[2], w[3]);
                            mine += 8;
                        }
                    }
                }
                mine = __reduce_add_sync(0xffffffffu, mine);
                if (lane == 0 && mine > 0) {
                    __threadfence();
                    fence_proxy_async_global();
                    red_release_gpu_add(L.in_counters + c, mine);
                }
            }
        }
        for (; alive; ++ordinal) {
            int u = 0;
            if (lane == 0) u = consume_unit(ordinal);
            u = __shfl_sync(0xffffffffu, u, 0);
            if (u == -2) {
                alive = false;
                break;
            }
            if (u < 0) break;
            int l = STACKED ? u / upl : 0;
            const int ul = STACKED ? u - l * upl : u;
            WUnit wu{};
            if (MODE == MODE_DW) wu = decode_w_any(p, u, STACKED, L.n_layers, l);
            const TcLayer& ly = L.layer[l];
            if (DWF) {
                const int ot = ul / p.n_nt, nt = ul - ot * p.n_nt;
                if (e < kDwHelpers &&
                    !helper_pass(2 * p.qb, ly.colsum != nullptr && nt == 0, ly.colsum,
                                 ot * kBlockM)) {
                    alive = false;
                    break;
                }
                if (!wait_acc()) {
                    alive = false;
                    break;
                }
                // every lane holds one row of the tile: 32 fp32 columns per TMEM load,
                // stored straight to global memory (no buffers in this mode); the
                // self part, then the partner part
                const int row = ot * kBlockM + quarter * 32 + lane;
#pragma unroll 1
                for (int which = 0; which < 2; ++which) {
                    float* base = which ? ly.dwn : ly.dws;
#pragma unroll 1
                    for (int c = 0; c < WCOLS / 32; ++c) {
                        uint32_t raw[32];
                        load_acc(which * BN + c * 32, raw);
                        if (which == 1 && c == WCOLS / 32 - 1) release_acc();
                        if (row < p.d) {
                            float4* dst = reinterpret_cast<float4*>(
                                base + (size_t)row * p.d + nt * BN + cslice * WCOLS + c * 32);
#pragma unroll
                            for (int m = 0; m < 8; ++m)
                                dst[m] = make_float4(__uint_as_float(raw[4 * m]),
                                                     __uint_as_float(raw[4 * m + 1]),
                                                     __uint_as_float(raw[4 * m + 2]),
                                                     __uint_as_float(raw[4 * m + 3]));
                        }
                    }
                }
            } else if (MODE != MODE_DW) {
                // One body per direction, each compiled with the direction fixed (a
                // fused launch picks one per unit): the epilogue sits on the layer
                // chain, and a run-time direction costs registers and instructions.
                auto row_epilogue = [&](auto fwd_tag) -> bool {
                constexpr bool fwd = decltype(fwd_tag)::value;
                constexpr int RB = WCOLS * 2;                  // patch row bytes (128 or 64)
                constexpr int SUB = WCOLS / 32;                // 32-column sub-chunks per patch
                RowUnit r = decode_row_unit(p, ul, STACKED, !fwd && MODE == MODE_FDX,
                                            STACKED && ly.shift > 0);
                if (PAIR) r.t = 2 * r.t + (int)rank;
                const int qw = r.t * kBlockM + quarter * 32;   // first compressed row of the warp
                const int lo_w = qw & (ly.k - 1), hi_w = qw >> ly.s;
                const int q_row = qw + lane;
                const int tok_row = q_row < p.Mh ? ((q_row >> ly.s) << (ly.s + 1)) +
                                                       (r.beta << ly.s) + (q_row & (ly.k - 1))
                                                 : -1;
                const int col0 = r.j * BN + cslice * WCOLS;
                // a patch entirely past the end (ragged tail) loads and stores nothing
                const bool inside = qw < p.Mh;
                const bool has_res = (p.flags & 2u) != 0 && inside;
                const bool has_mprev = !fwd && ly.mprev != nullptr && ly.dz_out;
                // fused launch: the last forward layer also writes the top layer's
                // dz = dy * act'(z), the first input-gradient layer's operand
                const bool top_dz = MODE == MODE_FDX && l == L.n_fwd - 1 && L.top_dy != nullptr;
                const CUtensorMap* mE0 = &L.maps[l][3];
                const CUtensorMap* mE1 = &L.maps[l][4];
                const CUtensorMap* mE2 = &L.maps[l][5];
                const int wpr = p.d >> 5;
                // the 128-token chunk that holds the patch's rows (32 compressed rows
                // lie in one chunk for every link distance)
                const int tok0 = ((qw >> ly.s) << (ly.s + 1)) + (r.beta << ly.s) + (qw & (ly.k - 1));
                const int chunk = tok0 >> 7;
                // every earlier store has finished reading the buffer: refill it
                if (lane == 0) bulk_wait_read<0>();
                __syncwarp();
                if (!wait_inputs(ordinal)) {
                    return false;
                }
                if (has_res) {
                    int okg = 1;
                    if (lane == 0) {
                        // stacked input gradient: the residual term g of these rows is
                        // stored by the layer above after its dz; wait until the chunk's g
                        // is complete (the dz the MMAs read was checked by the producer)
                        if (!fwd && STACKED && L.g_counters != nullptr && l > first_dx) {
                            okg = wait_counter(L.g_counters + (size_t)(l - 1) * L.n_chunks + chunk,
                                               min(128, L.tokens - (chunk << 7)) * p.d, abort, tmo);
                            if (okg) fence_proxy_async_global();
                        }
                        if (okg) {
                            mbar_arrive_expect_tx(&bars->epi_load[e], 32 * RB);
                            tma_load_4d(buf, mE0, &bars->epi_load[e], col0, lo_w, r.beta, hi_w);
                        }
                    }
                    if (__shfl_sync(0xffffffffu, okg, 0) == 0) {
                        return false;
                    }
                }
                uint32_t mp[SUB];
#pragma unroll
                for (int h = 0; h < SUB; ++h)
                    mp[h] = (has_mprev && tok_row >= 0)
                                ? __ldg(ly.mprev + (size_t)tok_row * wpr + (col0 >> 5) + h)
                                : 0u;
                // this warp's bias slice in registers, column h * 32 + lane in
                // bias_reg[h], handed to the lanes by shuffles (no shared memory:
                // the ring of the pair launches takes a fifth stage instead)
                float bias_reg[SUB];
#pragma unroll
                for (int h = 0; h < SUB; ++h)
                    bias_reg[h] = fwd && ly.bias ? __ldg(ly.bias + col0 + h * 32 + lane) : 0.f;
                if (!wait_acc()) {
                    return false;
                }
                // FWD z (layer API only): the pre-activation, row-wise stores; every
                // lane joins the warp-wide TMEM loads, rows past the end skip the store
                if (fwd && ly.zout) {
#pragma unroll 1
                    for (int h = 0; h < SUB; ++h) {
                        uint32_t raw[32];
                        load_acc(h * 32, raw);
#pragma unroll
                        for (int m = 0; m < 4; ++m) {
                            uint32_t w[4];
#pragma unroll
                            for (int i = 0; i < 4; ++i) {
                                const int e2 = 8 * m + 2 * i;
                                w[i] = pack_bf16x2(
                                    __uint_as_float(raw[e2]) +
                                        __shfl_sync(0xffffffffu, bias_reg[h], e2),
                                    __uint_as_float(raw[e2 + 1]) +
                                        __shfl_sync(0xffffffffu, bias_reg[h], e2 + 1));
                            }
                            if (tok_row >= 0)
                                reinterpret_cast<uint4*>(ly.zout + (size_t)tok_row * p.d + col0 +
                                                         h * 32)[m] = make_uint4(w[0], w[1], w[2], w[3]);
                        }
                    }
                }
                if (has_res) {
                    const bool okl = wait_bar(&bars->epi_load[e], ld_phase);
                    ld_phase ^= 1;
                    if (!okl) {
                        return false;
                    }
                    // a g row read for the last time: drop its line from L2 without
                    // writing it back (one 128-byte line per row of the patch)
                    if (!fwd && ly.g_discard != nullptr && tok_row >= 0 && RB == 128)
                        asm volatile("discard.global.L2 [%0], 128;" ::"l"(
                                         ly.g_discard + (size_t)tok_row * p.d + col0)
                                     : "memory");
                }
                const bool write_out = fwd || ly.out;
                uint32_t gw[SUB][16];
                uint32_t mbits[SUB];
#pragma unroll
                for (int h = 0; h < SUB; ++h) {
                    uint32_t raw[32];
                    load_acc(h * 32, raw);
                    if (h == SUB - 1) release_acc();
                    // The arithmetic runs on the FP32 pipe, two columns per instruction
                    // where it can (f32x2): the epilogue of a chained unit sits on the
                    // layer chain, and half-rate integer work (compares, selects, bit
                    // ors) made it issue-bound.  Eight columns at a time: column pairs
                    // q = 4m .. 4m + 3.
                    const bool relu = fwd && (p.flags & 4u);
                    uint64_t lo = f32x2_pack(0x1p23f, 0.f), hi = lo;   // mask-word halves
#pragma unroll
                    for (int m = 0; m < 4; ++m) {
                        uint32_t rw[4] = {0u, 0u, 0u, 0u};   // residual (bf16 pairs), or +0
                        if (has_res) {
                            const uint4 q4 = *patch_piece<RB>(buf, lane, 4 * h + m);
                            rw[0] = q4.x;
                            rw[1] = q4.y;
                            rw[2] = q4.z;
                            rw[3] = q4.w;
                        }
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            const int q = 4 * m + i;
                            uint64_t v2 = f32x2_pack(__uint_as_float(raw[2 * q]),
                                                     __uint_as_float(raw[2 * q + 1]));
                            if (fwd)
                                v2 = f32x2_add(
                                    v2, f32x2_pack(__shfl_sync(0xffffffffu, bias_reg[h], 2 * q),
                                                   __shfl_sync(0xffffffffu, bias_reg[h], 2 * q + 1)));
                            const uint64_t r2 = bf16x2_to_f32x2(rw[i]);
                            if (relu) {
                                // b = [z > 0] exactly as 1.0 / 0.0: z * 2^100 * 2^100 saturated
                                // to [0, 1] (every positive float, denormals included,
                                // reaches at least 2^51 before the clamp; zero, negative and
                                // NaN go to 0).  y = fma(z, b, x) is relu(z) + x with one
                                // rounding; with x = +0 a negative z gives (-0) + (+0) = +0.
                                const float2 t = f32x2_unpack(f32x2_mul(v2, kF32x2Pow100));
                                const uint64_t b2 =
                                    f32x2_pack(mul_sat_f32(t.x, 0x1p100f), mul_sat_f32(t.y, 0x1p100f));
                                // the mask word: sum of b_c 2^c, exact in fp32, as two 16-bit
                                // halves offset by 2^23 (the integer is the low mantissa)
                                const uint64_t w2 = f32x2_pack((float)(1u << ((2 * q) & 15)),
                                                               (float)(1u << ((2 * q + 1) & 15)));
                                if (q < 8)
                                    lo = f32x2_fma(b2, w2, lo);
                                else
                                    hi = f32x2_fma(b2, w2, hi);
                                v2 = f32x2_fma(v2, b2, r2);
                            } else if (has_res) {
                                v2 = f32x2_add(v2, r2);
                            }
                            const float2 t = f32x2_unpack(v2);
                            gw[h][q] = pack_bf16x2(t.x, t.y);
                        }
                    }
                    if (relu) {
                        const float2 l2 = f32x2_unpack(lo), h2 = f32x2_unpack(hi);
                        mbits[h] = __byte_perm(__float_as_uint(l2.x + l2.y),
                                               __float_as_uint(h2.x + h2.y), 0x5410);
                    } else {
                        mbits[h] = 0u;
                    }
                    // the lane's own row, the pieces just read: safe to overwrite now.
                    // With the ReLU gradient of the layer below, dz = dx * mask goes
                    // first; otherwise y (FWD) or dx (DX).
                    if (has_mprev) {
                        const PairMasks keep(mp[h]);
#pragma unroll
                        for (int m = 0; m < 4; ++m) {
                            uint32_t w4[4];
#pragma unroll
                            for (int i = 0; i < 4; ++i) w4[i] = gw[h][4 * m + i] & keep(4 * m + i);
                            *patch_piece<RB>(buf, lane, 4 * h + m) =
                                make_uint4(w4[0], w4[1], w4[2], w4[3]);
                        }
                    } else if (write_out) {
#pragma unroll
                        for (int m = 0; m < 4; ++m)
                            *patch_piece<RB>(buf, lane, 4 * h + m) =
                                make_uint4(gw[h][4 * m], gw[h][4 * m + 1], gw[h][4 * m + 2],
                                           gw[h][4 * m + 3]);
                    }
                }
                // Publish the CTA's rows of the unit to the next layer's units once
                // every patch's stores have landed.  Each warp waits for its own
                // stores and counts itself in a shared counter (release at CTA
                // scope); the last of the unit's warps issues one release at GPU
                // scope and adds the elements of the CTA's rows to the counters of
                // the (at most two) 128-token chunks they lie in.  One release per
                // CTA and unit instead of one per warp: each costs about a
                // microsecond on the layer chain.
                const bool signal = STACKED && l + 1 < L.n_layers;
                auto count = [&](int* ctr, int kind) {
                    if (lane == 0) {
                        if (inside) bulk_wait<0>();
                        fence_proxy_async_global();
                        int* done = &bars->pub_done[kind][ordinal % kUnitQ];
                        if (atom_add_acq_rel_cta_shared(done, 1) == EW - 1) {
                            *done = 0;   // next used by ordinal + kUnitQ, after this unit
                            const int cols = BN;
                            int c0 = -1, n0 = 0, c1 = -1, n1 = 0;
                            for (int qd = 0; qd < 4; ++qd) {
                                const int q = r.t * kBlockM + 32 * qd;
                                if (q >= p.Mh) break;
                                const int c = (((q >> ly.s) << (ly.s + 1)) + (r.beta << ly.s) +
                                               (q & (ly.k - 1))) >> 7;
                                const int n = min(32, p.Mh - q) * cols;
                                if (c0 < 0 || c == c0) {
                                    c0 = c;
                                    n0 += n;
                                } else {
                                    c1 = c;
                                    n1 += n;
                                }
                            }
                            fence_acq_rel_gpu();
                            int* base = ctr + (size_t)l * L.n_chunks;
                            if (n0) red_relaxed_gpu_add(base + c0, n0);
                            if (n1) red_relaxed_gpu_add(base + c1, n1);
                        }
                    }
                    __syncwarp();
                };
                if (has_mprev) {
                    // the dz patch (the next layer's MMA operand) first
                    publish();
                    if (lane == 0 && inside) {
                        tma_store_4d(mE2, buf, col0, lo_w, r.beta, hi_w);
                        bulk_commit();
                    }
                    const bool split_g = write_out && L.g_counters != nullptr;
                    if (signal && (!write_out || split_g)) count(L.counters, 0);
                    if (write_out) {
                        // then the output gradient g (the next layer's residual term)
                        if (lane == 0) bulk_wait_read<0>();
                        __syncwarp();
#pragma unroll
                        for (int h = 0; h < SUB; ++h)
#pragma unroll
                            for (int m = 0; m < 4; ++m)
                                *patch_piece<RB>(buf, lane, 4 * h + m) =
                                    make_uint4(gw[h][4 * m], gw[h][4 * m + 1], gw[h][4 * m + 2],
                                               gw[h][4 * m + 3]);
                        publish();
                        if (lane == 0 && inside) {
                            tma_store_4d(mE1, buf, col0, lo_w, r.beta, hi_w);
                            bulk_commit();
                        }
                        if (signal) count(split_g ? L.g_counters : L.counters, split_g ? 1 : 0);
                    }
                } else {
                    // the patch: y (FWD) or dx (DX), written over the residual rows
                    if (write_out) {
                        publish();
                        if (lane == 0 && inside) {
                            tma_store_4d(mE1, buf, col0, lo_w, r.beta, hi_w);
                            bulk_commit();
                        }
                    }
                    if (top_dz) {
                        // the top layer's dz = dy * [z > 0] (a copy of dy without the
                        // ReLU) for the same rows and columns, dy read straight from
                        // global memory, written over the buffer once the y store has
                        // read it; counted with y below
                        if (lane == 0) bulk_wait_read<0>();
                        __syncwarp();
#pragma unroll
                        for (int h = 0; h < SUB; ++h) {
                            uint4 q4[4] = {};
                            if (tok_row >= 0) {
                                const uint4* src = reinterpret_cast<const uint4*>(
                                    L.top_dy + (size_t)tok_row * p.d + col0 + h * 32);
#pragma unroll
                                for (int m = 0; m < 4; ++m) q4[m] = __ldg(src + m);
                            }
                            const PairMasks keep((p.flags & 4u) ? mbits[h] : ~0u);
#pragma unroll
                            for (int m = 0; m < 4; ++m) {
                                uint32_t w4[4] = {q4[m].x, q4[m].y, q4[m].z, q4[m].w};
#pragma unroll
                                for (int i = 0; i < 4; ++i) w4[i] &= keep(4 * m + i);
                                *patch_piece<RB>(buf, lane, 4 * h + m) =
                                    make_uint4(w4[0], w4[1], w4[2], w4[3]);
                            }
                        }
                        publish();
                        if (lane == 0 && inside) {
                            tma_store_4d(mE2, buf, col0, lo_w, r.beta, hi_w);
                            bulk_commit();
                        }
                    }
                    if (signal) count(L.counters, 0);
                }
                // FWD: the ReLU mask words, read only by the input gradient (a later
                // launch), after the signal so that they stay off the layer chain
                if (fwd && ly.mout && tok_row >= 0) {
#pragma unroll
                    for (int h = 0; h < SUB; ++h)
                        ly.mout[(size_t)tok_row * wpr + (col0 >> 5) + h] = mbits[h];
                }
                return true;
                };
                bool ok_unit;
                if (MODE == MODE_FDX)
                    ok_unit = is_fwd(l) ? row_epilogue(std::true_type{})
                                        : row_epilogue(std::false_type{});
                else
                    ok_unit = row_epilogue(std::integral_constant<bool, MODE == MODE_FWD>{});
                if (!ok_unit) {
                    alive = false;
                    break;
                }
            } else {
                const WUnit& w = wu;
                if (e < kDwHelpers &&
                    !helper_pass(w.kb1 - w.kb0,
                                 ly.colsum != nullptr && w.which == 0 && w.nt == 0,
                                 ly.colsum + (p.splits_self > 1 ? (size_t)w.split * p.d : 0),
                                 w.ot * kBlockM)) {
                    alive = false;
                    break;
                }
                if (!wait_acc()) {
                    alive = false;
                    break;
                }
                const int S = w.which ? p.splits_nbr : p.splits_self;
                const CUtensorMap* map = &L.maps[l][S > 1 ? 3 : (w.which ? 5 : 4)];
                const int row0 = (S > 1 ? (w.which * p.splits_max + w.split) * p.d : 0) +
                                 w.ot * kBlockM + quarter * 32;
                const int col0 = w.nt * BN + cslice * WCOLS;
#pragma unroll 1
                for (int c = 0; c < WCOLS / 32; ++c) {
                    uint32_t raw[32];
                    load_acc(c * 32, raw);
                    if (c == WCOLS / 32 - 1) release_acc();
                    // the buffer's previous store must have been read
                    if (lane == 0) bulk_wait_read<0>();
                    __syncwarp();
#pragma unroll
                    for (int m = 0; m < 8; ++m)
                        *patch_piece<128>(buf, lane, m) =
                            make_uint4(raw[4 * m], raw[4 * m + 1], raw[4 * m + 2], raw[4 * m + 3]);
                    publish();
                    // d is a multiple of 64, so a warp's 32 rows are all inside or all
                    // past the end (ragged o tile); the latter are not stored
                    if (lane == 0 && w.ot * kBlockM + quarter * 32 < p.d) {
                        tma_store_2d(map, buf, col0 + c * 32, row0);
                        bulk_commit();
                    }
                }
            }
            if (DWF) {
                acc_phase ^= 1;   // one accumulator pair per unit
            } else {
                acc ^= 1;
                if (acc == 0) acc_phase ^= 1;
            }
        }
        // every store of this warp has landed before the CTA exits
        if (lane == 0) bulk_wait<0>();
        __syncwarp();
    }

    tc_fence_before();
    __syncthreads();
    if (PAIR) cluster_sync_all();   // neither CTA frees the pair's TMEM while the other uses it
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        if (PAIR)
            tmem_dealloc_pair(tmem_base, TMEM_COLS);
        else
            tmem_dealloc(tmem_base, TMEM_COLS);
    }
}

// ---------------------------------------------------------------- CTA pairs
// Weight gradients of a run of layers on pairs of SMs (MODE_DWP): a cluster of
// two CTAs computes a 256 x BN tile of dW_self and of dW_nbr with
// tcgen05.mma.cta_group::2.  CTA r of the pair holds the dz rows of output
// tile 2 * tp + r (its half of A, M = 128 of 256) and input columns r * BN/2
// .. (r+1) * BN/2 - 1 of the column tile (its half of B); the leader (rank 0)
// issues the MMAs, and each CTA's TMEM receives its 128 rows of both
// accumulators.  Per 64-token stage an SM now takes in 32 KB instead of 48 KB
// for the same MMA work.  Token blocks go in pairs of stages (bit-0 rows, then
// bit-1 rows) as in MODE_DWF.
//
// Synchronisation.  Both CTAs' copies of a stage complete on the leader's
// full barrier (the leader expects the pair's bytes).  The leader's commits
// arrive, in both CTAs, on `consumed` (a stage's MMAs are done) and `tfull`
// (a tile is done).  Four helper warps per CTA wait for `consumed`, add up
// their dz tile's columns (dbias) and release the stage on their own CTA's
// `empty`; every epilogue warp of both CTAs releases the accumulators on the
// leader's `tempty`.  Every wait is bounded; an aborting CTA still reaches the
// final cluster barrier, which both CTAs need to free the pair's TMEM.
struct __align__(8) PairBarriers {
    uint64_t full[8];
    uint64_t consumed[8];
    uint64_t empty[8];
    uint64_t tfull;
    uint64_t tempty;
    uint64_t drain;
    uint64_t ring_idle;   // the helper warps are done with the CTA's last unit's stages
    uint32_t tmem_base;
    int abort;
};

// A stage: this CTA's dz rows (A), its input columns (B) and, in a launch
// with shift layers, the same columns of the rows `shift` positions earlier (B2).
template <int BN, bool SHIFT>
__host__ __device__ constexpr int pair_stage_bytes() {
    return kABytes + (SHIFT ? 2 : 1) * (BN / 2) * kBlockK * 2;
}
template <int BN, bool SHIFT>
__host__ __device__ constexpr int pair_stages() {
    return ((kRingBytesDwf / pair_stage_bytes<BN, SHIFT>()) > 8
                ? 8
                : (kRingBytesDwf / pair_stage_bytes<BN, SHIFT>())) &
           ~1;
}
template <int BN, bool SHIFT>
__host__ __device__ constexpr size_t pair_smem_total() {
    return 1024 + (size_t)pair_stages<BN, SHIFT>() * pair_stage_bytes<BN, SHIFT>() +
           sizeof(PairBarriers);
}

template <int BN, bool SHIFT>
__global__ void __launch_bounds__(cta_threads(BN), 1)
    hcw_dwp_kernel(const __grid_constant__ TcLaunch<kMaxStackLayers> L) {
    constexpr int STAGES = pair_stages<BN, SHIFT>();
    constexpr int SB = pair_stage_bytes<BN, SHIFT>();
    constexpr int B2_OFF = kABytes + (BN / 2) * kBlockK * 2;   // SHIFT: the B2 tile
    constexpr int NH = BN / 2;                          // B columns per CTA
    constexpr uint32_t TMEM_COLS = 2 * BN;              // self and partner accumulators
    constexpr uint32_t IDESC = idesc_bf16_f32(2 * kBlockM, BN, 1, 1);
    constexpr int EW = epi_warps(BN);
    constexpr int WCOLS = warp_cols(BN);
    static_assert(STAGES % 2 == 0 && STAGES >= 2, "pairs of stages");
    // the last unit's staging buffers per epilogue warp: as many 4 KB patches as
    // the idle ring holds, up to the warp's four stores
    constexpr int NBUF = (STAGES * SB) / (EW * kEpiBufBytes) >= 4
                             ? 4
                             : (STAGES * SB) / (EW * kEpiBufBytes);
    static_assert(NBUF >= 2 && EW * NBUF * kEpiBufBytes <= STAGES * SB,
                  "patch buffers inside the ring");
    const TcParams& p = L.p;
    const uint32_t rank = cluster_ctarank();
    const int pair = (int)blockIdx.x >> 1, n_pairs = (int)gridDim.x >> 1;
    const int tpl = p.n_ot / 2;                         // 256-row tiles per layer
    const int upl = tpl * p.n_nt;
    const int n_units = upl * L.n_layers;

    extern __shared__ uint8_t smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~(uintptr_t)1023);
    PairBarriers* bars = reinterpret_cast<PairBarriers*>(smem + (size_t)STAGES * SB);
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        // the operand maps of this pair's own units only (one unit a pair in
        // the training step), in the order the units come
        for (int u = pair; u < n_units; u += n_pairs) {
            const int lu = u / upl;
            const int l = L.dep_counters != nullptr ? L.n_layers - 1 - lu : lu;
            tma_prefetch_desc(&L.maps[l][0]);
            tma_prefetch_desc(&L.maps[l][1]);
            if (SHIFT && L.layer[l].shift > 0) tma_prefetch_desc(&L.maps[l][2]);
        }
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(&bars->full[s], 1);
            mbar_init(&bars->consumed[s], 1);
            mbar_init(&bars->empty[s], kDwHelpers);
        }
        mbar_init(&bars->tfull, 1);
        mbar_init(&bars->tempty, 2 * EW);
        mbar_init(&bars->drain, 1);
        mbar_init(&bars->ring_idle, kDwHelpers);
        bars->abort = 0;
        fence_mbar_init();
    }
    if (warp == 1) {
        tmem_alloc_pair(&bars->tmem_base, TMEM_COLS);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync_all();   // both CTAs' barriers exist before any cross-CTA arrive
    tc_fence_after();
    const uint32_t tmem_base = bars->tmem_base;
    volatile int* abort = &bars->abort;
    const uint64_t tmo = p.timeout_ns;

    // unit u -> (layer, tile); a launch behind the fused input gradient takes
    // the layers from the top down, the order in which their dz complete
    const bool dep = L.dep_counters != nullptr;
    auto unit_layer = [&](int u, int& ul) {
        const int lu = u / upl;
        ul = u - lu * upl;
        return dep ? L.n_layers - 1 - lu : lu;
    };

    if (warp == 0) {
        // ------------------------------------------------------------ producer (both CTAs)
        // lane 0 issues the copies; the whole warp waits for a unit's operands
        // when the launch started before they were complete
        int stage = 0;
        uint32_t phase = 0;
        uint32_t issued_mask = 0, issued_phase = 0;
        bool ok = true;
        for (int u = pair; u < n_units && ok; u += n_pairs) {
            int ul;
            const int l = unit_layer(u, ul);
            const int tp = ul / p.n_nt, nt = ul - tp * p.n_nt;
            const TcLayer& ly = L.layer[l];
            if (dep) {
                ok = wait_chunks_warp(L.dep_counters + (size_t)ly.dep_row * L.n_chunks,
                                      L.n_chunks, L.tokens, p.d, abort, tmo);
                if (!ok) break;
            }
            if (lane == 0) {
                if (dep) fence_proxy_async_global();   // the copies read what was acquired
                for (int pq = 0; pq < p.qb && ok; ++pq) {
                    const int q0 = pq * 64;
                    const int lo0 = q0 & (ly.k - 1), hi0 = q0 >> ly.s;
                    for (int bit = 0; bit < 2; ++bit) {
                        if (!mbar_wait(&bars->empty[stage], phase ^ 1, abort, tmo)) {
                            ok = false;
                            break;
                        }
                        uint8_t* sA = smem + (size_t)stage * SB;
                        const bool shl = SHIFT && ly.shift > 0;
                        if (rank == 0)
                            mbar_arrive_expect_tx(&bars->full[stage],
                                                  2 * (shl ? SB : B2_OFF));
                        issued_mask |= 1u << stage;
                        issued_phase = (issued_phase & ~(1u << stage)) | (phase << stage);
                        const uint32_t fb = mapa_shared(&bars->full[stage], 0);
                        tma_load_5d_pair(sA, &L.maps[l][0], fb, 0, lo0, bit, hi0,
                                         (2 * tp + (int)rank) * (kBlockM / 64));
                        tma_load_5d_pair(sA + kABytes, &L.maps[l][1], fb, 0, lo0, bit, hi0,
                                         nt * (BN / 64) + (int)rank * (NH / 64));
                        if (shl) {
                            // the stage's 64 positions p of one sample, and the same
                            // columns at p - shift (zeros before the sample's start)
                            const long long tok = (long long)hi0 * 2 * ly.k + bit * ly.k + lo0;
                            const int smp = (int)(tok / p.seq_n), pos = (int)(tok % p.seq_n);
                            tma_load_4d_pair(sA + B2_OFF, &L.maps[l][2], fb, 0, pos - ly.shift,
                                             smp, nt * (BN / 64) + (int)rank * (NH / 64));
                        }
                        if (++stage == STAGES) {
                            stage = 0;
                            phase ^= 1;
                        }
                    }
                }
            }
            ok = __shfl_sync(0xffffffffu, ok, 0) != 0;
        }
        if (!ok && rank == 0 && lane == 0) {
            // every copy of the pair completes on the leader's barriers: let them land
            for (int s = 0; s < STAGES; ++s)
                if (issued_mask & (1u << s))
                    mbar_wait_drain(&bars->full[s], (issued_phase >> s) & 1u, tmo);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer (leader)
        if (lane == 0 && rank == 0) {
            int stage = 0;
            uint32_t phase = 0, acc_phase = 0;
            bool ok = true, any = false;
            for (int u = pair; u < n_units && ok; u += n_pairs) {
                if (!mbar_wait(&bars->tempty, acc_phase ^ 1, abort, tmo)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t d_self = tmem_base, d_nbr = tmem_base + BN;
                for (int pq = 0; pq < p.qb && ok; ++pq) {
                    if (!mbar_wait(&bars->full[stage], phase, abort, tmo) ||
                        !mbar_wait(&bars->full[stage + 1], phase, abort, tmo)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t a0 = smem_u32(smem + (size_t)stage * SB), x0 = a0 + kABytes;
                    const uint32_t a1 = a0 + SB, x1 = a1 + kABytes;
                    auto dsc = [](uint32_t base, int kk) {
                        return smem_desc_sw128(base + kk * 2048, 8192, 1024);
                    };
#pragma unroll
                    for (int kk = 0; kk < kBlockK / 16; ++kk)
                        mma_bf16_f32_pair(d_self, dsc(a0, kk), dsc(x0, kk), IDESC, (pq | kk) != 0);
#pragma unroll
                    for (int kk = 0; kk < kBlockK / 16; ++kk)
                        mma_bf16_f32_pair(d_self, dsc(a1, kk), dsc(x1, kk), IDESC, 1);
                    int ul_unused;
                    if (SHIFT && L.layer[unit_layer(u, ul_unused)].shift > 0) {
                        // a shift layer: every row's partner is the row shift earlier
                        const uint32_t y0 = a0 + B2_OFF, y1 = a1 + B2_OFF;
#pragma unroll
                        for (int kk = 0; kk < kBlockK / 16; ++kk)
                            mma_bf16_f32_pair(d_nbr, dsc(a0, kk), dsc(y0, kk), IDESC, (pq | kk) != 0);
#pragma unroll
                        for (int kk = 0; kk < kBlockK / 16; ++kk)
                            mma_bf16_f32_pair(d_nbr, dsc(a1, kk), dsc(y1, kk), IDESC, 1);
                    } else {
#pragma unroll
                        for (int kk = 0; kk < kBlockK / 16; ++kk)
                            mma_bf16_f32_pair(d_nbr, dsc(a1, kk), dsc(x0, kk), IDESC, (pq | kk) != 0);
                        if (!p.causal) {
#pragma unroll
                            for (int kk = 0; kk < kBlockK / 16; ++kk)
                                mma_bf16_f32_pair(d_nbr, dsc(a0, kk), dsc(x1, kk), IDESC, 1);
                        }
                    }
                    any = true;
                    mma_commit_pair(&bars->consumed[stage], 3);
                    mma_commit_pair(&bars->consumed[stage + 1], 3);
                    stage += 2;
                    if (stage == STAGES) {
                        stage = 0;
                        phase ^= 1;
                    }
                }
                if (!ok) break;
                mma_commit_pair(&bars->tfull, 3);
                acc_phase ^= 1;
            }
            if (any) {
                // the pair's MMAs have completed before TMEM can be freed
                mma_commit_pair(&bars->drain, 1);
                mbar_wait_drain(&bars->drain, 0, tmo);
            }
        }
    } else {
        // ------------------------------------------------------------ epilogue (both CTAs)
        const int e = warp - 2;
        const int quarter = warp & 3;
        const int cslice = e >> 2;
        const uint32_t tempty_leader = mapa_shared(&bars->tempty, 0);
        int hstage = 0;
        uint32_t hphase = 0, acc_phase = 0;
        bool alive = true;
        for (int u = pair; u < n_units && alive; u += n_pairs) {
            int ul;
            const int l = unit_layer(u, ul);
            const int tp = ul / p.n_nt, nt = ul - tp * p.n_nt;
            const int ot = 2 * tp + (int)rank;
            const TcLayer& ly = L.layer[l];
            const bool last = u + n_pairs >= n_units;   // no further unit: the ring goes idle
            // the output maps of the last unit's staged stores, fetched while it runs
            if (last && e == EW - 1 && lane == 0) {
                tma_prefetch_desc(&L.maps[l][4]);
                tma_prefetch_desc(&L.maps[l][5]);
            }
            if (e < kDwHelpers) {
                // release this CTA's stages once the pair's MMAs have read them, and
                // sum the dz tile's columns on the way (dbias, output rows of tile ot)
                const bool do_cs = ly.colsum != nullptr && nt == 0;
                const int t = e * 32 + lane;
                const int box = t >> 6, c = (t >> 3) & 7, tph = t & 7;
                float cs[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) cs[i] = 0.f;
                for (int ks = 0; ks < 2 * p.qb; ++ks) {
                    const bool okw = mbar_wait(&bars->consumed[hstage], hphase, abort, tmo);
                    if (!__all_sync(0xffffffffu, okw)) {
                        alive = false;
                        break;
                    }
                    if (do_cs) {
                        const uint8_t* sA = smem + (size_t)hstage * SB + box * 8192;
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const int r = tph + 8 * i;
                            const uint4 q =
                                *reinterpret_cast<const uint4*>(sA + r * 128 + ((c ^ tph) << 4));
                            const uint32_t wv[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
                            for (int j = 0; j < 4; ++j) {
                                const float2 f = unpack_bf16x2(wv[j]);
                                cs[2 * j] += f.x;
                                cs[2 * j + 1] += f.y;
                            }
                        }
                    }
                    __syncwarp();
                    if (lane == 0) mbar_arrive(&bars->empty[hstage]);
                    if (++hstage == STAGES) {
                        hstage = 0;
                        hphase ^= 1;
                    }
                }
                if (!alive) break;
                if (do_cs) {
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        cs[i] += __shfl_xor_sync(0xffffffffu, cs[i], 1);
                        cs[i] += __shfl_xor_sync(0xffffffffu, cs[i], 2);
                        cs[i] += __shfl_xor_sync(0xffffffffu, cs[i], 4);
                    }
                    const int o0 = ot * kBlockM + box * 64 + c * 8;
                    if (tph == 0 && o0 < p.d) {
                        float4* dst = reinterpret_cast<float4*>(ly.colsum + o0);
                        dst[0] = make_float4(cs[0], cs[1], cs[2], cs[3]);
                        dst[1] = make_float4(cs[4], cs[5], cs[6], cs[7]);
                    }
                }
                __syncwarp();
                if (last && lane == 0) mbar_arrive(&bars->ring_idle);
            }
            const bool okt = mbar_wait(&bars->tfull, acc_phase, abort, tmo);
            if (!__all_sync(0xffffffffu, okt)) {
                alive = false;
                break;
            }
            tc_fence_after();
            // The CTA's last unit: the ring is idle once the helper warps are done
            // with it, so the tiles go out through shared memory by TMA (NBUF 4 KB
            // patch buffers per warp, whole 128-byte rows): per-lane row stores at
            // the end of the launch, all SMs at once, took ~13 us to drain.
            // Earlier units store from registers while the next unit's operands
            // stream into the ring.
            const bool staged =
                last && __all_sync(0xffffffffu, mbar_wait(&bars->ring_idle, 0, abort, tmo));
            uint8_t* sbuf = smem + (size_t)e * NBUF * kEpiBufBytes;
            int nbuf = 0;
            // this CTA's 128 rows of the tile: one row per lane, 32 fp32 columns per load
            const int row = ot * kBlockM + quarter * 32 + lane;
#pragma unroll 1
            for (int which = 0; which < 2; ++which) {
                float* base = which ? ly.dwn : ly.dws;
#pragma unroll 1
                for (int c = 0; c < WCOLS / 32; ++c) {
                    uint32_t raw[32];
                    __syncwarp();
                    tmem_ld_32x32b_x32(tmem_base + ((uint32_t)(quarter * 32) << 16) +
                                           (uint32_t)(which * BN + cslice * WCOLS + c * 32),
                                       raw);
                    tmem_ld_wait_regs(raw);
                    if (which == 1 && c == WCOLS / 32 - 1) {
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive_remote_tmem(tempty_leader);
                    }
                    if (staged) {
                        uint8_t* buf = sbuf + (nbuf % NBUF) * kEpiBufBytes;
                        // the buffer's store before last has been read
                        if (lane == 0 && nbuf >= NBUF) bulk_wait_read<NBUF - 1>();
                        __syncwarp();
#pragma unroll
                        for (int m = 0; m < 8; ++m)
                            *patch_piece<128>(buf, lane, m) = make_uint4(
                                raw[4 * m], raw[4 * m + 1], raw[4 * m + 2], raw[4 * m + 3]);
                        fence_proxy_async_smem();
                        __syncwarp();
                        // d is a multiple of 64: a warp's 32 rows are all inside or all
                        // past the end of a ragged tile
                        if (lane == 0 && ot * kBlockM + quarter * 32 < p.d) {
                            tma_store_2d(&L.maps[l][4 + which], buf, nt * BN + cslice * WCOLS + c * 32,
                                         ot * kBlockM + quarter * 32);
                            bulk_commit();
                        }
                        ++nbuf;
                        continue;
                    }
                    if (row < p.d) {
                        float4* dst = reinterpret_cast<float4*>(
                            base + (size_t)row * p.d + nt * BN + cslice * WCOLS + c * 32);
#pragma unroll
                        for (int m = 0; m < 8; ++m)
                            dst[m] = make_float4(__uint_as_float(raw[4 * m]),
                                                 __uint_as_float(raw[4 * m + 1]),
                                                 __uint_as_float(raw[4 * m + 2]),
                                                 __uint_as_float(raw[4 * m + 3]));
                    }
                }
            }
            acc_phase ^= 1;
        }
        // every TMA store of this warp has landed before the CTA exits
        if (lane == 0) bulk_wait<0>();
        __syncwarp();
    }

    tc_fence_before();
    __syncthreads();
    cluster_sync_all();   // neither CTA frees the pair's TMEM while the other uses it
    if (warp == 1) {
        __syncwarp();
        tc_fence_after();
        tmem_dealloc_pair(tmem_base, TMEM_COLS);
    }
}

// A launch with dep_counters is a programmatic dependent of the preceding
// kernel (the fused forward / input-gradient launch that triggers it).
template <int BN, bool SHIFT>
static cudaError_t launch_pair(const TcLaunch<kMaxStackLayers>& L, int grid, cudaStream_t st) {
    constexpr size_t smem = pair_smem_total<BN, SHIFT>();
    static_assert(smem <= 232448, "shared memory budget");
    auto kern = hcw_dwp_kernel<BN, SHIFT>;
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
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3((unsigned)cta_threads(BN));
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = L.dep_counters ? 2 : 1;
    return cudaLaunchKernelEx(&cfg, kern, L);
}

template <int MODE, int BN, int NL, bool PAIR = false>
static cudaError_t launch_one(const TcLaunch<NL>& L, int grid, cudaStream_t st) {
    constexpr size_t smem = smem_total<MODE, BN, PAIR>();
    static_assert(smem <= 232448, "shared memory budget");
    auto kern = hcw_tc_kernel<MODE, BN, NL, PAIR>;
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
    if (!PAIR) {
        kern<<<grid, cta_threads(BN), smem, st>>>(L);
        return cudaGetLastError();
    }
    // clusters of two CTAs (the grid is even)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3((unsigned)cta_threads(BN));
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

cudaError_t launch_tc(int mode, int BN, const TcLaunch<1>& L, int grid, cudaStream_t st) {
#define HCW_TC_CASE(M, N) \
    if (mode == M && BN == N) return launch_one<M, N, 1>(L, grid, st);
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

cudaError_t launch_tc_stack(int mode, int BN, const TcLaunch<kMaxStackLayers>& L, int grid,
                            cudaStream_t st) {
    if (mode == MODE_DWP) {
        bool shift = false;
        for (int i = 0; i < L.n_layers; ++i) shift = shift || L.layer[i].shift > 0;
        if (BN == 256) return shift ? launch_pair<256, true>(L, grid, st)
                                    : launch_pair<256, false>(L, grid, st);
        if (BN == 128) return shift ? launch_pair<128, true>(L, grid, st)
                                    : launch_pair<128, false>(L, grid, st);
        return cudaErrorInvalidValue;
    }
#define HCW_TC_STACK_CASE(M, N) \
    if (mode == M && BN == N) return launch_one<M, N, kMaxStackLayers>(L, grid, st);
    HCW_TC_STACK_CASE(MODE_FWD, 256)
    HCW_TC_STACK_CASE(MODE_FWD, 128)
    HCW_TC_STACK_CASE(MODE_FWD, 64)
    HCW_TC_STACK_CASE(MODE_DX, 256)
    HCW_TC_STACK_CASE(MODE_DX, 128)
    HCW_TC_STACK_CASE(MODE_DX, 64)
    HCW_TC_STACK_CASE(MODE_DW, 256)
    HCW_TC_STACK_CASE(MODE_DW, 128)
    HCW_TC_STACK_CASE(MODE_DW, 64)
    HCW_TC_STACK_CASE(MODE_DWF, 256)
    HCW_TC_STACK_CASE(MODE_DWF, 128)
    HCW_TC_STACK_CASE(MODE_DWF, 64)
#undef HCW_TC_STACK_CASE
    return cudaErrorInvalidValue;
}

cudaError_t launch_tc_stack_pair(int mode, int BN, const TcLaunch<kMaxStackLayers>& L, int grid,
                                 cudaStream_t st) {
    if (BN != 256 || grid % 2) return cudaErrorInvalidValue;
    if (mode == MODE_FWD) return launch_one<MODE_FWD, 256, kMaxStackLayers, true>(L, grid, st);
    if (mode == MODE_DX) return launch_one<MODE_DX, 256, kMaxStackLayers, true>(L, grid, st);
    return cudaErrorInvalidValue;
}

cudaError_t launch_tc_step_pair(int BN, const TcLaunch<kMaxStepLayers>& L, int grid,
                                cudaStream_t st) {
    if (grid % 2) return cudaErrorInvalidValue;
    if (BN == 256) return launch_one<MODE_FDX, 256, kMaxStepLayers, true>(L, grid, st);
    if (BN == 128) return launch_one<MODE_FDX, 128, kMaxStepLayers, true>(L, grid, st);
    return cudaErrorInvalidValue;
}

size_t tc_smem_bytes(int BN) {
    return BN == 256 ? smem_total<MODE_FWD, 256>()
                     : BN == 128 ? smem_total<MODE_FWD, 128>() : smem_total<MODE_FWD, 64>();
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
