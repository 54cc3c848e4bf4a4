// hcw_api.cu -- the C ABI of include/hcw.h: argument validation, TMA tensor
// maps, work decomposition and launches.  No device memory is allocated
// here; every buffer is the caller's.
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <atomic>
#include <mutex>

#include "hcw.h"
#include "hcw_internal.h"

namespace hcw {
namespace {

constexpr unsigned kAllFlags = HCW_CAUSAL | HCW_RESIDUAL | HCW_ACT_RELU;
constexpr unsigned long long kDefaultTimeoutNs = 2000000000ull;   // 2 s per wait

int log2_exact(long long n) {
    if (n < 2 || (n & (n - 1))) return -1;
    int b = 0;
    while ((1ll << b) < n) ++b;
    return b;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

bool overlaps(const void* a, size_t na, const void* b, size_t nb) {
    if (!a || !b || na == 0 || nb == 0) return false;
    const uintptr_t x = reinterpret_cast<uintptr_t>(a), y = reinterpret_cast<uintptr_t>(b);
    return x < y + nb && y < x + na;
}

size_t elem_size(int dtype) { return dtype == HCW_F32 ? 4 : 2; }

int sm_count() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 148;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1)
        return 148;
    return n;
}

// ------------------------------------------------------------ tensor maps
typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void* p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

// Token-major activations [B*n][d] bf16 viewed as (d, lo = k, bit = 2, HI),
// box (inner features, box_lo, 1, box_hi) with box_lo * box_hi = box_rows
// positions sharing bit s; the 128-byte swizzle for 64-feature (128-byte)
// boxes, the 64-byte swizzle for 32-feature ones.
bool map_rows(CUtensorMap* m, const void* base, long long tokens, int d, int k, int box_rows,
              int inner = 64) {
    EncodeTiledFn enc = encode_fn();
    if (!enc || !base) return false;
    const int box_lo = k < box_rows ? k : box_rows;
    const int box_hi = box_rows / box_lo;
    const long long HI = tokens / (2ll * k);
    cuuint64_t dims[4] = {(cuuint64_t)d, (cuuint64_t)k, 2, (cuuint64_t)HI};
    cuuint64_t strides[3] = {(cuuint64_t)d * 2, (cuuint64_t)k * d * 2, (cuuint64_t)2 * k * d * 2};
    cuuint32_t box[4] = {(cuuint32_t)inner, (cuuint32_t)box_lo, 1, (cuuint32_t)box_hi};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
               inner == 64 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// The same view with the features split into 64-wide blocks as the outermost
// dimension, (64, lo, bit, HI, d / 64): a box (64, box_lo, 1, box_hi, nblk)
// fetches nblk consecutive 64-feature blocks of the same 64 positions in one
// copy, laid out block after block (the MN-major operands of the weight
// gradient).
bool map_rows_blocks(CUtensorMap* m, const void* base, long long tokens, int d, int k,
                     int box_rows, int nblk) {
    EncodeTiledFn enc = encode_fn();
    if (!enc || !base) return false;
    const int box_lo = k < box_rows ? k : box_rows;
    const int box_hi = box_rows / box_lo;
    const long long HI = tokens / (2ll * k);
    cuuint64_t dims[5] = {64, (cuuint64_t)k, 2, (cuuint64_t)HI, (cuuint64_t)(d / 64)};
    cuuint64_t strides[4] = {(cuuint64_t)d * 2, (cuuint64_t)k * d * 2, (cuuint64_t)2 * k * d * 2,
                             128};
    cuuint32_t box[5] = {64, (cuuint32_t)box_lo, 1, (cuuint32_t)box_hi, (cuuint32_t)nblk};
    cuuint32_t estr[5] = {1, 1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, const_cast<void*>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Activations [samples][n][d] bf16 as (64 features, position, sample, d / 64
// blocks), box (64, 64 positions, 1, nblk): 64 consecutive positions of one
// sample; positions outside [0, n) load as zeros (a shift layer's partner rows,
// read at p - k).
bool map_positions_blocks(CUtensorMap* m, const void* base, long long tokens, int n, int d,
                          int nblk) {
    EncodeTiledFn enc = encode_fn();
    if (!enc || !base || n < 64) return false;
    cuuint64_t dims[4] = {64, (cuuint64_t)n, (cuuint64_t)(tokens / n), (cuuint64_t)(d / 64)};
    cuuint64_t strides[3] = {(cuuint64_t)d * 2, (cuuint64_t)n * d * 2, 128};
    cuuint32_t box[4] = {64, 64, 1, (cuuint32_t)nblk};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Activations [samples][n][d] bf16 as (d, position, sample, 1), box (64
// features, box_rows positions, 1, 1), 128-byte swizzle: box_rows consecutive
// positions of one sample; positions outside [0, n) load as zeros (the
// partner rows of a shift layer in a stacked launch).
bool map_positions(CUtensorMap* m, const void* base, long long tokens, int n, int d,
                   int box_rows) {
    EncodeTiledFn enc = encode_fn();
    if (!enc || !base || n < box_rows) return false;
    cuuint64_t dims[4] = {(cuuint64_t)d, (cuuint64_t)n, (cuuint64_t)(tokens / n), 1};
    cuuint64_t strides[3] = {(cuuint64_t)d * 2, (cuuint64_t)n * d * 2,
                             (cuuint64_t)tokens * d * 2};
    cuuint32_t box[4] = {64, (cuuint32_t)box_rows, 1, 1};
    cuuint32_t estr[4] = {1, 1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Weights W[o][i] as (64 i, o, d / 64 i-blocks), box (64, 64 o, nblk): nblk
// consecutive 64-column blocks of 64 rows in one copy (the MN-major B
// operand of the input gradient), 128-byte swizzle.
bool map_weight_blocks(CUtensorMap* m, const void* base, int d, int nblk) {
    EncodeTiledFn enc = encode_fn();
    if (!enc || !base) return false;
    cuuint64_t dims[3] = {64, (cuuint64_t)d, (cuuint64_t)(d / 64)};
    cuuint64_t strides[2] = {(cuuint64_t)d * 2, 128};
    cuuint32_t box[3] = {64, 64, (cuuint32_t)nblk};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Activations [tokens][d] bf16 as (8 features, tokens, d / 8): a box (8,
// box_tokens, nchunk) is a box_tokens x 8*nchunk-feature slice laid out chunk
// by chunk, 16 bytes per token and chunk -- the layout of the resident
// kernels' A tile.
bool map_rows16(CUtensorMap* m, const void* base, long long tokens, int d, int nchunk,
                int box_tokens) {
    EncodeTiledFn enc = encode_fn();
    if (!enc || !base) return false;
    cuuint64_t dims[3] = {8, (cuuint64_t)tokens, (cuuint64_t)(d / 8)};
    cuuint64_t strides[2] = {(cuuint64_t)d * 2, 16};
    cuuint32_t box[3] = {8, (cuuint32_t)box_tokens, (cuuint32_t)nchunk};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_NONE,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Weights W[o][k] bf16 [d][d], box (64 k, box_o), 128-byte swizzle.
bool map_weight(CUtensorMap* m, const void* base, int d, int box_o) {
    EncodeTiledFn enc = encode_fn();
    if (!enc || !base) return false;
    cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)d};
    cuuint64_t strides[1] = {(cuuint64_t)d * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)box_o};
    cuuint32_t estr[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// bf16 matrix [rows][d] viewed as (64 features, rows, d / 64 tiles), box
// (64, box_rows, box_tiles), 128-byte swizzle: one copy lands box_tiles
// consecutive 64-feature tiles of box_rows rows each (the decode's weight
// chunks, ring rows and inputs).
bool map_tiles_sw128(CUtensorMap* m, const void* base, long long rows, int d, int box_rows,
                     int box_tiles) {
    EncodeTiledFn enc = encode_fn();
    if (!enc || !base || rows < 1) return false;
    cuuint64_t dims[3] = {64, (cuuint64_t)rows, (cuuint64_t)(d / 64)};
    cuuint64_t strides[2] = {(cuuint64_t)d * 2, 128};
    cuuint32_t box[3] = {64, (cuuint32_t)box_rows, (cuuint32_t)box_tiles};
    cuuint32_t estr[3] = {1, 1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// fp32 matrix [rows][d], box (32 columns, 32 rows), 128-byte swizzle: the
// patches the weight-gradient epilogue stores.
bool map_f32_patches(CUtensorMap* m, const void* base, long long rows, int d) {
    EncodeTiledFn enc = encode_fn();
    if (!enc || !base) return false;
    cuuint64_t dims[2] = {(cuuint64_t)d, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)d * 4};
    cuuint32_t box[2] = {32, 32};
    cuuint32_t estr[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void*>(base), dims, strides,
               box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
               CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int pick_bn(int d) { return d % 256 == 0 ? 256 : d % 128 == 0 ? 128 : 64; }

// ------------------------------------------------------------ validation
struct Shape {
    int B, n, d, b, s;
    long long tokens;
    size_t act_bytes;
};

int check_shape(int layer, int dim_override, int B, int n, int d, int dtype, unsigned flags,
                Shape* sh) {
    if (dtype != HCW_BF16 && dtype != HCW_F32) return HCW_ERR_INVALID_ARG;
    if (flags & ~kAllFlags) return HCW_ERR_INVALID_ARG;
    const int b = log2_exact(n);
    if (b < 1 || n > (1 << 30)) return HCW_ERR_INVALID_ARG;
    if (B < 0 || d < 1 || layer < 0) return HCW_ERR_INVALID_ARG;
    if (dim_override < -1 || dim_override >= b) return HCW_ERR_INVALID_ARG;
    const long long tokens = (long long)B * n;
    if (tokens > (1ll << 31) - 1) return HCW_ERR_UNSUPPORTED;
    if (dtype == HCW_BF16 && (d % 64 != 0 || d > 16384)) return HCW_ERR_UNSUPPORTED;
    sh->B = B;
    sh->n = n;
    sh->d = d;
    sh->b = b;
    sh->s = dim_override >= 0 ? dim_override : layer % b;
    sh->tokens = tokens;
    sh->act_bytes = (size_t)tokens * d * elem_size(dtype);
    return HCW_OK;
}

// Layer schedule of a stack (Sec. 3.3, Sec. 4): stack layer l uses cube
// dimension dims[l] when a schedule array is given, else dim_override for
// every layer (the fixed control), else (layer0 + l) mod log2 n (rot).
struct Sched {
    const int* dims;
    int layer0;
    int dim_override;
    // s >= 0: hypercube dimension; s < 0: shift of Eq. (1) by -s (schedules only)
    int dim(const Shape& sh, int l) const {
        if (dims) return dims[l];
        return dim_override >= 0 ? dim_override : (layer0 + l) % sh.b;
    }
    bool has_shift(int L) const {
        if (!dims) return false;
        for (int l = 0; l < L; ++l)
            if (dims[l] < 0) return true;
        return false;
    }
};

// Row grouping of a shift layer's launches: any cube dimension serves (the
// partner rows come row-aligned from a second tensor); 2^6 = 64-row runs.
int shift_group_dim(const Shape& sh) { return sh.b - 1 < 6 ? sh.b - 1 : 6; }

// Stacked forward / input-gradient launches take shift layers when a 128-row
// unit lies inside one sample and the tokens form whole 256-token row-block
// pairs (the k = 128 grouping): n >= 128, tokens a multiple of 256.
constexpr int kShiftStackDim = 7;
bool shift_stackable(const Shape& sh) { return sh.n >= 128 && sh.tokens % 256 == 0; }

// Bytes of one layer's ReLU mask: ceil(d/32) 32-bit words per token.
size_t mask_bytes(const Shape& sh) { return (size_t)sh.tokens * ((sh.d + 31) / 32) * 4; }

// ------------------------------------------------------------ bf16 sizes
struct WPlan {
    int n_ot, n_nt, qb, nkb_self, nkb_nbr, kb_per_unit, splits_self, splits_nbr, splits_max,
        units;
};

// The split of the token range of the weight gradient into units: one layer's,
// or `layers` layers' sharing one launch.
WPlan plan_dw(long long tokens, int d, unsigned flags, int layers = 1) {
    WPlan w;
    const int BN = pick_bn(d);
    const long long Mh = tokens / 2;
    w.n_ot = (d + 127) / 128;
    w.n_nt = d / BN;
    w.qb = (int)((Mh + 63) / 64);
    w.nkb_self = 2 * w.qb;
    w.nkb_nbr = (flags & HCW_CAUSAL) ? w.qb : 2 * w.qb;
    const int tiles = w.n_ot * w.n_nt;
    const long long total_kb = (long long)layers * tiles * (w.nkb_self + w.nkb_nbr);
    const int sms = sm_count();
    // the fewest token blocks per unit (at least 4, i.e. 256 tokens) whose
    // units still fit in one wave of persistent CTAs: makespan = kpu blocks
    long long kpu = (total_kb + sms - 1) / sms;
    if (kpu < 4) kpu = 4;
    // (once kpu covers every block of both parts there is one split each and
    // the count cannot drop further, even if the tiles alone exceed the SMs)
    const long long kpu_max = w.nkb_self > w.nkb_nbr ? w.nkb_self : w.nkb_nbr;
    while (kpu < kpu_max &&
           (long long)layers * tiles *
                   ((w.nkb_self + kpu - 1) / kpu + (w.nkb_nbr + kpu - 1) / kpu) > sms)
        ++kpu;
    w.kb_per_unit = (int)kpu;
    w.splits_self = (int)((w.nkb_self + kpu - 1) / kpu);
    w.splits_nbr = (int)((w.nkb_nbr + kpu - 1) / kpu);
    if (w.splits_self < 1) w.splits_self = 1;
    if (w.splits_nbr < 1) w.splits_nbr = 1;
    w.splits_max = w.splits_self > w.splits_nbr ? w.splits_self : w.splits_nbr;
    w.units = tiles * (w.splits_self + w.splits_nbr);
    return w;
}

// SM pairs of the batched weight-gradient launch of a training step when it
// runs on pairs behind the fused forward / input-gradient launch (the
// conditions of stack_weight_bf16 for one launch of <= kMaxStackLayers
// layers), else 0.
int dw_early_pairs(const Shape& sh, unsigned flags, int L) {
    if (L > kMaxStackLayers || pick_bn(sh.d) < 128) return 0;
    const WPlan w = plan_dw(sh.tokens, sh.d, flags);
    const int tiles = w.n_ot * w.n_nt, sms = sm_count();
    if (L * tiles * 2 < sms || 5 * L * tiles < 3 * sms || w.n_ot % 2 != 0) return 0;
    const int total = tiles * L;
    return total / 2 < sms / 2 ? total / 2 : sms / 2;
}

// Workspace of the weight gradient (bf16: dW split partials, both dtypes:
// column-sum partials of dbias) and of the full layer backward, which adds
// the masked gradient dz = dy * act'(z) in front when an activation is used:
//   [dz (ReLU only)][dW partials (bf16, more than one split)][colsum partials]
struct WsLayout {
    size_t dz_off, dz_bytes, w_off, part_bytes, col_off, col_bytes, w_bytes, total;
};

size_t align256(size_t v) { return (v + 255) & ~(size_t)255; }

WsLayout ws_layout(long long tokens, int d, int dtype, unsigned flags) {
    WsLayout l;
    const size_t es = elem_size(dtype);
    l.dz_off = 0;
    l.dz_bytes = (flags & HCW_ACT_RELU) ? align256((size_t)tokens * d * es) : 0;
    l.w_off = l.dz_off + l.dz_bytes;
    if (dtype == HCW_BF16 && tokens > 0) {
        WPlan w = plan_dw(tokens, d, flags);
        l.part_bytes = (w.splits_max > 1) ? align256((size_t)2 * w.splits_max * d * d * 4) : 0;
    } else {
        l.part_bytes = 0;
    }
    l.col_off = l.part_bytes;   // relative to w_off
    l.col_bytes = align256(colsum_workspace_bytes(tokens, d));
    l.w_bytes = l.part_bytes + l.col_bytes;
    l.total = l.w_off + l.w_bytes;
    return l;
}

unsigned long long g_timeout_ns = kDefaultTimeoutNs;
std::atomic<unsigned long long> g_launches{0};

int cuda_status(cudaError_t e) { return e == cudaSuccess ? HCW_OK : HCW_ERR_CUDA; }

// Count `kernels` launches if the launch call succeeded.
int launched(cudaError_t e, int kernels) {
    if (e != cudaSuccess) return HCW_ERR_CUDA;
    g_launches.fetch_add((unsigned long long)kernels, std::memory_order_relaxed);
    return HCW_OK;
}

// ------------------------------------------------------------ layer internals
// Row-unit geometry of a forward (or input-gradient) pass: which bit value's
// rows take both parts.  Sec. 3.1 causal rule: in the forward, positions with
// bit s set receive (K = 2d) and the others do not (K = d); in the input
// gradient it is the mirror image (a bit-0 row takes dz from its partner).
void row_unit_params(TcParams& p, const Shape& sh, int BN, unsigned flags, bool backward) {
    const int d = sh.d;
    p.d = d;
    p.Mh = (int)(sh.tokens / 2);
    p.nK = d / 64;
    p.n_rb = (p.Mh + 127) / 128;
    p.n_nt = d / BN;
    if (flags & HCW_CAUSAL) {
        p.n_full = 1;
        p.full_bit0 = backward ? 0 : 1;
        p.half_bit = backward ? 1 : 0;
    } else {
        p.n_full = 2;
        p.full_bit0 = 0;
        p.full_bit1 = 1;
        p.half_bit = -1;
    }
    p.n_units = p.n_rb * p.n_nt * 2;
    p.timeout_ns = g_timeout_ns;
}

// The five forward maps of one layer: x rows (128-row boxes), W_self, W_nbr,
// x rows (32-row residual patches), y rows (32-row output patches).
// pair: the weight boxes hold half a column tile (each CTA of a pair loads
// its half of B)
bool fwd_maps(CUtensorMap* m, const Shape& sh, int s, const void* x, const void* Ws,
              const void* Wn, const void* y, bool pair = false, int bn = 0) {
    const int d = sh.d, BN = bn ? bn : pick_bn(d), k = 1 << s;
    const int pw = epi_patch_cols(BN);
    const int box_o = pair ? BN / 2 : BN;
    if (!map_rows(&m[0], x, sh.tokens, d, k, 128) || !map_weight(&m[1], Ws, d, box_o) ||
        !map_weight(&m[2], Wn, d, box_o) || !map_rows(&m[3], x, sh.tokens, d, k, 32, pw) ||
        !map_rows(&m[4], y, sh.tokens, d, k, 32, pw))
        return false;
    m[5] = m[4];   // unused by the forward
    return true;
}

// xpair (a shift layer): the partner part reads the same rows of xpair, and
// every row takes both parts.
int fwd_bf16(const Shape& sh, const void* x, const void* Ws, const void* Wn, const float* bias,
             unsigned flags, void* y, void* z, uint32_t* mask, cudaStream_t st,
             const void* xpair = nullptr) {
    const int BN = pick_bn(sh.d);
    TcLaunch<1> L;
    memset(&L, 0, sizeof(L));
    if (!fwd_maps(L.maps[0], sh, sh.s, x, Ws, Wn, y)) return HCW_ERR_CUDA;
    if (xpair && !map_rows(&L.maps[0][5], xpair, sh.tokens, sh.d, 1 << sh.s, 128))
        return HCW_ERR_CUDA;
    L.layer[0] = {sh.s, 1 << sh.s, bias, mask, static_cast<__nv_bfloat16*>(z), true, nullptr, false};
    L.layer[0].pair_rows = xpair != nullptr;
    row_unit_params(L.p, sh, BN, xpair ? flags & ~HCW_CAUSAL : flags, false);
    L.p.flags = flags;
    L.n_layers = 1;
    const int sms = sm_count();
    const int grid = L.p.n_units < sms ? L.p.n_units : sms;
    return launched(launch_tc(MODE_FWD, BN, L, grid, st), 1);
}

// Completion counters of a stacked-forward launch: one int per layer of the
// group and 128-token chunk.
size_t stack_counter_bytes(long long tokens, int L) {
    const int layers = L < kMaxStackLayers ? L : kMaxStackLayers;
    // per (layer, 128-token chunk) completion counters, the unit counter, the
    // chunk counters of the top layer's dz written by the launch itself, and
    // (input gradient) per (layer, chunk) counters of the output gradient g
    const size_t chunks = (size_t)((tokens + 127) / 128);
    return align256((2 * (size_t)layers * chunks + 1 + chunks) * sizeof(int) + 16);
}

// Whether a stacked forward / input-gradient launch runs on pairs of SMs
// (tcgen05 cta_group::2, 256-row tiles): 256-column tiles and at least two
// row blocks.  Each SM of a pair loads its own rows and half of the weight
// tile per stage.
bool use_pairs(const Shape& sh) {
    return pick_bn(sh.d) == 256 && sh.tokens / 2 > 128;
}

// Whether a bf16 stacked forward / input gradient runs on the resident
// kernels (hcw_res.cu): the shape fits them (d in {128, 256, 512}, n <= 256,
// whole 256-token tiles) and hcw_set_stack_kernels asked for them.
std::atomic<int> g_stack_kernels{HCW_STACK_AUTO};
std::atomic<int> g_decode_kernel{HCW_DECODE_WARP_MMA};

bool use_resident(const Shape& sh) {
    const int mode = g_stack_kernels.load(std::memory_order_relaxed);
    if (mode == HCW_STACK_STREAMING || !res_supported(sh.d, sh.n, sh.tokens)) return false;
    // measured on GB300 (char-LM shapes, d = 512): the streaming kernels are
    // faster, so they are the automatic choice
    return mode == HCW_STACK_RESIDENT;
}

// Row-unit geometry of a pair launch: units count row-block pairs.
void pair_units(TcParams& p) { p.n_units = ((p.n_rb + 1) / 2) * p.n_nt * 2; }

// Launch a stacked forward / input-gradient run, on pairs of SMs if `pair`.
int launch_rows(int mode, int BN, TcLaunch<kMaxStackLayers>& T, int n, bool pair,
                cudaStream_t st) {
    const int sms = sm_count();
    const int total = T.p.n_units * n;
    if (pair) {
        const int pairs = total < sms / 2 ? total : sms / 2;
        return launched(launch_tc_stack_pair(mode, BN, T, 2 * pairs, st), 1);
    }
    return launched(launch_tc_stack(mode, BN, T, total < sms ? total : sms, st), 1);
}

// Layers [l0, l0 + n) of a bf16 stack in one persistent launch.  in_ptr(l),
// out_ptr(l), mask_ptr(l) give each layer's input, output and mask.
template <class In, class Out, class Mask>
int stack_fwd_group(const Shape& sh, int l0, int n, const Sched& sc,
                    const uint8_t* Ws, const uint8_t* Wn, const float* bias, unsigned flags,
                    In in_ptr, Out out_ptr, Mask mask_ptr, int* counters, cudaStream_t st) {
    const int d = sh.d, BN = pick_bn(d);
    const size_t wb = (size_t)d * d * 2;
    const bool pair = use_pairs(sh);
    static thread_local TcLaunch<kMaxStackLayers> L;
    memset(&L, 0, sizeof(L));
    for (int i = 0; i < n; ++i) {
        const int l = l0 + i;
        const int sl = sc.dim(sh, l);
        // a shift layer: rows in runs of 128 positions, its input as positions
        const int s = sl >= 0 ? sl : kShiftStackDim;
        if (!fwd_maps(L.maps[i], sh, s, in_ptr(l), Ws + l * wb, Wn + l * wb, out_ptr(l), pair) ||
            (sl < 0 && !map_positions(&L.maps[i][0], in_ptr(l), sh.tokens, sh.n, d, 128)))
            return HCW_ERR_CUDA;
        L.layer[i] = {s, 1 << s, bias ? bias + (size_t)l * d : nullptr, mask_ptr(l), nullptr,
                      true, nullptr, false};
        L.layer[i].shift = sl < 0 ? -sl : 0;
    }
    row_unit_params(L.p, sh, BN, flags, false);
    L.p.seq_n = sh.n;
    if (pair) pair_units(L.p);
    L.p.flags = flags;
    L.n_layers = n;
    L.counters = counters;
    L.n_chunks = (int)((sh.tokens + 127) / 128);
    L.tokens = (int)sh.tokens;
    L.sched = counters + (size_t)n * L.n_chunks;
    cudaError_t e = cudaMemsetAsync(counters, 0, ((size_t)n * L.n_chunks + 1) * sizeof(int), st);
    if (e != cudaSuccess) return HCW_ERR_CUDA;
    return launch_rows(MODE_FWD, BN, L, n, pair, st);
}

// Layers [l0, l0 + n) of a bf16 stack in one resident launch (hcw_res.cu).
template <class In, class Out, class Mask>
int stack_fwd_resident(const Shape& sh, int l0, int n, const Sched& sc,
                       const uint8_t* Ws, const uint8_t* Wn, const float* bias, unsigned flags,
                       In in_ptr, Out out_ptr, Mask mask_ptr, cudaStream_t st) {
    const int d = sh.d, N = d >= 256 ? d / 2 : d;
    const size_t wb = (size_t)d * d * 2;
    static thread_local ResLaunch R;
    memset(&R, 0, sizeof(R));
    for (int i = 0; i < n; ++i) {
        const int l = l0 + i;
        const int s = sc.dim(sh, l);
        if (!map_weight(&R.wmap[i][0], Ws + l * wb, d, N / 2) ||
            !map_weight(&R.wmap[i][1], Wn + l * wb, d, N / 2) ||
            !map_rows16(&R.imap[i], out_ptr(l), sh.tokens, d, 1, 64))
            return HCW_ERR_CUDA;
        R.layer[i] = {s, RES_Y, out_ptr(l), bias ? bias + (size_t)l * d : nullptr, mask_ptr(l),
                      nullptr};
    }
    R.in = in_ptr(l0);
    R.n_layers = n;
    R.d = d;
    R.n = sh.n;
    R.tokens = (int)sh.tokens;
    R.flags = flags;
    R.timeout_ns = g_timeout_ns;
    return launched(launch_res(MODE_FWD, R, st), 1);
}

// dx: a row gathers dz from its partner exactly when the partner received from it
// dzpair (a shift layer): the partner part reads the same rows of dzpair
// (the dz of each row's reader), and every row takes both parts.
int dx_bf16(const Shape& sh, const void* dz, const void* dy, const void* Ws, const void* Wn,
            unsigned flags, void* dx, cudaStream_t st, const uint32_t* mprev = nullptr,
            void* dz_out = nullptr, const void* dzpair = nullptr) {
    const int d = sh.d, BN = pick_bn(d), k = 1 << sh.s;
    const int pw = epi_patch_cols(BN);
    TcLaunch<1> L;
    memset(&L, 0, sizeof(L));
    CUtensorMap* maps = L.maps[0];
    // maps of absent operands get a valid stand-in address; the kernel never uses them
    const void* res = (flags & HCW_RESIDUAL) ? dy : dz;
    if (!map_rows(&maps[0], dz, sh.tokens, d, k, 128) || !map_weight_blocks(&maps[1], Ws, d, BN / 64) ||
        !map_weight_blocks(&maps[2], Wn, d, BN / 64) ||
        !map_rows(&maps[3], res, sh.tokens, d, k, 32, pw) ||
        !map_rows(&maps[4], dx ? dx : dz_out, sh.tokens, d, k, 32, pw) ||
        !map_rows(&maps[5], dz_out ? dz_out : dx, sh.tokens, d, k, 32, pw))
        return HCW_ERR_CUDA;
    if (dzpair && !map_rows(&maps[5], dzpair, sh.tokens, d, k, 128)) return HCW_ERR_CUDA;
    L.layer[0] = {sh.s, k, nullptr, nullptr, nullptr, dx != nullptr, mprev, dz_out != nullptr};
    L.layer[0].pair_rows = dzpair != nullptr;
    row_unit_params(L.p, sh, BN, dzpair ? flags & ~HCW_CAUSAL : flags, true);
    L.p.flags = flags & HCW_RESIDUAL;
    L.n_layers = 1;
    const int sms = sm_count();
    const int grid = L.p.n_units < sms ? L.p.n_units : sms;
    return launched(launch_tc(MODE_DX, BN, L, grid, st), 1);
}

// dW: token-contracted, split over token blocks, fixed-order reduction; dbias
// by a deterministic two-pass column sum.  wws: weight workspace.
int dw_bf16(const Shape& sh, const void* x, const void* dz, unsigned flags, float* dWs,
            float* dWn, float* dbias, uint8_t* wws, cudaStream_t st) {
    const int d = sh.d, BN = pick_bn(d), k = 1 << sh.s;
    const WsLayout lay = ws_layout(sh.tokens, d, HCW_BF16, flags);
    const WPlan w = plan_dw(sh.tokens, d, flags);
    TcLaunch<1> L;
    memset(&L, 0, sizeof(L));
    CUtensorMap* maps = L.maps[0];
    float* part = reinterpret_cast<float*>(wws);
    if (!map_rows_blocks(&maps[0], dz, sh.tokens, d, k, 64, 2) ||
        !map_rows_blocks(&maps[1], x, sh.tokens, d, k, 64, BN / 64) ||
        !map_f32_patches(&maps[3], w.splits_max > 1 ? (const void*)part : (const void*)dWs,
                         w.splits_max > 1 ? 2ll * w.splits_max * d : d, d) ||
        !map_f32_patches(&maps[4], dWs, d, d) || !map_f32_patches(&maps[5], dWn, d, d))
        return HCW_ERR_CUDA;
    maps[2] = maps[1];   // unused by the weight gradient
    L.layer[0] = {sh.s, k, nullptr, nullptr, nullptr, false, nullptr, false};
    TcParams& p = L.p;
    p.d = d;
    p.Mh = (int)(sh.tokens / 2);
    p.n_nt = w.n_nt;
    p.n_ot = w.n_ot;
    p.qb = w.qb;
    p.nkb_self = w.nkb_self;
    p.nkb_nbr = w.nkb_nbr;
    p.kb_per_unit = w.kb_per_unit;
    p.splits_self = w.splits_self;
    p.splits_nbr = w.splits_nbr;
    p.splits_max = w.splits_max;
    p.causal = (flags & HCW_CAUSAL) ? 1 : 0;
    p.n_units = w.units;
    p.timeout_ns = g_timeout_ns;
    L.n_layers = 1;
    const int sms = sm_count();
    const int grid = p.n_units < sms ? p.n_units : sms;
    int rc = launched(launch_tc(MODE_DW, BN, L, grid, st), 1);
    if (rc) return rc;
    if (w.splits_max > 1) {
        rc = launched(launch_splitk_reduce(part, w.splits_max, w.splits_self,
                                           w.splits_nbr, d, dWs, dWn, st),
                      1);
        if (rc) return rc;
    }
    if (dbias)
        return launched(launch_colsum_bf16(static_cast<const __nv_bfloat16*>(dz), sh.tokens, d,
                                           reinterpret_cast<float*>(wws + lay.col_off), dbias,
                                           st),
                        2);
    return HCW_OK;
}

// dW[o][k] = sum_t a[t][o] x[t][k]: the self part of the weight gradient alone
// (dW_self with a = dz; for a shift layer also dW_nbr, with a = the readers' dz).
int dw_self_bf16(const Shape& sh, const void* x, const void* a, unsigned flags, float* dW,
                 uint8_t* wws, cudaStream_t st) {
    const int d = sh.d, BN = pick_bn(d), k = 1 << sh.s;
    const WPlan w = plan_dw(sh.tokens, d, flags);
    TcLaunch<1> L;
    memset(&L, 0, sizeof(L));
    CUtensorMap* maps = L.maps[0];
    float* part = reinterpret_cast<float*>(wws);
    if (!map_rows_blocks(&maps[0], a, sh.tokens, d, k, 64, 2) ||
        !map_rows_blocks(&maps[1], x, sh.tokens, d, k, 64, BN / 64) ||
        !map_f32_patches(&maps[3], w.splits_max > 1 ? (const void*)part : (const void*)dW,
                         w.splits_max > 1 ? 2ll * w.splits_max * d : d, d) ||
        !map_f32_patches(&maps[4], dW, d, d))
        return HCW_ERR_CUDA;
    maps[2] = maps[1];   // unused
    maps[5] = maps[4];   // unused: no partner part
    L.layer[0] = {sh.s, k, nullptr, nullptr, nullptr, false, nullptr, false};
    TcParams& p = L.p;
    p.d = d;
    p.Mh = (int)(sh.tokens / 2);
    p.n_nt = w.n_nt;
    p.n_ot = w.n_ot;
    p.qb = w.qb;
    p.nkb_self = w.nkb_self;
    p.nkb_nbr = w.nkb_nbr;
    p.kb_per_unit = w.kb_per_unit;
    p.splits_self = w.splits_self;   // the plan's split of the self part: fits the partials
    p.splits_nbr = 0;
    p.splits_max = w.splits_max;
    p.causal = 0;
    p.n_units = w.n_ot * w.n_nt * w.splits_self;
    p.timeout_ns = g_timeout_ns;
    L.n_layers = 1;
    const int sms = sm_count();
    const int grid = p.n_units < sms ? p.n_units : sms;
    int rc = launched(launch_tc(MODE_DW, BN, L, grid, st), 1);
    if (rc) return rc;
    if (w.splits_self > 1)
        rc = launched(launch_splitk_reduce(part, w.splits_max, w.splits_self, 0, d, dW, dW, st), 1);
    return rc;
}

int fwd_f32(const Shape& sh, const void* x, const void* Ws, const void* Wn, const float* bias,
            unsigned flags, void* y, void* z, uint32_t* mask, cudaStream_t st) {
    return launched(launch_f32_fwd(static_cast<const float*>(x), static_cast<const float*>(Ws),
                                   static_cast<const float*>(Wn), bias, sh.s, sh.B, sh.n, sh.d,
                                   flags, static_cast<float*>(y), static_cast<float*>(z), mask,
                                   st),
                    1);
}

int dx_f32(const Shape& sh, const void* dz, const void* dy, const void* Ws, const void* Wn,
           unsigned flags, void* dx, cudaStream_t st) {
    return launched(launch_f32_dx(static_cast<const float*>(dz), static_cast<const float*>(dy),
                                  static_cast<const float*>(Ws), static_cast<const float*>(Wn),
                                  sh.s, sh.B, sh.n, sh.d, flags, static_cast<float*>(dx), st),
                    1);
}

int dw_f32(const Shape& sh, const void* x, const void* dz, unsigned flags, float* dWs,
           float* dWn, float* dbias, uint8_t* wws, cudaStream_t st) {
    const WsLayout lay = ws_layout(sh.tokens, sh.d, HCW_F32, flags);
    int rc = launched(launch_f32_dw(static_cast<const float*>(x), static_cast<const float*>(dz),
                                    sh.s, sh.B, sh.n, sh.d, flags, dWs, dWn, st),
                      1);
    if (rc || !dbias) return rc;
    return launched(launch_colsum_f32(static_cast<const float*>(dz), sh.tokens, sh.d,
                                      reinterpret_cast<float*>(wws + lay.col_off), dbias, st),
                    2);
}

int layer_fwd_impl(const Shape& sh, int dtype, const void* x, const void* Ws, const void* Wn,
                   const float* bias, unsigned flags, void* y, void* z, cudaStream_t st,
                   uint32_t* mask = nullptr) {
    if (sh.tokens == 0) return HCW_OK;
    return dtype == HCW_BF16 ? fwd_bf16(sh, x, Ws, Wn, bias, flags, y, z, mask, st)
                             : fwd_f32(sh, x, Ws, Wn, bias, flags, y, z, mask, st);
}

int zero_weight_grads(const Shape& sh, float* dWs, float* dWn, float* dbias, cudaStream_t st) {
    // empty batch: the sums over no tokens are zero
    const size_t wbytes = (size_t)sh.d * sh.d * sizeof(float);
    cudaError_t e = cudaMemsetAsync(dWs, 0, wbytes, st);
    if (e == cudaSuccess) e = cudaMemsetAsync(dWn, 0, wbytes, st);
    if (e == cudaSuccess && dbias) e = cudaMemsetAsync(dbias, 0, sh.d * sizeof(float), st);
    return cuda_status(e);
}

int layer_dx_impl(const Shape& sh, int dtype, const void* dz, const void* dy, const void* Ws,
                  const void* Wn, unsigned flags, void* dx, cudaStream_t st) {
    if (sh.tokens == 0) return HCW_OK;
    return dtype == HCW_BF16 ? dx_bf16(sh, dz, dy, Ws, Wn, flags, dx, st)
                             : dx_f32(sh, dz, dy, Ws, Wn, flags, dx, st);
}

int layer_dw_impl(const Shape& sh, int dtype, const void* x, const void* dz, unsigned flags,
                  float* dWs, float* dWn, float* dbias, uint8_t* wws, cudaStream_t st) {
    if (sh.tokens == 0) return zero_weight_grads(sh, dWs, dWn, dbias, st);
    return dtype == HCW_BF16 ? dw_bf16(sh, x, dz, flags, dWs, dWn, dbias, wws, st)
                             : dw_f32(sh, x, dz, flags, dWs, dWn, dbias, wws, st);
}

int layer_bwd_impl(const Shape& sh, int dtype, const void* x, const void* z, const void* dy,
                   const void* Ws, const void* Wn, unsigned flags, void* dx, float* dWs,
                   float* dWn, float* dbias, void* ws, cudaStream_t st) {
    if (sh.tokens == 0) return zero_weight_grads(sh, dWs, dWn, dbias, st);
    const WsLayout lay = ws_layout(sh.tokens, sh.d, dtype, flags);
    uint8_t* wsb = static_cast<uint8_t*>(ws);
    const void* dz = dy;
    int rc;
    if (flags & HCW_ACT_RELU) {
        void* dzw = wsb + lay.dz_off;
        const size_t count = (size_t)sh.tokens * sh.d;
        rc = launched(dtype == HCW_BF16
                          ? launch_relu_grad_bf16(static_cast<const __nv_bfloat16*>(dy),
                                                  static_cast<const __nv_bfloat16*>(z),
                                                  static_cast<__nv_bfloat16*>(dzw), count, st)
                          : launch_relu_grad_f32(static_cast<const float*>(dy),
                                                 static_cast<const float*>(z),
                                                 static_cast<float*>(dzw), count, st),
                      1);
        if (rc) return rc;
        dz = dzw;
    }
    rc = layer_dx_impl(sh, dtype, dz, dy, Ws, Wn, flags, dx, st);
    if (rc) return rc;
    return layer_dw_impl(sh, dtype, x, dz, flags, dWs, dWn, dbias, wsb + lay.w_off, st);
}

// ------------------------------------------------------------ stack backward
// Workspaces of the stack backward.
//   input gradients, bf16: the output gradient g of every layer when both the
//   ReLU and the residual are on (the residual term of that layer's input
//   gradient; otherwise g is dz itself or dy), then the completion counters
//   of the stacked launch.  fp32: two g buffers used in turn.
//   weight gradients, bf16: the unit counter of the batched launch, then the
//   single-layer weight-gradient workspace (used when the layers are too few
//   to fill the GPU and run one by one).  fp32: the single-layer workspace.
//   hcw_stack_bwd: every layer's dz, then both of the above.
// bf16: bytes in front of the counters.  The streaming kernels keep every
// layer's g there (ReLU with the residual); the resident kernels use the first
// 2 act_bytes as one fp32 [tokens][d] buffer (g where rows change CTA, and
// between launches of more than 16 layers).
size_t stack_g_region(const Shape& sh, unsigned flags, int L) {
    const size_t a = align256(sh.act_bytes);
    const bool keep_g = (flags & HCW_ACT_RELU) && (flags & HCW_RESIDUAL);
    // two g buffers used in turn (see stack_data_bf16)
    size_t r = keep_g ? 2 * a : 0;
    // schedules with shift layers that the stacked launches cannot take run
    // layer by layer: two g buffers in turn and the readers' dz of a shift layer
    if (r < 3 * a) r = 3 * a;
    return r;
}

size_t stack_data_ws(const Shape& sh, int dtype, unsigned flags, int L) {
    const size_t a = align256(sh.act_bytes);
    if (dtype == HCW_BF16) return stack_g_region(sh, flags, L) + stack_counter_bytes(sh.tokens, L);
    return 2 * a;
}

// True when `cnt` layers' whole-range weight-gradient units (one per output
// tile) would leave most SMs idle: their launch then splits the token range
// of every layer (split_dw_ws).
bool split_dw_layers(const Shape& sh, unsigned flags, int cnt) {
    const WPlan w = plan_dw(sh.tokens, sh.d, flags);
    return cnt * w.n_ot * w.n_nt * 2 < sm_count();
}

// Workspace of the split launch over `cnt` layers: the fp32 partials
// [cnt][2][splits][d][d] and the dbias partials [cnt][splits of the self
// part][d] (when the token range is split).
size_t split_dw_ws(const Shape& sh, unsigned flags, int cnt) {
    const WPlan w = plan_dw(sh.tokens, sh.d, flags, cnt);
    const size_t dd = (size_t)sh.d * sh.d * 4;
    const size_t part = w.splits_max > 1 ? align256((size_t)cnt * 2 * w.splits_max * dd) : 0;
    const size_t bpart =
        w.splits_self > 1 ? align256((size_t)cnt * w.splits_self * sh.d * 4) : 0;
    return part + bpart;
}

// bf16: [unit counter (256 B)][weight-gradient workspace][the readers' dz of a
// shift layer (one activation buffer)], or [unit counter][the split launch's
// partials] when that is larger
size_t stack_weight_ws(const Shape& sh, int dtype, unsigned flags, int L) {
    const WsLayout w = ws_layout(sh.tokens, sh.d, dtype, flags);
    if (dtype != HCW_BF16) return w.w_bytes;
    size_t body = align256(w.w_bytes) + align256(sh.act_bytes);
    // the launches of kMaxStackLayers layers and the last, shorter one
    const int counts[2] = {L < kMaxStackLayers ? L : kMaxStackLayers, L % kMaxStackLayers};
    for (int cnt : counts)
        if (cnt > 0 && split_dw_layers(sh, flags, cnt)) {
            const size_t need = split_dw_ws(sh, flags, cnt);
            if (need > body) body = need;
        }
    return 256 + body;
}

size_t stack_dz_bytes(const Shape& sh, int L) { return align256((size_t)L * sh.act_bytes); }


struct StackData {
    const void* masks;
    const void* dy;
    const uint8_t* Ws;
    const uint8_t* Wn;
    Sched sc;
    int L;
    unsigned flags;
    void* dx;
    uint8_t* dz;   // [L][tokens][d], layer stride act_bytes
    uint8_t* ws;
};

struct StackWeight {
    const void* x;
    const void* acts;
    const uint8_t* dz;
    Sched sc;
    int L;
    unsigned flags;
    float* dWs;
    float* dWn;
    float* dbias;
    uint8_t* ws;
    // the fused forward / input-gradient launch just issued on the stream, or
    // null: its completion counters, where row 2 L - 2 - l counts dz_l.  A
    // batched launch on SM pairs then starts as its programmatic dependent
    // and waits on those counters instead of the launch's end.
    const int* fdx_counters = nullptr;
};

// bf16 input gradients on the resident kernels: one launch per run of <= 16
// layers, top down.  The first launch starts from dy; a run that stops above
// layer 0 leaves g (fp32) in the workspace for the next one.
int stack_data_resident(const Shape& sh, const StackData& a, cudaStream_t st) {
    const int d = sh.d, L = a.L, N = d >= 256 ? d / 2 : d;
    const bool relu = (a.flags & HCW_ACT_RELU) != 0;
    const size_t ab = sh.act_bytes, wb = (size_t)d * d * 2;
    const size_t mb = mask_bytes(sh);
    float* gs = reinterpret_cast<float*>(a.ws);
    auto dz = [&](int l) -> void* { return a.dz + (size_t)l * ab; };
    auto mask = [&](int l) {
        return reinterpret_cast<const uint32_t*>(static_cast<const uint8_t*>(a.masks) +
                                                 (size_t)l * mb);
    };
    static thread_local ResLaunch R;
    for (int top = L - 1; top >= 0; top -= kMaxStackLayers) {
        const int cnt = top + 1 < kMaxStackLayers ? top + 1 : kMaxStackLayers;
        memset(&R, 0, sizeof(R));
        for (int i = 0; i < cnt; ++i) {
            const int l = top - i;
            const int s = a.sc.dim(sh, l);
            if (!map_weight_blocks(&R.wmap[i][0], a.Ws + l * wb, d, N / 128) ||
                !map_weight_blocks(&R.wmap[i][1], a.Wn + l * wb, d, N / 128))
                return HCW_ERR_CUDA;
            ResLayer& y = R.layer[i];
            y.s = s;
            if (l == 0) {
                y.out_kind = RES_DX;
                y.out = a.dx;
            } else if (i == cnt - 1) {
                y.out_kind = RES_G;
                y.out = gs;
            } else {
                y.out_kind = RES_DZ;
                y.out = dz(l - 1);
                y.mprev = relu ? mask(l - 1) : nullptr;
            }
            // the stand-in for RES_G is never used (fp32 leaves row by row)
            const void* ob = y.out_kind == RES_G ? a.dx : y.out;
            if (!map_rows16(&R.imap[i], ob, sh.tokens, d, 1, 64))
                return HCW_ERR_CUDA;
        }
        R.in = top == L - 1 ? a.dy : static_cast<const void*>(gs);
        R.in_f32 = top == L - 1 ? 0 : 1;
        R.in_mask = relu ? mask(top) : nullptr;
        R.in_dz = static_cast<__nv_bfloat16*>(dz(top));
        R.gscratch = gs;
        R.n_layers = cnt;
        R.d = d;
        R.n = sh.n;
        R.tokens = (int)sh.tokens;
        R.flags = a.flags;
        R.timeout_ns = g_timeout_ns;
        const int rc = launched(launch_res(MODE_DX, R, st), 1);
        if (rc) return rc;
    }
    return HCW_OK;
}

// bf16 input gradients: the ReLU gradient of the top layer, then one stacked
// launch per run of <= 16 layers, top down, whose kernel also applies the
// ReLU gradient of the layer below.
// bf16 input gradients of a schedule with shift layers that the stacked
// launches cannot take (n < 128, or not whole 256-token row-block pairs, or
// the resident kernels chosen), layer by layer: dz_l
// from the ReLU gradient (or a copy of g), then the layer's input gradient --
// a shift layer with the readers' dz, S_{-k} dz, as its row-aligned partner.
int stack_data_layers_bf16(const Shape& sh, const StackData& a, cudaStream_t st) {
    const int d = sh.d, L = a.L;
    const bool relu = (a.flags & HCW_ACT_RELU) != 0;
    const size_t ab = sh.act_bytes, a256 = align256(ab), wb = (size_t)d * d * 2;
    const size_t mb = mask_bytes(sh);
    void* gbuf[2] = {a.ws, a.ws + a256};
    void* v = a.ws + 2 * a256;
    const void* g = a.dy;
    int rc;
    for (int l = L - 1; l >= 0; --l) {
        void* dzl = a.dz + (size_t)l * ab;
        if (relu)
            rc = launched(launch_relu_grad_mask_bf16(
                              static_cast<const __nv_bfloat16*>(g),
                              reinterpret_cast<const uint32_t*>(static_cast<const uint8_t*>(a.masks) +
                                                                (size_t)l * mb),
                              static_cast<__nv_bfloat16*>(dzl), sh.tokens, d, st),
                          1);
        else
            rc = cuda_status(cudaMemcpyAsync(dzl, g, ab, cudaMemcpyDeviceToDevice, st));
        if (rc) return rc;
        void* out = l == 0 ? a.dx : gbuf[l & 1];
        const int s = a.sc.dim(sh, l);
        Shape shl = sh;
        if (s >= 0) {
            shl.s = s;
            rc = dx_bf16(shl, dzl, g, a.Ws + l * wb, a.Wn + l * wb, a.flags, out, st);
        } else {
            rc = launched(launch_shift_rows_bf16(static_cast<const __nv_bfloat16*>(dzl),
                                                 static_cast<__nv_bfloat16*>(v), sh.tokens, sh.n,
                                                 d, s, st),
                          1);
            if (rc) return rc;
            shl.s = shift_group_dim(sh);
            rc = dx_bf16(shl, dzl, g, a.Ws + l * wb, a.Wn + l * wb, a.flags, out, st, nullptr,
                         nullptr, v);
        }
        if (rc) return rc;
        g = out;
    }
    return HCW_OK;
}

int stack_data_bf16(const Shape& sh, const StackData& a, cudaStream_t st) {
    if (a.sc.has_shift(a.L) && (!shift_stackable(sh) || use_resident(sh)))
        return stack_data_layers_bf16(sh, a, st);
    if (use_resident(sh)) return stack_data_resident(sh, a, st);
    const int d = sh.d, BN = pick_bn(d), L = a.L;
    const bool relu = (a.flags & HCW_ACT_RELU) != 0;
    const bool resid = (a.flags & HCW_RESIDUAL) != 0;
    const bool keep_g = relu && resid;
    const size_t ab = sh.act_bytes, a256 = align256(ab), wb = (size_t)d * d * 2;
    const size_t mb = mask_bytes(sh);
    auto dz = [&](int l) -> void* { return a.dz + (size_t)l * ab; };
    // Output gradients g in two buffers used in turn: layer l's units write
    // g_{l-1} over g_{l+1} only for rows whose dz_l chunks are complete, and the
    // layer-(l+1) units that wrote those chunks had read their g_{l+1} rows (the
    // residual term) before storing their outputs.
    auto gbuf = [&](int l) -> void* { return a.ws + (size_t)(l & 1) * a256; };
    auto mask = [&](int l) {
        return reinterpret_cast<const uint32_t*>(static_cast<const uint8_t*>(a.masks) +
                                                 (size_t)l * mb);
    };
    // output gradient g_l of layer l (the residual term of its input gradient)
    auto g = [&](int l) -> const void* {
        if (l == L - 1) return a.dy;
        return keep_g ? gbuf(l) : dz(l);
    };
    int rc;
    // the top layer's dz = dy * act'(z) is written by the first launch itself
    int* counters = reinterpret_cast<int*>(a.ws + stack_g_region(sh, a.flags, L));
    const int n_chunks = (int)((sh.tokens + 127) / 128);
    const bool pair = use_pairs(sh);
    const int pw = epi_patch_cols(BN);
    static thread_local TcLaunch<kMaxStackLayers> T;
    for (int top = L - 1; top >= 0; top -= kMaxStackLayers) {
        const int cnt = top + 1 < kMaxStackLayers ? top + 1 : kMaxStackLayers;
        memset(&T, 0, sizeof(T));
        for (int i = 0; i < cnt; ++i) {
            const int l = top - i;
            const int sl = a.sc.dim(sh, l);
            // a shift layer: rows in runs of 128 positions, dz as positions
            const int s = sl >= 0 ? sl : kShiftStackDim;
            const int k = 1 << s;
            // stores: g_{l-1} (map 4) and dz_{l-1} (map 5); at l = 0 the stack's dx
            void* out = l == 0 ? a.dx : (relu ? (resid ? gbuf(l - 1) : nullptr) : dz(l - 1));
            void* dzo = (l > 0 && relu) ? dz(l - 1) : nullptr;
            CUtensorMap* m = T.maps[i];
            const void* res = resid ? g(l) : dz(l);
            if (!map_rows(&m[0], dz(l), sh.tokens, d, k, 128) ||
                !map_weight_blocks(&m[1], a.Ws + l * wb, d, (pair ? BN / 2 : BN) / 64) ||
                !map_weight_blocks(&m[2], a.Wn + l * wb, d, (pair ? BN / 2 : BN) / 64) ||
                !map_rows(&m[3], res, sh.tokens, d, k, 32, pw) ||
                !map_rows(&m[4], out ? out : dzo, sh.tokens, d, k, 32, pw) ||
                !map_rows(&m[5], dzo ? dzo : out, sh.tokens, d, k, 32, pw))
                return HCW_ERR_CUDA;
            if (sl < 0 && !map_positions(&m[0], dz(l), sh.tokens, sh.n, d, 128))
                return HCW_ERR_CUDA;
            T.layer[i] = {s, k, nullptr, nullptr, nullptr, out != nullptr,
                          dzo ? mask(l - 1) : nullptr, dzo != nullptr};
            T.layer[i].shift = sl < 0 ? -sl : 0;
            // the g buffers written by this launch (not dy, not a previous launch's)
            if (keep_g && i > 0)
                T.layer[i].g_discard = static_cast<const __nv_bfloat16*>(res);
        }
        row_unit_params(T.p, sh, BN, a.flags, true);
        if (pair) pair_units(T.p);
        T.p.seq_n = sh.n;
        T.p.flags = a.flags & HCW_RESIDUAL;
        T.n_layers = cnt;
        T.counters = counters;
        T.n_chunks = n_chunks;
        T.tokens = (int)sh.tokens;
        T.sched = counters + (size_t)cnt * n_chunks;
        if (top == L - 1) {
            T.top_dy = static_cast<const __nv_bfloat16*>(a.dy);
            T.top_mask = relu ? mask(L - 1) : nullptr;
            T.top_dz = static_cast<__nv_bfloat16*>(dz(L - 1));
            T.in_counters = T.sched + 1;
        }
        // g apart from dz: with the ReLU and the residual, the kernel publishes
        // each patch's dz before it stores g
        if (keep_g) T.g_counters = T.sched + 1 + n_chunks;
        if (cudaMemsetAsync(counters, 0,
                            ((size_t)(keep_g ? 2 : 1) * cnt * n_chunks + 1 + n_chunks) *
                                sizeof(int),
                            st) != cudaSuccess)
            return HCW_ERR_CUDA;
        rc = launch_rows(MODE_DX, BN, T, cnt, pair, st);
        if (rc) return rc;
    }
    return HCW_OK;
}

// The weight gradients of layers l0 .. l0 + cnt - 1 when each has few output
// tiles (small d): one launch whose units split every layer's token range
// (units of one size over all the layers, claimed dynamically; the self
// part's units also sum their dz columns, the dbias of their split), then
// one reduction launch over all the layers' partials -- two launches in place
// of four per layer.  Hypercube layers only (a shift layer takes the launches
// of stack_weight_bf16).
int split_dw_launch(const Shape& sh, const StackWeight& a, int l0, int cnt, uint8_t* wws,
                    int* sched, cudaStream_t st) {
    const int d = sh.d, BN = pick_bn(d);
    const size_t ab = sh.act_bytes, dd = (size_t)d * d;
    const WPlan w = plan_dw(sh.tokens, d, a.flags, cnt);
    const bool split = w.splits_max > 1;
    const size_t part_floats = (size_t)2 * w.splits_max * dd;   // one layer's partials
    float* part = reinterpret_cast<float*>(wws);
    float* bpart = reinterpret_cast<float*>(wws + (split ? align256(cnt * part_floats * 4) : 0));
    static thread_local TcLaunch<kMaxStackLayers> T;
    memset(&T, 0, sizeof(T));
    for (int i = 0; i < cnt; ++i) {
        const int l = l0 + i;
        const int s = a.sc.dim(sh, l);
        if (s < 0) return HCW_ERR_UNSUPPORTED;
        const int k = 1 << s;
        const void* x = l == 0 ? a.x : static_cast<const uint8_t*>(a.acts) + (size_t)(l - 1) * ab;
        float* gs = a.dWs + (size_t)l * dd;
        CUtensorMap* m = T.maps[i];
        if (!map_rows_blocks(&m[0], a.dz + (size_t)l * ab, sh.tokens, d, k, 64, 2) ||
            !map_rows_blocks(&m[1], x, sh.tokens, d, k, 64, BN / 64) ||
            !map_f32_patches(&m[3], split ? (const void*)(part + i * part_floats) : (const void*)gs,
                             split ? 2ll * w.splits_max * d : d, d) ||
            !map_f32_patches(&m[4], gs, d, d) ||
            !map_f32_patches(&m[5], a.dWn + (size_t)l * dd, d, d))
            return HCW_ERR_CUDA;
        m[2] = m[1];   // unused by the weight gradient
        T.layer[i] = {s, k, nullptr, nullptr, nullptr, false, nullptr, false};
        // the self part's units sum dz's columns on the way (helper warps):
        // dbias itself for units over the whole token range, else the split's
        // partial sums
        if (a.dbias)
            T.layer[i].colsum = w.splits_self == 1 ? a.dbias + (size_t)l * d
                                                   : bpart + (size_t)i * w.splits_self * d;
    }
    TcParams& p = T.p;
    p.d = d;
    p.Mh = (int)(sh.tokens / 2);
    p.n_nt = w.n_nt;
    p.n_ot = w.n_ot;
    p.qb = w.qb;
    p.nkb_self = w.nkb_self;
    p.nkb_nbr = w.nkb_nbr;
    p.kb_per_unit = w.kb_per_unit;
    p.splits_self = w.splits_self;
    p.splits_nbr = w.splits_nbr;
    p.splits_max = w.splits_max;
    p.causal = (a.flags & HCW_CAUSAL) ? 1 : 0;
    p.n_units = w.units;
    p.seq_n = sh.n;
    p.timeout_ns = g_timeout_ns;
    T.n_layers = cnt;
    T.sched = sched;
    if (cudaMemsetAsync(sched, 0, sizeof(int), st) != cudaSuccess) return HCW_ERR_CUDA;
    const int sms = sm_count(), total = w.units * cnt;
    int rc = launched(launch_tc_stack(MODE_DW, BN, T, total < sms ? total : sms, st), 1);
    if (rc) return rc;
    if (split)
        rc = launched(launch_splitk_reduce(part, w.splits_max, w.splits_self, w.splits_nbr, d,
                                           a.dWs + (size_t)l0 * dd, a.dWn + (size_t)l0 * dd, st,
                                           cnt, part_floats, dd, a.dbias ? bpart : nullptr,
                                           a.dbias ? a.dbias + (size_t)l0 * d : nullptr),
                      1);
    return rc;
}

// bf16 weight gradients: runs of up to 16 independent layers in one launch
// (whole token range per tile, units handed out longest first; the kernel
// also sums dz's columns into dbias), or, when their tiles cannot fill the
// GPU, one launch over token splits of every layer (split_dw_launch); a
// schedule with shift layers that cannot take the batched launch runs layer
// by layer.
int stack_weight_bf16(const Shape& sh, const StackWeight& a, cudaStream_t st) {
    const int d = sh.d, BN = pick_bn(d), L = a.L;
    const size_t ab = sh.act_bytes;
    const WsLayout wl = ws_layout(sh.tokens, d, HCW_BF16, a.flags);
    int* sched = reinterpret_cast<int*>(a.ws);
    // Shift layers join the batched launch on SM pairs (their partner rows come
    // from a (position, sample) view, 64 positions of one sample per stage,
    // hence n >= 128); otherwise every layer runs on its own.
    const WPlan wp = plan_dw(sh.tokens, d, a.flags);
    const bool shift_batched = sh.n >= 128 && BN >= 128 && wp.n_ot % 2 == 0 && [&] {
        for (int l0 = 0; l0 < L; l0 += kMaxStackLayers) {
            const int cnt = L - l0 < kMaxStackLayers ? L - l0 : kMaxStackLayers;
            if (5 * cnt * wp.n_ot * wp.n_nt < 3 * sm_count()) return false;
        }
        return true;
    }();
    if (a.sc.has_shift(L) && !shift_batched) {
        // layer by layer; a shift layer's dW_nbr = sum_t (S_{-k} dz)_t^T x_t, the
        // self-part GEMM of the readers' dz against the layer input
        uint8_t* wws = a.ws + 256;
        void* v = a.ws + 256 + align256(wl.w_bytes);
        for (int l = 0; l < L; ++l) {
            const void* xl =
                l == 0 ? a.x : static_cast<const uint8_t*>(a.acts) + (size_t)(l - 1) * ab;
            const void* dzl = a.dz + (size_t)l * ab;
            float* gs = a.dWs + (size_t)l * d * d;
            float* gn = a.dWn + (size_t)l * d * d;
            float* gb = a.dbias ? a.dbias + (size_t)l * d : nullptr;
            const int s = a.sc.dim(sh, l);
            Shape shl = sh;
            int rc;
            if (s >= 0) {
                shl.s = s;
                rc = dw_bf16(shl, xl, dzl, a.flags, gs, gn, gb, wws, st);
            } else {
                shl.s = shift_group_dim(sh);
                rc = dw_self_bf16(shl, xl, dzl, a.flags, gs, wws, st);
                if (!rc)
                    rc = launched(launch_shift_rows_bf16(static_cast<const __nv_bfloat16*>(dzl),
                                                         static_cast<__nv_bfloat16*>(v),
                                                         sh.tokens, sh.n, d, s, st),
                                  1);
                if (!rc) rc = dw_self_bf16(shl, xl, v, a.flags, gn, wws, st);
                if (!rc && gb)
                    rc = launched(launch_colsum_bf16(static_cast<const __nv_bfloat16*>(dzl),
                                                     sh.tokens, d,
                                                     reinterpret_cast<float*>(wws + wl.col_off),
                                                     gb, st),
                                  2);
            }
            if (rc) return rc;
        }
        return HCW_OK;
    }
    uint8_t* wws = a.ws + 256;
    auto dz = [&](int l) -> const void* { return a.dz + (size_t)l * ab; };
    auto act = [&](int l) -> const void* {
        return l == 0 ? a.x : static_cast<const uint8_t*>(a.acts) + (size_t)(l - 1) * ab;
    };
    const WPlan w1 = plan_dw(sh.tokens, d, a.flags);
    const int tiles = w1.n_ot * w1.n_nt;
    const int sms = sm_count();
    static thread_local TcLaunch<kMaxStackLayers> T;
    int rc;
    for (int l0 = 0; l0 < L; l0 += kMaxStackLayers) {
        const int cnt = L - l0 < kMaxStackLayers ? L - l0 : kMaxStackLayers;
        if (split_dw_layers(sh, a.flags, cnt)) {
            rc = split_dw_launch(sh, a, l0, cnt, wws, sched, st);
            if (rc) return rc;
            continue;
        }
        memset(&T, 0, sizeof(T));
        for (int i = 0; i < cnt; ++i) {
            const int l = l0 + i;
            const int sl = a.sc.dim(sh, l);
            // a shift layer's rows are grouped as a hypercube view with k = 64
            const int s = sl >= 0 ? sl : 6;
            const int k = 1 << s;
            CUtensorMap* m = T.maps[i];
            if (!map_rows_blocks(&m[0], dz(l), sh.tokens, d, k, 64, 2) ||
                !map_rows_blocks(&m[1], act(l), sh.tokens, d, k, 64, BN / 64) ||
                !map_f32_patches(&m[4], a.dWs + (size_t)l * d * d, d, d) ||
                !map_f32_patches(&m[5], a.dWn + (size_t)l * d * d, d, d))
                return HCW_ERR_CUDA;
            m[2] = m[1];
            m[3] = m[4];
            if (sl < 0 && !map_positions_blocks(&m[2], act(l), sh.tokens, sh.n, d, BN / 128))
                return HCW_ERR_CUDA;
            T.layer[i] = {s, k, nullptr, nullptr, nullptr, false, nullptr, false,
                          a.dbias ? a.dbias + (size_t)l * d : nullptr,
                          a.dWs + (size_t)l * d * d, a.dWn + (size_t)l * d * d};
            T.layer[i].shift = sl < 0 ? -sl : 0;
        }
        // One unit per (layer, output tile) accumulating the self and the partner
        // part together reads each dz and input block once (the separate parts
        // read the receiving rows twice and leave a long tail of short units);
        // used when those units alone fill most of the GPU.  On pairs of SMs
        // (256-row tiles, cta_group::2) each SM takes in a third less per stage.
        const bool fused = 5 * cnt * tiles >= 3 * sms;
        const bool paired = fused && BN >= 128 && w1.n_ot % 2 == 0;
        if (paired)
            for (int i = 0; i < cnt; ++i) {
                const int l = l0 + i;
                const int k = 1 << T.layer[i].s;
                if (!map_rows_blocks(&T.maps[i][1], act(l), sh.tokens, d, k, 64, BN / 128))
                    return HCW_ERR_CUDA;
            }
        TcParams& p = T.p;
        memset(&p, 0, sizeof(p));
        p.d = d;
        p.Mh = (int)(sh.tokens / 2);
        p.n_nt = w1.n_nt;
        p.n_ot = w1.n_ot;
        p.qb = w1.qb;
        p.nkb_self = w1.nkb_self;
        p.nkb_nbr = w1.nkb_nbr;
        p.kb_per_unit = w1.nkb_self > w1.nkb_nbr ? w1.nkb_self : w1.nkb_nbr;
        p.splits_self = 1;
        p.splits_nbr = 1;
        p.splits_max = 1;
        p.causal = (a.flags & HCW_CAUSAL) ? 1 : 0;
        p.n_units = fused ? tiles : tiles * 2;
        p.seq_n = sh.n;
        p.timeout_ns = g_timeout_ns;
        T.n_layers = cnt;
        T.sched = sched;
        // the pair launch hands out its units statically (no unit counter); right
        // behind the fused launch it starts early, on the SMs that launch leaves
        const bool early = paired && a.fdx_counters != nullptr && L <= kMaxStackLayers;
        if (early) {
            T.dep_counters = a.fdx_counters;
            T.n_chunks = (int)((sh.tokens + 127) / 128);
            T.tokens = (int)sh.tokens;
            for (int i = 0; i < cnt; ++i) T.layer[i].dep_row = 2 * L - 2 - (l0 + i);
        } else if (cudaMemsetAsync(sched, 0, sizeof(int), st) != cudaSuccess) {
            return HCW_ERR_CUDA;
        }
        const int total = p.n_units * cnt;
        if (paired) {
            // clusters of two CTAs, one 256-row tile per cluster
            const int pairs = total / 2 < sms / 2 ? total / 2 : sms / 2;
            rc = launched(launch_tc_stack(MODE_DWP, BN, T, 2 * pairs, st), 1);
        } else {
            rc = launched(launch_tc_stack(fused ? MODE_DWF : MODE_DW, BN, T,
                                          total < sms ? total : sms, st),
                          1);
        }
        if (rc) return rc;
    }
    return HCW_OK;
}

// fp32 input gradients, layer by layer (the correctness path).
int stack_data_f32(const Shape& sh, const StackData& a, cudaStream_t st) {
    const int d = sh.d, L = a.L;
    const bool relu = (a.flags & HCW_ACT_RELU) != 0;
    const size_t ab = sh.act_bytes, a256 = align256(ab), wb = (size_t)d * d * 4;
    const size_t mb = mask_bytes(sh);
    uint8_t* g[2] = {a.ws, a.ws + a256};
    auto dz = [&](int l) -> void* { return a.dz + (size_t)l * ab; };
    auto mask = [&](int l) {
        return reinterpret_cast<const uint32_t*>(static_cast<const uint8_t*>(a.masks) +
                                                 (size_t)l * mb);
    };
    int rc;
    if (relu) {
        rc = launched(launch_relu_grad_mask_f32(static_cast<const float*>(a.dy), mask(L - 1),
                                                static_cast<float*>(dz(L - 1)), sh.tokens, d, st),
                      1);
    } else {
        rc = cuda_status(cudaMemcpyAsync(dz(L - 1), a.dy, ab, cudaMemcpyDeviceToDevice, st));
    }
    if (rc) return rc;
    const void* cur_g = a.dy;
    for (int l = L - 1; l >= 0; --l) {
        Shape shl = sh;
        shl.s = a.sc.dim(sh, l);
        void* out = l == 0 ? a.dx : (relu ? (void*)g[l & 1] : dz(l - 1));
        rc = layer_dx_impl(shl, HCW_F32, dz(l), cur_g, a.Ws + l * wb, a.Wn + l * wb, a.flags, out,
                           st);
        if (rc) return rc;
        if (l == 0) break;
        if (relu) {
            rc = launched(launch_relu_grad_mask_f32(static_cast<const float*>(out), mask(l - 1),
                                                    static_cast<float*>(dz(l - 1)), sh.tokens, d,
                                                    st),
                          1);
            if (rc) return rc;
        }
        cur_g = out;
    }
    return HCW_OK;
}

// fp32 weight gradients, layer by layer.
int stack_weight_f32(const Shape& sh, const StackWeight& a, cudaStream_t st) {
    const int d = sh.d;
    const size_t ab = sh.act_bytes;
    for (int l = 0; l < a.L; ++l) {
        Shape shl = sh;
        shl.s = a.sc.dim(sh, l);
        const void* in = l == 0 ? a.x : static_cast<const uint8_t*>(a.acts) + (size_t)(l - 1) * ab;
        const int rc = layer_dw_impl(shl, HCW_F32, in, a.dz + (size_t)l * ab, a.flags,
                                     a.dWs + (size_t)l * d * d, a.dWn + (size_t)l * d * d,
                                     a.dbias ? a.dbias + (size_t)l * d : nullptr, a.ws, st);
        if (rc) return rc;
    }
    return HCW_OK;
}

// Argument checks of the two halves (sizes, pointers, alignment, overlaps).
int check_stack_data(const Shape& sh, int dtype, unsigned flags, int L, const void* masks,
                     const void* dy, const void* Ws, const void* Wn, const void* dx,
                     const void* dz, const void* ws, size_t ws_bytes) {
    const bool relu = (flags & HCW_ACT_RELU) != 0;
    if (!dy || !Ws || !Wn || !dx || !dz || (relu && !masks)) return HCW_ERR_INVALID_ARG;
    const void* ptrs[] = {masks, dy, Ws, Wn, dx, dz};
    for (const void* q : ptrs)
        if (q && !aligned16(q)) return HCW_ERR_ALIGNMENT;
    const size_t need = stack_data_ws(sh, dtype, flags, L);
    if (ws_bytes < need || (need && !ws)) return HCW_ERR_WORKSPACE;
    if (ws && !aligned16(ws)) return HCW_ERR_ALIGNMENT;
    const size_t ab = sh.act_bytes, zb = (size_t)L * ab;
    const size_t mbs = relu ? (size_t)L * mask_bytes(sh) : 0;
    const size_t wb = (size_t)L * sh.d * sh.d * elem_size(dtype);
    const void* ins[][2] = {{dy, (const void*)ab}, {masks, (const void*)mbs},
                            {Ws, (const void*)wb}, {Wn, (const void*)wb}};
    for (auto& q : ins) {
        const size_t n = reinterpret_cast<size_t>(q[1]);
        if (overlaps(dx, ab, q[0], n) || overlaps(dz, zb, q[0], n) ||
            overlaps(ws, ws_bytes, q[0], n))
            return HCW_ERR_ALIASING;
    }
    if (overlaps(dx, ab, dz, zb) || overlaps(ws, ws_bytes, dx, ab) || overlaps(ws, ws_bytes, dz, zb))
        return HCW_ERR_ALIASING;
    return HCW_OK;
}

int check_stack_weight(const Shape& sh, int dtype, unsigned flags, int L, const void* x,
                       const void* acts, const void* dz, const float* dWs, const float* dWn,
                       const float* dbias, const void* ws, size_t ws_bytes) {
    if (!x || !dz || !dWs || !dWn || (L > 1 && !acts)) return HCW_ERR_INVALID_ARG;
    const void* ptrs[] = {x, acts, dz, dWs, dWn, dbias};
    for (const void* q : ptrs)
        if (q && !aligned16(q)) return HCW_ERR_ALIGNMENT;
    const size_t need = stack_weight_ws(sh, dtype, flags, L);
    if (ws_bytes < need || (need && !ws)) return HCW_ERR_WORKSPACE;
    if (ws && !aligned16(ws)) return HCW_ERR_ALIGNMENT;
    const size_t ab = sh.act_bytes, gb = (size_t)L * sh.d * sh.d * 4, bb = (size_t)L * sh.d * 4;
    const size_t acts_b = (size_t)(L - 1) * ab;
    const void* outs[][2] = {{dWs, (const void*)gb}, {dWn, (const void*)gb},
                             {dbias, (const void*)bb}, {ws, (const void*)ws_bytes}};
    const void* ins[][2] = {{x, (const void*)ab}, {acts, (const void*)acts_b},
                            {dz, (const void*)((size_t)L * ab)}};
    for (int i = 0; i < 4; ++i) {
        const size_t ni = reinterpret_cast<size_t>(outs[i][1]);
        for (auto& q : ins)
            if (overlaps(outs[i][0], ni, q[0], reinterpret_cast<size_t>(q[1])))
                return HCW_ERR_ALIASING;
        for (int j = i + 1; j < 4; ++j)
            if (overlaps(outs[i][0], ni, outs[j][0], reinterpret_cast<size_t>(outs[j][1])))
                return HCW_ERR_ALIASING;
    }
    return HCW_OK;
}

int zero_weight_grads(int L, int d, float* dWs, float* dWn, float* dbias, cudaStream_t st) {
    const size_t gbytes = (size_t)L * d * d * sizeof(float);
    cudaError_t e = cudaMemsetAsync(dWs, 0, gbytes, st);
    if (e == cudaSuccess) e = cudaMemsetAsync(dWn, 0, gbytes, st);
    if (e == cudaSuccess && dbias) e = cudaMemsetAsync(dbias, 0, (size_t)L * d * 4, st);
    return cuda_status(e);
}

int check_fwd_ptrs(const Shape& sh, int dtype, const void* x, const void* Ws, const void* Wn,
                   const float* bias, void* y, void* z) {
    if (!x || !Ws || !Wn || !y) return HCW_ERR_INVALID_ARG;
    if (!aligned16(x) || !aligned16(Ws) || !aligned16(Wn) || !aligned16(y) ||
        (bias && !aligned16(bias)) || (z && !aligned16(z)))
        return HCW_ERR_ALIGNMENT;
    const size_t wb = (size_t)sh.d * sh.d * elem_size(dtype);
    if (overlaps(y, sh.act_bytes, x, sh.act_bytes) || overlaps(y, sh.act_bytes, Ws, wb) ||
        overlaps(y, sh.act_bytes, Wn, wb) || overlaps(y, sh.act_bytes, bias, sh.d * 4) ||
        overlaps(y, sh.act_bytes, z, sh.act_bytes) || overlaps(z, sh.act_bytes, x, sh.act_bytes))
        return HCW_ERR_ALIASING;
    return HCW_OK;
}

int check_bwd_ptrs(const Shape& sh, int dtype, unsigned flags, const void* x, const void* z,
                   const void* dy, const void* Ws, const void* Wn, void* dx, float* dWs,
                   float* dWn, float* dbias) {
    if (!x || !dy || !Ws || !Wn || !dx || !dWs || !dWn) return HCW_ERR_INVALID_ARG;
    if ((flags & HCW_ACT_RELU) && !z) return HCW_ERR_INVALID_ARG;
    const void* ptrs[] = {x, z, dy, Ws, Wn, dx, dWs, dWn, dbias};
    for (const void* q : ptrs)
        if (q && !aligned16(q)) return HCW_ERR_ALIGNMENT;
    const size_t ab = sh.act_bytes, wb = (size_t)sh.d * sh.d * elem_size(dtype);
    const size_t gb = (size_t)sh.d * sh.d * 4;
    if (overlaps(dx, ab, x, ab) || overlaps(dx, ab, dy, ab) || overlaps(dx, ab, z, ab) ||
        overlaps(dx, ab, Ws, wb) || overlaps(dx, ab, Wn, wb) || overlaps(dWs, gb, dWn, gb) ||
        overlaps(dx, ab, dWs, gb) || overlaps(dx, ab, dWn, gb) ||
        overlaps(dbias, sh.d * 4, dWs, gb) || overlaps(dbias, sh.d * 4, dWn, gb))
        return HCW_ERR_ALIASING;
    return HCW_OK;
}

// A schedule array of L layers: a cube dimension in [0, log2 n), or a shift
// -k with 1 <= k < n.
int check_dims(const Shape& sh, const int* dims, int L) {
    if (!dims) return HCW_ERR_INVALID_ARG;
    for (int l = 0; l < L; ++l)
        if (dims[l] >= sh.b || (dims[l] < 0 && -(long long)dims[l] >= sh.n))
            return HCW_ERR_INVALID_ARG;
    return HCW_OK;
}

int stack_fwd_impl(const Shape& sh, const void* x, const void* W_self, const void* W_nbr,
                   const float* bias, const Sched& sc, int L, int dtype, unsigned flags, void* y,
                   void* acts, void* masks, void* workspace, size_t ws_bytes, void* stream) {
    const int B = sh.B, n = sh.n, d = sh.d;
    int rc;
    if (sh.tokens == 0) return HCW_OK;
    if (L > 1 && !acts) return HCW_ERR_INVALID_ARG;
    if ((acts && !aligned16(acts)) || (masks && !aligned16(masks)) ||
        (workspace && !aligned16(workspace)))
        return HCW_ERR_ALIGNMENT;
    const size_t ab = sh.act_bytes, wb = (size_t)d * d * elem_size(dtype);
    const size_t mb = mask_bytes(sh);
    const size_t need = hcw_stack_fwd_workspace_bytes(B, n, d, dtype, flags, L);
    if (ws_bytes < need || (need && !workspace)) return HCW_ERR_WORKSPACE;
    rc = check_fwd_ptrs(sh, dtype, x, W_self, W_nbr, bias, y, nullptr);
    if (rc) return rc;
    const size_t acts_b = (size_t)(L - 1) * ab, m_b = (size_t)L * mb;
    if (overlaps(acts, acts_b, x, ab) || overlaps(acts, acts_b, y, ab) ||
        overlaps(masks, m_b, x, ab) || overlaps(masks, m_b, y, ab) ||
        overlaps(masks, m_b, acts, acts_b) || overlaps(acts, acts_b, W_self, L * wb) ||
        overlaps(acts, acts_b, W_nbr, L * wb) || overlaps(workspace, need, x, ab) ||
        overlaps(workspace, need, y, ab) || overlaps(workspace, need, acts, acts_b) ||
        overlaps(workspace, need, masks, m_b))
        return HCW_ERR_ALIASING;
    cudaStream_t st = (cudaStream_t)stream;
    const bool want_mask = masks && (flags & HCW_ACT_RELU);
    auto in_ptr = [&](int l) -> const void* {
        return l == 0 ? x : static_cast<const uint8_t*>(acts) + (size_t)(l - 1) * ab;
    };
    auto out_ptr = [&](int l) -> void* {
        return l == L - 1 ? y : static_cast<uint8_t*>(acts) + (size_t)l * ab;
    };
    auto mask_ptr = [&](int l) -> uint32_t* {
        return want_mask ? reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(masks) + (size_t)l * mb)
                         : nullptr;
    };
    if (dtype == HCW_BF16 && sc.has_shift(L) && (!shift_stackable(sh) || use_resident(sh))) {
        // layer by layer; a shift layer reads its partner rows S_k x, materialised
        // row-aligned behind the counters of the workspace
        void* u = static_cast<uint8_t*>(workspace) + stack_counter_bytes(sh.tokens, L);
        for (int l = 0; l < L; ++l) {
            const int s = sc.dim(sh, l);
            Shape shl = sh;
            const uint8_t* ws_l = static_cast<const uint8_t*>(W_self) + l * wb;
            const uint8_t* wn_l = static_cast<const uint8_t*>(W_nbr) + l * wb;
            const float* b_l = bias ? bias + (size_t)l * d : nullptr;
            if (s >= 0) {
                shl.s = s;
                rc = fwd_bf16(shl, in_ptr(l), ws_l, wn_l, b_l, flags, out_ptr(l), nullptr,
                              mask_ptr(l), st);
            } else {
                rc = launched(launch_shift_rows_bf16(static_cast<const __nv_bfloat16*>(in_ptr(l)),
                                                     static_cast<__nv_bfloat16*>(u), sh.tokens,
                                                     n, d, -s, st),
                              1);
                if (rc) return rc;
                shl.s = shift_group_dim(sh);
                rc = fwd_bf16(shl, in_ptr(l), ws_l, wn_l, b_l, flags, out_ptr(l), nullptr,
                              mask_ptr(l), st, u);
            }
            if (rc) return rc;
        }
        return HCW_OK;
    }
    if (dtype == HCW_BF16) {
        // up to kMaxStackLayers layers per persistent launch
        for (int l0 = 0; l0 < L; l0 += kMaxStackLayers) {
            const int cnt = L - l0 < kMaxStackLayers ? L - l0 : kMaxStackLayers;
            if (use_resident(sh) && !sc.has_shift(L))
                rc = stack_fwd_resident(sh, l0, cnt, sc,
                                        static_cast<const uint8_t*>(W_self),
                                        static_cast<const uint8_t*>(W_nbr), bias, flags, in_ptr,
                                        out_ptr, mask_ptr, st);
            else
                rc = stack_fwd_group(sh, l0, cnt, sc,
                                     static_cast<const uint8_t*>(W_self),
                                     static_cast<const uint8_t*>(W_nbr), bias, flags, in_ptr,
                                     out_ptr, mask_ptr, static_cast<int*>(workspace), st);
            if (rc) return rc;
        }
        return HCW_OK;
    }
    for (int l = 0; l < L; ++l) {
        Shape shl = sh;
        shl.s = sc.dim(sh, l);
        rc = layer_fwd_impl(shl, dtype, in_ptr(l), static_cast<const uint8_t*>(W_self) + l * wb,
                            static_cast<const uint8_t*>(W_nbr) + l * wb,
                            bias ? bias + (size_t)l * d : nullptr, flags, out_ptr(l), nullptr, st,
                            mask_ptr(l));
        if (rc) return rc;
    }
    return HCW_OK;
}

int stack_bwd_impl(const Shape& sh, const void* x, const void* acts, const void* masks,
                   const void* dy, const void* W_self, const void* W_nbr, const Sched& sc, int L,
                   int dtype, unsigned flags, void* dx, float* dW_self, float* dW_nbr,
                   float* dbias, void* workspace, size_t ws_bytes, void* stream) {
    const int d = sh.d;
    int rc;
    cudaStream_t st = (cudaStream_t)stream;
    if (sh.tokens == 0) {
        if (!dW_self || !dW_nbr) return HCW_ERR_INVALID_ARG;
        return zero_weight_grads(L, d, dW_self, dW_nbr, dbias, st);
    }
    // workspace: [dz of every layer][input-gradient scratch][weight-gradient scratch]
    const size_t zb = stack_dz_bytes(sh, L);
    const size_t db = align256(stack_data_ws(sh, dtype, flags, L));
    const size_t wb = stack_weight_ws(sh, dtype, flags, L);
    if (ws_bytes < zb + db + wb || !workspace) return HCW_ERR_WORKSPACE;
    if (!aligned16(workspace)) return HCW_ERR_ALIGNMENT;
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    rc = check_stack_data(sh, dtype, flags, L, masks, dy, W_self, W_nbr, dx, ws, ws + zb, db);
    if (rc) return rc;
    rc = check_stack_weight(sh, dtype, flags, L, x, acts, ws, dW_self, dW_nbr, dbias, ws + zb + db,
                            wb);
    if (rc) return rc;
    // the weight gradients read x and acts; the input gradients write dx
    const size_t ab = sh.act_bytes;
    if (overlaps(dx, ab, x, ab) || overlaps(dx, ab, acts, (size_t)(L - 1) * ab) ||
        overlaps(ws, ws_bytes, x, ab) || overlaps(ws, ws_bytes, acts, (size_t)(L - 1) * ab) ||
        overlaps(dx, ab, dW_self, (size_t)L * d * d * 4) ||
        overlaps(dx, ab, dW_nbr, (size_t)L * d * d * 4) ||
        overlaps(dx, ab, dbias, dbias ? (size_t)L * d * 4 : 0))
        return HCW_ERR_ALIASING;
    StackData da{masks, dy, static_cast<const uint8_t*>(W_self),
                 static_cast<const uint8_t*>(W_nbr), sc, L, flags, dx, ws, ws + zb};
    rc = dtype == HCW_BF16 ? stack_data_bf16(sh, da, st) : stack_data_f32(sh, da, st);
    if (rc) return rc;
    StackWeight wa{x, acts, ws, sc, L, flags, dW_self, dW_nbr, dbias, ws + zb + db};
    return dtype == HCW_BF16 ? stack_weight_bf16(sh, wa, st) : stack_weight_f32(sh, wa, st);
}

// ------------------------------------------------------------ training step
// Counters of the fused forward + input-gradient launch: per (layer, chunk)
// completion counters of its 2L layers, the unit counter, the (unused) top-dz
// chunk counters, and per (layer, chunk) counters of g.
size_t step_counter_bytes(long long tokens, int L) {
    const size_t chunks = (size_t)((tokens + 127) / 128);
    return align256((4 * (size_t)L * chunks + 1 + chunks) * sizeof(int) + 16);
}

// Whether a training step runs its forward and input gradient as one launch:
// bf16, any schedule whose shift layers the stacked launches take
// (shift_stackable), the streaming kernels on SM pairs (d a multiple of 128),
// and up to kMaxStackLayers layers.
bool step_fused(const Shape& sh, int dtype, const Sched& sc, int L) {
    // 256- or 128-column tiles on pairs (d = 128 takes the latter), at least
    // two row blocks
    const bool pairs = use_pairs(sh) || (pick_bn(sh.d) == 128 && sh.tokens / 2 > 128);
    return dtype == HCW_BF16 && (!sc.has_shift(L) || shift_stackable(sh)) && !use_resident(sh) &&
           pairs && L <= kMaxStackLayers && sh.tokens > 0;
}

size_t step_fwd_region(const Shape& sh, int dtype, unsigned flags, int L) {
    const size_t f = hcw_stack_fwd_workspace_bytes(sh.B, sh.n, sh.d, dtype, flags, L);
    const size_t c = step_counter_bytes(sh.tokens, L);
    return align256(f > c ? f : c);
}

// The forward (layers 0 .. L-1) and the input gradient (layers L-1 .. 0) in one
// launch on pairs of SMs; the last forward layer writes the top layer's dz.
int step_fused_launch(const Shape& sh, const void* x, const uint8_t* Ws, const uint8_t* Wn,
                      const float* bias, const void* dy, const Sched& sc, int L, unsigned flags,
                      void* y, void* acts, void* masks, void* dx, uint8_t* dz, uint8_t* gws,
                      int* counters, cudaStream_t st, int dw_pairs = 0) {
    // 128-column tiles when 256-column ones would leave more than half of the
    // SM pairs without a unit of a layer (few tokens: the launch is the layer
    // chain, and narrower units shorten each of its steps)
    const int sms_all = sm_count();
    int BN = pick_bn(sh.d);
    {
        TcParams q;
        row_unit_params(q, sh, BN, flags, false);
        pair_units(q);
        if (BN == 256 && 2 * q.n_units <= sms_all / 2) BN = 128;
    }
    const int d = sh.d, pw = epi_patch_cols(BN);
    const size_t ab = sh.act_bytes, a256 = align256(ab), wb = (size_t)d * d * 2;
    const size_t mb = mask_bytes(sh);
    const bool relu = (flags & HCW_ACT_RELU) != 0;
    const bool resid = (flags & HCW_RESIDUAL) != 0;
    const bool keep_g = relu && resid;
    auto in_ptr = [&](int l) -> const void* {
        return l == 0 ? x : static_cast<const uint8_t*>(acts) + (size_t)(l - 1) * ab;
    };
    auto out_ptr = [&](int l) -> void* {
        return l == L - 1 ? y : static_cast<uint8_t*>(acts) + (size_t)l * ab;
    };
    auto mask = [&](int l) -> uint32_t* {
        return relu ? reinterpret_cast<uint32_t*>(static_cast<uint8_t*>(masks) + (size_t)l * mb)
                    : nullptr;
    };
    auto dzp = [&](int l) -> void* { return dz + (size_t)l * ab; };
    auto gbuf = [&](int l) -> void* { return gws + (size_t)(l & 1) * a256; };   // as stack_data_bf16
    auto g = [&](int l) -> const void* {
        if (l == L - 1) return dy;
        return keep_g ? gbuf(l) : dzp(l);
    };
    static thread_local TcLaunch<kMaxStepLayers> T;
    memset(&T, 0, sizeof(T));
    for (int l = 0; l < L; ++l) {
        const int sl = sc.dim(sh, l);
        // a shift layer: rows in runs of 128 positions, its input as positions
        const int s = sl >= 0 ? sl : kShiftStackDim;
        CUtensorMap* m = T.maps[l];
        if (!fwd_maps(m, sh, s, in_ptr(l), Ws + l * wb, Wn + l * wb, out_ptr(l), true, BN) ||
            (sl < 0 && !map_positions(&m[0], in_ptr(l), sh.tokens, sh.n, d, 128)))
            return HCW_ERR_CUDA;
        // the last forward layer also stores the top layer's dz (map 5)
        if (l == L - 1 && !map_rows(&m[5], dzp(L - 1), sh.tokens, d, 1 << s, 32, pw))
            return HCW_ERR_CUDA;
        T.layer[l] = {s, 1 << s, bias ? bias + (size_t)l * d : nullptr, mask(l), nullptr, true,
                      nullptr, false};
        T.layer[l].shift = sl < 0 ? -sl : 0;
    }
    for (int i = 0; i < L; ++i) {
        const int l = L - 1 - i;   // input-gradient layers from the top down
        const int sl = sc.dim(sh, l);
        const int s = sl >= 0 ? sl : kShiftStackDim;
        const int k = 1 << s;
        // stores: g_{l-1} (map 4) and dz_{l-1} (map 5); at l = 0 the stack's dx
        void* out = l == 0 ? dx : (relu ? (resid ? gbuf(l - 1) : nullptr) : dzp(l - 1));
        void* dzo = (l > 0 && relu) ? dzp(l - 1) : nullptr;
        CUtensorMap* m = T.maps[L + i];
        const void* res = resid ? g(l) : dzp(l);
        if (!map_rows(&m[0], dzp(l), sh.tokens, d, k, 128) ||
            !map_weight_blocks(&m[1], Ws + l * wb, d, BN / 2 / 64) ||
            !map_weight_blocks(&m[2], Wn + l * wb, d, BN / 2 / 64) ||
            !map_rows(&m[3], res, sh.tokens, d, k, 32, pw) ||
            !map_rows(&m[4], out ? out : dzo, sh.tokens, d, k, 32, pw) ||
            !map_rows(&m[5], dzo ? dzo : out, sh.tokens, d, k, 32, pw))
            return HCW_ERR_CUDA;
        if (sl < 0 && !map_positions(&m[0], dzp(l), sh.tokens, sh.n, d, 128))
            return HCW_ERR_CUDA;
        T.layer[L + i] = {s, k, nullptr, nullptr, nullptr, out != nullptr,
                          dzo ? mask(l - 1) : nullptr, dzo != nullptr};
        T.layer[L + i].shift = sl < 0 ? -sl : 0;
        // the g buffers written by this launch (not dy)
        if (keep_g && i > 0) T.layer[L + i].g_discard = static_cast<const __nv_bfloat16*>(res);
    }
    row_unit_params(T.p, sh, BN, flags, false);
    pair_units(T.p);
    T.p.flags = flags;
    T.p.seq_n = sh.n;
    T.n_layers = 2 * L;
    T.n_fwd = L;
    const int n_chunks = (int)((sh.tokens + 127) / 128);
    T.counters = counters;
    T.n_chunks = n_chunks;
    T.tokens = (int)sh.tokens;
    T.sched = counters + (size_t)2 * L * n_chunks;
    T.in_counters = T.sched + 1;
    T.g_counters = keep_g ? T.sched + 1 + n_chunks : nullptr;
    T.top_dy = static_cast<const __nv_bfloat16*>(dy);
    T.top_dz = static_cast<__nv_bfloat16*>(dzp(L - 1));
    if (cudaMemsetAsync(counters, 0, step_counter_bytes(sh.tokens, L), st) != cudaSuccess)
        return HCW_ERR_CUDA;
    const int sms = sm_count();
    const int total = T.p.n_units * 2 * L;
    const int pairs = total < sms / 2 ? total : sms / 2;
    // With a weight-gradient launch of dw_pairs pairs right behind: the last
    // layer runs on the pairs that launch leaves idle, when they get through it
    // in well under the weight gradient's time (its units take K = 2d or d
    // steps of 64; a weight-gradient unit takes three or four per 64 compressed
    // rows of each bit value); the rest of the SMs go to the weight gradient
    // as soon as they are done with the earlier layers.
    if (dw_pairs > 0 && pairs == sms / 2 && pairs > dw_pairs) {
        const int tail = pairs - dw_pairs;
        const long long tail_steps =
            (long long)T.p.n_units * (T.p.n_full == 2 ? 4 : 3) * T.p.nK / 2 / tail;
        const long long dw_steps =
            (long long)((T.p.Mh + 63) / 64) * ((flags & HCW_CAUSAL) ? 3 : 4);
        if (4 * tail_steps <= 3 * dw_steps) T.tail_pairs = tail;
    }
    return launched(launch_tc_step_pair(BN, T, 2 * pairs, st), 1);
}

int train_step_impl(const Shape& sh, const void* x, const void* W_self, const void* W_nbr,
                    const float* bias, const void* dy, const Sched& sc, int L, int dtype,
                    unsigned flags, void* y, void* acts, void* masks, void* dx, float* dW_self,
                    float* dW_nbr, float* dbias, void* workspace, size_t ws_bytes, void* stream) {
    const int d = sh.d;
    cudaStream_t st = (cudaStream_t)stream;
    // workspace: [backward (dz | input-gradient scratch | weight-gradient
    // scratch)][forward scratch, or the fused launch's counters]
    const size_t zb = stack_dz_bytes(sh, L);
    const size_t db = align256(stack_data_ws(sh, dtype, flags, L));
    const size_t wbb = stack_weight_ws(sh, dtype, flags, L);
    const size_t bwd = align256(zb + db + wbb);
    const size_t fwd = step_fwd_region(sh, dtype, flags, L);
    // no weight-gradient outputs: the forward and the input gradient only
    const bool want_dw = dW_self != nullptr || dW_nbr != nullptr;
    if (want_dw && (!dW_self || !dW_nbr)) return HCW_ERR_INVALID_ARG;
    if (!want_dw && dbias) return HCW_ERR_INVALID_ARG;
    if (sh.tokens == 0) return want_dw ? zero_weight_grads(L, d, dW_self, dW_nbr, dbias, st) : HCW_OK;
    if (ws_bytes < bwd + fwd || !workspace) return HCW_ERR_WORKSPACE;
    if (!aligned16(workspace)) return HCW_ERR_ALIGNMENT;
    uint8_t* ws = static_cast<uint8_t*>(workspace);
    if (!step_fused(sh, dtype, sc, L)) {
        int rc = stack_fwd_impl(sh, x, W_self, W_nbr, bias, sc, L, dtype, flags, y, acts, masks,
                                ws + bwd, fwd, stream);
        if (rc) return rc;
        if (want_dw)
            return stack_bwd_impl(sh, x, acts, masks, dy, W_self, W_nbr, sc, L, dtype, flags, dx,
                                  dW_self, dW_nbr, dbias, ws, bwd, stream);
        rc = check_stack_data(sh, dtype, flags, L, masks, dy, W_self, W_nbr, dx, ws, ws + zb, db);
        if (rc) return rc;
        StackData da{masks, dy, static_cast<const uint8_t*>(W_self),
                     static_cast<const uint8_t*>(W_nbr), sc, L, flags, dx, ws, ws + zb};
        return dtype == HCW_BF16 ? stack_data_bf16(sh, da, st) : stack_data_f32(sh, da, st);
    }
    // the checks of the forward and the backward calls, on the same buffers
    if (L > 1 && !acts) return HCW_ERR_INVALID_ARG;
    if ((acts && !aligned16(acts)) || (masks && !aligned16(masks))) return HCW_ERR_ALIGNMENT;
    int rc = check_fwd_ptrs(sh, dtype, x, W_self, W_nbr, bias, y, nullptr);
    if (rc) return rc;
    const size_t ab = sh.act_bytes, wb = (size_t)d * d * 2;
    const size_t acts_b = (size_t)(L - 1) * ab, m_b = (size_t)L * mask_bytes(sh);
    if (overlaps(acts, acts_b, x, ab) || overlaps(acts, acts_b, y, ab) ||
        overlaps(masks, m_b, x, ab) || overlaps(masks, m_b, y, ab) ||
        overlaps(masks, m_b, acts, acts_b) || overlaps(acts, acts_b, W_self, L * wb) ||
        overlaps(acts, acts_b, W_nbr, L * wb) || overlaps(ws, ws_bytes, x, ab) ||
        overlaps(ws, ws_bytes, y, ab) || overlaps(ws, ws_bytes, acts, acts_b) ||
        overlaps(ws, ws_bytes, masks, m_b) || overlaps(dx, ab, y, ab) ||
        overlaps(dx, ab, acts, acts_b) || overlaps(dx, ab, x, ab) ||
        overlaps(dx, ab, masks, m_b))
        return HCW_ERR_ALIASING;
    rc = check_stack_data(sh, dtype, flags, L, masks, dy, W_self, W_nbr, dx, ws, ws + zb, db);
    if (rc) return rc;
    if (want_dw) {
        rc = check_stack_weight(sh, dtype, flags, L, x, acts, ws, dW_self, dW_nbr, dbias,
                                ws + zb + db, wbb);
        if (rc) return rc;
    }
    if (overlaps(dx, ab, dW_self, (size_t)L * d * d * 4) ||
        overlaps(dx, ab, dW_nbr, (size_t)L * d * d * 4) ||
        overlaps(dx, ab, dbias, dbias ? (size_t)L * d * 4 : 0) ||
        overlaps(dy, ab, y, ab) || overlaps(dy, ab, acts, acts_b) || overlaps(dy, ab, masks, m_b))
        return HCW_ERR_ALIASING;
    rc = step_fused_launch(sh, x, static_cast<const uint8_t*>(W_self),
                           static_cast<const uint8_t*>(W_nbr), bias, dy, sc, L, flags, y, acts,
                           masks, dx, ws, ws + zb, reinterpret_cast<int*>(ws + bwd), st,
                           want_dw ? dw_early_pairs(sh, flags, L) : 0);
    if (rc || !want_dw) return rc;
    StackWeight wa{x, acts, ws, sc, L, flags, dW_self, dW_nbr, dbias, ws + zb + db,
                   reinterpret_cast<const int*>(ws + bwd)};
    return stack_weight_bf16(sh, wa, st);
}

// Link distance of decode layer l: 2^s for the hypercube link along
// dimension s, k for a shift by k.
int decode_link(const int* dims, int layer0, int b, int l) {
    const int s = dims ? dims[l] : (layer0 + l) % b;
    return s >= 0 ? 1 << s : -s;
}

int decode_check(const int* dims, int layer0, int L, int B, int n, int d, Shape* sh) {
    if (L < 1 || L > kMaxDecodeLayers || B < 1 || layer0 < 0) return HCW_ERR_INVALID_ARG;
    int rc = check_shape(0, -1, B, n, d, HCW_BF16, 0, sh);
    if (rc) return rc;
    if (dims) return check_dims(*sh, dims, L);
    return HCW_OK;
}

}  // namespace

int count_launch(cudaError_t e, int kernels) { return launched(e, kernels); }

}  // namespace hcw

using namespace hcw;

extern "C" {

int hcw_version(void) { return 100; }

const char* hcw_status_string(int s) {
    switch (s) {
        case HCW_OK: return "HCW_OK";
        case HCW_ERR_INVALID_ARG: return "HCW_ERR_INVALID_ARG";
        case HCW_ERR_UNSUPPORTED: return "HCW_ERR_UNSUPPORTED";
        case HCW_ERR_ALIGNMENT: return "HCW_ERR_ALIGNMENT";
        case HCW_ERR_ALIASING: return "HCW_ERR_ALIASING";
        case HCW_ERR_CUDA: return "HCW_ERR_CUDA";
        case HCW_ERR_TIMEOUT: return "HCW_ERR_TIMEOUT";
        case HCW_ERR_WORKSPACE: return "HCW_ERR_WORKSPACE";
        default: return "HCW_ERR_UNKNOWN";
    }
}

int hcw_partner_table(int layer, int dim_override, int n, unsigned flags, int* partner) {
    const int b = log2_exact(n);
    if (b < 1 || layer < 0 || dim_override < -1 || dim_override >= b || !partner ||
        (flags & ~kAllFlags))
        return HCW_ERR_INVALID_ARG;
    const int s = dim_override >= 0 ? dim_override : layer % b;
    for (int i = 0; i < n; ++i) {
        const int p = i ^ (1 << s);
        const bool recv = !(flags & HCW_CAUSAL) || ((i >> s) & 1);
        partner[i] = recv ? p : -1;
    }
    return HCW_OK;
}

int hcw_partner_table_device(int layer, int dim_override, int n, unsigned flags,
                             int* partner_dev, void* stream) {
    const int b = log2_exact(n);
    if (b < 1 || layer < 0 || dim_override < -1 || dim_override >= b || !partner_dev ||
        (flags & ~kAllFlags))
        return HCW_ERR_INVALID_ARG;
    if (!aligned16(partner_dev)) return HCW_ERR_ALIGNMENT;
    const int s = dim_override >= 0 ? dim_override : layer % b;
    return launched(launch_partner_table(s, n, flags, partner_dev, (cudaStream_t)stream), 1);
}

int hcw_layer_fwd(const void* x, const void* W_self, const void* W_nbr, const float* bias,
                  int layer, int dim_override, int B, int n, int d, int dtype, unsigned flags,
                  void* y, void* z_save, void* stream) {
    Shape sh;
    int rc = check_shape(layer, dim_override, B, n, d, dtype, flags, &sh);
    if (rc) return rc;
    if (sh.tokens == 0) return HCW_OK;   // empty batch: nothing to compute
    rc = check_fwd_ptrs(sh, dtype, x, W_self, W_nbr, bias, y, z_save);
    if (rc) return rc;
    return layer_fwd_impl(sh, dtype, x, W_self, W_nbr, bias, flags, y, z_save,
                          (cudaStream_t)stream);
}

size_t hcw_workspace_bytes(int B, int n, int d, int dtype, unsigned flags) {
    Shape sh;
    if (check_shape(0, -1, B, n, d, dtype, flags, &sh)) return 0;
    return ws_layout(sh.tokens, d, dtype, flags).total;
}

int hcw_layer_bwd(const void* x, const void* z_save, const void* dy, const void* W_self,
                  const void* W_nbr, int layer, int dim_override, int B, int n, int d, int dtype,
                  unsigned flags, void* dx, float* dW_self, float* dW_nbr, float* dbias,
                  void* workspace, size_t ws_bytes, void* stream) {
    Shape sh;
    int rc = check_shape(layer, dim_override, B, n, d, dtype, flags, &sh);
    if (rc) return rc;
    if (sh.tokens == 0) {
        // empty batch: only the weight gradients (sums over no tokens, zero) are written
        if (!dW_self || !dW_nbr) return HCW_ERR_INVALID_ARG;
        return layer_bwd_impl(sh, dtype, x, z_save, dy, W_self, W_nbr, flags, dx, dW_self,
                              dW_nbr, dbias, workspace, (cudaStream_t)stream);
    }
    rc = check_bwd_ptrs(sh, dtype, flags, x, z_save, dy, W_self, W_nbr, dx, dW_self, dW_nbr,
                        dbias);
    if (rc) return rc;
    const size_t need = ws_layout(sh.tokens, d, dtype, flags).total;
    if (ws_bytes < need || (need && !workspace)) return HCW_ERR_WORKSPACE;
    if (workspace && !aligned16(workspace)) return HCW_ERR_ALIGNMENT;
    if (overlaps(workspace, ws_bytes, dx, sh.act_bytes) ||
        overlaps(workspace, ws_bytes, dy, sh.act_bytes) ||
        overlaps(workspace, ws_bytes, x, sh.act_bytes))
        return HCW_ERR_ALIASING;
    return layer_bwd_impl(sh, dtype, x, z_save, dy, W_self, W_nbr, flags, dx, dW_self, dW_nbr,
                          dbias, workspace, (cudaStream_t)stream);
}

int hcw_layer_bwd_data(const void* dz, const void* dy, const void* W_self, const void* W_nbr,
                       int layer, int dim_override, int B, int n, int d, int dtype,
                       unsigned flags, void* dx, void* stream) {
    Shape sh;
    int rc = check_shape(layer, dim_override, B, n, d, dtype, flags, &sh);
    if (rc) return rc;
    if (sh.tokens == 0) return HCW_OK;
    if (!dz || !W_self || !W_nbr || !dx || ((flags & HCW_RESIDUAL) && !dy))
        return HCW_ERR_INVALID_ARG;
    const void* ptrs[] = {dz, dy, W_self, W_nbr, dx};
    for (const void* q : ptrs)
        if (q && !aligned16(q)) return HCW_ERR_ALIGNMENT;
    const size_t ab = sh.act_bytes, wb = (size_t)d * d * elem_size(dtype);
    if (overlaps(dx, ab, dz, ab) || overlaps(dx, ab, dy, ab) || overlaps(dx, ab, W_self, wb) ||
        overlaps(dx, ab, W_nbr, wb))
        return HCW_ERR_ALIASING;
    return layer_dx_impl(sh, dtype, dz, dy, W_self, W_nbr, flags, dx, (cudaStream_t)stream);
}

size_t hcw_layer_bwd_weight_workspace_bytes(int B, int n, int d, int dtype, unsigned flags) {
    Shape sh;
    if (check_shape(0, -1, B, n, d, dtype, flags, &sh)) return 0;
    return ws_layout(sh.tokens, d, dtype, flags).w_bytes;
}

int hcw_layer_bwd_weight(const void* x, const void* dz, int layer, int dim_override, int B,
                         int n, int d, int dtype, unsigned flags, float* dW_self,
                         float* dW_nbr, float* dbias, void* workspace, size_t ws_bytes,
                         void* stream) {
    Shape sh;
    int rc = check_shape(layer, dim_override, B, n, d, dtype, flags, &sh);
    if (rc) return rc;
    if (!dW_self || !dW_nbr) return HCW_ERR_INVALID_ARG;
    const void* ptrs[] = {x, dz, dW_self, dW_nbr, dbias, workspace};
    for (const void* q : ptrs)
        if (q && !aligned16(q)) return HCW_ERR_ALIGNMENT;
    if (sh.tokens > 0 && (!x || !dz)) return HCW_ERR_INVALID_ARG;
    const size_t need = ws_layout(sh.tokens, d, dtype, flags).w_bytes;
    if (sh.tokens > 0 && (ws_bytes < need || (need && !workspace))) return HCW_ERR_WORKSPACE;
    const size_t ab = sh.act_bytes, gb = (size_t)d * d * 4;
    // the column sums read dz while they write dbias: dbias must not overlap an input
    if (overlaps(dW_self, gb, dW_nbr, gb) || overlaps(dbias, (size_t)d * 4, dW_self, gb) ||
        overlaps(dbias, (size_t)d * 4, dW_nbr, gb) || overlaps(workspace, ws_bytes, x, ab) ||
        overlaps(workspace, ws_bytes, dz, ab) || overlaps(workspace, ws_bytes, dW_self, gb) ||
        overlaps(workspace, ws_bytes, dW_nbr, gb) || overlaps(workspace, ws_bytes, dbias, (size_t)d * 4) ||
        overlaps(dW_self, gb, x, ab) || overlaps(dW_nbr, gb, x, ab) ||
        overlaps(dW_self, gb, dz, ab) || overlaps(dW_nbr, gb, dz, ab) ||
        overlaps(dbias, (size_t)d * 4, x, ab) || overlaps(dbias, (size_t)d * 4, dz, ab))
        return HCW_ERR_ALIASING;
    return layer_dw_impl(sh, dtype, x, dz, flags, dW_self, dW_nbr, dbias,
                         static_cast<uint8_t*>(workspace), (cudaStream_t)stream);
}

size_t hcw_stack_fwd_workspace_bytes(int B, int n, int d, int dtype, unsigned flags, int L) {
    Shape sh;
    if (L < 1 || check_shape(0, -1, B, n, d, dtype, flags, &sh)) return 0;
    // bf16: the stacked launches' counters, then the shifted input of a shift layer
    return dtype == HCW_BF16 && sh.tokens > 0
               ? stack_counter_bytes(sh.tokens, L) + align256(sh.act_bytes)
               : 0;
}

int hcw_stack_fwd(const void* x, const void* W_self, const void* W_nbr, const float* bias,
                  int layer0, int L, int dim_override, int B, int n, int d, int dtype,
                  unsigned flags, void* y, void* acts, void* masks, void* workspace,
                  size_t ws_bytes, void* stream) {
    Shape sh;
    if (L < 1) return HCW_ERR_INVALID_ARG;
    int rc = check_shape(layer0, dim_override, B, n, d, dtype, flags, &sh);
    if (rc) return rc;
    return stack_fwd_impl(sh, x, W_self, W_nbr, bias, Sched{nullptr, layer0, dim_override}, L,
                          dtype, flags, y, acts, masks, workspace, ws_bytes, stream);
}

int hcw_stack_fwd_dims(const void* x, const void* W_self, const void* W_nbr, const float* bias,
                       const int* dims, int L, int B, int n, int d, int dtype, unsigned flags,
                       void* y, void* acts, void* masks, void* workspace, size_t ws_bytes,
                       void* stream) {
    Shape sh;
    if (L < 1) return HCW_ERR_INVALID_ARG;
    int rc = check_shape(0, -1, B, n, d, dtype, flags, &sh);
    if (rc) return rc;
    rc = check_dims(sh, dims, L);
    if (rc) return rc;
    return stack_fwd_impl(sh, x, W_self, W_nbr, bias, Sched{dims, 0, -1}, L, dtype, flags, y,
                          acts, masks, workspace, ws_bytes, stream);
}

size_t hcw_stack_bwd_data_workspace_bytes(int B, int n, int d, int dtype, unsigned flags,
                                          int L) {
    Shape sh;
    if (L < 1 || check_shape(0, -1, B, n, d, dtype, flags, &sh)) return 0;
    return stack_data_ws(sh, dtype, flags, L);
}

size_t hcw_stack_bwd_weight_workspace_bytes(int B, int n, int d, int dtype, unsigned flags,
                                            int L) {
    Shape sh;
    if (L < 1 || check_shape(0, -1, B, n, d, dtype, flags, &sh)) return 0;
    return stack_weight_ws(sh, dtype, flags, L);
}

size_t hcw_stack_workspace_bytes(int B, int n, int d, int dtype, unsigned flags, int L) {
    Shape sh;
    if (L < 1 || check_shape(0, -1, B, n, d, dtype, flags, &sh)) return 0;
    return stack_dz_bytes(sh, L) + align256(stack_data_ws(sh, dtype, flags, L)) +
           stack_weight_ws(sh, dtype, flags, L);
}

int hcw_stack_bwd_data(const void* masks, const void* dy, const void* W_self, const void* W_nbr,
                       int layer0, int L, int dim_override, int B, int n, int d, int dtype,
                       unsigned flags, void* dx, void* dz, void* workspace, size_t ws_bytes,
                       void* stream) {
    Shape sh;
    if (L < 1) return HCW_ERR_INVALID_ARG;
    int rc = check_shape(layer0, dim_override, B, n, d, dtype, flags, &sh);
    if (rc) return rc;
    if (sh.tokens == 0) return HCW_OK;
    rc = check_stack_data(sh, dtype, flags, L, masks, dy, W_self, W_nbr, dx, dz, workspace,
                          ws_bytes);
    if (rc) return rc;
    StackData a{masks, dy, static_cast<const uint8_t*>(W_self), static_cast<const uint8_t*>(W_nbr),
                Sched{nullptr, layer0, dim_override}, L, flags, dx, static_cast<uint8_t*>(dz),
                static_cast<uint8_t*>(workspace)};
    return dtype == HCW_BF16 ? stack_data_bf16(sh, a, (cudaStream_t)stream)
                             : stack_data_f32(sh, a, (cudaStream_t)stream);
}

int stack_bwd_weight_impl(const Shape& sh, const void* x, const void* acts, const void* dz,
                          const Sched& sc, int L, int dtype, unsigned flags, float* dW_self,
                          float* dW_nbr, float* dbias, void* workspace, size_t ws_bytes,
                          void* stream);

int hcw_stack_bwd_weight_dims(const void* x, const void* acts, const void* dz, const int* dims,
                              int L, int B, int n, int d, int dtype, unsigned flags,
                              float* dW_self, float* dW_nbr, float* dbias, void* workspace,
                              size_t ws_bytes, void* stream) {
    Shape sh;
    if (L < 1) return HCW_ERR_INVALID_ARG;
    int rc = check_shape(0, -1, B, n, d, dtype, flags, &sh);
    if (rc) return rc;
    rc = check_dims(sh, dims, L);
    if (rc) return rc;
    return stack_bwd_weight_impl(sh, x, acts, dz, Sched{dims, 0, -1}, L, dtype, flags, dW_self,
                                 dW_nbr, dbias, workspace, ws_bytes, stream);
}

int hcw_stack_bwd_weight(const void* x, const void* acts, const void* dz, int layer0, int L,
                         int dim_override, int B, int n, int d, int dtype, unsigned flags,
                         float* dW_self, float* dW_nbr, float* dbias, void* workspace,
                         size_t ws_bytes, void* stream) {
    Shape sh;
    if (L < 1) return HCW_ERR_INVALID_ARG;
    int rc = check_shape(layer0, dim_override, B, n, d, dtype, flags, &sh);
    if (rc) return rc;
    return stack_bwd_weight_impl(sh, x, acts, dz, Sched{nullptr, layer0, dim_override}, L, dtype,
                                 flags, dW_self, dW_nbr, dbias, workspace, ws_bytes, stream);
}

int stack_bwd_weight_impl(const Shape& sh, const void* x, const void* acts, const void* dz,
                          const Sched& sc, int L, int dtype, unsigned flags, float* dW_self,
                          float* dW_nbr, float* dbias, void* workspace, size_t ws_bytes,
                          void* stream) {
    const int d = sh.d;
    int rc;
    if (sh.tokens == 0) {
        if (!dW_self || !dW_nbr) return HCW_ERR_INVALID_ARG;
        return zero_weight_grads(L, d, dW_self, dW_nbr, dbias, (cudaStream_t)stream);
    }
    rc = check_stack_weight(sh, dtype, flags, L, x, acts, dz, dW_self, dW_nbr, dbias, workspace,
                            ws_bytes);
    if (rc) return rc;
    StackWeight a{x, acts, static_cast<const uint8_t*>(dz), sc, L,
                  flags, dW_self, dW_nbr, dbias, static_cast<uint8_t*>(workspace)};
    return dtype == HCW_BF16 ? stack_weight_bf16(sh, a, (cudaStream_t)stream)
                             : stack_weight_f32(sh, a, (cudaStream_t)stream);
}

size_t hcw_stack_train_step_workspace_bytes(int B, int n, int d, int dtype, unsigned flags,
                                            int L) {
    Shape sh;
    if (L < 1 || check_shape(0, -1, B, n, d, dtype, flags, &sh)) return 0;
    return align256(stack_dz_bytes(sh, L) + align256(stack_data_ws(sh, dtype, flags, L)) +
                    stack_weight_ws(sh, dtype, flags, L)) +
           step_fwd_region(sh, dtype, flags, L);
}

int hcw_stack_train_step(const void* x, const void* W_self, const void* W_nbr, const float* bias,
                         const void* dy, int layer0, int L, int dim_override, int B, int n, int d,
                         int dtype, unsigned flags, void* y, void* acts, void* masks, void* dx,
                         float* dW_self, float* dW_nbr, float* dbias, void* workspace,
                         size_t ws_bytes, void* stream) {
    Shape sh;
    if (L < 1) return HCW_ERR_INVALID_ARG;
    int rc = check_shape(layer0, dim_override, B, n, d, dtype, flags, &sh);
    if (rc) return rc;
    return train_step_impl(sh, x, W_self, W_nbr, bias, dy, Sched{nullptr, layer0, dim_override}, L,
                           dtype, flags, y, acts, masks, dx, dW_self, dW_nbr, dbias, workspace,
                           ws_bytes, stream);
}

int hcw_stack_train_step_dims(const void* x, const void* W_self, const void* W_nbr,
                              const float* bias, const void* dy, const int* dims, int L, int B,
                              int n, int d, int dtype, unsigned flags, void* y, void* acts,
                              void* masks, void* dx, float* dW_self, float* dW_nbr, float* dbias,
                              void* workspace, size_t ws_bytes, void* stream) {
    Shape sh;
    if (L < 1) return HCW_ERR_INVALID_ARG;
    int rc = check_shape(0, -1, B, n, d, dtype, flags, &sh);
    if (rc) return rc;
    rc = check_dims(sh, dims, L);
    if (rc) return rc;
    return train_step_impl(sh, x, W_self, W_nbr, bias, dy, Sched{dims, 0, -1}, L, dtype, flags, y,
                           acts, masks, dx, dW_self, dW_nbr, dbias, workspace, ws_bytes, stream);
}

int hcw_stack_bwd(const void* x, const void* acts, const void* masks, const void* dy,
                  const void* W_self, const void* W_nbr, int layer0, int L, int dim_override,
                  int B, int n, int d, int dtype, unsigned flags, void* dx, float* dW_self,
                  float* dW_nbr, float* dbias, void* workspace, size_t ws_bytes, void* stream) {
    Shape sh;
    if (L < 1) return HCW_ERR_INVALID_ARG;
    int rc = check_shape(layer0, dim_override, B, n, d, dtype, flags, &sh);
    if (rc) return rc;
    return stack_bwd_impl(sh, x, acts, masks, dy, W_self, W_nbr,
                          Sched{nullptr, layer0, dim_override}, L, dtype, flags, dx, dW_self,
                          dW_nbr, dbias, workspace, ws_bytes, stream);
}

int hcw_stack_bwd_dims(const void* x, const void* acts, const void* masks, const void* dy,
                       const void* W_self, const void* W_nbr, const int* dims, int L, int B,
                       int n, int d, int dtype, unsigned flags, void* dx, float* dW_self,
                       float* dW_nbr, float* dbias, void* workspace, size_t ws_bytes,
                       void* stream) {
    Shape sh;
    if (L < 1) return HCW_ERR_INVALID_ARG;
    int rc = check_shape(0, -1, B, n, d, dtype, flags, &sh);
    if (rc) return rc;
    rc = check_dims(sh, dims, L);
    if (rc) return rc;
    return stack_bwd_impl(sh, x, acts, masks, dy, W_self, W_nbr, Sched{dims, 0, -1}, L, dtype,
                          flags, dx, dW_self, dW_nbr, dbias, workspace, ws_bytes, stream);
}

size_t hcw_decode_cache_bytes(const int* dims, int layer0, int L, int B, int n, int d) {
    Shape sh;
    if (decode_check(dims, layer0, L, B, n, d, &sh)) return 0;
    size_t slots = 0;
    for (int l = 0; l < L; ++l) slots += (size_t)decode_link(dims, layer0, sh.b, l) + 1;
    return slots * (size_t)B * d * 2;
}

int hcw_decode_step(const void* x_t, const void* W_self, const void* W_nbr, const float* bias,
                    const int* dims, int layer0, int L, int t, int B, int n, int d,
                    unsigned flags, void* cache, void* y_t, void* stream) {
    Shape sh;
    int rc = decode_check(dims, layer0, L, B, n, d, &sh);
    if (rc) return rc;
    // decoding is causal: a hypercube link without the causal rule would read a
    // later position
    if (!(flags & HCW_CAUSAL) || (flags & ~kAllFlags) || t < 0 || t >= n) return HCW_ERR_INVALID_ARG;
    if (!x_t || !W_self || !W_nbr || !cache || !y_t) return HCW_ERR_INVALID_ARG;
    DecodeGeo geo;
    if (!decode_geometry(d, &geo)) return HCW_ERR_UNSUPPORTED;
    const void* ptrs[] = {x_t, W_self, W_nbr, bias, cache, y_t};
    for (const void* q : ptrs)
        if (q && !aligned16(q)) return HCW_ERR_ALIGNMENT;
    const size_t row_bytes = (size_t)B * d * 2;
    const size_t cache_b = hcw_decode_cache_bytes(dims, layer0, L, B, n, d);
    const size_t wb = (size_t)L * d * d * 2;
    if (overlaps(y_t, row_bytes, x_t, row_bytes) || overlaps(y_t, row_bytes, cache, cache_b) ||
        overlaps(cache, cache_b, x_t, row_bytes) || overlaps(cache, cache_b, W_self, wb) ||
        overlaps(cache, cache_b, W_nbr, wb))
        return HCW_ERR_ALIASING;
    cudaStream_t st = (cudaStream_t)stream;
    auto* ring = static_cast<__nv_bfloat16*>(cache);
    const size_t per = (size_t)B * d;
    DecodeLaunch p;
    // ring of layer l: k_l + 1 slots of [B][d] from off[l]; position q in slot q mod (k_l + 1)
    size_t off[kMaxDecodeLayers + 1];
    int kl[kMaxDecodeLayers];
    off[0] = 0;
    for (int l = 0; l < L; ++l) {
        kl[l] = decode_link(dims, layer0, sh.b, l);
        off[l + 1] = off[l] + (size_t)(kl[l] + 1) * per;
    }
    // element offset of the slot of position q in layer l's ring
    auto slot = [&](int l, int q) { return off[l] + (size_t)(q % (kl[l] + 1)) * per; };
    for (int l = 0; l < L; ++l) {
        const int s = dims ? dims[l] : (layer0 + l) % sh.b;
        const bool recv = s >= 0 ? ((t >> s) & 1) != 0 : t >= kl[l];
        p.prow[l] = recv ? (int)(slot(l, t + 1) / d) : -1;   // the slot of t - k_l
        p.out[l] = l == L - 1 ? static_cast<__nv_bfloat16*>(y_t) : ring + slot(l + 1, t);
    }
    if (!map_tiles_sw128(&p.mWs, W_self, (long long)L * d, d, geo.oc, geo.kc / 64) ||
        !map_tiles_sw128(&p.mWn, W_nbr, (long long)L * d, d, geo.oc, geo.kc / 64) ||
        !map_tiles_sw128(&p.mCache, cache, (long long)(off[L] / d), d, 16, d / 64) ||
        !map_tiles_sw128(&p.mX, x_t, B, d, 16, d / 64))
        return HCW_ERR_CUDA;
    p.bias = bias;
    p.ring0 = ring + slot(0, t);
    p.g = geo;
    p.L = L;
    p.B = B;
    p.flags = flags;
    p.timeout_ns = g_timeout_ns;
    p.tc = g_decode_kernel.load(std::memory_order_relaxed) == HCW_DECODE_TCGEN05;
    return launched(launch_decode(p, st), 1);
}

int hcw_set_decode_kernel(int mode) {
    if (mode != HCW_DECODE_WARP_MMA && mode != HCW_DECODE_TCGEN05) return -1;
    return g_decode_kernel.exchange(mode);
}

int hcw_set_stack_kernels(int mode) {
    if (mode != HCW_STACK_AUTO && mode != HCW_STACK_RESIDENT && mode != HCW_STACK_STREAMING)
        return -1;
    return g_stack_kernels.exchange(mode);
}

int hcw_stack_kernels_used(int B, int n, int d, int dtype) {
    Shape sh;
    if (check_shape(0, -1, B, n, d, dtype, 0, &sh)) return -1;
    return dtype == HCW_BF16 && use_resident(sh) ? HCW_STACK_RESIDENT : HCW_STACK_STREAMING;
}

unsigned long long hcw_launch_count(void) { return g_launches.load(); }

int hcw_sync_status(void* stream) {
    if (cudaStreamSynchronize((cudaStream_t)stream) != cudaSuccess) return HCW_ERR_CUDA;
    int word = 0, word_res = 0, word_dec = 0, word_blk = 0, word_gemm = 0;
    if (error_word_read_clear(&word) != cudaSuccess ||
        res_error_word_read_clear(&word_res) != cudaSuccess ||
        decode_error_word_read_clear(&word_dec) != cudaSuccess ||
        block_error_word_read_clear(&word_blk) != cudaSuccess ||
        gemm_error_word_read_clear(&word_gemm) != cudaSuccess)
        return HCW_ERR_CUDA;
    if (!word) word = word_res;
    if (!word) word = word_dec;
    if (!word) word = word_blk;
    if (!word) word = word_gemm;
    if (word == HCW_ERR_INVALID_ARG) return HCW_ERR_INVALID_ARG;
    if (word) return word == HCW_ERR_TIMEOUT ? HCW_ERR_TIMEOUT : HCW_ERR_CUDA;
    return HCW_OK;
}

int hcw_selftest_wait(long long timeout_ns, void* stream) {
    if (timeout_ns < 1000 || timeout_ns > 10000000000ll) return HCW_ERR_INVALID_ARG;
    return launched(launch_wait_selftest((unsigned long long)timeout_ns, (cudaStream_t)stream),
                    1);
}

}  // extern "C"

// ---------------------------------------------------------------------------
// Weight gradient without caller-provided workspace.
//
// Some callers cannot allocate device memory when they call in: a plugin
// host that hands out only its own input/output buffers, code running in an
// allocator-free section, or a process whose allocator is owned by someone
// else.  hcw_layer_bwd_weight needs a scratch workspace (split-K partial
// sums of dW and column-sum partials of dbias), so this variant keeps that
// scratch in a fixed array linked into the library instead.  Every device
// that loads the library reserves the array until the process exits.
static constexpr size_t kNoAllocScratchBytes = (size_t)32 << 20;   // 32 MiB
static __device__ __align__(256) unsigned char hcw_noalloc_scratch[kNoAllocScratchBytes];

namespace {
// The host-side name of the array is a stand-in, not a device address: ask
// the runtime for the address on the current device.  The first call on a
// device loads the module there (its set-up); later calls are a lookup.  The
// address is asked for on every call rather than kept, so that a context
// torn down and made again (cudaDeviceReset) never leaves a stale address.
int noalloc_scratch(void** out) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, hcw_noalloc_scratch) != cudaSuccess || !p) return HCW_ERR_CUDA;
    *out = p;
    return HCW_OK;
}
}  // namespace

extern "C" {

int hcw_layer_bwd_weight_noalloc(const void* x, const void* dz, int layer, int dim_override,
                                 int B, int n, int d, int dtype, unsigned flags,
                                 float* dW_self, float* dW_nbr, float* dbias, void* stream) {
    Shape sh;
    int rc = check_shape(layer, dim_override, B, n, d, dtype, flags, &sh);
    if (rc) return rc;
    // the fixed scratch must hold what the workspace would: larger sizes are
    // rejected first, before any pointer is looked at
    if (ws_layout(sh.tokens, d, dtype, flags).w_bytes > kNoAllocScratchBytes)
        return HCW_ERR_WORKSPACE;
    if (!dW_self || !dW_nbr) return HCW_ERR_INVALID_ARG;
    const void* ptrs[] = {x, dz, dW_self, dW_nbr, dbias};
    for (const void* q : ptrs)
        if (q && !aligned16(q)) return HCW_ERR_ALIGNMENT;
    if (sh.tokens > 0 && (!x || !dz)) return HCW_ERR_INVALID_ARG;
    const size_t ab = sh.act_bytes, gb = (size_t)d * d * 4;
    if (overlaps(dW_self, gb, dW_nbr, gb) || overlaps(dbias, (size_t)d * 4, dW_self, gb) ||
        overlaps(dbias, (size_t)d * 4, dW_nbr, gb) || overlaps(dW_self, gb, x, ab) ||
        overlaps(dW_nbr, gb, x, ab) || overlaps(dW_self, gb, dz, ab) ||
        overlaps(dW_nbr, gb, dz, ab) || overlaps(dbias, (size_t)d * 4, x, ab) ||
        overlaps(dbias, (size_t)d * 4, dz, ab))
        return HCW_ERR_ALIASING;
    void* scratch = nullptr;
    rc = noalloc_scratch(&scratch);
    if (rc) return rc;
    // Every scratch byte the kernels read is written earlier in the same call
    // (each split writes its whole slab, each column-sum chunk its row), so
    // nothing has to be cleared between calls.
    return layer_dw_impl(sh, dtype, x, dz, flags, dW_self, dW_nbr, dbias,
                         static_cast<uint8_t*>(scratch), (cudaStream_t)stream);
}

}  // extern "C"
