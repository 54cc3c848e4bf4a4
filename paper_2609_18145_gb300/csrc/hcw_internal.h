// hcw_internal.h -- launch interfaces shared by the translation units of
// libhcw (not part of the public ABI, which is include/hcw.h).
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

namespace hcw {

// MODE_DWF: weight gradients of a run of layers, one unit per (layer, output
// tile) that accumulates the self and the partner part together.
// MODE_DWP: the same on pairs of SMs (cta_group::2, 256-row tiles, BN >= 128).
// MODE_FDX: a stacked forward and the stack's input gradient in one launch on
// pairs of SMs: layers [0, n_fwd) are forward layers, the rest input-gradient
// layers from the top down.
enum TcMode { MODE_FWD = 0, MODE_DX = 1, MODE_DW = 2, MODE_DWF = 3, MODE_DWP = 4, MODE_FDX = 5 };

// Work description of one tensor-core launch (see hcw_tc.cu for the unit
// decomposition).  Row indices are "compressed": for a fixed value beta of
// bit s, q = HI * k + lo enumerates the Mh = B*n/2 positions whose bit s is
// beta; the position (within the flattened [B*n] token axis) is
// HI * 2k + beta * k + lo.
struct TcParams {
    int d;          // feature width
    int Mh;         // positions per value of bit s: B * n / 2
    int nK;         // d / 64: K-steps per part (FWD, DX)
    // FWD / DX units
    int n_rb;       // ceil(Mh / 128) row blocks per bit value
    int n_nt;       // d / BN output column tiles
    int n_full;     // number of bit values whose rows take both parts (1 or 2)
    int full_bit0;  // bit value of the first full group
    int full_bit1;  // bit value of the second full group (if n_full == 2)
    int half_bit;   // bit value of the rows that take only the self part, -1 if none
    // DW units
    int n_ot;       // ceil(d / 128) output row tiles (o)
    int qb;         // ceil(Mh / 64) token blocks per bit value
    int nkb_self;   // token blocks of the self part: 2 * qb
    int nkb_nbr;    // token blocks of the partner part: qb (causal) or 2 * qb
    int kb_per_unit;
    int splits_self;
    int splits_nbr;
    int causal;
    int n_units;    // units of one layer
    int seq_n;      // launches with shift layers: positions per sample
    // epilogue
    unsigned flags;
    int splits_max;
    unsigned long long timeout_ns;
};

// The per-layer part of a launch.  A forward launch may cover a run of
// layers (the stacked forward); every other launch covers one layer.
struct TcLayer {
    int s;                        // cube dimension
    int k;                        // 2^s
    const float* bias;            // FWD bias or null
    uint32_t* mout;               // FWD: ReLU mask words [tokens][d/32], bit e = (z > 0), or null
    __nv_bfloat16* zout;          // FWD: bf16 pre-activation (layer API), or null
    bool out;                     // DX: the input gradient dx is stored (map 4)
    const uint32_t* mprev;        // DX: ReLU mask words of the layer below (fused ReLU grad)
    bool dz_out;                  // DX: dz of the layer below = dx * mask is stored (map 5)
    float* colsum;                // DW: dbias = column sums of dz; with the self part split,
                                  // the sums of each split, [split][d]
    float* dws;                   // MODE_DWF: dW_self, dW_nbr [d][d] fp32 (stored directly)
    float* dwn;
    // FWD / DX of one layer: the partner part reads the same rows of a second
    // tensor (map 5) instead of the partner rows of map 0 -- a shift layer of
    // Eq. (1), whose partner rows are materialised row-aligned beforehand
    bool pair_rows;
    // DX of a stacked launch: the residual term (map 3) when it is one of the
    // launch's own g buffers, [tokens][d] bf16; each epilogue warp discards its
    // patch's L2 lines once it has read them (nothing reads them again, and
    // the buffer is written anew two layers later), or null
    const __nv_bfloat16* g_discard;
    // A shift layer of Eq. (1) by `shift` positions (0: a hypercube layer).
    // MODE_DWP: its rows are grouped as a hypercube view with k = 64 (64
    // consecutive positions per stage); map 2 views the layer input as (64
    // features, position, sample, d / 64 blocks), so the rows p - shift of a
    // stage's positions p load as one box, the ones before the sample's start
    // as zeros.  Stacked FWD / DX: the rows are grouped with k = 128 (runs of
    // 128 positions), and map 0 views the input as (features, position,
    // sample, 1), so the partner rows p - shift (forward) or p + shift (input
    // gradient) load as one box, zeros outside the sample
    int shift;
    // MODE_DWP started early (TcLaunch::dep_counters): the row of the
    // completion counters that counts this layer's dz
    int dep_row;
};

// Columns of one epilogue patch (the inner extent of the 32-row residual and
// output boxes of the row kernels): 64 for 256-column tiles, else 32.
constexpr int epi_patch_cols(int BN) { return BN >= 256 ? 64 : 32; }

constexpr int kMaxStackLayers = 16;   // layers per stacked-forward launch
constexpr int kMaxStepLayers = 2 * kMaxStackLayers;   // forward + input-gradient launch

// maps[l][0..5] = tmA, tmB0, tmB1, tmE0, tmE1, tmE2 of layer l, as documented
// at hcw_tc_kernel in hcw_tc.cu.
constexpr int kTcMaps = 6;
template <int NL>
struct TcLaunch {
    CUtensorMap maps[NL][kTcMaps];
    TcLayer layer[NL];
    TcParams p;
    int n_layers;
    // stacked forward: completion counters [n_layers][n_chunks] (zeroed before
    // the launch), one per layer and 128-token chunk, counting output elements
    int* counters;
    int n_chunks;
    int tokens;
    int* sched;   // stacked launches: next unit to hand out (zeroed per launch), or null
    // Stacked input gradient, first run of layers: the launch itself writes the
    // top layer's dz = dy * act'(z) (mask bits; a plain copy without them)
    // before its units read it, counting each 128-token chunk in in_counters
    // (zeroed before the launch).  Null top_dy: that dz is already in memory.
    const __nv_bfloat16* top_dy;
    const uint32_t* top_mask;
    __nv_bfloat16* top_dz;
    int* in_counters;
    // Stacked input gradient with ReLU and residual: completion counters
    // [n_layers][n_chunks] of each layer's output gradient g (the residual term
    // of the layer below), counted apart from dz so that dz -- the operand the
    // next layer's MMAs wait for -- is published before g is stored.  Null:
    // g is dz (or absent) and the counters above cover it.
    int* g_counters;
    // MODE_FDX: the number of forward layers; the last of them also writes the
    // top layer's dz = dy * act'(z) (top_dy, top_dz) for the layers after it
    int n_fwd;
    // MODE_DWP launched as a programmatic dependent of the MODE_FDX launch that
    // writes its dz: that launch's completion counters [rows][n_chunks]
    // (layer.dep_row picks a layer's row).  A unit first waits until every
    // chunk of its layer's dz is complete; the layers go from the top down (the
    // order in which the input gradient finishes them).  Null: the operands
    // are complete when the launch starts.
    const int* dep_counters;
    // MODE_FDX followed by such a weight-gradient launch: only pairs
    // [0, tail_pairs) take units of the last layer (the input gradient of
    // layer 0, which nothing in the step reads); the others leave once every
    // earlier unit is claimed, and the weight gradient starts on their SMs.
    // 0: every pair takes units to the end.
    int tail_pairs;
};

// Launch one tensor-core pass (one layer).
cudaError_t launch_tc(int mode, int BN, const TcLaunch<1>& L, int grid, cudaStream_t stream);
// Launch a run of layers: MODE_FWD (layers in order) or MODE_DX (layers from
// the top down) with chunk-level dependencies, or MODE_DW (independent
// layers, the long self-part units of every layer first).
// MODE_DWP with L.dep_counters set is launched as a programmatic dependent of
// the preceding kernel in the stream.
cudaError_t launch_tc_stack(int mode, int BN, const TcLaunch<kMaxStackLayers>& L, int grid,
                            cudaStream_t stream);
// The same for MODE_FWD / MODE_DX on clusters of two CTAs (256-row tiles,
// cta_group::2; BN 256, even grid).  L.p counts pair units: row-block pairs.
cudaError_t launch_tc_stack_pair(int mode, int BN, const TcLaunch<kMaxStackLayers>& L, int grid,
                                 cudaStream_t stream);
// MODE_FDX on clusters of two CTAs (BN 256 or 128, even grid): L.n_fwd forward
// layers followed by the input gradient of those layers, top down.
cudaError_t launch_tc_step_pair(int BN, const TcLaunch<kMaxStepLayers>& L, int grid,
                                cudaStream_t stream);

// ---- Resident stacked launches (hcw_res.cu) ----
// A cluster of two CTAs keeps 256 consecutive tokens (whole samples, n <= 256)
// of the running activations (forward) or gradient (input gradient) in shared
// memory through every layer of the run; only the weights stream in.
enum ResOut {
    RES_Y = 0,    // forward: y_l, bf16 [tokens][d] (+ ReLU mask words in mout)
    RES_DZ = 1,   // input gradient: dz_{l-1} = bf16(g_{l-1}) * mask_{l-1}, bf16
    RES_DX = 2,   // input gradient of the stack's first layer: dx = bf16(g_{-1})
    RES_G = 3     // input gradient continued by a later launch: g_{l-1}, fp32
};

struct ResLayer {
    int s;                    // cube dimension
    int out_kind;             // ResOut
    void* out;                // where the layer's result goes (see ResOut)
    const float* bias;        // forward: bias [d] or null
    uint32_t* mout;           // forward: ReLU mask words [tokens][d/32] or null
    const uint32_t* mprev;    // RES_DZ: mask words of the layer below, or null (no ReLU)
};

struct ResLaunch {
    // per layer (in processing order: the forward bottom up, the input
    // gradient top down): W_self and W_nbr as the B operand, half a column
    // chunk per CTA (forward: K-major 2-D boxes; input gradient: MN-major
    // 3-D block boxes)
    CUtensorMap wmap[kMaxStackLayers][2];
    // per layer: its bf16 output (y_l, dz_{l-1} or dx) as (8 features, tokens,
    // d/8) with 64-token x 1-chunk boxes: where the rows change CTA (n = 256),
    // the next layer's A tile is reloaded from it chunk by chunk
    CUtensorMap imap[kMaxStackLayers];
    ResLayer layer[kMaxStackLayers];
    const void* in;           // forward: the first layer's input, bf16 [tokens][d];
                              // input gradient: the top layer's output gradient,
                              // bf16 dy, or fp32 g (in_f32) from an earlier launch
    int in_f32;
    const uint32_t* in_mask;  // input gradient: the top layer's mask words, or null
    __nv_bfloat16* in_dz;     // input gradient: the top layer's dz is stored here
    float* gscratch;          // input gradient, residual: fp32 [tokens][d] used when the
                              // rows change CTA between layers (n = 256)
    int n_layers;
    int d, n, tokens;
    unsigned flags;           // HCW_CAUSAL | HCW_RESIDUAL | HCW_ACT_RELU
    unsigned long long timeout_ns;
};

// Whether the resident kernels take this shape: d in {128, 256, 512},
// n <= 256, whole 256-token tiles.
bool res_supported(int d, int n, long long tokens);
// Launch MODE_FWD or MODE_DX over tokens / 256 clusters of two CTAs.
cudaError_t launch_res(int mode, const ResLaunch& L, cudaStream_t stream);
// Read the resident kernels' error word and reset it to 0 (synchronous).
cudaError_t res_error_word_read_clear(int* word);

// ---- One-token decode (hcw_decode.cu) ----
constexpr int kMaxDecodeLayers = 64;   // layers of one decode step
// Split of one decode layer over a cluster: CTA q of csize owns output columns
// [q oc, (q + 1) oc); weights stream in K chunks of kc through `stages` stages.
struct DecodeGeo {
    int d, oc, csize, kc, nchunks, stages;
};
// false: no cluster split for this d (the decode supports d <= 1024)
bool decode_geometry(int d, DecodeGeo* g);
size_t decode_smem_bytes(const DecodeGeo& g);
// One position of a decode: per layer l, out[l] = act(in_l Ws_l^T +
// partner_l Wn_l^T + bias_l) (+ in_l) over B rows of width d (bf16 in and
// out, fp32 accumulation), in_0 = x_t and in_l = out[l - 1]; partner_l is the
// B rows from row prow[l] of the cache map (prow[l] < 0: no partner part).
// x_t is also copied to ring0.  Maps (128-byte swizzle, matrices viewed as
// (64 features, rows, 64-feature tiles)): mWs / mWn over [L d][d] with box
// (64, oc, kc / 64), mCache over the rings as [rows][d] and mX over x_t [B][d]
// with box (64, 16, d / 64).
struct DecodeLaunch {
    CUtensorMap mWs, mWn, mCache, mX;
    int prow[kMaxDecodeLayers];
    __nv_bfloat16* out[kMaxDecodeLayers];
    const float* bias;
    __nv_bfloat16* ring0;
    DecodeGeo g;
    int L, B;
    unsigned flags;
    unsigned long long timeout_ns;
    bool tc;   // contraction on tcgen05 (else the warp-level MMA)
};
// One launch of every layer of the step: a cluster per 16 rows.
cudaError_t launch_decode(const DecodeLaunch& p, cudaStream_t st);
// Read the decode kernel's error word and reset it to 0 (synchronous).
cudaError_t decode_error_word_read_clear(int* word);

// Launch `kern` with programmatic stream serialization: it may start while the
// kernel before it in the stream finishes, and must call pdl_wait()
// (hcw_ptx.cuh) before it touches memory that kernel reads or writes.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t st, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// ---- Plain GEMMs of the character-LM block (hcw_gemm.cu) ----
// Row-major C[M][N] (fp32) = op(A) op(B), bf16 operands, fp32 accumulation;
// A is [M][K] ([K][M] when ta), B is [K][N] ([N][K] when tb).  split_ws
// (split_ws_bytes, 16-byte aligned, may be NULL) holds the fp32 partial sums
// of a K split; *launches receives the kernels enqueued (1 or 2).
cudaError_t gemm_bf16_f32(int M, int N, int K, const void* A, bool ta, const void* B, bool tb,
                          float* C, float* split_ws, size_t split_ws_bytes, cudaStream_t st,
                          int* launches);
// `batch` independent products contracted over their rows, in one launch:
// C[b] (fp32 [M][N]) = A_b^T B_b with A_b the row-major [K][M] bf16 matrix at
// A + b * a_batch_bytes and B_b the row-major [K][N] at B + b * b_batch_bytes
// (the weight gradients of a run of layers); C[b] at C + b * M * N.  Each
// output tile takes the whole K range (no partial sums).
cudaError_t gemm_bf16_f32_batched(int M, int N, int K, const void* A, size_t a_batch_bytes,
                                  const void* B, size_t b_batch_bytes, float* C, int batch,
                                  cudaStream_t st, int* launches);
// Epilogues of the GEMM: fp32 C; out = bf16(relu(C + bias[col])); or
// out = bf16(aux[row][col] > 0 ? C : 0), with colsum[col] (if given) += the
// column sums of out.  out and aux are [M][N] bf16.
enum GemmEpiKind { EPI_F32 = 0, EPI_BIAS_RELU = 1, EPI_RELU_GRAD = 2 };
struct GemmEpi {
    int kind;
    const float* bias;
    const __nv_bfloat16* aux;
    __nv_bfloat16* out;
    float* colsum;
};
// gemm_bf16_f32 with an epilogue (C unused unless epi.kind is EPI_F32; only
// fp32 output splits K).
cudaError_t gemm_bf16(int M, int N, int K, const void* A, bool ta, const void* B, bool tb,
                      float* C, const GemmEpi& epi, float* split_ws, size_t split_ws_bytes,
                      cudaStream_t st, int* launches);
// Read the GEMM kernel's error word and reset it to 0 (synchronous).
cudaError_t gemm_error_word_read_clear(int* word);

// ---- Character-LM block (hcw_block.cu) ----
// Read the block kernels' error word and reset it to 0 (synchronous).
cudaError_t block_error_word_read_clear(int* word);
// HCW_OK after counting `kernels` launches if e is cudaSuccess, else HCW_ERR_CUDA
// (the launch counter lives with the C API in hcw_api.cu).
int count_launch(cudaError_t e, int kernels);

// Dynamic shared memory the tensor-core kernel uses for this N tile.
size_t tc_smem_bytes(int BN);
int tc_stages(int BN);

// ---- SIMT kernels (hcw_simt.cu) ----
cudaError_t launch_f32_fwd(const float* x, const float* Ws, const float* Wn, const float* bias,
                           int s, int B, int n, int d, unsigned flags, float* y, float* z,
                           uint32_t* mout, cudaStream_t st);
// dz = dy where the ReLU mask bit is set, else 0 (masks [rows][ceil(d/32)] words)
cudaError_t launch_relu_grad_mask_f32(const float* dy, const uint32_t* mask, float* dz,
                                      long long rows, int d, cudaStream_t st);
cudaError_t launch_relu_grad_mask_bf16(const __nv_bfloat16* dy, const uint32_t* mask,
                                       __nv_bfloat16* dz, long long rows, int d,
                                       cudaStream_t st);
cudaError_t launch_f32_dx(const float* dz, const float* dy, const float* Ws, const float* Wn,
                          int s, int B, int n, int d, unsigned flags, float* dx,
                          cudaStream_t st);
cudaError_t launch_f32_dw(const float* x, const float* dz, int s, int B, int n, int d,
                          unsigned flags, float* dWs, float* dWn, cudaStream_t st);
// dz = dy * (z > 0), elementwise over count elements (T = float or bf16)
cudaError_t launch_relu_grad_f32(const float* dy, const float* z, float* dz, size_t count,
                                 cudaStream_t st);
cudaError_t launch_relu_grad_bf16(const __nv_bfloat16* dy, const __nv_bfloat16* z,
                                  __nv_bfloat16* dz, size_t count, cudaStream_t st);
// dbias[o] = sum_t dz[t][o], deterministic two-pass column sum.
size_t colsum_workspace_bytes(long long rows, int d);
cudaError_t launch_colsum_f32(const float* dz, long long rows, int d, float* partial,
                              float* out, cudaStream_t st);
cudaError_t launch_colsum_bf16(const __nv_bfloat16* dz, long long rows, int d, float* partial,
                               float* out, cudaStream_t st);
// The same for `batch` consecutive [rows][d] matrices: out [batch][d], partial
// batch * colsum_workspace_bytes(rows, d).
cudaError_t launch_colsum_bf16_batched(const __nv_bfloat16* dz, int batch, long long rows, int d,
                                       float* partial, float* out, cudaStream_t st);
// out_w[o][k] = sum_{s < splits_w} partial[w][s][o][k] for w in {self, nbr};
// `layers` such problems, partials part_stride floats apart, outputs
// out_stride floats apart; with bpart, also dbias[l][o] = sum over the
// splits_self splits of bpart[l][s][o]
cudaError_t launch_splitk_reduce(const float* partial, int splits_max, int splits_self,
                                 int splits_nbr, int d, float* dWs, float* dWn,
                                 cudaStream_t st, int layers = 1, size_t part_stride = 0,
                                 size_t out_stride = 0, const float* bpart = nullptr,
                                 float* dbias = nullptr);
cudaError_t launch_partner_table(int s, int n, unsigned flags, int* out, cudaStream_t st);
// out[b][i] = in[b][i - k] where 0 <= i - k < n, else 0 (bf16 [rows][d], k of
// either sign): the row-aligned partner operand of a shift layer.
cudaError_t launch_shift_rows_bf16(const __nv_bfloat16* in, __nv_bfloat16* out, long long rows,
                                   int n, int d, int k, cudaStream_t st);
cudaError_t launch_wait_selftest(unsigned long long timeout_ns, cudaStream_t st);
// Read the current device's error word and reset it to 0 (synchronous).
cudaError_t error_word_read_clear(int* word);

}  // namespace hcw
