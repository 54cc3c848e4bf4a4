/*
 * hcw.h -- C ABI of the rotated-hypercube mixing layer on GB300 (sm_103a).
 *
 * Method (arXiv 2609.18145, "Reaching Every Position Without Searching"):
 *   Sec. 3.1  positions i = 0..n-1 of a sample (n = 2^b) are vertices of a
 *             b-cube; layer l links i with its partner p(i) = i XOR 2^s,
 *             s = l mod b.  Causal rule: only the earlier endpoint is kept,
 *             so i receives from p(i) iff bit s of i is set (p(i) = i - 2^s).
 *   Eq. (1)   y_i = W_self x_i + W_off x_{i-k}: two d x d linear maps, no
 *             input-dependent routing.  W_off is called W_nbr here.
 *   Sec. 3.3  stacks: "rot" (s = l mod b) and the "fixed" control (one
 *             dimension at every layer, selected by dim_override >= 0).
 *
 * Conventions for every entry point
 *   - Matrices act on column vectors as in Eq. (1) and are stored row-major
 *     as W[o][k] (d_out x d_in), i.e. z[i][o] = sum_k W[o][k] x[i][k].
 *   - Activations are [B][n][d] row-major (d contiguous), samples
 *     independent (no link crosses a sample).
 *   - Optional epilogue (the paper states none; flags select it):
 *       z = W_self x_i + m_i W_nbr x_{p(i)} + bias,  y = act(z) + (RESIDUAL ? x_i : 0)
 *     with act = identity, or ReLU (ReLU'(0) = 0) under HCW_ACT_RELU.
 *   - dtype HCW_BF16: x, W, y, z, dy, dx are bf16; products accumulate in
 *     fp32; stored activations are rounded to bf16 (nearest, ties to even).
 *     Needs d % 64 == 0.  dtype HCW_F32: all of those are fp32 (any d >= 1).
 *     bias, dW_self, dW_nbr and dbias are always fp32.
 *   - Pointers are device pointers unless stated; all must be 16-byte
 *     aligned.  The caller owns every buffer; the library allocates no
 *     device memory.  Outputs are overwritten, never accumulated into.
 *   - Calls are asynchronous on `stream` (a cudaStream_t passed as void*,
 *     NULL = legacy default stream).  The return value reports argument
 *     validation and launch errors.  A kernel that gives up on a bounded
 *     wait records HCW_ERR_TIMEOUT in a per-device error word, read (and
 *     cleared) by hcw_sync_status.
 *   - n must be a power of two >= 2; B >= 0 (B = 0 does nothing); a
 *     violated requirement returns a non-zero hcw_status and launches
 *     nothing.
 */
#ifndef HCW_H
#define HCW_H

#include <stddef.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    HCW_OK = 0,
    HCW_ERR_INVALID_ARG = 1,   /* bad size, NULL required pointer, bad flag or dimension */
    HCW_ERR_UNSUPPORTED = 2,   /* valid request this build does not handle (e.g. bf16 with d % 64) */
    HCW_ERR_ALIGNMENT = 3,     /* a pointer is not 16-byte aligned */
    HCW_ERR_ALIASING = 4,      /* an output overlaps an input it must not overlap */
    HCW_ERR_CUDA = 5,          /* a CUDA runtime/driver call failed */
    HCW_ERR_TIMEOUT = 6,       /* a kernel gave up on a bounded wait (see hcw_sync_status) */
    HCW_ERR_WORKSPACE = 7      /* workspace NULL or smaller than hcw_workspace_bytes */
} hcw_status;

typedef enum { HCW_BF16 = 0, HCW_F32 = 1 } hcw_dtype;

#define HCW_CAUSAL   1u   /* Sec. 3.1 causal rule: receive only from the earlier endpoint */
#define HCW_RESIDUAL 2u   /* y = act(z) + x */
#define HCW_ACT_RELU 4u   /* act = ReLU (else identity, which is Eq. (1) itself) */

/* Library version (major * 10000 + minor * 100 + patch). */
int hcw_version(void);

/* Human-readable name of a status code.  Never NULL. */
const char* hcw_status_string(int status);

/*
 * Partner table of one layer, computed on the HOST (Sec. 3.1).
 *   partner[i] = i XOR 2^s if position i receives at this layer, else -1,
 *   for i = 0..n-1; s = layer mod log2 n, or dim_override if >= 0.
 *   partner: host array of n ints, written.
 * Returns HCW_ERR_INVALID_ARG for n not a power of two >= 2, dim_override >= log2 n,
 * layer < 0 or partner NULL.
 */
int hcw_partner_table(int layer, int dim_override, int n, unsigned flags, int* partner);

/*
 * The same table computed by the device index code that the kernels use,
 * written to device memory partner_dev[n] (int32) on `stream`.
 */
int hcw_partner_table_device(int layer, int dim_override, int n, unsigned flags,
                             int* partner_dev, void* stream);

/*
 * One mixing layer forward (Sec. 3.1 wiring, Eq. (1) maps, epilogue above).
 *   x       [B][n][d]  input (dtype)
 *   W_self  [d][d]     W[o][k] (dtype)
 *   W_nbr   [d][d]     W[o][k] (dtype)
 *   bias    [d] fp32 or NULL (no bias)
 *   layer   layer index l >= 0 (dimension s = l mod log2 n)
 *   dim_override  -1 for the rotated rule, else the fixed dimension s
 *   y       [B][n][d]  output (dtype); must not overlap x, W, bias or z_save
 *   z_save  [B][n][d]  pre-activation z (dtype) or NULL; needed by
 *                      hcw_layer_bwd when HCW_ACT_RELU is set
 */
int hcw_layer_fwd(const void* x, const void* W_self, const void* W_nbr, const float* bias,
                  int layer, int dim_override, int B, int n, int d, int dtype, unsigned flags,
                  void* y, void* z_save, void* stream);

/*
 * Bytes of device workspace hcw_layer_bwd / hcw_stack_bwd need for these
 * sizes and flags (0 is possible).  Depends on the device's SM count, so
 * query it with the target device current.
 */
size_t hcw_workspace_bytes(int B, int n, int d, int dtype, unsigned flags);

/*
 * One mixing layer backward (the chain rule through the forward above):
 *   dz = dy * act'(z)
 *   dx_i = W_self^T dz_i + m_{p(i)} W_nbr^T dz_{p(i)} + (RESIDUAL ? dy_i : 0)
 *          -- a gather, since p is an involution: no atomics
 *   dW_self = sum_i dz_i x_i^T, dW_nbr = sum_i m_i dz_i x_{p(i)}^T, dbias = sum_i dz_i
 *   x, dy   [B][n][d] (dtype); z_save [B][n][d] (dtype), required iff HCW_ACT_RELU
 *   dx      [B][n][d] (dtype) output; must not overlap any input
 *   dW_self, dW_nbr  [d][d] fp32 outputs (same W[o][k] layout as the weights)
 *   dbias   [d] fp32 output or NULL
 *   workspace/ws_bytes  device scratch of at least hcw_workspace_bytes(...)
 *   bytes (NULL allowed when that is 0); contents need not be initialised.
 * dW sums are reduced in a fixed order: results are deterministic.
 */
int hcw_layer_bwd(const void* x, const void* z_save, const void* dy,
                  const void* W_self, const void* W_nbr,
                  int layer, int dim_override, int B, int n, int d, int dtype, unsigned flags,
                  void* dx, float* dW_self, float* dW_nbr, float* dbias,
                  void* workspace, size_t ws_bytes, void* stream);

/*
 * The two halves of hcw_layer_bwd, for callers that schedule them
 * separately (e.g. the weight gradient on a second stream).
 *
 * hcw_layer_bwd_data: dx_i = W_self^T dz_i + m_{p(i)} W_nbr^T dz_{p(i)}
 *                            + (RESIDUAL ? dy_i : 0)
 *   dz [B][n][d] (dtype): gradient at the pre-activation, dy * act'(z)
 *   dy [B][n][d] (dtype): gradient at the output, read only under
 *                         HCW_RESIDUAL (may be NULL otherwise)
 *   dx [B][n][d] (dtype) output.  One kernel launch; no workspace.
 *
 * hcw_layer_bwd_weight: dW_self = sum_i dz_i x_i^T,
 *   dW_nbr = sum_i m_i dz_i x_{p(i)}^T, dbias = sum_i dz_i (if not NULL).
 *   workspace of at least hcw_layer_bwd_weight_workspace_bytes(...) bytes.
 *   Deterministic (fixed-order reductions).
 */
int hcw_layer_bwd_data(const void* dz, const void* dy, const void* W_self, const void* W_nbr,
                       int layer, int dim_override, int B, int n, int d, int dtype,
                       unsigned flags, void* dx, void* stream);

size_t hcw_layer_bwd_weight_workspace_bytes(int B, int n, int d, int dtype, unsigned flags);

int hcw_layer_bwd_weight(const void* x, const void* dz, int layer, int dim_override, int B,
                         int n, int d, int dtype, unsigned flags, float* dW_self,
                         float* dW_nbr, float* dbias, void* workspace, size_t ws_bytes,
                         void* stream);

/*
 * Stack of L layers (Sec. 3.3 "rot": layer l uses s = (layer0 + l) mod log2 n,
 * or dim_override for every layer).
 *   W_self, W_nbr  [L][d][d]; bias [L][d] fp32 or NULL
 *   y      [B][n][d] output of the last layer
 *   acts   [L-1][B][n][d] outputs of layers 0..L-2 (= inputs of layers
 *          1..L-1), written; required when L > 1 (kept for the backward)
 *   masks  with HCW_ACT_RELU: [L][B][n][ceil(d/32)] uint32 words, written:
 *          bit (o % 32) of word o/32 of token t is (z[t][o] > 0) -- the
 *          one bit per activation that the ReLU backward needs (d/8 bytes
 *          per token instead of the pre-activation itself); may be NULL
 *          when no backward follows.  Ignored without HCW_ACT_RELU.
 *   workspace/ws_bytes  at least hcw_stack_fwd_workspace_bytes(...) bytes of
 *          device scratch (NULL allowed when that is 0).
 * bf16: runs of up to 16 layers go in one persistent launch; a tile of
 * layer l starts as soon as the rows it reads (its own and its partners')
 * have been written by layer l-1, tracked per 128-token chunk.
 */
int hcw_stack_fwd(const void* x, const void* W_self, const void* W_nbr, const float* bias,
                  int layer0, int L, int dim_override, int B, int n, int d, int dtype,
                  unsigned flags, void* y, void* acts, void* masks, void* workspace,
                  size_t ws_bytes, void* stream);

/*
 * hcw_stack_fwd with an explicit schedule (Sec. 3.3 "Schedules", and the
 * variants of Sec. 4, "Order does not matter; coverage does": a random
 * permutation of the dimensions, a Gray-code order): stack layer l uses cube
 * dimension dims[l] instead of (layer0 + l) mod log2 n.
 *   dims   host array of L ints, read during the call (HCW_ERR_INVALID_ARG if
 *          NULL or out of range).  An entry s in [0, log2 n) is the hypercube
 *          link along dimension s ("jump 2^s" of App. A); an entry -k with
 *          1 <= k < n is Eq. (1)'s shift itself: position i takes x_{i-k}
 *          when i >= k within its sample ("near" of App. A is -1, the
 *          "local" schedule of Sec. 3.3).  A shift links the earlier position
 *          to the later one whether or not HCW_CAUSAL is set.
 * Schedules with a shift layer run layer by layer (bf16: the single-layer
 * tensor-core launches, the shifted partner rows materialised row-aligned in
 * the workspace); others run on the stacked launches.
 * Every other argument, the workspace and the outputs as for hcw_stack_fwd;
 * hcw_stack_bwd_dims with the same dims is its backward.
 */
int hcw_stack_fwd_dims(const void* x, const void* W_self, const void* W_nbr, const float* bias,
                       const int* dims, int L, int B, int n, int d, int dtype, unsigned flags,
                       void* y, void* acts, void* masks, void* workspace, size_t ws_bytes,
                       void* stream);

/* Workspace bytes hcw_stack_fwd needs for these sizes and L layers (0 is possible). */
size_t hcw_stack_fwd_workspace_bytes(int B, int n, int d, int dtype, unsigned flags, int L);

/*
 * Backward of hcw_stack_fwd, layers L-1 down to 0.
 *   x, acts, masks as given to / written by hcw_stack_fwd (masks required
 *   iff HCW_ACT_RELU); dy [B][n][d] gradient of y.
 *   dx [B][n][d] gradient of x (output); dW_self, dW_nbr [L][d][d] and
 *   dbias [L][d] (or NULL) fp32 outputs.
 *   workspace: at least hcw_stack_workspace_bytes(...) bytes.
 * bf16: the input gradients of runs of up to 16 layers go in one persistent
 * launch (top down, a tile starting as soon as the rows it reads are
 * written), whose kernel also applies the ReLU gradient of the layer below;
 * then one launch computes the weight and bias gradients of up to 16 layers
 * (whole token range per tile, no split reduction).  The workspace keeps
 * every layer's dz.
 */
int hcw_stack_bwd(const void* x, const void* acts, const void* masks, const void* dy,
                  const void* W_self, const void* W_nbr, int layer0, int L, int dim_override,
                  int B, int n, int d, int dtype, unsigned flags,
                  void* dx, float* dW_self, float* dW_nbr, float* dbias,
                  void* workspace, size_t ws_bytes, void* stream);

/*
 * Backward of hcw_stack_fwd_dims: hcw_stack_bwd with the schedule dims (host
 * array of L layers, as given to the forward).
 */
int hcw_stack_bwd_dims(const void* x, const void* acts, const void* masks, const void* dy,
                       const void* W_self, const void* W_nbr, const int* dims, int L, int B,
                       int n, int d, int dtype, unsigned flags, void* dx, float* dW_self,
                       float* dW_nbr, float* dbias, void* workspace, size_t ws_bytes,
                       void* stream);

/* Workspace bytes hcw_stack_bwd needs for L layers. */
size_t hcw_stack_workspace_bytes(int B, int n, int d, int dtype, unsigned flags, int L);

/*
 * One training step of a stack: hcw_stack_fwd followed by hcw_stack_bwd
 * (Sec. 3.1 wiring and Eq. (1) maps forward, the chain rule backward), same
 * layer schedule (layer0, dim_override) and flags.
 *   Inputs x [B][n][d], W_self, W_nbr [L][d][d], bias [L][d] (or NULL), dy
 *   [B][n][d] (the gradient of y).  Outputs y, acts, masks exactly as
 *   hcw_stack_fwd writes them, dx, dW_self, dW_nbr, dbias (or NULL) exactly as
 *   hcw_stack_bwd writes them.  All buffers are the caller's; dy must not
 *   overlap y, acts or masks.
 *   workspace: at least hcw_stack_train_step_workspace_bytes(...) bytes.
 *   dW_self = dW_nbr = dbias = NULL: the forward and the input gradient only
 *   (no weight gradients); dW_self and dW_nbr are given together or not at all.
 * The results equal those of the two separate calls bit for bit.  bf16 on
 * pairs of SMs with up to 16 layers: the forward and the
 * input gradient run as one persistent launch (the input gradient of a
 * 512-token window starts as soon as its forward is done, and the last
 * forward layer writes the top layer's dz = dy * act'(z) itself), then one
 * launch computes the weight and bias gradients.  That launch starts behind
 * the first as a programmatic dependent and waits on its completion counters;
 * when its units leave SM pairs idle, the first launch's last layer runs on
 * those pairs alone.  Other shapes run the two calls.  Errors as for
 * hcw_stack_fwd and hcw_stack_bwd.
 */
int hcw_stack_train_step(const void* x, const void* W_self, const void* W_nbr, const float* bias,
                         const void* dy, int layer0, int L, int dim_override, int B, int n, int d,
                         int dtype, unsigned flags, void* y, void* acts, void* masks, void* dx,
                         float* dW_self, float* dW_nbr, float* dbias, void* workspace,
                         size_t ws_bytes, void* stream);
size_t hcw_stack_train_step_workspace_bytes(int B, int n, int d, int dtype, unsigned flags,
                                            int L);

/*
 * hcw_stack_train_step on the schedule dims (host array of L layers, as for
 * hcw_stack_fwd_dims: dims[l] >= 0 a hypercube dimension, -k a shift of Eq. (1)
 * by k positions).  The results equal those of hcw_stack_fwd_dims followed by
 * hcw_stack_bwd_dims bit for bit.  The one-launch forward + input gradient
 * also takes shift layers when n >= 128 and B n is a multiple of 256.  The
 * workspace is hcw_stack_train_step_workspace_bytes(...).  Errors as for those
 * two calls.
 */
int hcw_stack_train_step_dims(const void* x, const void* W_self, const void* W_nbr,
                              const float* bias, const void* dy, const int* dims, int L, int B,
                              int n, int d, int dtype, unsigned flags, void* y, void* acts,
                              void* masks, void* dx, float* dW_self, float* dW_nbr, float* dbias,
                              void* workspace, size_t ws_bytes, void* stream);

/*
 * The two halves of hcw_stack_bwd, for callers that want them apart (frozen
 * weights need only the first; the second can run later or elsewhere).
 *
 * hcw_stack_bwd_data: input gradients through the stack (the chain rule of
 * Eq. (1), layers L-1 down to 0).
 *   masks, dy, W_self, W_nbr as for hcw_stack_bwd.
 *   dx [B][n][d] gradient of the stack's input (output).
 *   dz [L][B][n][d] (output): every layer's pre-activation gradient
 *      dz_l = g_l * act'(z_l), where g_l is the gradient of layer l's
 *      output -- the input of hcw_stack_bwd_weight.
 *   workspace: at least hcw_stack_bwd_data_workspace_bytes(...) bytes.
 */
int hcw_stack_bwd_data(const void* masks, const void* dy, const void* W_self, const void* W_nbr,
                       int layer0, int L, int dim_override, int B, int n, int d, int dtype,
                       unsigned flags, void* dx, void* dz, void* workspace, size_t ws_bytes,
                       void* stream);
size_t hcw_stack_bwd_data_workspace_bytes(int B, int n, int d, int dtype, unsigned flags,
                                          int L);

/*
 * hcw_stack_bwd_weight: every layer's weight gradients from its input (x for
 * layer 0, acts[l-1] above) and its dz as written by hcw_stack_bwd_data:
 *   dW_self[l] = sum_i dz_l,i x_l,i^T,  dW_nbr[l] = sum_i m_i dz_l,i x_l,p(i)^T,
 *   dbias[l] = sum_i dz_l,i (dbias may be NULL).  fp32 outputs [L][d][d], [L][d].
 *   workspace: at least hcw_stack_bwd_weight_workspace_bytes(...) bytes.
 * bf16: up to 16 layers per launch, whole token range per tile (no split
 * reduction); the same kernel sums dz's columns into dbias.  Layers with few
 * output tiles (small d, few layers: fewer than 76 tiles in the launch)
 * instead split every layer's token range over one launch and add the fp32
 * partials of weights and dbias in a second one, in split order.  Either way
 * deterministic: the same inputs give the same bits.
 */
int hcw_stack_bwd_weight(const void* x, const void* acts, const void* dz, int layer0, int L,
                         int dim_override, int B, int n, int d, int dtype, unsigned flags,
                         float* dW_self, float* dW_nbr, float* dbias, void* workspace,
                         size_t ws_bytes, void* stream);
size_t hcw_stack_bwd_weight_workspace_bytes(int B, int n, int d, int dtype, unsigned flags,
                                            int L);
/* hcw_stack_bwd_weight on the schedule dims (host array of L layers, as for
 * hcw_stack_fwd_dims); same workspace, results and errors. */
int hcw_stack_bwd_weight_dims(const void* x, const void* acts, const void* dz, const int* dims,
                              int L, int B, int n, int d, int dtype, unsigned flags,
                              float* dW_self, float* dW_nbr, float* dbias, void* workspace,
                              size_t ws_bytes, void* stream);

/*
 * hcw_layer_bwd_weight for callers that cannot allocate device memory (a
 * host that only lends its own input and output buffers, or code that must
 * not call an allocator): same arguments and results, minus the workspace.
 * The paper has no counterpart; this is an interface convenience.
 *   Scratch: a fixed 32 MiB array inside the library, reserved on every
 *   device that loads it until the process exits.  Sizes whose weight
 *   gradient needs more scratch than that (hcw_layer_bwd_weight_workspace_bytes
 *   > 32 MiB) are rejected with HCW_ERR_WORKSPACE before anything runs.
 *   Allocates nothing: no cudaMalloc, cudaFree or allocating library call.
 *   Every call asks the runtime for the array's device address on the
 *   current device; the first call on a device also loads the library's
 *   device code there (a one-time set-up per device, with that device
 *   current): make that first call before any stream capture.  Because the
 *   address is looked up on every call, a device reset (cudaDeviceReset)
 *   does not leave a stale address behind.
 *   dbias, when given, must not overlap x or dz (HCW_ERR_ALIASING).
 *   All calls share the one array: calls whose kernels may overlap on the
 *   GPU (different streams without ordering, or several host threads) race
 *   on it and must be serialised by the caller.  No part of the array needs
 *   to start at zero; whatever a previous call left there is overwritten
 *   before it is read.
 */
int hcw_layer_bwd_weight_noalloc(const void* x, const void* dz, int layer, int dim_override,
                                 int B, int n, int d, int dtype, unsigned flags,
                                 float* dW_self, float* dW_nbr, float* dbias, void* stream);

/*
 * Which kernels run the bf16 stacked forward and input gradient
 * (hcw_stack_fwd, hcw_stack_bwd_data, hcw_stack_bwd).  Process-wide.
 *   HCW_STACK_AUTO       the faster family as measured on GB300 for the
 *                        shape; currently streaming everywhere.  The default.
 *   HCW_STACK_RESIDENT   resident wherever the shape fits.
 *   HCW_STACK_STREAMING  streaming only.
 * Resident: a cluster of two CTAs keeps 256 consecutive tokens (whole
 * samples) in shared memory through a run of up to 16 layers.  Only the
 * weights stream in, and each layer's output is written once.  The shape must
 * have d in {128, 256, 512}, n <= 256 and B*n a multiple of 256.  The causal
 * partner product costs 4d^2 flops per token there (every lane computed, half
 * kept) instead of 3d^2.
 * Streaming: every layer's tiles pass through global memory (L2); any shape.
 * The two families add the products in different orders (resident: the self
 * and partner products K block by K block; streaming: the self part first),
 * and the resident input gradient keeps the residual stream g in fp32 between
 * layers where the streaming kernels round it to bf16 at every layer: their
 * results differ at bf16 rounding level.
 * Returns the previous mode, or -1 (mode unchanged) for an unknown mode.
 */
#define HCW_STACK_AUTO      0
#define HCW_STACK_RESIDENT  1
#define HCW_STACK_STREAMING 2
int hcw_set_stack_kernels(int mode);

/*
 * Which family the bf16 stacked forward and input gradient of these sizes
 * would run on under the current setting (on the current device):
 * HCW_STACK_RESIDENT or HCW_STACK_STREAMING; -1 for invalid sizes or dtype.
 */
int hcw_stack_kernels_used(int B, int n, int d, int dtype);

/*
 * One decode step of a causal stack, bf16 (Sec. 6, "Deployability": the
 * decode path runs one token at a time, and a sparse layer needs only the
 * last k inputs it links to, so its cache does not grow).
 * B sequences advance together to position t (0 <= t < n of their windows).
 * Layer l links t to t - k_l (k_l = 2^s for the hypercube link along
 * dimension s, which t takes when bit s of t is set; k_l = k for a shift,
 * taken when t >= k); the layers are dims[l] as for hcw_stack_fwd_dims, or
 * (dims NULL) dimension (layer0 + l) mod log2 n.
 *   x_t     [B][d]: the layer-0 input at position t.
 *   y_t     [B][d]: the stack's output at position t (written).
 *   cache   hcw_decode_cache_bytes(...) bytes: per layer a ring of k_l + 1
 *           slots, [k_l + 1][B][d] one after another in layer order; slot
 *           (p mod (k_l + 1)) holds the layer's input at position p.  The
 *           step reads the slot of t - k_l, (t + 1) mod (k_l + 1), and writes
 *           the input at t into slot t mod (k_l + 1), a different one, so every
 *           layer's output goes straight into the next layer's ring.  Slots are
 *           read only for partners p >= 0, so the ring needs no
 *           initialisation; steps must come in order t = 0, 1, ....
 * The whole step (every layer) is one kernel launch: a cluster of up to 16
 * CTAs per 16 sequences, exchanging each layer's output in distributed
 * shared memory.  Needs HCW_CAUSAL (without it a hypercube link reads a later
 * position), L <= 64 and d <= 1024 (HCW_ERR_UNSUPPORTED above).  y_t equals
 * row t of hcw_stack_fwd over the window to bf16 rounding.  Calls are
 * asynchronous on `stream`.
 */
int hcw_decode_step(const void* x_t, const void* W_self, const void* W_nbr, const float* bias,
                    const int* dims, int layer0, int L, int t, int B, int n, int d,
                    unsigned flags, void* cache, void* y_t, void* stream);
/* Bytes of the decode rings for this schedule (0 for invalid sizes). */
size_t hcw_decode_cache_bytes(const int* dims, int layer0, int L, int B, int n, int d);

/*
 * The contraction hcw_decode_step runs, for this process:
 *   HCW_DECODE_WARP_MMA (default): eight warps per CTA share the K range with
 *     the warp-level bf16 MMA and add their partial blocks;
 *   HCW_DECODE_TCGEN05: one thread issues tcgen05.mma (M = 64 over the 16
 *     rows of a row block, N = the CTA's output columns) into TMEM.
 * Both accumulate in fp32 and round the same tensors to bf16; they add the
 * products in different orders, so their results differ at bf16 rounding
 * level.  Returns the previous mode, or -1 (mode unchanged) for an unknown mode.
 */
#define HCW_DECODE_WARP_MMA 0
#define HCW_DECODE_TCGEN05  1
int hcw_set_decode_kernel(int mode);

/*
 * One training step (forward, loss, backward) of the character-LM block
 * around the mixing stack, bf16 (App. A: width d, hidden h = 1024 = 2d at
 * d = 512; the weight counts of Table B2ecost / B1cost fit token and position
 * embeddings, two LayerNorms and an FFN with biases per layer, a final
 * LayerNorm and an output head with bias):
 *   x = E[ids[:, :n]] + P
 *   per layer l:  x += M_l(LN1_l(x))     M_l: Eq. (1) without bias or activation,
 *                                        causal, cube dimension l mod log2 n
 *                 x += W2_l relu(W1_l LN2_l(x) + b1_l) + b2_l
 *   logits = LNf(x) Wh^T + bh
 *   loss = mean over the B n positions of logsumexp(logits) - logits[next symbol]
 * LayerNorm: biased variance, eps = 1e-5, per-feature scale and shift.
 * Shapes (all device memory, row-major; ids and loss 4-byte aligned, the
 * rest 16-byte aligned):
 *   ids [B][n + 1] int32 in [0, V): inputs ids[:, :n], targets ids[:, 1:]
 *   E [V][d], P [n][d], W_self / W_nbr [L][d][d], W1 [L][h][d], W2 [L][d][h],
 *   Wh [V][d]: bf16;  LayerNorm scales / shifts ln1_*, ln2_* [L][d], lnf_* [d],
 *   b1 [L][h], b2 [L][d], bh [V]: fp32.
 * Gradients (hcw_block_grads, same shapes, fp32) are overwritten, not
 * accumulated; *loss (one fp32 on the device) is overwritten.  The mixing
 * products run on this library's tcgen05 layer kernels, the FFN and head
 * products on its tcgen05 GEMM (bf16 operands, fp32 accumulation and output;
 * a weight gradient that splits the tokens adds its partial sums in a fixed
 * order).
 * Needs n a power of two, d a multiple of 64 and <= 1024, h a multiple of 8,
 * V >= 2.  An id outside [0, V) is read as 0 and reported by hcw_sync_status
 * as HCW_ERR_INVALID_ARG.  Asynchronous on `stream`; no state is shared
 * between calls other than the workspace each one is given.
 */
typedef struct {
    const void* E;
    const void* P;
    const float* ln1_g;
    const float* ln1_b;
    const void* W_self;
    const void* W_nbr;
    const float* ln2_g;
    const float* ln2_b;
    const void* W1;
    const float* b1;
    const void* W2;
    const float* b2;
    const float* lnf_g;
    const float* lnf_b;
    const void* Wh;
    const float* bh;
} hcw_block_params;

typedef struct {
    float* E;
    float* P;
    float* ln1_g;
    float* ln1_b;
    float* W_self;
    float* W_nbr;
    float* ln2_g;
    float* ln2_b;
    float* W1;
    float* b1;
    float* W2;
    float* b2;
    float* lnf_g;
    float* lnf_b;
    float* Wh;
    float* bh;
} hcw_block_grads;

/* Workspace bytes of hcw_block_step (0 for invalid sizes). */
size_t hcw_block_workspace_bytes(int B, int n, int d, int h, int V, int L);
int hcw_block_step(const int* ids, const hcw_block_params* params, const hcw_block_grads* grads,
                   int B, int n, int d, int h, int V, int L, float* loss, void* workspace,
                   size_t ws_bytes, void* stream);

/*
 * The block step's plain GEMM on its own (App. A's FFN and head products and
 * their gradients): row-major C[M][N] = op(A) op(B) in fp32 from bf16
 * operands with fp32 accumulation, where A is [M][K] (ta = 0) or [K][M]
 * (ta = 1) and B is [K][N] (tb = 0) or [N][K] (tb = 1), all row-major device
 * memory.  C is overwritten and must not overlap A, B or the workspace
 * (HCW_ERR_ALIASING).  M, N, K >= 1 (HCW_ERR_INVALID_ARG).  The workspace (may
 * be NULL; 16-byte aligned otherwise) holds fp32 partial sums when the K range
 * is split across CTAs: hcw_gemm_workspace_bytes gives the size that allows
 * the best split; a smaller one allows fewer splits, NULL none.  Partial sums
 * are added in split order.  Operands whose rows TMA cannot read (a K-major
 * row not a multiple of 16 bytes, an MN-major one not a multiple of 64
 * elements, a pointer not 16-byte aligned) take a plain tiled kernel.
 * Asynchronous on `stream`.
 */
size_t hcw_gemm_workspace_bytes(int M, int N, int K);
int hcw_gemm_bf16(int M, int N, int K, const void* A, int ta, const void* B, int tb, float* C,
                  void* workspace, size_t ws_bytes, void* stream);

/*
 * `batch` products contracted over their rows, in one launch (the weight
 * gradients of App. A's FFN for every layer of the block at once):
 *   C[b] = A_b^T B_b,   b = 0 .. batch - 1
 * A_b is the row-major [K][M] bf16 matrix at A + b * a_stride elements, B_b
 * the row-major [K][N] bf16 matrix at B + b * b_stride elements, C[b] the
 * row-major [M][N] fp32 matrix at C + b * M * N (overwritten).  Every output
 * tile takes the whole K range in one fp32 accumulator (no partial sums, no
 * workspace).  M, N, K, batch >= 1 and strides >= 0 (HCW_ERR_INVALID_ARG);
 * C must not overlap the operands' spans (HCW_ERR_ALIASING).  Shapes TMA
 * cannot read (M or N not a multiple of 64, a pointer or a stride not
 * 16-byte aligned) run one product at a time on hcw_gemm_bf16's path.
 * Asynchronous on `stream`.
 */
int hcw_gemm_bf16_batched(int M, int N, int K, const void* A, long long a_stride, const void* B,
                          long long b_stride, float* C, int batch, void* stream);

/* Number of kernels this library has launched in this process (all devices). */
unsigned long long hcw_launch_count(void);

/*
 * Synchronise `stream`, then read and clear the current device's error
 * word.  Returns HCW_ERR_TIMEOUT if a kernel gave up on a bounded wait since
 * the last call, HCW_ERR_CUDA if the synchronisation failed, else HCW_OK.
 */
int hcw_sync_status(void* stream);

/*
 * Self-test of the bounded-wait path the kernels use: launches one CTA that
 * waits on an mbarrier nothing ever arrives on.  After timeout_ns
 * nanoseconds (1e3 .. 1e10) it records HCW_ERR_TIMEOUT in the error word and
 * exits normally, leaving the context usable.  Follow with hcw_sync_status.
 */
int hcw_selftest_wait(long long timeout_ns, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* HCW_H */
