// hcw_decode.cu -- one-token decode of a causal stack (Sec. 6, "Deployability":
// the decode path runs one token at a time, and a sparse layer needs only the
// last k inputs it links to, so its cache does not grow).
//
// B sequences advance together by one position t.  Layer l with link distance
// k_l (2^s for the hypercube link along dimension s, k for a shift layer) keeps
// a ring of its last k_l inputs; position t's partner input, when t receives
// (bit s of t set, or t >= k), is the input of position t - k_l, i.e. ring slot
// (t - k_l) mod k_l = t mod k_l.  After the step every layer's input at t is
// written into that same slot.
//
// At decode sizes (B <= a few hundred rows) a layer is bound by streaming its
// two d x d weight matrices from memory, not by arithmetic, so the layer is a
// CUDA-core kernel spread over many CTAs: each CTA computes a 16 x 16 block of
// outputs over K = d (self) plus d (partner), staging 64-deep slices of the
// inputs and the weights through shared memory, fp32 accumulation.
#include "hcw_internal.h"

namespace hcw {

namespace {

constexpr int DT = 16;   // output tile: 16 rows x 16 columns, one thread each
constexpr int DK = 64;   // K slice staged in shared memory

__device__ __forceinline__ float bf(const __nv_bfloat16 v) { return __bfloat162float(v); }

// out[r][o] = act(sum_k Ws[o][k] x[r][k] + sum_k Wn[o][k] p[r][k] + bias[o]) (+ x[r][o])
// p (the partner rows) may be null: the position does not receive at this layer.
__global__ void __launch_bounds__(DT * DT)
    decode_layer_kernel(const __nv_bfloat16* __restrict__ x, const __nv_bfloat16* __restrict__ p,
                        const __nv_bfloat16* __restrict__ Ws, const __nv_bfloat16* __restrict__ Wn,
                        const float* __restrict__ bias, int B, int d, unsigned flags,
                        __nv_bfloat16* __restrict__ out) {
    __shared__ float xs[DT][DK + 1], ws[DT][DK + 1];
    const int tx = threadIdx.x % DT, ty = threadIdx.x / DT;
    const int r0 = blockIdx.y * DT, o0 = blockIdx.x * DT;
    float acc = 0.f;
    for (int part = 0; part < (p ? 2 : 1); ++part) {
        const __nv_bfloat16* A = part ? p : x;
        const __nv_bfloat16* W = part ? Wn : Ws;
        for (int k0 = 0; k0 < d; k0 += DK) {
            // 16 rows x 64 inputs and 16 weight rows x 64, four elements a thread
            for (int e = threadIdx.x; e < DT * DK; e += DT * DT) {
                const int rr = e / DK, kk = e % DK;
                const int r = r0 + rr, o = o0 + rr, k = k0 + kk;
                xs[rr][kk] = (r < B && k < d) ? bf(A[(size_t)r * d + k]) : 0.f;
                ws[rr][kk] = (o < d && k < d) ? bf(W[(size_t)o * d + k]) : 0.f;
            }
            __syncthreads();
#pragma unroll 16
            for (int kk = 0; kk < DK; ++kk) acc = fmaf(xs[ty][kk], ws[tx][kk], acc);
            __syncthreads();
        }
    }
    const int r = r0 + ty, o = o0 + tx;
    if (r >= B || o >= d) return;
    float v = acc + (bias ? bias[o] : 0.f);
    if (flags & 4u) v = v > 0.f ? v : 0.f;
    if (flags & 2u) v += bf(x[(size_t)r * d + o]);
    out[(size_t)r * d + o] = __float2bfloat16_rn(v);
}

// ring slot of every layer <- that layer's input at this step: in[l] [B][d]
// (layer 0: x_t, else inputs + (l - 1) * B * d), slot[l] = ring + slot offset
struct CommitArgs {
    const __nv_bfloat16* x0;
    const __nv_bfloat16* inputs;
    __nv_bfloat16* slot[kMaxDecodeLayers];
    int L;
    long long per_layer;   // B * d elements
};

__global__ void decode_commit_kernel(const __grid_constant__ CommitArgs a) {
    const long long per16 = a.per_layer / 8;   // 16-byte pieces per layer (d % 8 == 0)
    const long long total = per16 * a.L;
    for (long long t = (long long)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (long long)gridDim.x * blockDim.x) {
        const int l = (int)(t / per16);
        const long long e = t - (long long)l * per16;
        const uint4* src = reinterpret_cast<const uint4*>(
            l == 0 ? a.x0 : a.inputs + (size_t)(l - 1) * a.per_layer);
        reinterpret_cast<uint4*>(a.slot[l])[e] = src[e];
    }
}

}  // namespace

cudaError_t launch_decode_layer(const __nv_bfloat16* x, const __nv_bfloat16* partner,
                                const __nv_bfloat16* Ws, const __nv_bfloat16* Wn,
                                const float* bias, int B, int d, unsigned flags,
                                __nv_bfloat16* out, cudaStream_t st) {
    dim3 grid((unsigned)((d + DT - 1) / DT), (unsigned)((B + DT - 1) / DT));
    decode_layer_kernel<<<grid, DT * DT, 0, st>>>(x, partner, Ws, Wn, bias, B, d, flags, out);
    return cudaGetLastError();
}

cudaError_t launch_decode_commit(const __nv_bfloat16* x0, const __nv_bfloat16* inputs,
                                 __nv_bfloat16* const* slots, int L, int B, int d,
                                 cudaStream_t st) {
    if (L < 1 || L > kMaxDecodeLayers) return cudaErrorInvalidValue;
    CommitArgs a;
    a.x0 = x0;
    a.inputs = inputs;
    for (int l = 0; l < L; ++l) a.slot[l] = slots[l];
    a.L = L;
    a.per_layer = (long long)B * d;
    const long long pieces = a.per_layer / 8 * L;
    long long blocks = (pieces + 255) / 256;
    if (blocks > 152 * 8) blocks = 152 * 8;
    decode_commit_kernel<<<(unsigned)blocks, 256, 0, st>>>(a);
    return cudaGetLastError();
}

}  // namespace hcw
