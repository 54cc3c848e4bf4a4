// hcw_block.cu -- one training step (forward, loss, backward) of the
// character-LM block around the mixing stack (App. A: width d, hidden 1024 =
// 2d at d = 512; the weight counts of Table B2ecost / B1cost fit token and
// position embeddings, two LayerNorms and an FFN with biases per layer, a
// final LayerNorm and an output head with bias):
//
//   x = E[ids] + P
//   per layer l:  x += M_l(LN1_l(x))                M_l: Eq. (1), causal, rotated
//                 x += W2_l relu(W1_l LN2_l(x) + b1_l) + b2_l
//   logits = LNf(x) Wh^T + bh,   loss = mean next-symbol cross-entropy
//
// The mixing sublayer runs on this library's layer kernels (hcw_layer_fwd /
// hcw_layer_bwd: tcgen05, bf16); the FFN and head products run on this
// library's tcgen05 GEMM (hcw_gemm.cu), whose epilogue also applies the FFN's
// bias + ReLU and its gradient; the row kernels here (embedding, residual
// add + LayerNorm, cross-entropy, their gradients, column sums) are
// memory-bound and each makes one pass over its rows.  The residual stream x
// and its gradient are fp32; the GEMM operands are bf16 (h, M(h), g, relu(u),
// hf, dlogits, bf16(dx), the FFN pre-activation gradient); the other GEMM
// outputs are fp32.
#include <mutex>
#include <vector>

#include "hcw.h"
#include "hcw_internal.h"
#include "hcw_ptx.cuh"

namespace hcw {

namespace {

constexpr float kLnEps = 1e-5f;
constexpr int kRowWarps = 8;   // rows (one warp each) per CTA of the row kernels
// CTAs of the fused LayerNorm backward at most (rows of its partial sums), and
// its shared memory at the largest d (1024) with three sums
constexpr int kLnBwdMaxGrid = 1024;
constexpr size_t kLnBwdMaxSmem = (size_t)kRowWarps * 3 * 1024 * sizeof(float);

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}
__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

// symbol of input position t of sequence b (ids: [B][n + 1]); an id outside
// [0, V) reads symbol 0 and records HCW_ERR_INVALID_ARG in the error word
__device__ __forceinline__ int symbol(const int* ids, int b, int t, int n, int V) {
    const int v = ids[(size_t)b * (n + 1) + t];
    if (v < 0 || v >= V) {
        atomicExch(&g_error_word, HCW_ERR_INVALID_ARG);
        return 0;
    }
    return v;
}

// x[b n + t][c] = E[ids[b][t]][c] + P[t][c]   (fp32 out)
__global__ void embed_fwd_kernel(const int* ids, const __nv_bfloat16* E, const __nv_bfloat16* P,
                                 float* x, int B, int n, int d, int V) {
    pdl_wait();   // until the kernel before it in the stream has finished
    pdl_trigger();
    const size_t total = (size_t)B * n * d;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (size_t)gridDim.x * blockDim.x) {
        const int c = (int)(i % d);
        const size_t r = i / d;
        const int t = (int)(r % n), b = (int)(r / n);
        const int v = symbol(ids, b, t, n, V);
        x[i] = __bfloat162float(E[(size_t)v * d + c]) + __bfloat162float(P[(size_t)t * d + c]);
    }
}

// One warp per row: x = x_in (+ add1 bf16) (+ add2 fp32) (+ badd[c]); x_out = x
// when given; y = bf16((x - mean) rstd g + b); stats = (mean, rstd).  d <= 1024.
__global__ void __launch_bounds__(kRowWarps * 32)
    ln_fwd_kernel(const float* x_in, const __nv_bfloat16* add1, const float* add2,
                  const float* badd, float* x_out, const float* g, const float* b,
                  __nv_bfloat16* y, float2* stats, int T, int d) {
    pdl_wait();   // until the kernel before it in the stream has finished
    pdl_trigger();
    const int lane = threadIdx.x & 31;
    const int row = blockIdx.x * kRowWarps + (threadIdx.x >> 5);
    if (row >= T) return;
    const int nv = d >> 5;
    const size_t base = (size_t)row * d;
    float v[32];
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        if (i < nv) {
            const int c = i * 32 + lane;
            float t = x_in[base + c];
            if (add1) t += __bfloat162float(add1[base + c]);
            if (add2) t += add2[base + c];
            if (badd) t += badd[c];
            v[i] = t;
            s += t;
        }
    }
    const float mean = warp_sum(s) / d;
    float q = 0.f;
#pragma unroll
    for (int i = 0; i < 32; ++i)
        if (i < nv) q += (v[i] - mean) * (v[i] - mean);
    const float rstd = rsqrtf(warp_sum(q) / d + kLnEps);
#pragma unroll
    for (int i = 0; i < 32; ++i) {
        if (i < nv) {
            const int c = i * 32 + lane;
            if (x_out) x_out[base + c] = v[i];
            y[base + c] = __float2bfloat16_rn((v[i] - mean) * rstd * g[c] + b[c]);
        }
    }
    if (lane == 0) stats[row] = make_float2(mean, rstd);
}

// Four consecutive features at element e (a multiple of 4): fp32 as one
// 16-byte access, bf16 as one 8-byte access.
__device__ __forceinline__ float4 ld4(const float* p, size_t e) {
    return *reinterpret_cast<const float4*>(p + e);
}
__device__ __forceinline__ float4 ld4(const __nv_bfloat16* p, size_t e) {
    const uint2 u = *reinterpret_cast<const uint2*>(p + e);
    const float2 a = unpack_bf16x2(u.x), b = unpack_bf16x2(u.y);
    return make_float4(a.x, a.y, b.x, b.y);
}
__device__ __forceinline__ void st4(float* p, size_t e, float4 v) {
    *reinterpret_cast<float4*>(p + e) = v;
}
__device__ __forceinline__ void st4(__nv_bfloat16* p, size_t e, float4 v) {
    *reinterpret_cast<uint2*>(p + e) = make_uint2(pack_bf16x2(v.x, v.y), pack_bf16x2(v.z, v.w));
}
__device__ __forceinline__ float4 add4(float4 a, float4 b) {
    return make_float4(a.x + b.x, a.y + b.y, a.z + b.z, a.w + b.w);
}
__device__ __forceinline__ float sum4(float4 a) { return a.x + a.y + a.z + a.w; }

// ln_fwd_kernel for d a multiple of 128: lane holds features 4 (i 32 + lane) ..
// + 3 for i < d / 128 <= NV4.
template <int NV4>
__global__ void __launch_bounds__(kRowWarps * 32)
    ln_fwd4_kernel(const float* x_in, const __nv_bfloat16* add1, const float* add2,
                   const float* badd, float* x_out, const float* g, const float* b,
                   __nv_bfloat16* y, float2* stats, int T, int d) {
    pdl_wait();   // until the kernel before it in the stream has finished
    pdl_trigger();
    const int lane = threadIdx.x & 31;
    const int row = blockIdx.x * kRowWarps + (threadIdx.x >> 5);
    if (row >= T) return;
    const int nv = d >> 7;
    const size_t base = (size_t)row * d;
    float4 v[NV4];
    float s = 0.f;
#pragma unroll
    for (int i = 0; i < NV4; ++i) {
        if (i < nv) {
            const int c = (i * 32 + lane) * 4;
            float4 t = ld4(x_in, base + c);
            if (add1) t = add4(t, ld4(add1, base + c));
            if (add2) t = add4(t, ld4(add2, base + c));
            if (badd) t = add4(t, ld4(badd, (size_t)c));
            v[i] = t;
            s += sum4(t);
        }
    }
    const float mean = warp_sum(s) / d;
    float q = 0.f;
#pragma unroll
    for (int i = 0; i < NV4; ++i) {
        if (i < nv) {
            const float4 t = v[i];
            q += (t.x - mean) * (t.x - mean) + (t.y - mean) * (t.y - mean) +
                 (t.z - mean) * (t.z - mean) + (t.w - mean) * (t.w - mean);
        }
    }
    const float rstd = rsqrtf(warp_sum(q) / d + kLnEps);
#pragma unroll
    for (int i = 0; i < NV4; ++i) {
        if (i < nv) {
            const int c = (i * 32 + lane) * 4;
            const float4 t = v[i], gg = ld4(g, (size_t)c), bb = ld4(b, (size_t)c);
            if (x_out) st4(x_out, base + c, t);
            st4(y, base + c,
                make_float4((t.x - mean) * rstd * gg.x + bb.x, (t.y - mean) * rstd * gg.y + bb.y,
                            (t.z - mean) * rstd * gg.z + bb.z, (t.w - mean) * rstd * gg.w + bb.w));
        }
    }
    if (lane == 0) stats[row] = make_float2(mean, rstd);
}

// One warp per position r = b n + t: z = logits[r] + bh, target v* =
// ids[b][t + 1]; loss += (logsumexp(z) - z[v*]) / N; dlog[r][v] =
// bf16((softmax(z)[v] - [v == v*]) / N).
__global__ void __launch_bounds__(kRowWarps * 32)
    ce_kernel(const float* logits, const float* bh, const int* ids, __nv_bfloat16* dlog,
              float* loss, int B, int n, int V, float inv_N) {
    pdl_wait();   // until the kernel before it in the stream has finished
    pdl_trigger();
    const int lane = threadIdx.x & 31;
    const int r = blockIdx.x * kRowWarps + (threadIdx.x >> 5);
    if (r >= B * n) return;
    const int b = r / n, t = r % n;
    const int tgt = symbol(ids, b, t + 1, n, V);
    const float* z = logits + (size_t)r * V;
    float m = -INFINITY;
    for (int v = lane; v < V; v += 32) m = fmaxf(m, z[v] + bh[v]);
    m = warp_max(m);
    float s = 0.f;
    for (int v = lane; v < V; v += 32) s += expf(z[v] + bh[v] - m);
    const float lse = m + logf(warp_sum(s));
    for (int v = lane; v < V; v += 32) {
        const float p = expf(z[v] + bh[v] - lse) - (v == tgt ? 1.f : 0.f);
        dlog[(size_t)r * V + v] = __float2bfloat16_rn(p * inv_N);
    }
    if (lane == 0) atomicAdd(loss, (lse - (z[tgt] + bh[tgt])) * inv_N);
}

// out[c] += sum over a tile of kColRows rows of M[r][c] (bf16 M [T][C]; out
// zeroed before the launch): grid (ceil(C / 256), ceil(T / kColRows)), a
// thread per column of its tile, the rows' loads independent of each other
constexpr int kColRows = 64;
__global__ void colsum_kernel(const __nv_bfloat16* M, float* out, int T, int C) {
    pdl_wait();   // until the kernel before it in the stream has finished
    pdl_trigger();
    const int c = blockIdx.x * blockDim.x + threadIdx.x;
    if (c >= C) return;
    const int r0 = blockIdx.y * kColRows;
    const int r1 = min(T, r0 + kColRows);
    float s = 0.f;
#pragma unroll 8
    for (int r = r0; r < r1; ++r) s += __bfloat162float(M[(size_t)r * C + c]);
    atomicAdd(out + c, s);
}

// W consecutive features at element e (W = 2 or 4; e a multiple of W).
template <int W>
__device__ __forceinline__ void ldv(const float* p, size_t e, float (&v)[W]) {
    if constexpr (W == 4) {
        const float4 t = *reinterpret_cast<const float4*>(p + e);
        v[0] = t.x, v[1] = t.y, v[2] = t.z, v[3] = t.w;
    } else {
        const float2 t = *reinterpret_cast<const float2*>(p + e);
        v[0] = t.x, v[1] = t.y;
    }
}
template <int W>
__device__ __forceinline__ void ldv(const __nv_bfloat16* p, size_t e, float (&v)[W]) {
    if constexpr (W == 4) {
        const uint2 u = *reinterpret_cast<const uint2*>(p + e);
        const float2 a = unpack_bf16x2(u.x), b = unpack_bf16x2(u.y);
        v[0] = a.x, v[1] = a.y, v[2] = b.x, v[3] = b.y;
    } else {
        const float2 a = unpack_bf16x2(*reinterpret_cast<const uint32_t*>(p + e));
        v[0] = a.x, v[1] = a.y;
    }
}
template <int W>
__device__ __forceinline__ void stv(float* p, size_t e, const float (&v)[W]) {
    if constexpr (W == 4)
        *reinterpret_cast<float4*>(p + e) = make_float4(v[0], v[1], v[2], v[3]);
    else
        *reinterpret_cast<float2*>(p + e) = make_float2(v[0], v[1]);
}
template <int W>
__device__ __forceinline__ void stv(__nv_bfloat16* p, size_t e, const float (&v)[W]) {
    if constexpr (W == 4)
        *reinterpret_cast<uint2*>(p + e) =
            make_uint2(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]));
    else
        *reinterpret_cast<uint32_t*>(p + e) = pack_bf16x2(v[0], v[1]);
}

// LayerNorm backward and its parameter sums in one pass over the rows.  Per
// row (one warp), with xhat = (x - mean) rstd and dxhat = dy g,
//   dx = rstd (dxhat - mean(dxhat) - xhat mean(dxhat xhat))  (+ dres)
// written to dx_out (fp32) and, when dxb is given, as bf16; dy is fp32 or
// bf16.  Every load of a row comes before its stores: dres and dx_out may be
// the same buffer (the gradient updated in place).  Lane l holds features
// W (32 i + l) .. + W - 1, i < d / (32 W) <= NV.  Warps take rows
// blockIdx.x * kRowWarps + warp, then every gridDim.x * kRowWarps further on,
// summing per feature dy xhat (the scale gradient), dy (the shift gradient)
// and, with ncol = 3, bf16(dx) (the column sums of dxb); the CTA adds its
// warps' sums in warp order into row blockIdx.x of part [gridDim.x][ncol d],
// which ln_part_reduce_kernel adds up in row order.
template <int NV, int W, typename DY>
__global__ void __launch_bounds__(kRowWarps * 32)
    ln_bwd_fused_kernel(const DY* dy, const float* x, const float2* stats, const float* g,
                        const float* dres, float* dx_out, __nv_bfloat16* dxb, int T, int d,
                        int ncol, float* part) {
    pdl_wait();   // until the kernel before it in the stream has finished
    pdl_trigger();
    extern __shared__ float red[];   // [kRowWarps][ncol d]: each warp's sums, then the CTA's
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int nv = d / (32 * W);
    const int width = ncol * d;
    float* mine = red + (size_t)warp * width;   // this warp's sums, kept in shared memory
    for (int c = lane; c < width; c += 32) mine[c] = 0.f;
    __syncwarp();
    for (int row = blockIdx.x * kRowWarps + warp; row < T; row += gridDim.x * kRowWarps) {
        const size_t base = (size_t)row * d;
        const float2 st = stats[row];
        float xh[NV][W], dh[NV][W], rv[NV][W];
        float s1 = 0.f, s2 = 0.f;
#pragma unroll
        for (int i = 0; i < NV; ++i) {
            if (i < nv) {
                const int c = (i * 32 + lane) * W;
                float xx[W], gg[W], yv[W], sg[W], sb[W];
                if (dres) {
                    ldv<W>(dres, base + c, rv[i]);
                } else {
#pragma unroll
                    for (int j = 0; j < W; ++j) rv[i][j] = 0.f;
                }
                ldv<W>(dy, base + c, yv);
                ldv<W>(x, base + c, xx);
                ldv<W>(g, (size_t)c, gg);
                ldv<W>(mine, (size_t)c, sg);
                ldv<W>(mine, (size_t)d + c, sb);
#pragma unroll
                for (int j = 0; j < W; ++j) {
                    xh[i][j] = (xx[j] - st.x) * st.y;
                    dh[i][j] = yv[j] * gg[j];
                    s1 += dh[i][j];
                    s2 += dh[i][j] * xh[i][j];
                    sg[j] += yv[j] * xh[i][j];
                    sb[j] += yv[j];
                }
                stv<W>(mine, (size_t)c, sg);
                stv<W>(mine, (size_t)d + c, sb);
            }
        }
        const float m1 = warp_sum(s1) / d, m2 = warp_sum(s2) / d;
#pragma unroll
        for (int i = 0; i < NV; ++i) {
            if (i < nv) {
                const int c = (i * 32 + lane) * W;
                float v[W];
#pragma unroll
                for (int j = 0; j < W; ++j) v[j] = st.y * (dh[i][j] - m1 - xh[i][j] * m2) + rv[i][j];
                stv<W>(dx_out, base + c, v);
                if (dxb) {
                    stv<W>(dxb, base + c, v);
                    if (ncol == 3) {
                        float sc[W];
                        ldv<W>(mine, (size_t)2 * d + c, sc);
#pragma unroll
                        for (int j = 0; j < W; ++j)
                            sc[j] += __bfloat162float(__float2bfloat16_rn(v[j]));
                        stv<W>(mine, (size_t)2 * d + c, sc);
                    }
                }
            }
        }
    }
    __syncthreads();
    for (int c = threadIdx.x; c < width; c += blockDim.x) {
        float t = 0.f;
#pragma unroll
        for (int w = 0; w < kRowWarps; ++w) t += red[(size_t)w * width + c];
        part[(size_t)blockIdx.x * width + c] = t;
    }
}

// Sum of the nblk rows of part [nblk][ncol d] per column, in row order:
// columns [0, d) -> dgam, [d, 2d) -> dbet, [2d, 3d) -> dcol.  A CTA of 32
// warps per 32 columns, a column a lane: warp w adds rows w, w + 32, ...
// (sixteen loads in flight), then the 32 warp sums meet in shared memory in
// warp order.
constexpr int kReduceWarps = 32;
__global__ void __launch_bounds__(kReduceWarps * 32)
    ln_part_reduce_kernel(const float* part, int nblk, int d, int ncol, float* dgam, float* dbet,
                          float* dcol) {
    pdl_wait();   // until the kernel before it in the stream has finished
    pdl_trigger();
    __shared__ float acc[kReduceWarps][33];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int width = ncol * d;
    const int c = blockIdx.x * 32 + lane;
    float s = 0.f;
    if (c < width) {
        for (int b0 = warp; b0 < nblk; b0 += 16 * kReduceWarps) {
            float v[16];
#pragma unroll
            for (int k = 0; k < 16; ++k) {
                const int b = b0 + k * kReduceWarps;
                v[k] = b < nblk ? part[(size_t)b * width + c] : 0.f;
            }
#pragma unroll
            for (int k = 0; k < 16; ++k) s += v[k];
        }
    }
    acc[warp][lane] = s;
    __syncthreads();
    if (warp == 0 && c < width) {
        float t = 0.f;
#pragma unroll
        for (int w = 0; w < kReduceWarps; ++w) t += acc[w][lane];
        const int seg = c / d, cc = c - seg * d;
        (seg == 0 ? dgam : (seg == 1 ? dbet : dcol))[cc] = t;
    }
}

// The same sums for a list of LayerNorm backward passes at once: job
// blockIdx.y adds up its own partial rows (in row order, as above).
constexpr int kMaxLnJobs = 64;
struct LnJob {
    const float* part;
    int nblk, ncol;
    float* dgam;
    float* dbet;
    float* dcol;
};
struct LnJobs {
    LnJob job[kMaxLnJobs];
    int d;
};
__global__ void __launch_bounds__(kReduceWarps * 32)
    ln_part_reduce_batched_kernel(const __grid_constant__ LnJobs J) {
    pdl_wait();   // until the kernel before it in the stream has finished
    pdl_trigger();
    __shared__ float acc[kReduceWarps][33];
    const LnJob& jb = J.job[blockIdx.y];
    const int d = J.d;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int width = jb.ncol * d;
    const int c = blockIdx.x * 32 + lane;
    if (blockIdx.x * 32 >= width) return;   // block-uniform: this job is narrower
    float s = 0.f;
    if (c < width) {
        for (int b0 = warp; b0 < jb.nblk; b0 += 16 * kReduceWarps) {
            float v[16];
#pragma unroll
            for (int k = 0; k < 16; ++k) {
                const int b = b0 + k * kReduceWarps;
                v[k] = b < jb.nblk ? jb.part[(size_t)b * width + c] : 0.f;
            }
#pragma unroll
            for (int k = 0; k < 16; ++k) s += v[k];
        }
    }
    acc[warp][lane] = s;
    __syncthreads();
    if (warp == 0 && c < width) {
        float t = 0.f;
#pragma unroll
        for (int w = 0; w < kReduceWarps; ++w) t += acc[w][lane];
        const int seg = c / d, cc = c - seg * d;
        (seg == 0 ? jb.dgam : (seg == 1 ? jb.dbet : jb.dcol))[cc] = t;
    }
}

// dE[ids[b][t]] += dx[b n + t]   (dE zeroed before the launch)
__global__ void embed_bwd_kernel(const int* ids, const float* dx, float* dE, int B, int n, int d,
                                 int V) {
    pdl_wait();   // until the kernel before it in the stream has finished
    pdl_trigger();
    const size_t total = (size_t)B * n * d;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (size_t)gridDim.x * blockDim.x) {
        const int c = (int)(i % d);
        const size_t r = i / d;
        const int v = symbol(ids, (int)(r / n), (int)(r % n), n, V);
        atomicAdd(dE + (size_t)v * d + c, dx[i]);
    }
}

// dP[t][c] = sum over b of dx[b n + t][c]
__global__ void pos_bwd_kernel(const float* dx, float* dP, int B, int n, int d) {
    pdl_wait();   // until the kernel before it in the stream has finished
    pdl_trigger();
    const size_t total = (size_t)n * d;
    for (size_t i = (size_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (size_t)gridDim.x * blockDim.x) {
        float s = 0.f;
        for (int b = 0; b < B; ++b) s += dx[(size_t)b * n * d + i];
        dP[i] = s;
    }
}

}  // namespace

namespace {

// Row-major C[M][N] (fp32) = op(A) op(B) with bf16 operands and fp32
// accumulation; A is [M][K] ([K][M] when ta), B is [K][N] ([N][K] when tb).
// split_ws holds the partial sums when the GEMM splits K.  HCW_OK after
// counting its launches, else HCW_ERR_CUDA.
int gemm(float* split_ws, size_t split_bytes, cudaStream_t st, int M, int N, int K, const void* A,
         bool ta, const void* B, bool tb, float* C) {
    int launches = 0;
    const cudaError_t e =
        gemm_bf16_f32(M, N, K, A, ta, B, tb, C, split_ws, split_bytes, st, &launches);
    return count_launch(e, launches);
}

// The FFN's products with their elementwise step in the epilogue, bf16 out:
// a = relu(G W1^T + b1) (aux NULL), or dpre = (a > 0) * (dy W2) (bias NULL),
// whose column sums (the gradient of b1) go into colsum (zeroed before).
int gemm_ffn(cudaStream_t st, int M, int N, int K, const void* A, const void* B, bool tb,
             const float* bias, const __nv_bfloat16* aux, __nv_bfloat16* out,
             float* colsum = nullptr) {
    GemmEpi epi;
    epi.kind = bias ? EPI_BIAS_RELU : EPI_RELU_GRAD;
    epi.bias = bias;
    epi.aux = aux;
    epi.out = out;
    epi.colsum = colsum;
    int launches = 0;
    const cudaError_t e =
        gemm_bf16(M, N, K, A, false, B, tb, nullptr, epi, nullptr, 0, st, &launches);
    return count_launch(e, launches);
}

int sms_now() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1)
        return 148;
    return n;
}

size_t round256(size_t v) { return (v + 255) & ~(size_t)255; }

// Workspace of one step (byte offsets; T = B n tokens):
//   xs   [2L + 1][T][d] fp32   x_0 .. x_L (layer inputs, x_L the head's), then
//                              the L mid-layer streams (after the mixing)
//   h1, g [L][T][d] bf16       LN1 / LN2 outputs (mixing and FFN inputs)
//   a    [L][T][h] bf16        relu(u), the FFN's hidden activations
//   st1, st2 [L][T], stf [T]   LayerNorm (mean, rstd)
//   m, hf [T][d] bf16          mixing output (per layer), head input
//   U    [T][max(h, V, d)] fp32  every GEMM output with T rows, in turn
//   dlog [T][V] bf16; dx [T][d] fp32
//   dxf  [L][T][d] bf16        each FFN output's gradient (bf16 of dx)
//   dpre [L][T][h] bf16        each FFN pre-activation gradient
//   dh [T][d] bf16; the LayerNorm backward's partial sums
//   dzm  [L][T][d] bf16        each mixing layer's output gradient (its dz),
//                              read by the batched weight-gradient launch,
//                              and that launch's scratch; the fp32 partial
//   sums of the GEMMs that split K (the weight gradients)
constexpr size_t kSplitWs = (size_t)32 << 20;
struct BlockWs {
    size_t xs, h1, g, a, st1, st2, stf, m, hf, U, dlog, dx, dxf, dpre, dh, lnp, dzm, sws,
        sws_bytes, split, total;
};

BlockWs block_ws(int B, int n, int d, int h, int V, int L) {
    const size_t T = (size_t)B * n;
    const size_t wide = (size_t)(h > V ? (h > d ? h : d) : (V > d ? V : d));
    BlockWs w;
    size_t o = 0;
    auto take = [&](size_t bytes) {
        const size_t at = o;
        o += round256(bytes);
        return at;
    };
    w.xs = take((2 * (size_t)L + 1) * T * d * 4);
    w.h1 = take((size_t)L * T * d * 2);
    w.g = take((size_t)L * T * d * 2);
    w.a = take((size_t)L * T * h * 2);
    w.st1 = take((size_t)L * T * 8);
    w.st2 = take((size_t)L * T * 8);
    w.stf = take(T * 8);
    w.m = take(T * d * 2);
    w.hf = take(T * d * 2);
    w.U = take(T * wide * 4);
    w.dlog = take(T * V * 2);
    w.dx = take(T * d * 4);
    // per layer: the FFN output's gradient (bf16) and the pre-activation
    // gradient, the operands of the batched FFN weight gradients after the loop
    w.dxf = take((size_t)L * T * d * 2);
    w.dpre = take((size_t)L * T * h * 2);
    w.dh = take(T * d * 2);
    // LayerNorm backward partial sums, one slice per pass (2 L + 1 of them),
    // added up together after the backward loop
    w.lnp = take((2 * (size_t)L + 1) * kLnBwdMaxGrid * 3 * d * 4);
    // every mixing layer's output gradient, kept for one batched weight-gradient
    // launch at the end of the backward, and that launch's scratch
    w.dzm = take((size_t)L * T * d * 2);
    w.sws_bytes = hcw_stack_bwd_weight_workspace_bytes(B, n, d, HCW_BF16, HCW_CAUSAL, L);
    w.sws = take(w.sws_bytes);
    w.split = take(kSplitWs);
    w.total = o;
    return w;
}

}  // namespace

namespace {

bool block_sizes_ok(int B, int n, int d, int h, int V, int L) {
    return B >= 1 && n >= 2 && (n & (n - 1)) == 0 && d >= 64 && d % 64 == 0 && d <= 1024 &&
           h >= 8 && h % 8 == 0 && V >= 2 && L >= 1 && (long long)B * n * (n + 1) < (1ll << 40);
}

bool a16(const void* p) { return p && (reinterpret_cast<uintptr_t>(p) & 15) == 0; }


unsigned elem_grid(size_t total) {
    const size_t want = (total + 255) / 256, cap = (size_t)sms_now() * 16;
    return (unsigned)(want < cap ? (want ? want : 1) : cap);
}

// LayerNorm forward rows: four features a lane and access when d is a
// multiple of 128, else one (ln_fwd_kernel)
cudaError_t launch_ln_fwd(cudaStream_t st, const float* x_in, const __nv_bfloat16* add1,
                          const float* add2, const float* badd, float* x_out, const float* g,
                          const float* b, __nv_bfloat16* y, float2* stats, int T, int d) {
    const dim3 grid((T + kRowWarps - 1) / kRowWarps), blk(kRowWarps * 32);
    const int v4 = d / 128;
#define HCW_LNF(K) \
    return launch_pdl(K, grid, blk, 0, st, x_in, add1, add2, badd, x_out, g, b, y, stats, T, d)
    if (d % 128 != 0) HCW_LNF(ln_fwd_kernel);
    if (v4 <= 1) HCW_LNF(ln_fwd4_kernel<1>);
    if (v4 <= 2) HCW_LNF(ln_fwd4_kernel<2>);
    if (v4 <= 4) HCW_LNF(ln_fwd4_kernel<4>);
    HCW_LNF(ln_fwd4_kernel<8>);
#undef HCW_LNF
}

template <int NV, int W, typename DY>
cudaError_t launch_ln_bwd_fused(cudaStream_t st, int grid, const DY* dy, const float* x,
                                const float2* stats, const float* g, const float* dres,
                                float* dx_out, __nv_bfloat16* dxb, int T, int d, int ncol,
                                float* part) {
    auto kern = ln_bwd_fused_kernel<NV, W, DY>;
    static std::once_flag once[64];
    static cudaError_t set_err[64];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
    std::call_once(once[dev], [&] {
        set_err[dev] = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                            (int)kLnBwdMaxSmem);
    });
    if (set_err[dev] != cudaSuccess) return set_err[dev];
    const size_t smem = (size_t)kRowWarps * ncol * d * sizeof(float);
    return launch_pdl(kern, dim3(grid), dim3(kRowWarps * 32), smem, st, dy, x, stats, g, dres,
                      dx_out, dxb, T, d, ncol, part);
}

// Resident CTAs per SM of the fused LayerNorm backward for this d (its
// register use and shared memory), at least 1.
template <int NV, int W, typename DY>
int ln_bwd_occupancy(int d, int ncol) {
    int n = 0;
    const size_t smem = (size_t)kRowWarps * ncol * d * sizeof(float);
    if (cudaFuncSetAttribute(ln_bwd_fused_kernel<NV, W, DY>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)kLnBwdMaxSmem) != cudaSuccess ||
        cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, ln_bwd_fused_kernel<NV, W, DY>,
                                                      kRowWarps * 32, smem) != cudaSuccess)
        return 1;
    return n > 0 ? n : 1;
}

int ln_bwd_ctas_per_sm(bool f32, int d, int ncol) {
#define HCW_OCC(NV, W) \
    return f32 ? ln_bwd_occupancy<NV, W, float>(d, ncol) : ln_bwd_occupancy<NV, W, __nv_bfloat16>(d, ncol)
    if (d % 128 == 0) {
        const int nv = d / 128;
        if (nv <= 1) HCW_OCC(1, 4);
        if (nv <= 2) HCW_OCC(2, 4);
        if (nv <= 4) HCW_OCC(4, 4);
        HCW_OCC(8, 4);
    }
    const int nv = d / 64;
    if (nv <= 4) HCW_OCC(4, 2);
    if (nv <= 8) HCW_OCC(8, 2);
    HCW_OCC(16, 2);
#undef HCW_OCC
}

template <typename DY>
cudaError_t launch_ln_bwd_rows(cudaStream_t st, int grid, const DY* dy, const float* x,
                               const float2* stats, const float* g, const float* dres,
                               float* dx_out, __nv_bfloat16* dxb, int T, int d, int ncol,
                               float* part) {
#define HCW_LNB(NV, W) \
    return launch_ln_bwd_fused<NV, W, DY>(st, grid, dy, x, stats, g, dres, dx_out, dxb, T, d, ncol, part)
    if (d % 128 == 0) {   // four features a lane and access
        const int nv = d / 128;
        if (nv <= 1) HCW_LNB(1, 4);
        if (nv <= 2) HCW_LNB(2, 4);
        if (nv <= 4) HCW_LNB(4, 4);
        HCW_LNB(8, 4);
    }
    const int nv = d / 64;   // d % 64 == 0: two
    if (nv <= 4) HCW_LNB(4, 2);
    if (nv <= 8) HCW_LNB(8, 2);
    HCW_LNB(16, 2);
#undef HCW_LNB
}

// The LayerNorm backward: rows and per-CTA parameter sums in one pass
// (ln_bwd_fused_kernel), then their fixed-order sum (ln_part_reduce_kernel)
// into dgam, dbet and, when dcol is given, the column sums of dxb.  Two
// launches (*nk).
cudaError_t launch_ln_bwd(cudaStream_t st, const float* dyf, const __nv_bfloat16* dyb,
                          const float* x, const float2* stats, const float* g, const float* dres,
                          float* dx_out, __nv_bfloat16* dxb, float* part, float* dgam, float* dbet,
                          float* dcol, int T, int d, int* nk, LnJob* defer = nullptr) {
    *nk = 0;
    if (dcol && !dxb) return cudaErrorInvalidValue;
    const int ncol = dcol ? 3 : 2;
    // one wave: as many CTAs as fit on the SMs at once, at most one a row group
    int grid = (T + kRowWarps - 1) / kRowWarps;
    const int wave = ln_bwd_ctas_per_sm(dyf != nullptr, d, ncol) * sms_now();
    grid = grid < wave ? grid : wave;
    grid = grid < kLnBwdMaxGrid ? grid : kLnBwdMaxGrid;
    cudaError_t e = dyf ? launch_ln_bwd_rows<float>(st, grid, dyf, x, stats, g, dres, dx_out, dxb,
                                                    T, d, ncol, part)
                        : launch_ln_bwd_rows<__nv_bfloat16>(st, grid, dyb, x, stats, g, dres,
                                                            dx_out, dxb, T, d, ncol, part);
    if (e != cudaSuccess) return e;
    *nk = 1;
    if (defer) {
        // the sums are added up later, with other passes' (part stays untouched)
        *defer = LnJob{part, grid, ncol, dgam, dbet, dcol};
        return cudaSuccess;
    }
    e = launch_pdl(ln_part_reduce_kernel, dim3((ncol * d + 31) / 32), dim3(kReduceWarps * 32), 0,
                   st, static_cast<const float*>(part), grid, d, ncol, dgam, dbet, dcol);
    if (e == cudaSuccess) *nk = 2;
    return e;
}

int block_step(const int* ids, const hcw_block_params& p, const hcw_block_grads& gr, int B, int n,
               int d, int h, int V, int L, float* loss, uint8_t* ws, cudaStream_t st) {
    const int T = B * n;
    const BlockWs w = block_ws(B, n, d, h, V, L);
    const size_t Td = (size_t)T * d, Th = (size_t)T * h;
    float* xs = reinterpret_cast<float*>(ws + w.xs);
    auto X = [&](int l) { return xs + (size_t)l * Td; };              // x_l, l = 0..L
    auto XM = [&](int l) { return xs + (size_t)(L + 1 + l) * Td; };   // mid-layer stream
    auto H1 = [&](int l) { return reinterpret_cast<__nv_bfloat16*>(ws + w.h1) + (size_t)l * Td; };
    auto G = [&](int l) { return reinterpret_cast<__nv_bfloat16*>(ws + w.g) + (size_t)l * Td; };
    auto A = [&](int l) { return reinterpret_cast<__nv_bfloat16*>(ws + w.a) + (size_t)l * Th; };
    auto DZM = [&](int l) { return reinterpret_cast<__nv_bfloat16*>(ws + w.dzm) + (size_t)l * Td; };
    auto S1 = [&](int l) { return reinterpret_cast<float2*>(ws + w.st1) + (size_t)l * T; };
    auto S2 = [&](int l) { return reinterpret_cast<float2*>(ws + w.st2) + (size_t)l * T; };
    float2* sf = reinterpret_cast<float2*>(ws + w.stf);
    auto* m = reinterpret_cast<__nv_bfloat16*>(ws + w.m);
    auto* hf = reinterpret_cast<__nv_bfloat16*>(ws + w.hf);
    float* U = reinterpret_cast<float*>(ws + w.U);
    auto* dlog = reinterpret_cast<__nv_bfloat16*>(ws + w.dlog);
    float* dx = reinterpret_cast<float*>(ws + w.dx);
    float* lnp = reinterpret_cast<float*>(ws + w.lnp);
    auto DXF = [&](int l) { return reinterpret_cast<__nv_bfloat16*>(ws + w.dxf) + (size_t)l * Td; };
    auto DPRE = [&](int l) { return reinterpret_cast<__nv_bfloat16*>(ws + w.dpre) + (size_t)l * Th; };
    auto* dh = reinterpret_cast<__nv_bfloat16*>(ws + w.dh);
    auto bf = [](const void* q, size_t off) {
        return static_cast<const __nv_bfloat16*>(q) + off;
    };
    float* split = reinterpret_cast<float*>(ws + w.split);
    const unsigned rows_grid = (unsigned)((T + kRowWarps - 1) / kRowWarps);
    int rc;
#define HCW_TRY(expr)          \
    do {                       \
        rc = (expr);           \
        if (rc) return rc;     \
    } while (0)
#define HCW_CU(expr) HCW_TRY((expr) == cudaSuccess ? HCW_OK : HCW_ERR_CUDA)
#define HCW_GEMM(...) HCW_TRY(gemm(split, kSplitWs, st, __VA_ARGS__))
    // gradients that are sums (atomics) start at zero; so does the loss
    HCW_CU(cudaMemsetAsync(loss, 0, sizeof(float), st));
    HCW_CU(cudaMemsetAsync(gr.E, 0, (size_t)V * d * 4, st));
    float* zero_d[] = {gr.ln1_g, gr.ln1_b, gr.ln2_g, gr.ln2_b, gr.b2};
    for (float* q : zero_d) HCW_CU(cudaMemsetAsync(q, 0, (size_t)L * d * 4, st));
    HCW_CU(cudaMemsetAsync(gr.lnf_g, 0, (size_t)d * 4, st));
    HCW_CU(cudaMemsetAsync(gr.lnf_b, 0, (size_t)d * 4, st));
    HCW_CU(cudaMemsetAsync(gr.b1, 0, (size_t)L * h * 4, st));
    HCW_CU(cudaMemsetAsync(gr.bh, 0, (size_t)V * 4, st));

    // ------------------------------------------------------------ forward
    HCW_TRY(count_launch(launch_pdl(embed_fwd_kernel, dim3(elem_grid(Td)), dim3(256), 0, st, ids,
                                    bf(p.E, 0), bf(p.P, 0), X(0), B, n, d, V),
                         1));
    HCW_TRY(count_launch(launch_ln_fwd(st, X(0), nullptr, nullptr, nullptr, nullptr, p.ln1_g,
                                       p.ln1_b, H1(0), S1(0), T, d),
                         1));
    for (int l = 0; l < L; ++l) {
        HCW_TRY(hcw_layer_fwd(H1(l), bf(p.W_self, (size_t)l * d * d), bf(p.W_nbr, (size_t)l * d * d),
                              nullptr, l, -1, B, n, d, HCW_BF16, HCW_CAUSAL, m, nullptr, st));
        HCW_TRY(count_launch(launch_ln_fwd(st, X(l), m, nullptr, nullptr, XM(l),
                                           p.ln2_g + (size_t)l * d, p.ln2_b + (size_t)l * d, G(l),
                                           S2(l), T, d),
                             1));
        HCW_TRY(gemm_ffn(st, T, h, d, G(l), bf(p.W1, (size_t)l * h * d), true,
                         p.b1 + (size_t)l * h, nullptr, A(l)));   // a = relu(g W1^T + b1)
        HCW_GEMM(T, d, h, A(l), false, bf(p.W2, (size_t)l * d * h), true, U);
        const bool top = l + 1 == L;
        HCW_TRY(count_launch(
            launch_ln_fwd(st, XM(l), nullptr, U, p.b2 + (size_t)l * d, X(l + 1),
                          top ? p.lnf_g : p.ln1_g + (size_t)(l + 1) * d,
                          top ? p.lnf_b : p.ln1_b + (size_t)(l + 1) * d, top ? hf : H1(l + 1),
                          top ? sf : S1(l + 1), T, d),
            1));
    }
    HCW_GEMM(T, V, d, hf, false, p.Wh, true, U);
    HCW_TRY(count_launch(launch_pdl(ce_kernel, dim3(rows_grid), dim3(kRowWarps * 32), 0, st,
                                    static_cast<const float*>(U), p.bh, ids, dlog, loss, B, n, V,
                                    1.f / T),
                         1));

    // ----------------------------------------------------------- backward
    const unsigned gridT = (unsigned)((T + kColRows - 1) / kColRows);
    HCW_GEMM(V, d, T, dlog, true, hf, false, gr.Wh);   // dWh = dlog^T hf
    HCW_TRY(count_launch(launch_pdl(colsum_kernel, dim3((V + 255) / 256, gridT), dim3(256), 0, st,
                                    static_cast<const __nv_bfloat16*>(dlog), gr.bh, T, V),
                         1));
    HCW_GEMM(T, d, V, dlog, false, p.Wh, false, U);    // dhf = dlog Wh
    // each LayerNorm backward that writes the gradient of x_{l+1} (LNf, then
    // LN1 of layer l + 1) also sums its bf16 copy's columns: db2 of layer l
    int nk = 0;
    // every LayerNorm backward pass leaves its partial sums in its own slice;
    // one launch adds them all up after the loop
    static thread_local std::vector<LnJob> jobs;
    jobs.assign(2 * (size_t)L + 1, LnJob{});
    int njobs = 0;
    auto lnp_slice = [&](int i) { return lnp + (size_t)i * kLnBwdMaxGrid * 3 * d; };
    cudaError_t le = launch_ln_bwd(st, U, nullptr, X(L), sf, p.lnf_g, nullptr, dx, DXF(L - 1),
                                   lnp_slice(njobs), gr.lnf_g, gr.lnf_b,
                                   gr.b2 + (size_t)(L - 1) * d, T, d, &nk, &jobs[njobs]);
    ++njobs;
    HCW_TRY(count_launch(le, nk));
    for (int l = L - 1; l >= 0; --l) {
        // FFN sublayer: DXF(l) = bf16(dx) is the gradient of its output;
        // dpre = (a > 0) * (DXF(l) W2), and db1 = its column sums.  Its weight
        // gradients W2 (DXF(l)^T a) and W1 (dpre^T g) come after the loop.
        HCW_TRY(gemm_ffn(st, T, h, d, DXF(l), bf(p.W2, (size_t)l * d * h), false, nullptr, A(l),
                         DPRE(l), gr.b1 + (size_t)l * h));
        HCW_GEMM(T, d, h, DPRE(l), false, bf(p.W1, (size_t)l * h * d), false, U);  // dg
        le = launch_ln_bwd(st, U, nullptr, XM(l), S2(l), p.ln2_g + (size_t)l * d, dx, dx,
                           DZM(l), lnp_slice(njobs), gr.ln2_g + (size_t)l * d,
                           gr.ln2_b + (size_t)l * d, nullptr, T, d, &nk, &jobs[njobs]);
        ++njobs;
        HCW_TRY(count_launch(le, nk));
        // mixing sublayer: DZM(l) = bf16(dx) is the gradient of M_l(h) (its dz: no
        // activation); its input gradient now, its weight gradient with the other
        // layers' after the loop
        HCW_TRY(hcw_layer_bwd_data(DZM(l), nullptr, bf(p.W_self, (size_t)l * d * d),
                                   bf(p.W_nbr, (size_t)l * d * d), l, -1, B, n, d, HCW_BF16,
                                   HCW_CAUSAL, dh, st));
        le = launch_ln_bwd(st, nullptr, dh, X(l), S1(l), p.ln1_g + (size_t)l * d, dx, dx,
                           l > 0 ? DXF(l - 1) : nullptr, lnp_slice(njobs),
                           gr.ln1_g + (size_t)l * d, gr.ln1_b + (size_t)l * d,
                           l > 0 ? gr.b2 + (size_t)(l - 1) * d : nullptr, T, d, &nk,
                           &jobs[njobs]);
        ++njobs;
        HCW_TRY(count_launch(le, nk));
    }
    // the LayerNorm parameter gradients (and db2) of every pass, in launches of
    // up to kMaxLnJobs passes
    for (int j0 = 0; j0 < njobs; j0 += kMaxLnJobs) {
        const int cnt = njobs - j0 < kMaxLnJobs ? njobs - j0 : kMaxLnJobs;
        static thread_local LnJobs part;
        part.d = d;
        for (int j = 0; j < cnt; ++j) part.job[j] = jobs[j0 + j];
        HCW_TRY(count_launch(launch_pdl(ln_part_reduce_batched_kernel,
                                        dim3((3 * d + 31) / 32, cnt), dim3(kReduceWarps * 32), 0,
                                        st, part),
                             1));
    }
    // the FFN weight gradients of all layers, two batched launches (every
    // output tile over the whole token range, no partial sums):
    // dW2_l = DXF(l)^T a_l [d][h], dW1_l = dpre_l^T g_l [h][d]
    {
        int nl = 0;
        HCW_CU(gemm_bf16_f32_batched(d, h, T, DXF(0), Td * 2, A(0), Th * 2, gr.W2, L, st, &nl));
        HCW_TRY(count_launch(cudaSuccess, nl));
        HCW_CU(gemm_bf16_f32_batched(h, d, T, DPRE(0), Th * 2, G(0), Td * 2, gr.W1, L, st, &nl));
        HCW_TRY(count_launch(cudaSuccess, nl));
    }
    // the mixing layers' weight gradients, all layers in one batched launch: x_l =
    // H1(l) (contiguous over l), dz_l = DZM(l)
    HCW_TRY(hcw_stack_bwd_weight(H1(0), L > 1 ? H1(1) : nullptr, DZM(0), 0, L, -1, B, n, d,
                                 HCW_BF16, HCW_CAUSAL, gr.W_self, gr.W_nbr, nullptr,
                                 w.sws_bytes ? ws + w.sws : nullptr, w.sws_bytes, st));
    HCW_TRY(count_launch(launch_pdl(embed_bwd_kernel, dim3(elem_grid(Td)), dim3(256), 0, st, ids,
                                    static_cast<const float*>(dx), gr.E, B, n, d, V),
                         1));
    return count_launch(launch_pdl(pos_bwd_kernel, dim3(elem_grid((size_t)n * d)), dim3(256), 0,
                                   st, static_cast<const float*>(dx), gr.P, B, n, d),
                        1);
#undef HCW_TRY
#undef HCW_CU
#undef HCW_GEMM
}

}  // namespace

cudaError_t block_error_word_read_clear(int* word) {
    const int zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(word, g_error_word, sizeof(int));
    if (e == cudaSuccess && *word) e = cudaMemcpyToSymbol(g_error_word, &zero, sizeof(int));
    return e;
}

}  // namespace hcw

using namespace hcw;

extern "C" {

size_t hcw_block_workspace_bytes(int B, int n, int d, int h, int V, int L) {
    if (!block_sizes_ok(B, n, d, h, V, L)) return 0;
    return block_ws(B, n, d, h, V, L).total;
}

int hcw_block_step(const int* ids, const hcw_block_params* params, const hcw_block_grads* grads,
                   int B, int n, int d, int h, int V, int L, float* loss, void* workspace,
                   size_t ws_bytes, void* stream) {
    if (!params || !grads || !ids || !loss) return HCW_ERR_INVALID_ARG;
    if (!block_sizes_ok(B, n, d, h, V, L))
        return (d > 1024 && d % 64 == 0) ? HCW_ERR_UNSUPPORTED : HCW_ERR_INVALID_ARG;
    const hcw_block_params& p = *params;
    const hcw_block_grads& g = *grads;
    const void* in[] = {p.E, p.P, p.ln1_g, p.ln1_b, p.W_self, p.W_nbr, p.ln2_g, p.ln2_b, p.W1,
                        p.b1, p.W2, p.b2, p.lnf_g, p.lnf_b, p.Wh, p.bh};
    const void* out[] = {g.E, g.P, g.ln1_g, g.ln1_b, g.W_self, g.W_nbr, g.ln2_g, g.ln2_b, g.W1,
                         g.b1, g.W2, g.b2, g.lnf_g, g.lnf_b, g.Wh, g.bh, loss};
    for (const void* q : in)
        if (!q) return HCW_ERR_INVALID_ARG;
    for (const void* q : out)
        if (!q) return HCW_ERR_INVALID_ARG;
    for (const void* q : in)
        if (!a16(q)) return HCW_ERR_ALIGNMENT;
    for (const void* q : out)
        if (q != loss && !a16(q)) return HCW_ERR_ALIGNMENT;
    // ids and the loss are read and written as 4-byte scalars
    if ((reinterpret_cast<uintptr_t>(loss) & 3) || (reinterpret_cast<uintptr_t>(ids) & 3))
        return HCW_ERR_ALIGNMENT;
    const size_t need = block_ws(B, n, d, h, V, L).total;
    if (!workspace || ws_bytes < need || !a16(workspace)) return HCW_ERR_WORKSPACE;
    return block_step(ids, p, g, B, n, d, h, V, L, loss, static_cast<uint8_t*>(workspace),
                      (cudaStream_t)stream);
}

}  // extern "C"
