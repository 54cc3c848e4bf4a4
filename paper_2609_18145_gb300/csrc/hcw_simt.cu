// hcw_simt.cu -- CUDA-core kernels of libhcw:
//   * the fp32 path of the layer (forward, input gradient, weight gradient),
//     tiled FFMA with fp32 accumulation, for callers that need fp32 accuracy;
//   * the elementwise / reduction helpers of the bf16 path: ReLU gradient
//     mask, deterministic column sums (dbias), split-K reduction of dW;
//   * the device partner table (same index code as the kernels).
//
// Index rules, per layer link s inside each sample of n positions:
//   s >= 0 (Sec. 3.1): partner p(i) = i XOR 2^s; causal: i receives from p(i)
//          iff bit s of i is set;
//   s < 0  (Eq. (1) with k = -s, "near" of App. A is k = 1): p(i) = i - k, and
//          i receives iff i >= k (a shift always links earlier to later).
#include "hcw_internal.h"

namespace hcw {

namespace {

__device__ __forceinline__ int partner_of(int i, int s) { return s >= 0 ? i ^ (1 << s) : i + s; }

__device__ __forceinline__ bool receives(int i, int s, unsigned flags) {
    if (s < 0) return i + s >= 0;
    return !(flags & 1u) || ((i >> s) & 1);
}

// the position that takes x_i as its partner input at link s, or -1
__device__ __forceinline__ int reader_of(int i, int s, int n, unsigned flags) {
    if (s < 0) return i - s < n ? i - s : -1;
    const int p = i ^ (1 << s);
    return receives(p, s, flags) ? p : -1;
}

constexpr int T = 32;   // tile edge of the fp32 kernels

// z[r][o] = sum_k Ws[o][k] x[r][k] + m_r sum_k Wn[o][k] x[p(r)][k] + bias[o]
// Block: 32 rows x 32 outputs, 32 x 8 threads, 4 outputs per thread.
// mout (optional): ReLU mask words [rows][ceil(d/32)], bit o%32 of word o/32 = (z > 0).
__global__ void f32_fwd_kernel(const float* __restrict__ x, const float* __restrict__ Ws,
                               const float* __restrict__ Wn, const float* __restrict__ bias,
                               int s, int n, int d, long long rows, unsigned flags,
                               float* __restrict__ y, float* __restrict__ z,
                               uint32_t* __restrict__ mout) {
    __shared__ float xs[T][T + 1], xp[T][T + 1], ws[T][T + 1], wn[T][T + 1];
    const long long r0 = (long long)blockIdx.y * T;
    const int o0 = blockIdx.x * T;
    const int tx = threadIdx.x, ty = threadIdx.y;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int k0 = 0; k0 < d; k0 += T) {
        for (int rr = ty; rr < T; rr += 8) {
            const long long r = r0 + rr;
            const int k = k0 + tx;
            float a = 0.f, b = 0.f;
            if (r < rows && k < d) {
                const int i = (int)(r % n);
                a = x[r * d + k];
                b = receives(i, s, flags) ? x[(r - i + partner_of(i, s)) * d + k] : 0.f;
            }
            xs[rr][tx] = a;
            xp[rr][tx] = b;
            const int o = o0 + rr;
            ws[rr][tx] = (o < d && k < d) ? Ws[(long long)o * d + k] : 0.f;
            wn[rr][tx] = (o < d && k < d) ? Wn[(long long)o * d + k] : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int kk = 0; kk < T; ++kk) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int rr = ty + 8 * q;
                acc[q] = fmaf(xs[rr][kk], ws[tx][kk], acc[q]);
                acc[q] = fmaf(xp[rr][kk], wn[tx][kk], acc[q]);
            }
        }
        __syncthreads();
    }
    const int o = o0 + tx;
    const int wpr = (d + 31) >> 5;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const long long r = r0 + ty + 8 * q;
        const bool ok = r < rows && o < d;
        float v = ok ? acc[q] + (bias ? bias[o] : 0.f) : 0.f;
        if (mout) {
            // the warp covers the 32 columns of one mask word of row r
            const unsigned bits = __ballot_sync(0xffffffffu, ok && v > 0.f);
            if (tx == 0 && r < rows) mout[r * wpr + (o0 >> 5)] = bits;
        }
        if (!ok) continue;
        if (z) z[r * d + o] = v;
        if (flags & 4u) v = v > 0.f ? v : 0.f;
        if (flags & 2u) v += x[r * d + o];
        y[r * d + o] = v;
    }
}

// dx[r][k] = sum_o dz[r][o] Ws[o][k] + m_{p(r)} sum_o dz[p(r)][o] Wn[o][k] (+ dy[r][k])
__global__ void f32_dx_kernel(const float* __restrict__ dz, const float* __restrict__ dy,
                              const float* __restrict__ Ws, const float* __restrict__ Wn, int s,
                              int n, int d, long long rows, unsigned flags,
                              float* __restrict__ dx) {
    __shared__ float gs[T][T + 1], gp[T][T + 1], ws[T][T + 1], wn[T][T + 1];
    const long long r0 = (long long)blockIdx.y * T;
    const int k0 = blockIdx.x * T;
    const int tx = threadIdx.x, ty = threadIdx.y;
    float acc[4] = {0.f, 0.f, 0.f, 0.f};
    for (int o0 = 0; o0 < d; o0 += T) {
        for (int rr = ty; rr < T; rr += 8) {
            const long long r = r0 + rr;
            const int o = o0 + tx;
            float a = 0.f, b = 0.f;
            if (r < rows && o < d) {
                const int i = (int)(r % n);
                const int j = reader_of(i, s, n, flags);
                a = dz[r * d + o];
                b = j >= 0 ? dz[(r - i + j) * d + o] : 0.f;
            }
            gs[rr][tx] = a;
            gp[rr][tx] = b;
            const int oo = o0 + rr, k = k0 + tx;
            ws[rr][tx] = (oo < d && k < d) ? Ws[(long long)oo * d + k] : 0.f;
            wn[rr][tx] = (oo < d && k < d) ? Wn[(long long)oo * d + k] : 0.f;
        }
        __syncthreads();
#pragma unroll 8
        for (int oo = 0; oo < T; ++oo) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int rr = ty + 8 * q;
                acc[q] = fmaf(gs[rr][oo], ws[oo][tx], acc[q]);
                acc[q] = fmaf(gp[rr][oo], wn[oo][tx], acc[q]);
            }
        }
        __syncthreads();
    }
    const int k = k0 + tx;
    if (k >= d) return;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const long long r = r0 + ty + 8 * q;
        if (r >= rows) continue;
        float v = acc[q];
        if (flags & 2u) v += dy[r * d + k];
        dx[r * d + k] = v;
    }
}

// dWs[o][k] = sum_r dz[r][o] x[r][k];  dWn[o][k] = sum_r m_r dz[r][o] x[p(r)][k]
// Block: 32 o x 32 k; the token loop is sequential (fixed order).
__global__ void f32_dw_kernel(const float* __restrict__ x, const float* __restrict__ dz, int s,
                              int n, int d, long long rows, unsigned flags,
                              float* __restrict__ dWs, float* __restrict__ dWn) {
    __shared__ float gz[T][T + 1], xs[T][T + 1], xp[T][T + 1];
    const int o0 = blockIdx.y * T, k0 = blockIdx.x * T;
    const int tx = threadIdx.x, ty = threadIdx.y;
    float as[4] = {0.f, 0.f, 0.f, 0.f}, an[4] = {0.f, 0.f, 0.f, 0.f};
    for (long long r0 = 0; r0 < rows; r0 += T) {
        for (int rr = ty; rr < T; rr += 8) {
            const long long r = r0 + rr;
            float g = 0.f, a = 0.f, b = 0.f;
            if (r < rows) {
                const int i = (int)(r % n);
                if (o0 + tx < d) g = dz[r * d + o0 + tx];
                if (k0 + tx < d) {
                    a = x[r * d + k0 + tx];
                    b = receives(i, s, flags) ? x[(r - i + partner_of(i, s)) * d + k0 + tx] : 0.f;
                }
            }
            gz[rr][tx] = g;
            xs[rr][tx] = a;
            xp[rr][tx] = b;
        }
        __syncthreads();
#pragma unroll 8
        for (int rr = 0; rr < T; ++rr) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const float g = gz[rr][ty + 8 * q];
                as[q] = fmaf(g, xs[rr][tx], as[q]);
                an[q] = fmaf(g, xp[rr][tx], an[q]);
            }
        }
        __syncthreads();
    }
    const int k = k0 + tx;
    if (k >= d) return;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int o = o0 + ty + 8 * q;
        if (o >= d) continue;
        dWs[(long long)o * d + k] = as[q];
        dWn[(long long)o * d + k] = an[q];
    }
}

template <typename V>
__device__ __forceinline__ float to_f(V v);
template <>
__device__ __forceinline__ float to_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 v) {
    return __bfloat162float(v);
}

template <typename V>
__global__ void relu_grad_kernel(const V* __restrict__ dy, const V* __restrict__ z,
                                 V* __restrict__ dz, size_t count) {
    const V zero = V(0.f);
    for (size_t t = (size_t)blockIdx.x * blockDim.x + threadIdx.x; t < count;
         t += (size_t)gridDim.x * blockDim.x)
        dz[t] = to_f(z[t]) > 0.f ? dy[t] : zero;
}

// dz[t][o] = mask bit (t, o) ? dy[t][o] : 0, masks as written by the forward
// (any d: rows of ceil(d / 32) mask words).
__global__ void relu_grad_mask_f32_kernel(const float* __restrict__ dy,
                                          const uint32_t* __restrict__ mask,
                                          float* __restrict__ dz, long long rows, int d) {
    const int wpr = (d + 31) >> 5;
    const size_t count = (size_t)rows * d;
    for (size_t t = (size_t)blockIdx.x * blockDim.x + threadIdx.x; t < count;
         t += (size_t)gridDim.x * blockDim.x) {
        const size_t r = t / d;
        const int o = (int)(t - r * d);
        dz[t] = (mask[r * wpr + (o >> 5)] >> (o & 31)) & 1u ? dy[t] : 0.f;
    }
}

// The same for bf16 rows (d a multiple of 64): one thread per 16 bytes of a
// row, so a group never straddles a mask word.
template <typename V>
__global__ void relu_grad_mask_kernel(const V* __restrict__ dy, const uint32_t* __restrict__ mask,
                                      V* __restrict__ dz, long long rows, int d) {
    constexpr int VEC = 16 / sizeof(V);
    const int wpr = d >> 5;
    const int gpr = d / VEC;   // groups per row
    const size_t count = (size_t)rows * gpr;
    for (size_t t = (size_t)blockIdx.x * blockDim.x + threadIdx.x; t < count;
         t += (size_t)gridDim.x * blockDim.x) {
        const size_t r = t / gpr;
        const int o = (int)(t - r * gpr) * VEC;
        const uint32_t bits = (mask[r * wpr + (o >> 5)] >> (o & 31)) & ((1u << VEC) - 1u);
        uint4 v = reinterpret_cast<const uint4*>(dy)[t];
        uint32_t w[4] = {v.x, v.y, v.z, v.w};
        if (VEC == 8) {
#pragma unroll
            for (int i = 0; i < 4; ++i)
                w[i] &= ((bits >> (2 * i)) & 1u ? 0x0000FFFFu : 0u) |
                        ((bits >> (2 * i + 1)) & 1u ? 0xFFFF0000u : 0u);
        } else {
#pragma unroll
            for (int i = 0; i < 4; ++i) w[i] = (bits >> i) & 1u ? w[i] : 0u;
        }
        reinterpret_cast<uint4*>(dz)[t] = make_uint4(w[0], w[1], w[2], w[3]);
    }
}

// rows per partial of the column sum: 64 up to 65,536 rows (enough CTAs to
// fill the GPU), 256 above (the partials stay small)
inline long long col_rows(long long rows) { return rows <= 65536 ? 64 : 256; }

// partial[c][o] = sum_{r in chunk c} dz[r][o] for any d (block: 32 columns x
// 8 row lanes).
__global__ void colsum_partial_f32_kernel(const float* __restrict__ dz, long long rows, int d,
                                          int crows, float* __restrict__ partial) {
    __shared__ float red[8][33];
    const int o = blockIdx.x * 32 + threadIdx.x;
    const long long r0 = (long long)blockIdx.y * crows;
    const long long r1 = min(rows, r0 + crows);
    float acc = 0.f;
    if (o < d)
        for (long long r = r0 + threadIdx.y; r < r1; r += 8) acc += dz[r * d + o];
    red[threadIdx.y][threadIdx.x] = acc;
    __syncthreads();
    if (threadIdx.y == 0 && o < d) {
        float s = 0.f;
        for (int q = 0; q < 8; ++q) s += red[q][threadIdx.x];
        partial[(long long)blockIdx.y * d + o] = s;
    }
}

// The same for bf16 rows (d a multiple of 64), 16-byte loads.  Block: 64
// column groups of 16 bytes x 4 row lanes; each thread sums its group over every 4th row of
// the chunk, then the 4 row lanes are added in a fixed order.
template <typename V>
__global__ void colsum_partial_kernel(const V* __restrict__ dz, long long rows, int d, int crows,
                                      float* __restrict__ partial) {
    constexpr int VEC = 16 / sizeof(V);
    __shared__ float red[4][64][VEC + 1];
    // blockIdx.z selects one of several equally shaped matrices (layers)
    dz += (size_t)blockIdx.z * rows * d;
    partial += (size_t)blockIdx.z * gridDim.y * d;
    const int gpr = d / VEC;
    const int g = blockIdx.x * 64 + threadIdx.x;
    const long long r0 = (long long)blockIdx.y * crows;
    const long long r1 = min(rows, r0 + crows);
    float acc[VEC];
#pragma unroll
    for (int i = 0; i < VEC; ++i) acc[i] = 0.f;
    if (g < gpr) {
        const uint4* src = reinterpret_cast<const uint4*>(dz) + g;
        for (long long r = r0 + threadIdx.y; r < r1; r += 4) {
            const uint4 q = src[(size_t)r * gpr];
            const V* e = reinterpret_cast<const V*>(&q);
#pragma unroll
            for (int i = 0; i < VEC; ++i) acc[i] += to_f(e[i]);
        }
    }
#pragma unroll
    for (int i = 0; i < VEC; ++i) red[threadIdx.y][threadIdx.x][i] = acc[i];
    __syncthreads();
    if (threadIdx.y == 0 && g < gpr) {
#pragma unroll
        for (int i = 0; i < VEC; ++i) {
            const float s = ((red[0][threadIdx.x][i] + red[1][threadIdx.x][i]) +
                             red[2][threadIdx.x][i]) + red[3][threadIdx.x][i];
            partial[(long long)blockIdx.y * d + (long long)g * VEC + i] = s;
        }
    }
}

// out[o] = sum over the chunks c of partial[c][o], in chunk order: a CTA of 32
// warps per 32 columns, a column a lane; warp w adds chunks w, w + 32, ...,
// then the warp sums meet in shared memory in warp order.
__global__ void __launch_bounds__(1024) colsum_final_kernel(const float* __restrict__ partial,
                                                            int chunks, int d,
                                                            float* __restrict__ out) {
    __shared__ float red[32][33];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int o = blockIdx.x * 32 + lane;
    partial += (size_t)blockIdx.y * chunks * d;
    out += (size_t)blockIdx.y * d;
    float s = 0.f;
    if (o < d) {
#pragma unroll 4
        for (int c = warp; c < chunks; c += 32) s += partial[(long long)c * d + o];
    }
    red[warp][lane] = s;
    __syncthreads();
    if (warp == 0 && o < d) {
        float t = 0.f;
        for (int w = 0; w < 32; ++w) t += red[w][lane];
        out[o] = t;
    }
}

// out_w[l][o][k] = sum over the splits s of partial[l][w][s][o][k], w in {self,
// partner}; grid.y = 3 adds dbias[l][o] = sum over the self part's splits of
// bpart[l][s][o].  Block: 64 float4 columns x 8 split lanes; lane y adds the
// splits y, y + 8, ... in order, then the 8 lane sums meet in shared memory
// in lane order (deterministic).  grid.y = the part, grid.z = the layer.
__global__ void __launch_bounds__(512) splitk_reduce_kernel(
    const float* __restrict__ partial, int splits_max, int splits_self, int splits_nbr, int d,
    size_t part_stride, float* __restrict__ dWs, float* __restrict__ dWn, size_t out_stride,
    const float* __restrict__ bpart, float* __restrict__ dbias) {
    __shared__ float4 red[8][64];
    const int which = blockIdx.y;
    const int S = which == 1 ? splits_nbr : splits_self;
    if (S <= 1) return;   // written directly by the GEMM
    const size_t total4 = which == 2 ? (size_t)d / 4 : (size_t)d * d / 4;
    const size_t e4 = (size_t)blockIdx.x * 64 + threadIdx.x;
    if ((size_t)blockIdx.x * 64 >= total4) return;   // (the dbias rows are short)
    const float4* src = reinterpret_cast<const float4*>(
        which == 2 ? bpart + (size_t)blockIdx.z * splits_self * d
                   : partial + blockIdx.z * part_stride + (size_t)which * splits_max * d * d);
    float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
    if (e4 < total4) {
        for (int sp = threadIdx.y; sp < S; sp += 8) {
            const float4 b = src[(size_t)sp * total4 + e4];
            a.x += b.x;
            a.y += b.y;
            a.z += b.z;
            a.w += b.w;
        }
    }
    red[threadIdx.y][threadIdx.x] = a;
    __syncthreads();
    if (threadIdx.y == 0 && e4 < total4) {
#pragma unroll
        for (int y = 1; y < 8; ++y) {
            const float4 b = red[y][threadIdx.x];
            a.x += b.x;
            a.y += b.y;
            a.z += b.z;
            a.w += b.w;
        }
        float* out = which == 2 ? dbias + (size_t)blockIdx.z * d
                                : (which ? dWn : dWs) + blockIdx.z * out_stride;
        reinterpret_cast<float4*>(out)[e4] = a;
    }
}

// out[b][i] = in[b][i - k] for 0 <= i - k < n, else 0 (k of either sign):
// the partner rows of a shift layer (k > 0) or their readers (k < 0), as a
// row-aligned second operand.  One thread per 16-byte piece.
__global__ void shift_rows_kernel(const uint4* __restrict__ in, uint4* __restrict__ out,
                                  long long rows, int n, int pieces, int k) {
    const long long total = rows * pieces;
    for (long long t = (long long)blockIdx.x * blockDim.x + threadIdx.x; t < total;
         t += (long long)gridDim.x * blockDim.x) {
        const long long r = t / pieces;
        const int c = (int)(t - r * pieces);
        const int i = (int)(r % n);
        const int j = i - k;
        out[t] = (j >= 0 && j < n) ? in[(r - i + j) * pieces + c] : make_uint4(0, 0, 0, 0);
    }
}

__global__ void partner_table_kernel(int s, int n, unsigned flags, int* out) {
    const int i = blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n) out[i] = receives(i, s, flags) ? partner_of(i, s) : -1;
}

inline int blocks_for(size_t count, int threads, int cap = 152 * 16) {
    size_t b = (count + threads - 1) / threads;
    return (int)(b < (size_t)cap ? (b == 0 ? 1 : b) : cap);
}

}  // namespace

cudaError_t launch_f32_fwd(const float* x, const float* Ws, const float* Wn, const float* bias,
                           int s, int B, int n, int d, unsigned flags, float* y, float* z,
                           uint32_t* mout, cudaStream_t st) {
    const long long rows = (long long)B * n;
    dim3 grid((d + T - 1) / T, (unsigned)((rows + T - 1) / T));
    f32_fwd_kernel<<<grid, dim3(T, 8), 0, st>>>(x, Ws, Wn, bias, s, n, d, rows, flags, y, z,
                                                 mout);
    return cudaGetLastError();
}

cudaError_t launch_relu_grad_mask_f32(const float* dy, const uint32_t* mask, float* dz,
                                      long long rows, int d, cudaStream_t st) {
    relu_grad_mask_f32_kernel<<<blocks_for((size_t)rows * d, 256), 256, 0, st>>>(dy, mask, dz,
                                                                              rows, d);
    return cudaGetLastError();
}

cudaError_t launch_relu_grad_mask_bf16(const __nv_bfloat16* dy, const uint32_t* mask,
                                       __nv_bfloat16* dz, long long rows, int d,
                                       cudaStream_t st) {
    relu_grad_mask_kernel<__nv_bfloat16>
        <<<blocks_for((size_t)rows * d / 8, 256), 256, 0, st>>>(dy, mask, dz, rows, d);
    return cudaGetLastError();
}

cudaError_t launch_f32_dx(const float* dz, const float* dy, const float* Ws, const float* Wn,
                          int s, int B, int n, int d, unsigned flags, float* dx,
                          cudaStream_t st) {
    const long long rows = (long long)B * n;
    dim3 grid((d + T - 1) / T, (unsigned)((rows + T - 1) / T));
    f32_dx_kernel<<<grid, dim3(T, 8), 0, st>>>(dz, dy, Ws, Wn, s, n, d, rows, flags, dx);
    return cudaGetLastError();
}

cudaError_t launch_f32_dw(const float* x, const float* dz, int s, int B, int n, int d,
                          unsigned flags, float* dWs, float* dWn, cudaStream_t st) {
    const long long rows = (long long)B * n;
    dim3 grid((d + T - 1) / T, (d + T - 1) / T);
    f32_dw_kernel<<<grid, dim3(T, 8), 0, st>>>(x, dz, s, n, d, rows, flags, dWs, dWn);
    return cudaGetLastError();
}

cudaError_t launch_relu_grad_f32(const float* dy, const float* z, float* dz, size_t count,
                                 cudaStream_t st) {
    relu_grad_kernel<float><<<blocks_for(count, 256), 256, 0, st>>>(dy, z, dz, count);
    return cudaGetLastError();
}

cudaError_t launch_relu_grad_bf16(const __nv_bfloat16* dy, const __nv_bfloat16* z,
                                  __nv_bfloat16* dz, size_t count, cudaStream_t st) {
    relu_grad_kernel<__nv_bfloat16><<<blocks_for(count, 256), 256, 0, st>>>(dy, z, dz, count);
    return cudaGetLastError();
}

size_t colsum_workspace_bytes(long long rows, int d) {
    const long long chunks = (rows + col_rows(rows) - 1) / col_rows(rows);
    return (size_t)(chunks < 1 ? 1 : chunks) * (size_t)d * sizeof(float);
}

template <typename V>
static cudaError_t colsum(const V* dz, long long rows, int d, float* partial, float* out,
                          cudaStream_t st, int batch = 1) {
    const int crows = (int)col_rows(rows);
    const long long chunks = (rows + crows - 1) / crows;
    if (chunks == 0) {
        cudaError_t e = cudaMemsetAsync(out, 0, (size_t)batch * d * sizeof(float), st);
        return e;
    }
    if (sizeof(V) == 4) {
        colsum_partial_f32_kernel<<<dim3((d + 31) / 32, (unsigned)chunks, 1), dim3(32, 8), 0, st>>>(
            reinterpret_cast<const float*>(dz), rows, d, crows, partial);
    } else {
        constexpr int VEC = 16 / sizeof(V);
        dim3 grid((d / VEC + 63) / 64, (unsigned)chunks, (unsigned)batch);
        colsum_partial_kernel<V><<<grid, dim3(64, 4), 0, st>>>(dz, rows, d, crows, partial);
    }
    colsum_final_kernel<<<dim3((d + 31) / 32, batch), 1024, 0, st>>>(partial, (int)chunks, d, out);
    return cudaGetLastError();
}

cudaError_t launch_colsum_bf16_batched(const __nv_bfloat16* dz, int batch, long long rows, int d,
                                       float* partial, float* out, cudaStream_t st) {
    return colsum<__nv_bfloat16>(dz, rows, d, partial, out, st, batch);
}

cudaError_t launch_colsum_f32(const float* dz, long long rows, int d, float* partial,
                              float* out, cudaStream_t st) {
    return colsum<float>(dz, rows, d, partial, out, st);
}

cudaError_t launch_colsum_bf16(const __nv_bfloat16* dz, long long rows, int d, float* partial,
                               float* out, cudaStream_t st) {
    return colsum<__nv_bfloat16>(dz, rows, d, partial, out, st);
}

cudaError_t launch_splitk_reduce(const float* partial, int splits_max, int splits_self,
                                 int splits_nbr, int d, float* dWs, float* dWn,
                                 cudaStream_t st, int layers, size_t part_stride,
                                 size_t out_stride, const float* bpart, float* dbias) {
    const size_t total4 = (size_t)d * d / 4;
    if (layers < 1) return cudaSuccess;
    const unsigned parts = (bpart && dbias) ? 3 : 2;
    splitk_reduce_kernel<<<dim3((unsigned)((total4 + 63) / 64), parts, (unsigned)layers),
                           dim3(64, 8), 0, st>>>(partial, splits_max, splits_self, splits_nbr, d,
                                                 part_stride, dWs, dWn, out_stride, bpart, dbias);
    return cudaGetLastError();
}

cudaError_t launch_shift_rows_bf16(const __nv_bfloat16* in, __nv_bfloat16* out, long long rows,
                                   int n, int d, int k, cudaStream_t st) {
    const int pieces = d / 8;   // d % 64 == 0 on the bf16 path
    shift_rows_kernel<<<blocks_for((size_t)rows * pieces, 256), 256, 0, st>>>(
        reinterpret_cast<const uint4*>(in), reinterpret_cast<uint4*>(out), rows, n, pieces, k);
    return cudaGetLastError();
}

cudaError_t launch_partner_table(int s, int n, unsigned flags, int* out, cudaStream_t st) {
    partner_table_kernel<<<(n + 255) / 256, 256, 0, st>>>(s, n, flags, out);
    return cudaGetLastError();
}

}  // namespace hcw
