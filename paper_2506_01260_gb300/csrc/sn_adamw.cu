// sn_adamw.cu — the row-constant AdamW step that keeps W_p2 inside the
// subspace (Sec. 5), memory-bound, on the CUDA cores.
//
// W is the torch weight [rows = d, cols = n]; its columns are the paper's rows
// of W_p2 (the d-vectors that live in S).  One step t >= 1:
//   M = b1 M + (1 - b1) g,  V = b2 V + (1 - b2) g^2          (in place, fp32)
//   mu[c] = mean over the column of V / (1 - b2^t)             (the paper's row mean)
//   W = W - lr (M / (1 - b1^t)) / (sqrt(mu[c]) + eps) - lambda W
// Pass 1 updates V and adds each block's column sums of V^ to a zeroed [cols]
// fp32 workspace with one atomic per column and block; pass 2 updates M (it
// reads g again, 2 bytes, instead of reading back an updated M, 4 bytes) and
// W: 28 bytes moved per element with a bf16 gradient.  Each thread owns four
// adjacent columns (16-byte accesses, rows unrolled by four) of a block of rows
// when the column count is a multiple of 4, else one column; every access is
// coalesced along the columns.
#include "sn_internal.cuh"

namespace sn {
namespace {

constexpr int kCols = 256;   // columns per block (one per thread)
constexpr int kRows = 64;    // rows per block

template <typename GT>
__device__ __forceinline__ float load_grad(const GT *g, int64_t e);
template <>
__device__ __forceinline__ float load_grad<float>(const float *g, int64_t e)
{
    return __ldg(g + e);
}
template <>
__device__ __forceinline__ float load_grad<__nv_bfloat16>(const __nv_bfloat16 *g, int64_t e)
{
    return __bfloat162float(g[e]);
}

template <typename GT>
__global__ void __launch_bounds__(kCols) k_adamw_moments(const GT *__restrict__ g,
                                                          float *__restrict__ M,
                                                          float *__restrict__ V, int64_t rows,
                                                          int64_t cols, float b1, float b2,
                                                          float vcorr, float *__restrict__ colsum)
{
    const int64_t c = (int64_t)blockIdx.x * kCols + threadIdx.x;
    const int64_t r0 = (int64_t)blockIdx.y * kRows;
    if (c >= cols)
        return;
    const int64_t r1 = r0 + kRows < rows ? r0 + kRows : rows;
    float s = 0.f;
    for (int64_t r = r0; r < r1; ++r) {
        const int64_t e = r * cols + c;
        const float gv = load_grad(g, e);
        const float m = b1 * M[e] + (1.f - b1) * gv;
        const float v = b2 * V[e] + (1.f - b2) * gv * gv;
        M[e] = m;
        V[e] = v;
        s += v * vcorr;
    }
    atomicAdd(colsum + c, s);
}

__global__ void __launch_bounds__(kCols) k_adamw_apply(float *__restrict__ W,
                                                        const float *__restrict__ M, int64_t rows,
                                                        int64_t cols, float lr, float mcorr,
                                                        float eps, float lam, float inv_rows,
                                                        const float *__restrict__ colsum)
{
    const int64_t c = (int64_t)blockIdx.x * kCols + threadIdx.x;
    const int64_t r0 = (int64_t)blockIdx.y * kRows;
    if (c >= cols)
        return;
    const float alpha = 1.f / (sqrtf(colsum[c] * inv_rows) + eps);
    const float step = lr * mcorr * alpha;
    const int64_t r1 = r0 + kRows < rows ? r0 + kRows : rows;
    for (int64_t r = r0; r < r1; ++r) {
        const int64_t e = r * cols + c;
        const float w = W[e];
        W[e] = w - step * M[e] - lam * w;
    }
}

// ---- four columns per thread ------------------------------------------------

template <typename GT>
__device__ __forceinline__ float4 load_grad4(const GT *g, int64_t e);
template <>
__device__ __forceinline__ float4 load_grad4<float>(const float *g, int64_t e)
{
    return __ldg((const float4 *)(g + e));
}
template <>
__device__ __forceinline__ float4 load_grad4<__nv_bfloat16>(const __nv_bfloat16 *g, int64_t e)
{
    const uint2 u = __ldg((const uint2 *)(g + e));
    return make_float4(__uint_as_float(u.x << 16), __uint_as_float(u.x & 0xFFFF0000u),
                       __uint_as_float(u.y << 16), __uint_as_float(u.y & 0xFFFF0000u));
}

constexpr int kRowsV = 64;   // rows per block (vector kernels)
constexpr int kUnroll = 4;

template <typename GT>
__global__ void __launch_bounds__(kCols) k_adamw_v4(const GT *__restrict__ g, float *__restrict__ V,
                                                     int64_t rows, int64_t cols, float b2, float vcorr,
                                                     float *__restrict__ colsum)
{
    const int64_t c = 4 * ((int64_t)blockIdx.x * kCols + threadIdx.x);
    const int64_t r0 = (int64_t)blockIdx.y * kRowsV;
    if (c >= cols)
        return;
    const int64_t r1 = r0 + kRowsV < rows ? r0 + kRowsV : rows;
    float4 s = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int64_t rb = r0; rb < r1; rb += kUnroll) {
        float4 gv[kUnroll], vv[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u)
            if (rb + u < r1) {
                gv[u] = load_grad4(g, (rb + u) * cols + c);
                vv[u] = *(const float4 *)(V + (rb + u) * cols + c);
            }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u)
            if (rb + u < r1) {
                float4 v;
                v.x = b2 * vv[u].x + (1.f - b2) * gv[u].x * gv[u].x;
                v.y = b2 * vv[u].y + (1.f - b2) * gv[u].y * gv[u].y;
                v.z = b2 * vv[u].z + (1.f - b2) * gv[u].z * gv[u].z;
                v.w = b2 * vv[u].w + (1.f - b2) * gv[u].w * gv[u].w;
                *(float4 *)(V + (rb + u) * cols + c) = v;
                s.x += v.x * vcorr;
                s.y += v.y * vcorr;
                s.z += v.z * vcorr;
                s.w += v.w * vcorr;
            }
    }
    atomicAdd(colsum + c, s.x);
    atomicAdd(colsum + c + 1, s.y);
    atomicAdd(colsum + c + 2, s.z);
    atomicAdd(colsum + c + 3, s.w);
}

template <typename GT>
__global__ void __launch_bounds__(kCols) k_adamw_mw4(const GT *__restrict__ g, float *__restrict__ W,
                                                      float *__restrict__ M, int64_t rows,
                                                      int64_t cols, float b1, float lr, float mcorr,
                                                      float eps, float lam, float inv_rows,
                                                      const float *__restrict__ colsum)
{
    const int64_t c = 4 * ((int64_t)blockIdx.x * kCols + threadIdx.x);
    const int64_t r0 = (int64_t)blockIdx.y * kRowsV;
    if (c >= cols)
        return;
    const float4 cs = *(const float4 *)(colsum + c);
    const float4 st = make_float4(lr * mcorr / (sqrtf(cs.x * inv_rows) + eps),
                                  lr * mcorr / (sqrtf(cs.y * inv_rows) + eps),
                                  lr * mcorr / (sqrtf(cs.z * inv_rows) + eps),
                                  lr * mcorr / (sqrtf(cs.w * inv_rows) + eps));
    const int64_t r1 = r0 + kRowsV < rows ? r0 + kRowsV : rows;
    for (int64_t rb = r0; rb < r1; rb += kUnroll) {
        float4 gv[kUnroll], mv[kUnroll], wv[kUnroll];
#pragma unroll
        for (int u = 0; u < kUnroll; ++u)
            if (rb + u < r1) {
                const int64_t e = (rb + u) * cols + c;
                gv[u] = load_grad4(g, e);
                mv[u] = *(const float4 *)(M + e);
                wv[u] = *(const float4 *)(W + e);
            }
#pragma unroll
        for (int u = 0; u < kUnroll; ++u)
            if (rb + u < r1) {
                const int64_t e = (rb + u) * cols + c;
                float4 m, w;
                m.x = b1 * mv[u].x + (1.f - b1) * gv[u].x;
                m.y = b1 * mv[u].y + (1.f - b1) * gv[u].y;
                m.z = b1 * mv[u].z + (1.f - b1) * gv[u].z;
                m.w = b1 * mv[u].w + (1.f - b1) * gv[u].w;
                w.x = wv[u].x - st.x * m.x - lam * wv[u].x;
                w.y = wv[u].y - st.y * m.y - lam * wv[u].y;
                w.z = wv[u].z - st.z * m.z - lam * wv[u].z;
                w.w = wv[u].w - st.w * m.w - lam * wv[u].w;
                *(float4 *)(M + e) = m;
                *(float4 *)(W + e) = w;
            }
    }
}

}  // namespace

cudaError_t adamw_rowconst(bool grad_bf16, float *W, const void *g, float *M, float *V,
                           int64_t rows, int64_t cols, int64_t t, float lr, float b1, float b2,
                           float eps, float lam, float *colsum, cudaStream_t s)
{
    cudaError_t e = cudaMemsetAsync(colsum, 0, sizeof(float) * (size_t)cols, s);
    if (e != cudaSuccess)
        return e;
    // bias corrections of step t, in double before rounding to fp32
    const float vcorr = (float)(1.0 / (1.0 - pow((double)b2, (double)t)));
    const float mcorr = (float)(1.0 / (1.0 - pow((double)b1, (double)t)));
    if (cols % 4 == 0) {
        const dim3 grid((unsigned)((cols / 4 + kCols - 1) / kCols),
                        (unsigned)((rows + kRowsV - 1) / kRowsV));
        const float inv_rows = (float)(1.0 / (double)rows);
        if (grad_bf16) {
            k_adamw_v4<__nv_bfloat16><<<grid, kCols, 0, s>>>((const __nv_bfloat16 *)g, V, rows,
                                                             cols, b2, vcorr, colsum);
            k_adamw_mw4<__nv_bfloat16><<<grid, kCols, 0, s>>>((const __nv_bfloat16 *)g, W, M, rows,
                                                              cols, b1, lr, mcorr, eps, lam,
                                                              inv_rows, colsum);
        } else {
            k_adamw_v4<float><<<grid, kCols, 0, s>>>((const float *)g, V, rows, cols, b2, vcorr,
                                                     colsum);
            k_adamw_mw4<float><<<grid, kCols, 0, s>>>((const float *)g, W, M, rows, cols, b1, lr,
                                                      mcorr, eps, lam, inv_rows, colsum);
        }
        count_launch(2);
        return cudaGetLastError();
    }
    const dim3 grid((unsigned)((cols + kCols - 1) / kCols), (unsigned)((rows + kRows - 1) / kRows));
    if (grad_bf16)
        k_adamw_moments<__nv_bfloat16><<<grid, kCols, 0, s>>>(
            (const __nv_bfloat16 *)g, M, V, rows, cols, b1, b2, vcorr, colsum);
    else
        k_adamw_moments<float><<<grid, kCols, 0, s>>>((const float *)g, M, V, rows, cols, b1, b2,
                                                     vcorr, colsum);
    k_adamw_apply<<<grid, kCols, 0, s>>>(W, M, rows, cols, lr, mcorr, eps, lam,
                                         (float)(1.0 / (double)rows), colsum);
    count_launch(2);
    return cudaGetLastError();
}

}  // namespace sn
